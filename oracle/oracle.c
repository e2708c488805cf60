/*
 * oracle.c -- CPU oracle for the rank-compensation hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is built into oracle/liboracle.so and
 * may be loaded only by tests/, __graft_entry__.smoke() and the CPU-baseline
 * legs of bench.py.  The GPU library never links, loads or calls it, and the
 * two share no code, header, table or helper.
 *
 * Everything here is plain, unblocked IEEE binary64 arithmetic written from
 * the definitions in the paper (Low-Precision Rank Compensation for Matrices
 * and Tensor Trains):
 *
 *   - storage rounding (Sec. 3.2-3.3 and the remark after Thm 4.1: U, Sigma
 *     and V^T are rounded individually): IEEE 754 binary64 -> binary32 /
 *     binary16 conversion, round to nearest with ties to even, gradual
 *     underflow, overflow to infinity, written with integer operations from
 *     the format definition (never via an intermediate format);
 *   - matrix apply (Sec. 4.4, Eq. gpu_matrix_apply): Y = [(X V) diag(s)] U^T;
 *   - TT reconstruction (Sec. 7.5, Eq. gpu_tt_reconstruction): the
 *     reshape / matrix-product chain Z_1 = G_1, B_l = Z_{l-1} K_l,
 *     Z_l = reshape(B_l); and, independently, the entry definition of
 *     Sec. 5.1, T(i_1..i_d) = G_1(i_1) G_2(i_2) ... G_d(i_d);
 *   - Frobenius norm / difference (Sec. 5.1, "Frobenius norm") with a
 *     Neumaier-compensated sum;
 *   - the certificates (Thm 4.1 Eq. matrix_condition, Thm 6.1
 *     Eq. tt_condition), the tail error E_k (Sec. 4) and the storage counts
 *     (Eq. matrix_storage_ratio, Sec. 5.1 TT core count).
 *
 * Parallelism is OpenMP over independent output rows only; no sum is split.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------- */
/* IEEE 754 rounding from binary64 (Sec. 3.2: u = 2^-p, round to nearest)     */
/* ------------------------------------------------------------------------- */

/*
 * Round the binary64 value x to a binary format with p significand bits
 * (implicit bit included), minimum normal exponent emin, maximum exponent
 * emax and an exponent field of ebits bits; return the encoding.
 *
 * The finite nonzero input is |x| = M * 2^E with M an integer below 2^53.
 * The target keeps the bits of weight >= 2^q, where q is the exponent of the
 * last significand bit (lead - (p-1)), never below the subnormal quantum
 * emin - (p-1).  The dropped bits decide the rounding: above half -> up,
 * exactly half -> up only if the kept integer is odd (ties to even).
 */
static uint64_t round_binary(double x, int p, int emin, int emax, int ebits, int total_bits)
{
    uint64_t bits;
    memcpy(&bits, &x, sizeof bits);
    const uint64_t sign_out = (bits >> 63) << (total_bits - 1);
    const int e = (int)((bits >> 52) & 0x7ffu);
    const uint64_t frac = bits & ((1ull << 52) - 1);
    const uint64_t exp_ones = ((1ull << ebits) - 1) << (p - 1);

    if (e == 0x7ff) {
        if (frac != 0) return sign_out | exp_ones | (1ull << (p - 2)); /* quiet NaN */
        return sign_out | exp_ones;                                    /* infinity  */
    }
    if (e == 0 && frac == 0) return sign_out;                          /* +-0 */

    const uint64_t M = (e == 0) ? frac : (frac | (1ull << 52));
    const int E = (e == 0) ? -1074 : e - 1075;
    int len = 0;
    for (uint64_t t = M; t != 0; t >>= 1) ++len;                       /* bit length of M */
    const int lead = E + len - 1;                                      /* exponent of leading bit */
    int q = lead - (p - 1);
    if (q < emin - (p - 1)) q = emin - (p - 1);                        /* gradual underflow */
    const int shift = q - E;                                           /* > 0 for p < 53 */

    uint64_t R;
    if (shift >= 64) {
        R = 0;                                   /* below half the quantum */
    } else {
        R = M >> shift;
        const uint64_t rem = M & ((1ull << shift) - 1);
        const uint64_t half = 1ull << (shift - 1);
        if (rem > half || (rem == half && (R & 1u))) R += 1;
    }
    if (R == (1ull << p)) { R >>= 1; q += 1; }  /* carry into a new binade */
    if (R < (1ull << (p - 1))) return sign_out | R;                    /* subnormal or zero */
    const int lead_out = q + (p - 1);
    if (lead_out > emax) return sign_out | exp_ones;                   /* overflow */
    const uint64_t biased = (uint64_t)(lead_out - emin + 1);
    return sign_out | (biased << (p - 1)) | (R - (1ull << (p - 1)));
}

uint32_t oracle_f64_to_f32_bits(double x) { return (uint32_t)round_binary(x, 24, -126, 127, 8, 32); }
uint16_t oracle_f64_to_f16_bits(double x) { return (uint16_t)round_binary(x, 11, -14, 15, 5, 16); }
/* bfloat16 (Sec. 3.2 precision table): 8 significand bits, binary32's exponent range */
uint16_t oracle_f64_to_bf16_bits(double x) { return (uint16_t)round_binary(x, 8, -126, 127, 8, 16); }

/* Value of a binary16 / binary32 encoding, from the format definition. */
double oracle_f16_bits_to_f64(uint16_t h)
{
    const int s = h >> 15, e = (h >> 10) & 0x1f, f = h & 0x3ff;
    double v;
    if (e == 0) v = ldexp((double)f, -24);
    else if (e == 31) v = f ? NAN : INFINITY;
    else v = ldexp((double)(f | 0x400), e - 25);
    return s ? -v : v;
}

double oracle_f32_bits_to_f64(uint32_t w)
{
    const int s = (int)(w >> 31), e = (int)((w >> 23) & 0xff);
    const uint32_t f = w & 0x7fffffu;
    double v;
    if (e == 0) v = ldexp((double)f, -149);
    else if (e == 255) v = f ? NAN : INFINITY;
    else v = ldexp((double)(f | 0x800000u), e - 150);
    return s ? -v : v;
}

/* Value of a bfloat16 encoding: sign, 8-bit biased exponent, 7 fraction bits. */
double oracle_bf16_bits_to_f64(uint16_t h)
{
    const int s = h >> 15, e = (h >> 7) & 0xff, f = h & 0x7f;
    double v;
    if (e == 0) v = ldexp((double)f, -133);
    else if (e == 255) v = f ? NAN : INFINITY;
    else v = ldexp((double)(f | 0x80), e - 134);
    return s ? -v : v;
}

/* fmt: 0 = binary64 (copy), 1 = binary32, 2 = binary16, 3 = bfloat16.  Packed layout:
 * dst row r holds the rounded src[r, 0..cols) followed by +0 up to ld_dst. */
void oracle_round_pack(const double* src, int64_t rows, int64_t cols, int64_t ld_src,
                       void* dst, int64_t ld_dst, int fmt)
{
    for (int64_t r = 0; r < rows; ++r) {
        for (int64_t c = 0; c < ld_dst; ++c) {
            const double v = (c < cols) ? src[r * ld_src + c] : 0.0;
            if (fmt == 0) ((double*)dst)[r * ld_dst + c] = v;
            else if (fmt == 1) ((uint32_t*)dst)[r * ld_dst + c] = oracle_f64_to_f32_bits(v);
            else if (fmt == 3) ((uint16_t*)dst)[r * ld_dst + c] = oracle_f64_to_bf16_bits(v);
            else ((uint16_t*)dst)[r * ld_dst + c] = oracle_f64_to_f16_bits(v);
        }
    }
}

void oracle_decode(const void* src, int64_t count, int fmt, double* dst)
{
    for (int64_t i = 0; i < count; ++i) {
        if (fmt == 0) dst[i] = ((const double*)src)[i];
        else if (fmt == 1) dst[i] = oracle_f32_bits_to_f64(((const uint32_t*)src)[i]);
        else if (fmt == 3) dst[i] = oracle_bf16_bits_to_f64(((const uint16_t*)src)[i]);
        else dst[i] = oracle_f16_bits_to_f64(((const uint16_t*)src)[i]);
    }
}

/* ------------------------------------------------------------------------- */
/* Matrix apply, Sec. 4.4 Eq. gpu_matrix_apply:  Y = [(X V) diag(s)] U^T     */
/* ------------------------------------------------------------------------- */

/* One query row c: w = X[c,:] V (V = Vt^T), w <- w diag(s), Y[c,:] = w U^T. */
static void apply_row(const double* U, int64_t ldu, const double* s, const double* Vt, int64_t ldv,
                      const double* xrow, double* yrow, int64_t m, int64_t n, int64_t k, double* w)
{
    for (int64_t j = 0; j < k; ++j) {
        double acc = 0.0;
        for (int64_t i = 0; i < n; ++i) acc += xrow[i] * Vt[j * ldv + i];
        w[j] = acc;
    }
    for (int64_t j = 0; j < k; ++j) w[j] *= s[j];
    for (int64_t r = 0; r < m; ++r) {
        double acc = 0.0;
        for (int64_t j = 0; j < k; ++j) acc += w[j] * U[r * ldu + j];
        yrow[r] = acc;
    }
}

/* U: m x k (ld ldu), s: k, Vt: k x n (ld ldv), X: b x n (ld ldx), Y: b x m (ld ldy). */
void oracle_apply(const double* U, int64_t ldu, const double* s, const double* Vt, int64_t ldv,
                  const double* X, int64_t ldx, double* Y, int64_t ldy,
                  int64_t m, int64_t n, int64_t k, int64_t b)
{
    #pragma omp parallel
    {
        double* w = (double*)malloc((size_t)(k > 0 ? k : 1) * sizeof(double));
        #pragma omp for schedule(dynamic, 1)
        for (int64_t c = 0; c < b; ++c)
            apply_row(U, ldu, s, Vt, ldv, X + c * ldx, Y + c * ldy, m, n, k, w);
        free(w);
    }
}

/* Only the listed query rows; output row t is Y[rows[t], :]. */
void oracle_apply_rows(const double* U, int64_t ldu, const double* s, const double* Vt, int64_t ldv,
                       const double* X, int64_t ldx, const int64_t* rows, int64_t count,
                       double* Yrows, int64_t m, int64_t n, int64_t k)
{
    #pragma omp parallel
    {
        double* w = (double*)malloc((size_t)(k > 0 ? k : 1) * sizeof(double));
        #pragma omp for schedule(dynamic, 1)
        for (int64_t t = 0; t < count; ++t)
            apply_row(U, ldu, s, Vt, ldv, X + rows[t] * ldx, Yrows + t * m, m, n, k, w);
        free(w);
    }
}

/* ------------------------------------------------------------------------- */
/* TT reconstruction                                                          */
/* ------------------------------------------------------------------------- */

/*
 * Sec. 7.5, Eq. gpu_tt_reconstruction.  cores[l] is G_{l+1}, C order
 * ranks[l] x dims[l] x ranks[l+1]; ranks[0] = ranks[d] = 1.
 *   Z_1 = reshape(G_1, n_1 x r_1)
 *   B_l = Z_{l-1} K_l,  K_l = reshape(G_l, r_{l-1} x (n_l r_l))
 *   Z_l = reshape(B_l, (n_1...n_l) x r_l)            (a no-op in row-major storage)
 * The final Z_d (r_d = 1) is the tensor, C order with i_1 slowest.
 */
int oracle_tt_chain(const double* const* cores, const int64_t* dims, const int64_t* ranks, int d,
                    double* out)
{
    if (d < 2) return -1;
    int64_t P = dims[0];
    double* Z = (double*)malloc((size_t)(P * ranks[1]) * sizeof(double));
    if (!Z) return -2;
    memcpy(Z, cores[0], (size_t)(P * ranks[1]) * sizeof(double));
    for (int l = 1; l < d; ++l) {
        const int64_t r0 = ranks[l], nl = dims[l], r1 = ranks[l + 1];
        const int64_t cols = nl * r1;
        const double* K = cores[l];
        double* B = (l == d - 1) ? out : (double*)malloc((size_t)(P * cols) * sizeof(double));
        if (!B) { free(Z); return -2; }
        #pragma omp parallel for schedule(static)
        for (int64_t p = 0; p < P; ++p) {
            for (int64_t c = 0; c < cols; ++c) {
                double acc = 0.0;
                for (int64_t a = 0; a < r0; ++a) acc += Z[p * r0 + a] * K[a * cols + c];
                B[p * cols + c] = acc;
            }
        }
        free(Z);
        Z = B;
        P *= nl;
    }
    return 0;
}

/*
 * Sec. 5.1 entry definition, evaluated independently of the chain above:
 * T(i_1,...,i_d) = G_1(i_1) G_2(i_2) ... G_d(i_d), as a row vector times
 * matrices, left to right.  flat[t] is a C-order flat index (i_d fastest).
 */
int oracle_tt_entries(const double* const* cores, const int64_t* dims, const int64_t* ranks, int d,
                      const int64_t* flat, int64_t count, double* out)
{
    int64_t rmax = 1;
    for (int l = 0; l <= d; ++l) if (ranks[l] > rmax) rmax = ranks[l];
    int err = 0;
    #pragma omp parallel
    {
        double* v = (double*)malloc((size_t)rmax * sizeof(double));
        double* w = (double*)malloc((size_t)rmax * sizeof(double));
        int64_t* idx = (int64_t*)malloc((size_t)d * sizeof(int64_t));
        if (!v || !w || !idx) {
            #pragma omp atomic write
            err = -2;
        } else {
            #pragma omp for schedule(static)
            for (int64_t t = 0; t < count; ++t) {
                int64_t f = flat[t];
                for (int l = d - 1; l >= 0; --l) { idx[l] = f % dims[l]; f /= dims[l]; }
                v[0] = 1.0;
                for (int l = 0; l < d; ++l) {
                    const int64_t r0 = ranks[l], nl = dims[l], r1 = ranks[l + 1];
                    const double* G = cores[l];
                    for (int64_t b = 0; b < r1; ++b) {
                        double acc = 0.0;
                        for (int64_t a = 0; a < r0; ++a) acc += v[a] * G[(a * nl + idx[l]) * r1 + b];
                        w[b] = acc;
                    }
                    for (int64_t b = 0; b < r1; ++b) v[b] = w[b];
                }
                out[t] = v[0];
            }
        }
        free(v); free(w); free(idx);
    }
    return err;
}

/* ------------------------------------------------------------------------- */
/* Frobenius norm / difference (Sec. 5.1), Neumaier-compensated               */
/* ------------------------------------------------------------------------- */

static void neumaier_add(double* s, double* c, double t)
{
    const double u = *s + t;
    if (fabs(*s) >= fabs(t)) *c += (*s - u) + t;
    else *c += (t - u) + *s;
    *s = u;
}

/* diff = ||a - b||_F (b may be NULL: b = 0), norm_a = ||a||_F (nullable). */
void oracle_fro_diff(const double* a, const double* b, int64_t count, double* diff, double* norm_a)
{
    double s = 0.0, c = 0.0, s2 = 0.0, c2 = 0.0;
    for (int64_t i = 0; i < count; ++i) {
        const double dd = a[i] - (b ? b[i] : 0.0);
        neumaier_add(&s, &c, dd * dd);
        neumaier_add(&s2, &c2, a[i] * a[i]);
    }
    *diff = sqrt(s + c);
    if (norm_a) *norm_a = sqrt(s2 + c2);
}

/* ------------------------------------------------------------------------- */
/* Certificate and accounting                                                 */
/* ------------------------------------------------------------------------- */

/* Sec. 4: E_k = ||A - A_k||_F = (sum_{j>k} sigma_j^2)^(1/2); sigma[0] = sigma_1.
 * Summed from the smallest term upwards. */
double oracle_tail_error(const double* sigma, int64_t len, int64_t k)
{
    double s = 0.0, c = 0.0;
    for (int64_t j = len - 1; j >= k; --j) neumaier_add(&s, &c, sigma[j] * sigma[j]);
    return sqrt(s + c);
}

/* Thm 4.1 Eq. matrix_condition (E_{k+1} + eta <= E_k) and Thm 6.1
 * Eq. tt_condition (E_{R+} + eta_TT <= E_R): the same test on scalars. */
int oracle_certified(double e_base, double e_aug, double eta) { return (e_aug + eta <= e_base) ? 1 : 0; }

/* Thm 4.1 Eq. matrix_universal_bound: ||A - Ahat_{k+1}||_F <= (E_k^2 - sigma_{k+1}^2)^(1/2) + eta. */
double oracle_matrix_bound(double e_k, double sigma_next, double eta)
{
    return sqrt(e_k * e_k - sigma_next * sigma_next) + eta;
}

/* Sec. 4.2: rank-k factors stored with `bits` per scalar cost bits * k (m + n + 1). */
double oracle_matrix_storage_bits(int64_t m, int64_t n, int64_t k, int bits)
{
    return (double)bits * (double)k * (double)(m + n + 1);
}

/* Sec. 5.1: TT storage sum_l R_{l-1} n_l R_l scalars, times bits. */
double oracle_tt_storage_bits(const int64_t* dims, const int64_t* ranks, int d, int bits)
{
    double s = 0.0;
    for (int l = 0; l < d; ++l) s += (double)ranks[l] * (double)dims[l] * (double)ranks[l + 1];
    return s * (double)bits;
}

/* Thread count of the OpenMP loops (timing of the oracle on 1 and on all
 * host cores); no effect on any result, every loop writes disjoint outputs. */
void oracle_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

int oracle_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
