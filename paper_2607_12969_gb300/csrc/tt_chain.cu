// tt_chain.cu -- TT reconstruction as a chain of matrix products (Sec. 5.1:
// T(i_1..i_d) = G_1(i_1)...G_d(i_d); Sec. 7.5, Eq. gpu_tt_reconstruction:
// B_l = Z_{l-1} K_l) contracted from both ends toward one bond c:
//   left   Z(1) = G_1,      Z(j+1) = Z(j) K_j            (P_j x r_j rows)
//   right  S(d) = G_d,      S(j)   = K'_j S(j+1)         (r_{j-1} x Q_j)
//   output T = Z(c) S(c+1), a (n_1...n_c) x (n_{c+1}...n_d) matrix, which is
//          the C-order tensor.
// K_j is core j viewed as r_{j-1} x (n_j r_j) and K'_j the same core viewed
// as (r_{j-1} n_j) x r_j -- both are the stored C-order array, so every
// reshape is free.  The bond c minimises the multiply count; the last
// product writes the output and carries nearly all the work.  For the 16^6
// tensor with ranks (1,16,26,26,26,16,1) the chain meets at the middle bond:
// 0.88 GFLOP, against 1.50 GFLOP for the left-to-right chain.
//
// Every product runs on the product kernels of gemm_cc.cu (register-tiled
// binary32, DFMA-bound binary64); intermediates live in the stream's
// workspace (two buffers per side, alternating).
#include <math.h>

#include "common.cuh"

namespace lrc {

namespace {

struct ChainPlan {
    int c;                  // bond: left cores 0..c-1, right cores c..d-1 (0-based)
    double flops;
};

// Multiply-adds x 2 of the chain that meets at bond c.
double chain_flops(const TTShape& sh, int c) {
    const int d = sh.d;
    double f = 0.0, P = (double)sh.dims[0];
    for (int j = 1; j <= c - 1; ++j) {
        f += 2.0 * P * (double)sh.ranks[j] * (double)sh.dims[j] * (double)sh.ranks[j + 1];
        P *= (double)sh.dims[j];
    }
    double Q = (double)sh.dims[d - 1];
    for (int j = d - 2; j >= c; --j) {
        f += 2.0 * (double)sh.ranks[j] * (double)sh.dims[j] * (double)sh.ranks[j + 1] * Q;
        Q *= (double)sh.dims[j];
    }
    return f + 2.0 * P * Q * (double)sh.ranks[c];
}

ChainPlan plan_chain(const TTShape& sh) {
    ChainPlan best{sh.d - 1, INFINITY};
    for (int c = 1; c <= sh.d - 1; ++c) {
        const double f = chain_flops(sh, c);
        if (f <= best.flops) best = ChainPlan{c, f};   // ties: the larger c (fewer right products)
    }
    return best;
}

size_t round256(size_t bytes) { return (bytes + 255) / 256 * 256; }

}  // namespace

double tt_chain_flops(const TTShape& sh) { return plan_chain(sh).flops; }

int tt_chain_bond(const TTShape& sh) { return plan_chain(sh).c; }

namespace {

lrc_status product(const float* A, int64_t lda, const float* B, int64_t ldb, float* C, int64_t ldc, int64_t M,
                   int64_t N, int64_t K, cudaStream_t s) {
    return gemm_cc_f32(A, lda, B, ldb, false, C, ldc, M, N, K, 1, 0, s);
}
lrc_status product(const double* A, int64_t lda, const double* B, int64_t ldb, double* C, int64_t ldc, int64_t M,
                   int64_t N, int64_t K, cudaStream_t s) {
    return gemm_cc_f64(A, lda, B, ldb, C, ldc, M, N, K, s);
}

// tc_final (binary32 only): the output product on the tensor cores through
// the scaled binary16 split (LRC_F32_TC) when the product kernel takes it.
template <typename T>
lrc_status launch_chain(const TTShape& sh, T* out, cudaStream_t s, bool tc_final = false) {
    const int d = sh.d;
    const int c = plan_chain(sh).c;
    const T* const* G = reinterpret_cast<const T* const*>(sh.cores);
    // P[j]: rows of Z(j); Q[j]: columns of S(j) (0-based core index j)
    int64_t P[17] = {0}, Q[17] = {0};
    P[1] = sh.dims[0];
    for (int j = 1; j <= c - 1; ++j) P[j + 1] = P[j] * sh.dims[j];
    Q[d - 1] = sh.dims[d - 1];
    for (int j = d - 2; j >= c; --j) Q[j] = sh.dims[j] * Q[j + 1];
    size_t lsz[2] = {0, 0}, rsz[2] = {0, 0};
    for (int j = 2; j <= c; ++j) {
        const size_t b = round256((size_t)P[j] * (size_t)sh.ranks[j] * sizeof(T));
        if (b > lsz[j & 1]) lsz[j & 1] = b;
    }
    for (int j = c; j <= d - 2; ++j) {
        const size_t b = round256((size_t)sh.ranks[j] * (size_t)Q[j] * sizeof(T));
        if (b > rsz[j & 1]) rsz[j & 1] = b;
    }
    unsigned char* ws = nullptr;
    const int64_t rc = sh.ranks[c];
    const bool tc = tc_final && sizeof(T) == 4 && split_product_fits(P[c], Q[c], rc);
    const size_t tsz = tc ? round256(split_product_bytes(P[c], Q[c], rc)) : 0;
    const size_t total = lsz[0] + lsz[1] + rsz[0] + rsz[1] + tsz;
    if (total > 0) {
        void* p = nullptr;
        lrc_status st = stream_workspace(s, total, &p);
        if (st != LRC_OK) return st;
        ws = static_cast<unsigned char*>(p);
    }
    T* L[2] = {reinterpret_cast<T*>(ws), reinterpret_cast<T*>(ws + lsz[0])};
    T* R[2] = {reinterpret_cast<T*>(ws + lsz[0] + lsz[1]), reinterpret_cast<T*>(ws + lsz[0] + lsz[1] + rsz[0])};
    lrc_status st = LRC_OK;
    const T* Z = G[0];   // Z(1) = G_1: n_1 x r_1
    for (int j = 1; j <= c - 1; ++j) {
        const int64_t w = sh.dims[j] * sh.ranks[j + 1];
        T* dst = L[(j + 1) & 1];
        if ((st = product(Z, sh.ranks[j], G[j], w, dst, w, P[j], w, sh.ranks[j], s)) != LRC_OK) return st;
        Z = dst;
    }
    const T* S = G[d - 1];   // S(d) = G_d: r_{d-1} x n_d
    for (int j = d - 2; j >= c; --j) {
        T* dst = R[j & 1];
        if ((st = product(G[j], sh.ranks[j + 1], S, Q[j + 1], dst, Q[j + 1], sh.ranks[j] * sh.dims[j], Q[j + 1],
                          sh.ranks[j + 1], s)) != LRC_OK)
            return st;
        S = dst;
    }
    if constexpr (sizeof(T) == 4) {
        // Z is P x r (row pitch r), S is r x Q (row pitch Q): B = S^T
        if (tc)
            return launch_split_product(Z, rc, 1, S, 1, Q[c], P[c], Q[c], rc,
                                        ws + lsz[0] + lsz[1] + rsz[0] + rsz[1], out, s);
    }
    return product(Z, sh.ranks[c], S, Q[c], out, Q[c], P[c], Q[c], sh.ranks[c], s);
}

}  // namespace

lrc_status launch_tt_chain_f32(const TTShape& sh, float* out, cudaStream_t s) {
    bool handled = false;
    const lrc_status st = launch_tt_side_f32(sh, out, s, &handled);
    if (handled) return st;
    return launch_chain<float>(sh, out, s);
}

lrc_status launch_tt_chain_f32tc(const TTShape& sh, float* out, cudaStream_t s) {
    return launch_chain<float>(sh, out, s, true);
}

lrc_status launch_tt_chain_f64(const TTShape& sh, double* out, cudaStream_t s) {
    return launch_chain<double>(sh, out, s);
}

bool tt_chain_saves(const TTShape& sh) { return plan_chain(sh).flops <= 0.8 * chain_flops(sh, sh.d - 1); }

}  // namespace lrc
