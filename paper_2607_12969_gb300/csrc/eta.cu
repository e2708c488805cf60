// eta.cu -- the storage perturbation eta of Thm 4.1 and eta_TT of Thm 6.1
// without forming either the dense matrix or the dense tensor.
//
// Matrix (remark after Thm 4.1: U, Sigma, V^T rounded individually).  With
// dU = U - Uh, dV = V - Vh, ds = s - sh (exact in binary64: the rounding
// error of a binary64 value to a narrower format is representable),
//
//   A - Ah = U S V^T - Uh Sh Vh^T
//          = [dU, Uh] . [[S, S], [S, dS]] . [dV, Vh]^T,
//
// so with Gu = [dU, Uh]^T [dU, Uh] and Gv = [dV, Vh]^T [dV, Vh] (2k x 2k)
// and the block-diagonal middle matrix M,  eta^2 = tr(M^T Gu M Gv).  Every
// term of that trace carries the rounding errors explicitly, so no large
// quantities cancel (the expansion ||A||^2 - 2<A, Ah> + ||Ah||^2 would lose
// everything for FP32 factors).
//
// Tensor Train (Sec. 5.1, Thm 6.1).  With D_l = Z_l - Zh_l the difference of
// the partial products (Sec. 7.5, Eq. gpu_tt_reconstruction) the pair
// [D_l, Zh_l] obeys [D_l, Zh_l] = [D_{l-1}, Zh_{l-1}] C_l(i_l) with the
// block core C_l(i) = [[G_l(i), 0], [dG_l(i), Gh_l(i)]], and
// T - Th = [D_{d-1}, Zh_{d-1}] [G_d; dG_d].  The Gram matrix
// M_l = sum over prefixes of [D_l, Zh_l]^T [D_l, Zh_l] (2 r_l x 2 r_l)
// follows from M_l = sum_i C_l(i)^T M_{l-1} C_l(i), so eta_TT^2 =
// sum_i [G_d(i); dG_d(i)]^T M_{d-1} [G_d(i); dG_d(i)].
//
// All arithmetic is binary64 (CUDA-core DFMA); the sums are deterministic
// (fixed per-CTA ranges, partials added in a fixed order).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>
#include <vector>

#include "common.cuh"

namespace lrc {

namespace {

constexpr int kGT = 16;          // largest Gram output tile (T x T, one entry per thread)
constexpr int kGRows = 32;       // rows of the reduction per chunk
constexpr int kGThreads = 256;
constexpr int kMaxProbs = 3;     // products per batched launch
constexpr int kMmT = 16;         // GEMM tile: up to 16 rows x 16 columns, one entry per thread
constexpr int kMmK = 16;         // GEMM k-chunk
constexpr int kCombineBlocks = 304;

__device__ __forceinline__ double wide(double v) { return v; }
__device__ __forceinline__ double wide(float v) { return (double)v; }
__device__ __forceinline__ double wide(__half v) { return (double)__half2float(v); }
__device__ __forceinline__ double wide(__nv_bfloat16 v) { return (double)__bfloat162float(v); }

// ---- operand packing --------------------------------------------------------
// P (L x 2k, row pitch 2k) from the row-major L x k factors X (binary64) and
// Xh (stored format): order 0 -> [X - Xh, Xh], order 1 -> [X, X - Xh].
template <typename T>
__global__ void eta_pack_rows_kernel(const double* __restrict__ X, int64_t ldx, const T* __restrict__ Xh,
                                     int64_t ldh, int64_t L, int k, int order, double* __restrict__ P) {
    const int64_t total = L * (int64_t)k;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = e / k;
        const int j = (int)(e - r * k);
        const double x = X[r * ldx + j];
        const double xh = wide(Xh[r * ldh + j]);
        const double dx = x - xh;
        double* row = P + r * (2 * (int64_t)k);
        row[j] = order == 0 ? dx : x;
        row[k + j] = order == 0 ? xh : dx;
    }
}

// P (L x 2k) from the k x L factors X, Xh (the columns of X are the vectors):
// P[c][j] = first block (X - Xh or X) at (j, c), P[c][k + j] = second block.
// 32 x 32 tiles transposed through shared memory; block (32, 8).
template <typename T>
__global__ void eta_pack_cols_kernel(const double* __restrict__ X, int64_t ldx, const T* __restrict__ Xh,
                                     int64_t ldh, int64_t L, int k, int order, double* __restrict__ P) {
    __shared__ double s0[32][33];
    __shared__ double s1[32][33];
    const int64_t c0 = (int64_t)blockIdx.x * 32;
    const int j0 = blockIdx.y * 32;
    const int tx = threadIdx.x, ty = threadIdx.y;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int j = j0 + ty + 8 * q;
        const int64_t c = c0 + tx;
        double a = 0.0, b = 0.0;
        if (j < k && c < L) {
            const double x = X[(int64_t)j * ldx + c];
            const double xh = wide(Xh[(int64_t)j * ldh + c]);
            const double dx = x - xh;
            a = order == 0 ? dx : x;
            b = order == 0 ? xh : dx;
        }
        s0[ty + 8 * q][tx] = a;
        s1[ty + 8 * q][tx] = b;
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int64_t c = c0 + ty + 8 * q;
        const int j = j0 + tx;
        if (c < L && j < k) {
            double* row = P + c * (2 * (int64_t)k);
            row[j] = s0[tx][ty + 8 * q];
            row[k + j] = s1[tx][ty + 8 * q];
        }
    }
}

// Operands of one interior TT level from G (ra x n x rb, binary64) and Gh
// (stored format): CD (2ra x n x rb) holds G in rows a < ra and G - Gh in
// rows ra + a (the D-columns of the block cores [[G, 0], [dG, Gh]]), CZ
// (ra x n x rb) holds Gh in binary64 (their Z-columns; the zero block is not
// stored).
template <typename T>
__global__ void eta_tt_blocks_kernel(const double* __restrict__ G, const T* __restrict__ Gh, int64_t cnt,
                                     double* __restrict__ CD, double* __restrict__ CZ) {
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < cnt;
         e += (int64_t)gridDim.x * blockDim.x) {
        const double g = G[e];
        const double gh = wide(Gh[e]);
        CD[e] = g;
        CD[cnt + e] = g - gh;
        CZ[e] = gh;
    }
}

// ---- C = A^T B over a long reduction, split over CTAs --------------------
// Up to three products per launch.  Product j: A (L x p, pitch lda), B (L x p,
// pitch ldb), binary64; C (p x p, pitch ldc).  Output tiles are T x T with
// T = ceil(p / ceil(p / 16)) so that padding stays small; with `sym` only
// tiles ta <= tb are formed (C symmetric), otherwise C2 (may be null)
// receives C^T.  The units (product, tile pair, 32-row chunk) are laid end to
// end and cut into equal contiguous ranges, one per CTA; a CTA writes one
// partial tile per pair it touches at slot blockIdx.x + global pair index,
// which is distinct for every (CTA, pair).
struct GramProb {
    const double* A;
    const double* B;
    double* C;
    double* C2;
    int64_t lda, ldb, ldc, L;
    int p, T, nt, sym;
    int npairs, t0;            // tile pairs; first global pair index
    int64_t nchunks, u0, e0;   // chunks per pair; first unit; first output entry
};

struct GramBatch {
    GramProb pr[kMaxProbs];
    int np;
    int G;
    int64_t Q;                 // units of all products
    int64_t E;                 // output entries of all products
    double* part;
};

__device__ __forceinline__ void pair_tiles(const GramProb& P, int t, int* ta, int* tb) {
    if (!P.sym) {
        *ta = t / P.nt;
        *tb = t - *ta * P.nt;
        return;
    }
    int a = 0, rem = t;
    while (rem >= P.nt - a) {
        rem -= P.nt - a;
        ++a;
    }
    *ta = a;
    *tb = a + rem;
}

__host__ __device__ __forceinline__ int64_t cta_of_unit(int64_t u, int64_t Q, int G) {
    return ((u + 1) * (int64_t)G + Q - 1) / Q - 1;
}

__global__ void __launch_bounds__(kGThreads) eta_gram_kernel(const __grid_constant__ GramBatch g) {
    __shared__ double sA[2][kGRows][kGT];
    __shared__ double sB[2][kGRows][kGT];
    const int tid = threadIdx.x;
    const int64_t q0 = (int64_t)blockIdx.x * g.Q / g.G;
    const int64_t q1 = (int64_t)(blockIdx.x + 1) * g.Q / g.G;
    int buf = 0;
    int j = 0;
    int64_t u = q0;
    while (u < q1) {
        while (j + 1 < g.np && u >= g.pr[j + 1].u0) ++j;
        const GramProb& P = g.pr[j];
        const double* A = P.A;
        const double* B = P.B;
        const int64_t lda = P.lda, ldb = P.ldb, L = P.L, nch = P.nchunks;
        const int T = P.T, p = P.p;
        const int64_t lu = u - P.u0;
        const int t = (int)(lu / nch);
        const int64_t ce = min(q1, P.u0 + (int64_t)(t + 1) * nch);
        int ta, tb;
        pair_tiles(P, t, &ta, &tb);
        const bool compute = tid < T * T;
        const int tx = compute ? tid % T : 0, ty = compute ? tid / T : 0;
        // loader: elements e = tid and tid + 256 of the 32 x T chunk
        int lr[2], lc[2];
        bool lv[2];
#pragma unroll
        for (int x = 0; x < 2; ++x) {
            const int e = tid + kGThreads * x;
            lv[x] = e < kGRows * T;
            lr[x] = lv[x] ? e / T : 0;
            lc[x] = lv[x] ? e % T : 0;
        }
        double acc = 0.0;
        double ra[2], rb[2];
        auto fetch = [&](int64_t chunk) {
#pragma unroll
            for (int x = 0; x < 2; ++x) {
                const int64_t r = chunk * kGRows + lr[x];
                const int ca = ta * T + lc[x], cb = tb * T + lc[x];
                const bool ok = lv[x] && r < L;
                ra[x] = (ok && ca < p) ? A[r * lda + ca] : 0.0;
                rb[x] = (ok && cb < p) ? B[r * ldb + cb] : 0.0;
            }
        };
        fetch(lu - (int64_t)t * nch);
        for (int64_t v = u; v < ce; ++v) {
#pragma unroll
            for (int x = 0; x < 2; ++x) {
                if (lv[x]) {
                    sA[buf][lr[x]][lc[x]] = ra[x];
                    sB[buf][lr[x]][lc[x]] = rb[x];
                }
            }
            __syncthreads();
            if (v + 1 < ce) fetch(v + 1 - P.u0 - (int64_t)t * nch);
            if (compute) {
#pragma unroll
                for (int r = 0; r < kGRows; ++r) acc = fma(sA[buf][r][ty], sB[buf][r][tx], acc);
            }
            buf ^= 1;
        }
        if (compute) g.part[((int64_t)blockIdx.x + P.t0 + t) * (kGT * kGT) + ty * T + tx] = acc;
        u = ce;
    }
}

// Every output entry: the partial tiles of its pair added in CTA order.
__global__ void eta_gram_reduce_kernel(const __grid_constant__ GramBatch g) {
    const int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (e >= g.E) return;
    int jp = 0;
    while (jp + 1 < g.np && e >= g.pr[jp + 1].e0) ++jp;
    const GramProb& P = g.pr[jp];
    const int64_t le = e - P.e0;
    const int i0 = (int)(le / P.p), j0 = (int)(le % P.p);
    int i = i0, j = j0;
    if (P.sym && i > j) {
        i = j0;
        j = i0;
    }
    const int T = P.T;
    const int ta = i / T, tb = j / T;
    const int t = P.sym ? ta * P.nt - ta * (ta - 1) / 2 + (tb - ta) : ta * P.nt + tb;
    const int64_t c0 = cta_of_unit(P.u0 + (int64_t)t * P.nchunks, g.Q, g.G);
    const int64_t c1 = cta_of_unit(P.u0 + (int64_t)(t + 1) * P.nchunks - 1, g.Q, g.G);
    const int off = (i % T) * T + (j % T);
    const int64_t tg = P.t0 + t;
    double s = 0.0;
    for (int64_t c = c0; c <= c1; ++c) s += g.part[(c + tg) * (kGT * kGT) + off];
    P.C[(int64_t)i0 * P.ldc + j0] = s;
    if (P.C2) P.C2[(int64_t)j0 * P.ldc + i0] = s;
}

// ---- C = A B, A p x K (small), B K x N (wide), binary64 ------------------
// Up to two products per launch; tiles of TR x 16 entries (TR = ceil(p /
// ceil(p / 16))), one entry per thread, row tiles of one column block in
// consecutive CTAs.
struct MmProb {
    const double* A;
    const double* B;
    double* C;
    int64_t lda, ldb, ldc, N;
    int p, K, TR, ntr;
    int64_t b0;                // first CTA
};

struct MmBatch {
    MmProb pr[2];
    int np;
};

__global__ void __launch_bounds__(256) eta_gemm_kernel(const __grid_constant__ MmBatch g) {
    __shared__ double sA[kMmK][kMmT];
    __shared__ double sB[kMmK][kMmT];
    const int jp = (g.np > 1 && (int64_t)blockIdx.x >= g.pr[1].b0) ? 1 : 0;
    const MmProb& P = g.pr[jp];
    const double* A = P.A;
    const double* B = P.B;
    const int64_t lb = (int64_t)blockIdx.x - P.b0;
    const int row0 = (int)(lb % P.ntr) * P.TR;
    const int64_t col0 = (lb / P.ntr) * kMmT;
    const int tid = threadIdx.x;
    const int ty = tid / kMmT, tx = tid % kMmT;
    const int TR = P.TR, p = P.p, K = P.K;
    const int64_t N = P.N;
    double acc = 0.0;
    for (int k0 = 0; k0 < K; k0 += kMmK) {
        {
            const int r = tid / kMmK, kk = tid % kMmK;       // A: TR rows x 16 k
            const int gr = row0 + r, gk = k0 + kk;
            sA[kk][r] = (r < TR && gr < p && gk < K) ? A[(int64_t)gr * P.lda + gk] : 0.0;
            const int kb = tid / kMmT, c = tid % kMmT;       // B: 16 k x 16 columns
            const int64_t gc = col0 + c;
            sB[kb][c] = (k0 + kb < K && gc < N) ? B[(int64_t)(k0 + kb) * P.ldb + gc] : 0.0;
        }
        __syncthreads();
        if (ty < TR) {
#pragma unroll
            for (int kk = 0; kk < kMmK; ++kk) acc = fma(sA[kk][ty], sB[kk][tx], acc);
        }
        __syncthreads();
    }
    const int gr = row0 + ty;
    const int64_t gc = col0 + tx;
    if (ty < TR && gr < p && gc < N) P.C[(int64_t)gr * P.ldc + gc] = acc;
}

// ---- final contractions ------------------------------------------------------
// Fixed-order block sum of (v0, v1) over 256 threads; result in thread 0.
__device__ __forceinline__ void block_sum2(double& v0, double& v1) {
    __shared__ double r0[8], r1[8];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        v0 += __shfl_xor_sync(0xffffffffu, v0, o);
        v1 += __shfl_xor_sync(0xffffffffu, v1, o);
    }
    const int w = threadIdx.x / 32;
    if ((threadIdx.x & 31) == 0) {
        r0[w] = v0;
        r1[w] = v1;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double a = 0.0, b = 0.0;
        for (int x = 0; x < (int)(blockDim.x / 32); ++x) {
            a += r0[x];
            b += r1[x];
        }
        v0 = a;
        v1 = b;
    }
}

// Matrix: eta^2 = sum_{i,j} sum_{p,p',q,q'} mu_pq(i) mu_p'q'(j) Gu_pp'(i,j) Gv_qq'(i,j)
// with mu_00 = mu_01 = mu_10 = s, mu_11 = s - sh (block 0 = difference,
// block 1 = stored factor); ||A||^2 = sum s_i s_j (U^T U)_ij (V^T V)_ij with
// U^T U = sum of the four Gu blocks (U = dU + Uh), likewise V^T V.
template <typename T>
__global__ void __launch_bounds__(256) eta_lowrank_combine_kernel(const double* __restrict__ Gu,
                                                                  const double* __restrict__ Gv,
                                                                  const double* __restrict__ s,
                                                                  const T* __restrict__ sh, int k,
                                                                  double* __restrict__ part) {
    const int64_t ld = 2 * (int64_t)k;
    double e2 = 0.0, n2 = 0.0;
    for (int i = blockIdx.x; i < k; i += gridDim.x) {
        const double si = s[i];
        const double di = si - wide(sh[i]);
        for (int j = threadIdx.x; j < k; j += blockDim.x) {
            const double sj = s[j];
            const double dj = sj - wide(sh[j]);
            const double u00 = Gu[i * ld + j], u01 = Gu[i * ld + k + j];
            const double u10 = Gu[(k + i) * ld + j], u11 = Gu[(k + i) * ld + k + j];
            const double v00 = Gv[i * ld + j], v01 = Gv[i * ld + k + j];
            const double v10 = Gv[(k + i) * ld + j], v11 = Gv[(k + i) * ld + k + j];
            // W_pp' = sum_{q,q'} mu_pq(i) mu_p'q'(j) Gv_qq'
            const double v_all = (v00 + v01) + (v10 + v11);
            const double w00 = si * sj * v_all;                          // p = p' = 0
            const double w01 = si * (sj * (v00 + v10) + dj * (v01 + v11));   // p = 0, p' = 1
            const double w10 = sj * (si * (v00 + v01) + di * (v10 + v11));   // p = 1, p' = 0
            const double w11 = si * sj * v00 + si * dj * v01 + di * sj * v10 + di * dj * v11;
            e2 += u00 * w00 + u01 * w01 + u10 * w10 + u11 * w11;
            n2 += si * sj * ((u00 + u01) + (u10 + u11)) * v_all;
        }
    }
    block_sum2(e2, n2);
    if (threadIdx.x == 0) {
        part[2 * blockIdx.x] = e2;
        part[2 * blockIdx.x + 1] = n2;
    }
}

// TT: eta^2 = <M_DD, H_GG> + 2 <M_DZ, H_GdG> + <M_ZZ, H_dGdG>,
// ||T||^2 = <M_DD + M_DZ + M_ZD + M_ZZ, H_GG>, with M the Gram matrix of
// [D, Zh] and H that of the columns [G_d; dG_d] (both 2r x 2r, pitch 2r).
__global__ void __launch_bounds__(256) eta_tt_combine_kernel(const double* __restrict__ M,
                                                             const double* __restrict__ H, int r,
                                                             double* __restrict__ part) {
    const int64_t ld = 2 * (int64_t)r;
    double e2 = 0.0, n2 = 0.0;
    for (int a = blockIdx.x; a < r; a += gridDim.x) {
        for (int b = threadIdx.x; b < r; b += blockDim.x) {
            const double mdd = M[a * ld + b], mdz = M[a * ld + r + b];
            const double mzd = M[(r + a) * ld + b], mzz = M[(r + a) * ld + r + b];
            const double hgg = H[a * ld + b], hgd = H[a * ld + r + b], hdd = H[(r + a) * ld + r + b];
            e2 += mdd * hgg + 2.0 * mdz * hgd + mzz * hdd;
            n2 += ((mdd + mdz) + (mzd + mzz)) * hgg;
        }
    }
    block_sum2(e2, n2);
    if (threadIdx.x == 0) {
        part[2 * blockIdx.x] = e2;
        part[2 * blockIdx.x + 1] = n2;
    }
}

__global__ void eta_finish_kernel(const double* __restrict__ part, int nparts, double* __restrict__ res) {
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    double e2 = 0.0, n2 = 0.0;
    for (int b = 0; b < nparts; ++b) {
        e2 += part[2 * b];
        n2 += part[2 * b + 1];
    }
    res[0] = sqrt(fmax(e2, 0.0));
    res[1] = sqrt(fmax(n2, 0.0));
}

// ---- host side ---------------------------------------------------------------

int grid_for(int64_t work, int threads) {
    const int64_t cap = (int64_t)sm_count() * 8;
    int64_t g = (work + threads - 1) / threads;
    return (int)std::max<int64_t>(1, std::min<int64_t>(g, cap));
}

struct GramSpec {
    const double* A;
    const double* B;
    int64_t lda, ldb, L;
    int p;
    bool sym;
    double* C;
    double* C2;
    int64_t ldc;
};

GramBatch plan_gram(const GramSpec* sp, int np, double* part) {
    GramBatch g{};
    g.np = np;
    int64_t u = 0, e = 0;
    int t0 = 0;
    for (int j = 0; j < np; ++j) {
        GramProb& P = g.pr[j];
        P.A = sp[j].A;
        P.B = sp[j].B;
        P.C = sp[j].C;
        P.C2 = sp[j].C2;
        P.lda = sp[j].lda;
        P.ldb = sp[j].ldb;
        P.ldc = sp[j].ldc;
        P.L = sp[j].L;
        P.p = sp[j].p;
        P.sym = sp[j].sym ? 1 : 0;
        const int nt = (P.p + kGT - 1) / kGT;
        P.T = (P.p + nt - 1) / nt;
        P.nt = (P.p + P.T - 1) / P.T;
        P.npairs = P.sym ? P.nt * (P.nt + 1) / 2 : P.nt * P.nt;
        P.nchunks = std::max<int64_t>(1, (P.L + kGRows - 1) / kGRows);
        P.u0 = u;
        P.t0 = t0;
        P.e0 = e;
        u += (int64_t)P.npairs * P.nchunks;
        t0 += P.npairs;
        e += (int64_t)P.p * P.p;
    }
    g.Q = u;
    g.E = e;
    g.G = (int)std::max<int64_t>(1, std::min<int64_t>(g.Q, 2 * (int64_t)sm_count()));
    g.part = part;
    return g;
}

// Partial-slot entries a batch needs (computed without a device pointer).
int64_t gram_slots(const GramSpec* sp, int np) {
    const GramBatch g = plan_gram(sp, np, nullptr);
    int pairs = 0;
    for (int j = 0; j < np; ++j) pairs += g.pr[j].npairs;
    return ((int64_t)g.G + pairs - 1) * (kGT * kGT);
}

lrc_status run_gram(const GramSpec* sp, int np, double* part, cudaStream_t s) {
    const GramBatch g = plan_gram(sp, np, part);
    eta_gram_kernel<<<g.G, kGThreads, 0, s>>>(g);
    lrc_status st = after_launch("eta_gram_kernel");
    if (st != LRC_OK) return st;
    eta_gram_reduce_kernel<<<(unsigned)((g.E + 255) / 256), 256, 0, s>>>(g);
    return after_launch("eta_gram_reduce_kernel");
}

struct MmSpec {
    const double* A;
    const double* B;
    double* C;
    int64_t lda, ldb, ldc, N;
    int p, K;
};

lrc_status run_gemm(const MmSpec* sp, int np, cudaStream_t s) {
    MmBatch g{};
    g.np = np;
    int64_t b = 0;
    for (int j = 0; j < np; ++j) {
        MmProb& P = g.pr[j];
        P.A = sp[j].A;
        P.B = sp[j].B;
        P.C = sp[j].C;
        P.lda = sp[j].lda;
        P.ldb = sp[j].ldb;
        P.ldc = sp[j].ldc;
        P.N = sp[j].N;
        P.p = sp[j].p;
        P.K = sp[j].K;
        const int nt = (P.p + kMmT - 1) / kMmT;
        P.TR = (P.p + nt - 1) / nt;
        P.ntr = (P.p + P.TR - 1) / P.TR;
        P.b0 = b;
        b += (int64_t)P.ntr * ((P.N + kMmT - 1) / kMmT);
    }
    if (b > 0x7fffffffLL) {
        set_error("eta GEMM grid too large");
        return LRC_ERR_UNSUPPORTED;
    }
    eta_gemm_kernel<<<(unsigned)b, 256, 0, s>>>(g);
    return after_launch("eta_gemm_kernel");
}

template <typename T>
lrc_status pack_rows(const double* X, int64_t ldx, const void* Xh, int64_t ldh, int64_t L, int k, int order,
                     double* P, cudaStream_t s) {
    eta_pack_rows_kernel<T><<<grid_for(L * k, 256), 256, 0, s>>>(X, ldx, (const T*)Xh, ldh, L, k, order, P);
    return after_launch("eta_pack_rows_kernel");
}

template <typename T>
lrc_status pack_cols(const double* X, int64_t ldx, const void* Xh, int64_t ldh, int64_t L, int k, int order,
                     double* P, cudaStream_t s) {
    dim3 grid((unsigned)((L + 31) / 32), (unsigned)((k + 31) / 32));
    eta_pack_cols_kernel<T><<<grid, dim3(32, 8), 0, s>>>(X, ldx, (const T*)Xh, ldh, L, k, order, P);
    return after_launch("eta_pack_cols_kernel");
}

// The last step of an eta: eta_finish_kernel adds the block sums in order
// and writes (eta, norm) into the stream's mapped result slot; the host reads
// them once the stream has synchronised (no copy-engine transfer).
lrc_status finish_eta(const double* cpart, int nparts, double* eta_out, double* norm_out, cudaStream_t s) {
    double* host = nullptr;
    double* dev = nullptr;
    lrc_status st = stream_result_slot(s, &host, &dev);
    if (st != LRC_OK) return st;
    eta_finish_kernel<<<1, 32, 0, s>>>(cpart, nparts, dev);
    if ((st = after_launch("eta_finish_kernel")) != LRC_OK) return st;
    const cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize (eta)");
    *eta_out = host[0];
    if (norm_out) *norm_out = host[1];
    return LRC_OK;
}

size_t align_up(size_t v) { return (v + 255) & ~(size_t)255; }

// Carves consecutive 256-byte aligned regions out of one workspace.
struct Carve {
    size_t off = 0;
    size_t take(size_t bytes) {
        const size_t o = off;
        off = align_up(off + bytes);
        return o;
    }
};

template <typename T>
lrc_status lowrank_eta_t(const double* U, const double* S, const double* Vt, const void* Uh, const void* Sh,
                         const void* Vht, int64_t m, int64_t n, int64_t k, double* eta_out, double* norm_out,
                         cudaStream_t s) {
    const int kk = (int)k;
    const int w = 2 * kk;
    const int64_t ldk = lrc_packed_ld(k), ldn = lrc_packed_ld(n);
    GramSpec sp[2] = {{nullptr, nullptr, w, w, m, w, true, nullptr, nullptr, w},
                      {nullptr, nullptr, w, w, n, w, true, nullptr, nullptr, w}};
    Carve c;
    const size_t o_pu = c.take((size_t)m * w * 8), o_pv = c.take((size_t)n * w * 8);
    const size_t o_gu = c.take((size_t)w * w * 8), o_gv = c.take((size_t)w * w * 8);
    const size_t o_part = c.take((size_t)gram_slots(sp, 2) * 8);
    const size_t o_cp = c.take((size_t)2 * kCombineBlocks * 8);
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, c.off, &ws);
    if (st != LRC_OK) return st;
    char* base = (char*)ws;
    double* Pu = (double*)(base + o_pu);
    double* Pv = (double*)(base + o_pv);
    double* Gu = (double*)(base + o_gu);
    double* Gv = (double*)(base + o_gv);
    double* cpart = (double*)(base + o_cp);
    sp[0].A = sp[0].B = Pu;
    sp[0].C = Gu;
    sp[1].A = sp[1].B = Pv;
    sp[1].C = Gv;

    if ((st = pack_rows<T>(U, ldk, Uh, ldk, m, kk, 0, Pu, s)) != LRC_OK) return st;
    if ((st = pack_cols<T>(Vt, ldn, Vht, ldn, n, kk, 0, Pv, s)) != LRC_OK) return st;
    if ((st = run_gram(sp, 2, (double*)(base + o_part), s)) != LRC_OK) return st;
    const int cb = std::min(kCombineBlocks, kk);
    eta_lowrank_combine_kernel<T><<<cb, 256, 0, s>>>(Gu, Gv, S, (const T*)Sh, kk, cpart);
    if ((st = after_launch("eta_lowrank_combine_kernel")) != LRC_OK) return st;
    return finish_eta(cpart, cb, eta_out, norm_out, s);
}

// The three products of one interior level (D-columns: CD, X_D; Z-columns:
// CZ, X_Z), written into the blocks of Mn (pitch 2 rb).
void interior_gram_specs(int ra, int64_t n, int rb, const double* CD, const double* CZ, const double* XD,
                         const double* XZ, double* Mn, GramSpec* sp) {
    const int64_t ld = 2 * (int64_t)rb;
    const int64_t L2 = 2 * (int64_t)ra * n, L1 = (int64_t)ra * n;
    sp[0] = {CD, XD, rb, rb, L2, rb, true, Mn, nullptr, ld};                              // M'_DD
    sp[1] = {CD, XZ, rb, rb, L2, rb, false, Mn + rb, Mn + (int64_t)rb * ld, ld};          // M'_DZ, M'_ZD
    sp[2] = {CZ, XZ + L1 * rb, rb, rb, L1, rb, true, Mn + (int64_t)rb * ld + rb, nullptr, ld};   // M'_ZZ
}

template <typename T>
lrc_status tt_eta_t(const TTShape& sh, const void* const* hats, double* eta_out, double* norm_out,
                    cudaStream_t s) {
    const int d = sh.d;
    int rmax = 1;
    for (int l = 0; l <= d; ++l) rmax = std::max<int>(rmax, (int)sh.ranks[l]);
    const int r1 = (int)sh.ranks[1], rl = (int)sh.ranks[d - 1];
    const int64_t n1 = sh.dims[0], nl = sh.dims[d - 1];
    // workspace sizes: packed first / last core, per-level operands, slots
    int64_t lev_max = 0, slots = 0;
    {
        GramSpec a = {nullptr, nullptr, 2 * r1, 2 * r1, n1, 2 * r1, true, nullptr, nullptr, 2 * r1};
        GramSpec b = {nullptr, nullptr, 2 * rl, 2 * rl, nl, 2 * rl, true, nullptr, nullptr, 2 * rl};
        slots = std::max(gram_slots(&a, 1), gram_slots(&b, 1));
    }
    for (int l = 1; l < d - 1; ++l) {
        const int ra = (int)sh.ranks[l], rb = (int)sh.ranks[l + 1];
        const int64_t n = sh.dims[l];
        lev_max = std::max(lev_max, 7 * (int64_t)ra * n * rb);
        GramSpec sp[3];
        interior_gram_specs(ra, n, rb, nullptr, nullptr, nullptr, nullptr, nullptr, sp);
        slots = std::max(slots, gram_slots(sp, 3));
    }
    const int64_t pack_max = std::max(n1 * 2 * r1, nl * 2 * rl);
    Carve c;
    const size_t o_pk = c.take((size_t)pack_max * 8), o_lev = c.take((size_t)lev_max * 8);
    const size_t o_m0 = c.take((size_t)4 * rmax * rmax * 8), o_m1 = c.take((size_t)4 * rmax * rmax * 8);
    const size_t o_part = c.take((size_t)slots * 8);
    const size_t o_cp = c.take((size_t)2 * kCombineBlocks * 8);
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, c.off, &ws);
    if (st != LRC_OK) return st;
    char* base = (char*)ws;
    double* Pk = (double*)(base + o_pk);
    double* lev = (double*)(base + o_lev);
    double* Mcur = (double*)(base + o_m0);
    double* Mnext = (double*)(base + o_m1);
    double* part = (double*)(base + o_part);
    double* cpart = (double*)(base + o_cp);

    // level 1: M_1 = [dG_1, Gh_1]^T [dG_1, Gh_1]  (G_1 is n_1 x r_1)
    if ((st = pack_rows<T>((const double*)sh.cores[0], r1, hats[0], r1, n1, r1, 0, Pk, s)) != LRC_OK) return st;
    {
        GramSpec a = {Pk, Pk, 2 * r1, 2 * r1, n1, 2 * r1, true, Mcur, nullptr, 2 * r1};
        if ((st = run_gram(&a, 1, part, s)) != LRC_OK) return st;
    }
    // interior levels: M_l = sum_i C_l(i)^T M_{l-1} C_l(i)
    for (int l = 1; l < d - 1; ++l) {
        const int ra = (int)sh.ranks[l], rb = (int)sh.ranks[l + 1];
        const int64_t n = sh.dims[l];
        const int64_t cnt = (int64_t)ra * n * rb, N = n * rb;
        double* CD = lev;
        double* CZ = CD + 2 * cnt;
        double* XD = CZ + cnt;
        double* XZ = XD + 2 * cnt;
        eta_tt_blocks_kernel<T><<<grid_for(cnt, 256), 256, 0, s>>>((const double*)sh.cores[l], (const T*)hats[l],
                                                                    cnt, CD, CZ);
        if ((st = after_launch("eta_tt_blocks_kernel")) != LRC_OK) return st;
        // X_D = M [G; dG], X_Z = M[:, Z] Gh  (2ra x n rb each)
        MmSpec mm[2] = {{Mcur, CD, XD, 2 * ra, N, N, N, 2 * ra, 2 * ra},
                        {Mcur + ra, CZ, XZ, 2 * ra, N, N, N, 2 * ra, ra}};
        if ((st = run_gemm(mm, 2, s)) != LRC_OK) return st;
        GramSpec sp[3];
        interior_gram_specs(ra, n, rb, CD, CZ, XD, XZ, Mnext, sp);
        if ((st = run_gram(sp, 3, part, s)) != LRC_OK) return st;
        std::swap(Mcur, Mnext);
    }
    // level d: H = Gram of the columns [G_d(:, i); dG_d(:, i)] (G_d is r x n_d)
    if ((st = pack_cols<T>((const double*)sh.cores[d - 1], nl, hats[d - 1], nl, nl, rl, 1, Pk, s)) != LRC_OK)
        return st;
    {
        GramSpec b = {Pk, Pk, 2 * rl, 2 * rl, nl, 2 * rl, true, Mnext, nullptr, 2 * rl};
        if ((st = run_gram(&b, 1, part, s)) != LRC_OK) return st;
    }
    const int cb = std::min(kCombineBlocks, rl);
    eta_tt_combine_kernel<<<cb, 256, 0, s>>>(Mcur, Mnext, rl, cpart);
    if ((st = after_launch("eta_tt_combine_kernel")) != LRC_OK) return st;
    return finish_eta(cpart, cb, eta_out, norm_out, s);
}

}  // namespace

lrc_status run_lowrank_eta(const double* U, const double* S, const double* Vt, const void* Uh, const void* Sh,
                           const void* Vht, lrc_fmt fmt, int64_t m, int64_t n, int64_t k, double* eta_out,
                           double* norm_out, cudaStream_t s) {
    switch (fmt) {
        case LRC_F64: return lowrank_eta_t<double>(U, S, Vt, Uh, Sh, Vht, m, n, k, eta_out, norm_out, s);
        case LRC_F32: return lowrank_eta_t<float>(U, S, Vt, Uh, Sh, Vht, m, n, k, eta_out, norm_out, s);
        case LRC_F16:
        case LRC_F16_O16: return lowrank_eta_t<__half>(U, S, Vt, Uh, Sh, Vht, m, n, k, eta_out, norm_out, s);
        case LRC_BF16: return lowrank_eta_t<__nv_bfloat16>(U, S, Vt, Uh, Sh, Vht, m, n, k, eta_out, norm_out, s);
    }
    set_error("unknown format");
    return LRC_ERR_INVALID_ARG;
}

lrc_status run_tt_eta(const TTShape& sh, const void* const* hats, lrc_fmt fmt, double* eta_out, double* norm_out,
                      cudaStream_t s) {
    switch (fmt) {
        case LRC_F64: return tt_eta_t<double>(sh, hats, eta_out, norm_out, s);
        case LRC_F32: return tt_eta_t<float>(sh, hats, eta_out, norm_out, s);
        case LRC_F16:
        case LRC_F16_O16: return tt_eta_t<__half>(sh, hats, eta_out, norm_out, s);
        case LRC_BF16: return tt_eta_t<__nv_bfloat16>(sh, hats, eta_out, norm_out, s);
    }
    set_error("unknown format");
    return LRC_ERR_INVALID_ARG;
}

}  // namespace lrc
