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
#include <cuda_fp16.h>

#include <algorithm>
#include <vector>

#include "common.cuh"

namespace lrc {

namespace {

constexpr int kGT = 16;          // Gram output tile (kGT x kGT), one entry per thread
constexpr int kGRows = 32;       // rows of the reduction per chunk
constexpr int kGThreads = kGT * kGT;
constexpr int kMmR = 32;         // GEMM tile rows
constexpr int kMmC = 128;        // GEMM tile columns
constexpr int kMmK = 16;         // GEMM k-chunk
constexpr int kCombineBlocks = 304;

__device__ __forceinline__ double wide(double v) { return v; }
__device__ __forceinline__ double wide(float v) { return (double)v; }
__device__ __forceinline__ double wide(__half v) { return (double)__half2float(v); }

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

// Block cores of one interior TT level: Cb (2ra x n x 2rb) from G (ra x n x rb,
// binary64) and Gh (stored format): rows a < ra hold [G(a,i,:), 0], rows
// ra + a hold [G - Gh, Gh].
template <typename T>
__global__ void eta_tt_blocks_kernel(const double* __restrict__ G, const T* __restrict__ Gh, int ra, int64_t n,
                                     int rb, double* __restrict__ Cb) {
    const int64_t total = (int64_t)ra * n * rb;
    const int64_t w = 2 * (int64_t)rb;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t ai = e / rb;              // a * n + i
        const int b = (int)(e - ai * rb);
        const double g = G[e];
        const double gh = wide(Gh[e]);
        double* top = Cb + ai * w;
        double* bot = Cb + (ai + (int64_t)ra * n) * w;
        top[b] = g;
        top[rb + b] = 0.0;
        bot[b] = g - gh;
        bot[rb + b] = gh;
    }
}

// ---- C = A^T B over a long reduction, split over CTAs --------------------
// A: L x p (pitch lda), B: L x q (pitch ldb), binary64.  Output tiles of
// kGT x kGT; with `sym` only tiles ta <= tb are formed (C symmetric).  The
// units (tile pair, 32-row chunk) are ordered pair-major and cut into equal
// contiguous ranges, one per CTA; a CTA writes one partial tile per pair it
// touches, at slot blockIdx.x + pair (distinct for every (CTA, pair)).
struct GramArgs {
    const double* A;
    const double* B;
    int64_t lda, ldb, L;
    int p, q, tq, sym;
    int npairs;
    int64_t nchunks, Q;
    int G;
    double* part;
};

__device__ __forceinline__ void pair_tiles(const GramArgs& g, int t, int* ta, int* tb) {
    if (!g.sym) {
        *ta = t / g.tq;
        *tb = t - *ta * g.tq;
        return;
    }
    int a = 0, rem = t;
    while (rem >= g.tq - a) {
        rem -= g.tq - a;
        ++a;
    }
    *ta = a;
    *tb = a + rem;
}

__host__ __device__ __forceinline__ int64_t cta_of_unit(int64_t u, int64_t Q, int G) {
    return ((u + 1) * (int64_t)G + Q - 1) / Q - 1;
}

__global__ void __launch_bounds__(kGThreads) eta_gram_kernel(const __grid_constant__ GramArgs g) {
    __shared__ double sA[2][kGRows][kGT];
    __shared__ double sB[2][kGRows][kGT];
    const int tid = threadIdx.x;
    const int tx = tid % kGT, ty = tid / kGT;
    // loader mapping: 2 elements of A and 2 of B per thread per chunk
    const int lr = tid / kGT, lc = tid % kGT;     // rows lr and lr + 16
    const int64_t q0 = (int64_t)blockIdx.x * g.Q / g.G;
    const int64_t q1 = (int64_t)(blockIdx.x + 1) * g.Q / g.G;
    int buf = 0;
    int64_t u = q0;
    while (u < q1) {
        const int t = (int)(u / g.nchunks);
        const int64_t ce = min(q1, (int64_t)(t + 1) * g.nchunks);
        int ta, tb;
        pair_tiles(g, t, &ta, &tb);
        const int ca = ta * kGT + lc, cb = tb * kGT + lc;
        const bool va = ca < g.p, vb = cb < g.q;
        double acc = 0.0;
        double ra0, ra1, rb0, rb1;
        auto fetch = [&](int64_t chunk) {
            const int64_t r0 = chunk * kGRows + lr, r1 = r0 + 16;
            ra0 = (va && r0 < g.L) ? g.A[r0 * g.lda + ca] : 0.0;
            ra1 = (va && r1 < g.L) ? g.A[r1 * g.lda + ca] : 0.0;
            rb0 = (vb && r0 < g.L) ? g.B[r0 * g.ldb + cb] : 0.0;
            rb1 = (vb && r1 < g.L) ? g.B[r1 * g.ldb + cb] : 0.0;
        };
        fetch(u - (int64_t)t * g.nchunks);
        for (int64_t v = u; v < ce; ++v) {
            sA[buf][lr][lc] = ra0;
            sA[buf][lr + 16][lc] = ra1;
            sB[buf][lr][lc] = rb0;
            sB[buf][lr + 16][lc] = rb1;
            __syncthreads();
            if (v + 1 < ce) fetch(v + 1 - (int64_t)t * g.nchunks);
#pragma unroll
            for (int r = 0; r < kGRows; ++r) acc = fma(sA[buf][r][ty], sB[buf][r][tx], acc);
            buf ^= 1;
        }
        g.part[((int64_t)blockIdx.x + t) * (kGT * kGT) + ty * kGT + tx] = acc;
        u = ce;
    }
}

// C (p x q, pitch ldc) = sum of the partial tiles in CTA order; with `sym`
// both C[i][j] and C[j][i] take the entry formed for i <= j.
__global__ void eta_gram_reduce_kernel(const __grid_constant__ GramArgs g, double* __restrict__ C, int64_t ldc) {
    const int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (e >= (int64_t)g.p * g.q) return;
    int i = (int)(e / g.q), j = (int)(e % g.q);
    if (g.sym && i > j) {
        const int s = i;
        i = j;
        j = s;
    }
    const int ta = i / kGT, tb = j / kGT;
    int t;
    if (!g.sym) {
        t = ta * g.tq + tb;
    } else {
        t = ta * g.tq - ta * (ta - 1) / 2 + (tb - ta);
    }
    const int64_t c0 = cta_of_unit((int64_t)t * g.nchunks, g.Q, g.G);
    const int64_t c1 = cta_of_unit((int64_t)(t + 1) * g.nchunks - 1, g.Q, g.G);
    const int off = (i % kGT) * kGT + (j % kGT);
    double s = 0.0;
    for (int64_t c = c0; c <= c1; ++c) s += g.part[(c + t) * (kGT * kGT) + off];
    C[(e / g.q) * ldc + (e % g.q)] = s;
}

// ---- C = A B, A p x K (small), B K x N (wide), binary64 ------------------
__global__ void __launch_bounds__(256) eta_gemm_kernel(const double* __restrict__ A, int64_t lda,
                                                       const double* __restrict__ B, int64_t ldb,
                                                       double* __restrict__ C, int64_t ldc, int p, int K,
                                                       int64_t N) {
    __shared__ double sA[kMmK][kMmR];
    __shared__ double sB[kMmK][kMmC];
    const int tid = threadIdx.x;
    const int tx = tid % 32, ty = tid / 32;       // 32 x 8 threads, 4 x 4 outputs each
    const int row0 = blockIdx.y * kMmR;
    const int64_t col0 = (int64_t)blockIdx.x * kMmC;
    double acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = 0.0;
    for (int k0 = 0; k0 < K; k0 += kMmK) {
        // A tile: 32 rows x 16 k -> 2 per thread
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int e = tid + 256 * q;
            const int r = e / kMmK, kk = e % kMmK;
            const int gr = row0 + r, gk = k0 + kk;
            sA[kk][r] = (gr < p && gk < K) ? A[(int64_t)gr * lda + gk] : 0.0;
        }
        // B tile: 16 k x 128 columns -> 8 per thread
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int e = tid + 256 * q;
            const int kk = e / kMmC, c = e % kMmC;
            const int gk = k0 + kk;
            const int64_t gc = col0 + c;
            sB[kk][c] = (gk < K && gc < N) ? B[(int64_t)gk * ldb + gc] : 0.0;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kMmK; ++kk) {
            double a[4], b[4];
#pragma unroll
            for (int x = 0; x < 4; ++x) a[x] = sA[kk][ty * 4 + x];
#pragma unroll
            for (int x = 0; x < 4; ++x) b[x] = sB[kk][tx + 32 * x];
#pragma unroll
            for (int x = 0; x < 4; ++x)
#pragma unroll
                for (int y = 0; y < 4; ++y) acc[x][y] = fma(a[x], b[y], acc[x][y]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int x = 0; x < 4; ++x) {
        const int gr = row0 + ty * 4 + x;
        if (gr >= p) continue;
#pragma unroll
        for (int y = 0; y < 4; ++y) {
            const int64_t gc = col0 + tx + 32 * y;
            if (gc < N) C[(int64_t)gr * ldc + gc] = acc[x][y];
        }
    }
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

// Plan of one A^T B reduction; slot count written to *slots.
GramArgs plan_gram(const double* A, int64_t lda, const double* B, int64_t ldb, int64_t L, int p, int q,
                   bool sym, double* part) {
    GramArgs g{};
    g.A = A;
    g.B = B;
    g.lda = lda;
    g.ldb = ldb;
    g.L = L;
    g.p = p;
    g.q = q;
    g.sym = sym ? 1 : 0;
    const int tp = (p + kGT - 1) / kGT;
    g.tq = (q + kGT - 1) / kGT;
    g.npairs = sym ? tp * (tp + 1) / 2 : tp * g.tq;
    g.nchunks = (L + kGRows - 1) / kGRows;
    g.Q = (int64_t)g.npairs * g.nchunks;
    g.G = (int)std::max<int64_t>(1, std::min<int64_t>(g.Q, 2 * (int64_t)sm_count()));
    g.part = part;
    return g;
}

int64_t gram_slots(int64_t L, int p, int q, bool sym) {
    const int tp = (p + kGT - 1) / kGT, tq = (q + kGT - 1) / kGT;
    const int64_t npairs = sym ? (int64_t)tp * (tp + 1) / 2 : (int64_t)tp * tq;
    const int64_t nchunks = (L + kGRows - 1) / kGRows;
    const int64_t G = std::max<int64_t>(1, std::min<int64_t>(npairs * nchunks, 2 * (int64_t)sm_count()));
    return (G + npairs - 1) * (int64_t)(kGT * kGT);
}

lrc_status run_gram(const GramArgs& g, double* C, int64_t ldc, cudaStream_t s) {
    eta_gram_kernel<<<g.G, kGThreads, 0, s>>>(g);
    lrc_status st = after_launch("eta_gram_kernel");
    if (st != LRC_OK) return st;
    const int64_t n = (int64_t)g.p * g.q;
    eta_gram_reduce_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(g, C, ldc);
    return after_launch("eta_gram_reduce_kernel");
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

template <typename T>
lrc_status tt_blocks(const double* G, const void* Gh, int ra, int64_t n, int rb, double* Cb, cudaStream_t s) {
    eta_tt_blocks_kernel<T><<<grid_for((int64_t)ra * n * rb, 256), 256, 0, s>>>(G, (const T*)Gh, ra, n, rb, Cb);
    return after_launch("eta_tt_blocks_kernel");
}

lrc_status gemm(const double* A, int64_t lda, const double* B, int64_t ldb, double* C, int64_t ldc, int p, int K,
                int64_t N, cudaStream_t s) {
    dim3 grid((unsigned)((N + kMmC - 1) / kMmC), (unsigned)((p + kMmR - 1) / kMmR));
    eta_gemm_kernel<<<grid, 256, 0, s>>>(A, lda, B, ldb, C, ldc, p, K, N);
    return after_launch("eta_gemm_kernel");
}

lrc_status read_result(const double* res, double* eta_out, double* norm_out, cudaStream_t s) {
    double host[2];
    cudaError_t e = cudaMemcpyAsync(host, res, sizeof host, cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync (eta result)");
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize (eta)");
    *eta_out = host[0];
    if (norm_out) *norm_out = host[1];
    return LRC_OK;
}

size_t align_up(size_t v) { return (v + 255) & ~(size_t)255; }

template <typename T>
lrc_status lowrank_eta_t(const double* U, const double* S, const double* Vt, const void* Uh, const void* Sh,
                         const void* Vht, int64_t m, int64_t n, int64_t k, double* eta_out, double* norm_out,
                         cudaStream_t s) {
    const int kk = (int)k;
    const int w = 2 * kk;
    const int64_t ldk = lrc_packed_ld(k), ldn = lrc_packed_ld(n);
    const int64_t slots = std::max(gram_slots(m, w, w, true), gram_slots(n, w, w, true));
    size_t off = 0;
    const size_t o_pu = off;
    off = align_up(off + (size_t)m * w * 8);
    const size_t o_pv = off;
    off = align_up(off + (size_t)n * w * 8);
    const size_t o_gu = off;
    off = align_up(off + (size_t)w * w * 8);
    const size_t o_gv = off;
    off = align_up(off + (size_t)w * w * 8);
    const size_t o_part = off;
    off = align_up(off + (size_t)slots * 8);
    const size_t o_cp = off;
    off = align_up(off + (size_t)2 * kCombineBlocks * 8);
    const size_t o_res = off;
    off = align_up(off + 16);
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, off, &ws);
    if (st != LRC_OK) return st;
    char* base = (char*)ws;
    double* Pu = (double*)(base + o_pu);
    double* Pv = (double*)(base + o_pv);
    double* Gu = (double*)(base + o_gu);
    double* Gv = (double*)(base + o_gv);
    double* part = (double*)(base + o_part);
    double* cpart = (double*)(base + o_cp);
    double* res = (double*)(base + o_res);

    if ((st = pack_rows<T>(U, ldk, Uh, ldk, m, kk, 0, Pu, s)) != LRC_OK) return st;
    if ((st = run_gram(plan_gram(Pu, w, Pu, w, m, w, w, true, part), Gu, w, s)) != LRC_OK) return st;
    if ((st = pack_cols<T>(Vt, ldn, Vht, ldn, n, kk, 0, Pv, s)) != LRC_OK) return st;
    if ((st = run_gram(plan_gram(Pv, w, Pv, w, n, w, w, true, part), Gv, w, s)) != LRC_OK) return st;
    const int cb = std::min(kCombineBlocks, kk);
    eta_lowrank_combine_kernel<T><<<cb, 256, 0, s>>>(Gu, Gv, S, (const T*)Sh, kk, cpart);
    if ((st = after_launch("eta_lowrank_combine_kernel")) != LRC_OK) return st;
    eta_finish_kernel<<<1, 32, 0, s>>>(cpart, cb, res);
    if ((st = after_launch("eta_finish_kernel")) != LRC_OK) return st;
    return read_result(res, eta_out, norm_out, s);
}

template <typename T>
lrc_status tt_eta_t(const TTShape& sh, const void* const* hats, double* eta_out, double* norm_out,
                    cudaStream_t s) {
    const int d = sh.d;
    int rmax = 1;
    int64_t blocks_max = 0, slots = 0;
    for (int l = 0; l <= d; ++l) rmax = std::max<int>(rmax, (int)sh.ranks[l]);
    // level 1: Gram of [dG_1, Gh_1] over n_1 rows; levels 2..d-1: block cores
    // and M C over 2 r_{l-1} n_l rows; level d: Gram of [G_d; dG_d] columns
    slots = std::max(slots, gram_slots(sh.dims[0], 2 * (int)sh.ranks[1], 2 * (int)sh.ranks[1], true));
    for (int l = 1; l < d - 1; ++l) {
        const int64_t ra = sh.ranks[l], rb = sh.ranks[l + 1], n = sh.dims[l];
        blocks_max = std::max(blocks_max, 4 * ra * n * rb);
        slots = std::max(slots, gram_slots(2 * ra * n, 2 * (int)rb, 2 * (int)rb, true));
    }
    const int64_t rl = sh.ranks[d - 1], nl = sh.dims[d - 1];
    slots = std::max(slots, gram_slots(nl, 2 * (int)rl, 2 * (int)rl, true));
    const int64_t pack_max = std::max(sh.dims[0] * 2 * sh.ranks[1], nl * 2 * rl);
    size_t off = 0;
    const size_t o_pk = off;
    off = align_up(off + (size_t)pack_max * 8);
    const size_t o_cb = off;
    off = align_up(off + (size_t)blocks_max * 8);
    const size_t o_x = off;
    off = align_up(off + (size_t)blocks_max * 8);
    const size_t o_m0 = off;
    off = align_up(off + (size_t)4 * rmax * rmax * 8);
    const size_t o_m1 = off;
    off = align_up(off + (size_t)4 * rmax * rmax * 8);
    const size_t o_part = off;
    off = align_up(off + (size_t)slots * 8);
    const size_t o_cp = off;
    off = align_up(off + (size_t)2 * kCombineBlocks * 8);
    const size_t o_res = off;
    off = align_up(off + 16);
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, off, &ws);
    if (st != LRC_OK) return st;
    char* base = (char*)ws;
    double* Pk = (double*)(base + o_pk);
    double* Cb = (double*)(base + o_cb);
    double* Xb = (double*)(base + o_x);
    double* Mcur = (double*)(base + o_m0);
    double* Mnext = (double*)(base + o_m1);
    double* part = (double*)(base + o_part);
    double* cpart = (double*)(base + o_cp);
    double* res = (double*)(base + o_res);

    // level 1: M_1 = [dG_1, Gh_1]^T [dG_1, Gh_1]  (G_1 is n_1 x r_1)
    {
        const int r1 = (int)sh.ranks[1];
        const int64_t n1 = sh.dims[0];
        if ((st = pack_rows<T>((const double*)sh.cores[0], r1, hats[0], r1, n1, r1, 0, Pk, s)) != LRC_OK) return st;
        if ((st = run_gram(plan_gram(Pk, 2 * r1, Pk, 2 * r1, n1, 2 * r1, 2 * r1, true, part), Mcur, 2 * r1, s)) !=
            LRC_OK)
            return st;
    }
    // interior levels: M_l = sum_i C_l(i)^T M_{l-1} C_l(i)
    for (int l = 1; l < d - 1; ++l) {
        const int ra = (int)sh.ranks[l], rb = (int)sh.ranks[l + 1];
        const int64_t n = sh.dims[l];
        if ((st = tt_blocks<T>((const double*)sh.cores[l], hats[l], ra, n, rb, Cb, s)) != LRC_OK) return st;
        const int64_t N = n * 2 * rb;
        if ((st = gemm(Mcur, 2 * ra, Cb, N, Xb, N, 2 * ra, 2 * ra, N, s)) != LRC_OK) return st;
        const int64_t L = 2 * (int64_t)ra * n;
        if ((st = run_gram(plan_gram(Cb, 2 * rb, Xb, 2 * rb, L, 2 * rb, 2 * rb, true, part), Mnext, 2 * rb, s)) !=
            LRC_OK)
            return st;
        std::swap(Mcur, Mnext);
    }
    // level d: H = Gram of the columns [G_d(:, i); dG_d(:, i)] (G_d is r x n_d)
    {
        const int r = (int)rl;
        if ((st = pack_cols<T>((const double*)sh.cores[d - 1], nl, hats[d - 1], nl, nl, r, 1, Pk, s)) != LRC_OK)
            return st;
        if ((st = run_gram(plan_gram(Pk, 2 * r, Pk, 2 * r, nl, 2 * r, 2 * r, true, part), Mnext, 2 * r, s)) !=
            LRC_OK)
            return st;
        const int cb = std::min(kCombineBlocks, r);
        eta_tt_combine_kernel<<<cb, 256, 0, s>>>(Mcur, Mnext, r, cpart);
        if ((st = after_launch("eta_tt_combine_kernel")) != LRC_OK) return st;
        eta_finish_kernel<<<1, 32, 0, s>>>(cpart, cb, res);
        if ((st = after_launch("eta_finish_kernel")) != LRC_OK) return st;
    }
    return read_result(res, eta_out, norm_out, s);
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
    }
    set_error("unknown format");
    return LRC_ERR_INVALID_ARG;
}

}  // namespace lrc
