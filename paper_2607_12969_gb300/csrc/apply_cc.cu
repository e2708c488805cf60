// apply_cc.cu -- fused low-rank apply on the CUDA cores, binary64 and binary32
// (Sec. 4.4, Eq. gpu_matrix_apply: Y = [(X V) diag(s)] U^T).
//
// A CTA owns BM query rows (a row tile) and a range of Y's columns; CTAs loop
// over row tiles (persistent grid).
//   phase 1: W = X[rows, :] V, reduced over n in BK1-wide slabs staged in
//            shared memory, in BN-wide chunks of the rank dimension; the last
//            chunk only computes the 16-wide column groups below k rounded
//            up to 16, so no arithmetic is spent on rank padding.
//            W <- W diag(s) is applied as each chunk finishes and the scaled
//            chunk is kept (transposed) in shared memory -- it never reaches
//            global memory;
//   phase 2: Y[rows, m-tile] = W U[m-tile, :]^T for every BN-wide m-tile of
//            the CTA's range, with U staged through shared memory and the
//            reduction running over k rounded up to 16 only.
// Each thread owns a TM x TN register tile of the current output tile, rows
// strided by BM/TM and columns strided by BN/TN, so that the shared-memory
// reads of a warp are conflict-free; staging buffers are padded by one
// element per row so that the transposing stores are conflict-free too.
//
// binary64 (DFMA-bound: the GB300 issues about 2 DFMA per clock per SM) uses
// this generic kernel with thin 8-row tiles and many CTAs per SM, so the work
// spreads evenly over the SMs.  binary32 has its own kernel below
// (apply_f32_kernel) with vectorised shared loads and prefetching; it adds
// each slab's partial sums to the running sums separately (blocked
// accumulation, rounding error growing like sqrt(n / BK1)).
#include "common.cuh"

namespace lrc {
namespace {

template <typename T>
struct Cfg;
template <>
struct Cfg<double> {
    // phase 1 handles TN1 16-wide rank groups per pass (TN1 is a template
    // parameter chosen so the passes divide k rounded up to 16 evenly, at most
    // kMaxTN1 groups: predicated-off FMAs still occupy the FP64 pipe, so no
    // pass may carry idle groups); phase 2 uses 64-wide column tiles
    static constexpr int BM = 8, TN2 = 4, BK1 = 16, BK2 = 16, TM = 1, THREADS = 128;
    static constexpr int kMaxTN1 = 12;
    static constexpr bool kBlocked = false;
    static constexpr int kCtasPerSm = 8;
};

template <typename T, int TN1>
__global__ void __launch_bounds__(Cfg<T>::THREADS)
apply_cc_kernel(const T* __restrict__ U, const T* __restrict__ S, const T* __restrict__ Vt,
                const T* __restrict__ X, T* __restrict__ Y, int64_t m, int64_t n, int k, int64_t b,
                int64_t ldk, int64_t ldn, int kp16, int64_t ntiles, int64_t m_chunk) {
    using P = Cfg<T>;
    constexpr int BM = P::BM, BK1 = P::BK1, BK2 = P::BK2, TM = P::TM, TN2 = P::TN2;
    constexpr int NT = P::THREADS;
    constexpr int TX = 16;                 // threads along columns: 16-wide column groups
    constexpr int TY = BM / TM;            // threads along rows
    constexpr int BN1 = TX * TN1, BN2 = TX * TN2;
    constexpr int LDA = BM + 1, LDB = (BN1 > BN2 ? BN1 : BN2) + 1;
    static_assert(TY * TX == NT, "thread tile");
    extern __shared__ __align__(16) unsigned char smem_raw[];
    T* Ws = reinterpret_cast<T*>(smem_raw);            // [kp16][BM]   scaled W, transposed
    T* As = Ws + (size_t)kp16 * BM;                     // [BK1][LDA]   X slab, transposed
    T* Bs = As + BK1 * LDA;                             // [BK][LDB]    Vt / U slab, transposed

    const int tid = threadIdx.x;
    const int tx = tid % TX, ty = tid / TX;
    const int64_t mbeg = (int64_t)blockIdx.y * m_chunk;
    const int64_t mend = (mbeg + m_chunk < m) ? mbeg + m_chunk : m;

    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int64_t row0 = tile * BM;
        // ------------- phase 1: W = X V, BN1 rank columns per pass ----------------
        for (int kc = 0; kc < kp16; kc += BN1) {
            const int rows_v = TN1 * TX;       // passes are full by construction
            T acc[TM][TN1];
#pragma unroll
            for (int i = 0; i < TM; ++i)
#pragma unroll
                for (int j = 0; j < TN1; ++j) acc[i][j] = T(0);
            for (int64_t k0 = 0; k0 < n; k0 += BK1) {
                for (int e = tid; e < BM * BK1; e += NT) {
                    const int r = e / BK1, c = e % BK1;
                    const int64_t gr = row0 + r, gc = k0 + c;
                    As[c * LDA + r] = (gr < b && gc < n) ? X[gr * ldn + gc] : T(0);
                }
                for (int e = tid; e < rows_v * BK1; e += NT) {
                    const int j = e / BK1, c = e % BK1;
                    const int gj = kc + j;
                    const int64_t gc = k0 + c;
                    Bs[c * LDB + j] = (gj < k && gc < n) ? Vt[(int64_t)gj * ldn + gc] : T(0);
                }
                __syncthreads();
                T part[TM][TN1];
#pragma unroll
                for (int i = 0; i < TM; ++i)
#pragma unroll
                    for (int j = 0; j < TN1; ++j) part[i][j] = P::kBlocked ? T(0) : acc[i][j];
#pragma unroll 4
                for (int c = 0; c < BK1; ++c) {
                    T a[TM], bb[TN1];
#pragma unroll
                    for (int i = 0; i < TM; ++i) a[i] = As[c * LDA + ty + i * TY];
#pragma unroll
                    for (int j = 0; j < TN1; ++j) bb[j] = Bs[c * LDB + tx + j * TX];
#pragma unroll
                    for (int i = 0; i < TM; ++i)
#pragma unroll
                        for (int j = 0; j < TN1; ++j) part[i][j] = fma(a[i], bb[j], part[i][j]);
                }
#pragma unroll
                for (int i = 0; i < TM; ++i)
#pragma unroll
                    for (int j = 0; j < TN1; ++j)
                        acc[i][j] = P::kBlocked ? acc[i][j] + part[i][j] : part[i][j];
                __syncthreads();
            }
            // W <- W diag(s), kept transposed in shared memory
#pragma unroll
            for (int j = 0; j < TN1; ++j) {
                const int gj = kc + tx + j * TX;
                const T sj = (gj < k) ? S[gj] : T(0);
#pragma unroll
                for (int i = 0; i < TM; ++i) Ws[(size_t)gj * BM + ty + i * TY] = acc[i][j] * sj;
            }
        }
        __syncthreads();

        // ------------- phase 2: Y[rows, m-tile] = W U[m-tile, :]^T ---------------
        for (int64_t mt = mbeg; mt < mend; mt += BN2) {
            T acc[TM][TN2];
#pragma unroll
            for (int i = 0; i < TM; ++i)
#pragma unroll
                for (int j = 0; j < TN2; ++j) acc[i][j] = T(0);
            for (int k0 = 0; k0 < kp16; k0 += BK2) {
                for (int e = tid; e < BN2 * BK2; e += NT) {
                    const int j = e / BK2, c = e % BK2;
                    const int64_t gm = mt + j;
                    const int gc = k0 + c;
                    Bs[c * LDB + j] = (gm < mend && gc < k) ? U[gm * ldk + gc] : T(0);
                }
                __syncthreads();
#pragma unroll
                for (int c = 0; c < BK2; ++c) {
                    T a[TM], bb[TN2];
#pragma unroll
                    for (int i = 0; i < TM; ++i) a[i] = Ws[(size_t)(k0 + c) * BM + ty + i * TY];
#pragma unroll
                    for (int j = 0; j < TN2; ++j) bb[j] = Bs[c * LDB + tx + j * TX];
#pragma unroll
                    for (int i = 0; i < TM; ++i)
#pragma unroll
                        for (int j = 0; j < TN2; ++j) acc[i][j] = fma(a[i], bb[j], acc[i][j]);
                }
                __syncthreads();
            }
#pragma unroll
            for (int i = 0; i < TM; ++i) {
                const int64_t gr = row0 + ty + i * TY;
                if (gr >= b) continue;
#pragma unroll
                for (int j = 0; j < TN2; ++j) {
                    const int64_t gm = mt + tx + j * TX;
                    if (gm < mend) Y[gr * m + gm] = acc[i][j];
                }
            }
        }
        __syncthreads();   // Ws is rewritten by the next row tile
    }
}

// ---------------------------------------------------------------------------
// binary32: FFMA-bound (128 FMA per clock per SM), so shared-memory traffic
// per FMA matters.  Each thread owns a contiguous 4 x 4 register tile and
// reads its operands as 128-bit shared loads (the A operand is the same for
// the 16 threads of a half-warp row group, a broadcast); the next global
// slab is fetched into registers while the current one is multiplied.
// ---------------------------------------------------------------------------
namespace f32k {
constexpr int BM = 32, BN = 64, BK1 = 32, BK2 = 16, TM = 4, TN = 4, TX = 16, NT = 128;
constexpr int LDA = BM + 4, LDB = BN + 4;     // 16-byte aligned rows
}

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }

// Loads 8 consecutive floats of row `r` (of `rows`), columns c0..c0+7 (of
// `cols`), zero outside.  Rows have pitch `ld` (a multiple of 16 floats).
__device__ __forceinline__ void load8(const float* __restrict__ base, int64_t ld, int64_t r, int64_t rows,
                                      int64_t c0, int64_t cols, float (&v)[8]) {
    if (r < rows && c0 + 8 <= cols) {
        const float4 a = __ldg(reinterpret_cast<const float4*>(base + r * ld + c0));
        const float4 b = __ldg(reinterpret_cast<const float4*>(base + r * ld + c0 + 4));
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = (r < rows && c0 + j < cols) ? __ldg(base + r * ld + c0 + j) : 0.0f;
    }
}

// X slab (32 x 32) row xr cols xc..+7, and Vt slab rows xr and xr+32 of the
// chunk starting at rank kc (only rows below cols_v are real).
__device__ __forceinline__ void fetch_phase1(const float* __restrict__ X, const float* __restrict__ Vt, int64_t ldn,
                                             int64_t row0, int64_t b, int64_t n, int k, int kc, int cols_v,
                                             int xr, int xc, int64_t k0, float (&xv)[8], float (&v0)[8],
                                             float (&v1)[8]) {
    load8(X, ldn, row0 + xr, b, k0 + xc, n, xv);
    if (xr < cols_v) {
        load8(Vt, ldn, kc + xr, k, k0 + xc, n, v0);
    } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) v0[j] = 0.0f;
    }
    if (xr + 32 < cols_v) {
        load8(Vt, ldn, kc + xr + 32, k, k0 + xc, n, v1);
    } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) v1[j] = 0.0f;
    }
}

__global__ void __launch_bounds__(f32k::NT, 3)
apply_f32_kernel(const float* __restrict__ U, const float* __restrict__ S, const float* __restrict__ Vt,
                 const float* __restrict__ X, float* __restrict__ Y, int64_t m, int64_t n, int k, int64_t b,
                 int64_t ldk, int64_t ldn, int kp16, int64_t ntiles, int64_t m_chunk) {
    using namespace f32k;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    float* Ws = reinterpret_cast<float*>(smem_raw);    // [kp16][BM]   scaled W, transposed
    float* As = Ws + (size_t)kp16 * BM;                 // [BK1][LDA]   X slab, transposed
    float* Bs = As + BK1 * LDA;                         // [BK1][LDB]   Vt / U slab, transposed
    const int tid = threadIdx.x;
    const int tx = tid % TX, ty = tid / TX;
    const int64_t mbeg = (int64_t)blockIdx.y * m_chunk;
    const int64_t mend = (mbeg + m_chunk < m) ? mbeg + m_chunk : m;
    // slab-load mapping: X slab 32 x 32 -> thread loads row tid/4, columns (tid%4)*8 .. +7
    const int xr = tid / 4, xc = (tid % 4) * 8;

    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int64_t row0 = tile * BM;
        // ---------------- phase 1 -----------------------------------------------
        for (int kc = 0; kc < kp16; kc += BN) {
            const int cols_v = (kp16 - kc) < BN ? (kp16 - kc) : BN;     // rank columns in this chunk
            float acc[TM][TN] = {};
            float xv[8], v0[8], v1[8];
            fetch_phase1(X, Vt, ldn, row0, b, n, k, kc, cols_v, xr, xc, 0, xv, v0, v1);
            for (int64_t k0 = 0; k0 < n; k0 += BK1) {
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    As[(xc + j) * LDA + xr] = xv[j];
                    Bs[(xc + j) * LDB + xr] = v0[j];
                    Bs[(xc + j) * LDB + xr + 32] = v1[j];
                }
                __syncthreads();
                if (k0 + BK1 < n) fetch_phase1(X, Vt, ldn, row0, b, n, k, kc, cols_v, xr, xc, k0 + BK1, xv, v0, v1);
                float part[TM][TN] = {};
#pragma unroll 8
                for (int c = 0; c < BK1; ++c) {
                    const float4 a = ld4(As + c * LDA + ty * TM);
                    const float4 bb = ld4(Bs + c * LDB + tx * TN);
                    part[0][0] = fmaf(a.x, bb.x, part[0][0]); part[0][1] = fmaf(a.x, bb.y, part[0][1]);
                    part[0][2] = fmaf(a.x, bb.z, part[0][2]); part[0][3] = fmaf(a.x, bb.w, part[0][3]);
                    part[1][0] = fmaf(a.y, bb.x, part[1][0]); part[1][1] = fmaf(a.y, bb.y, part[1][1]);
                    part[1][2] = fmaf(a.y, bb.z, part[1][2]); part[1][3] = fmaf(a.y, bb.w, part[1][3]);
                    part[2][0] = fmaf(a.z, bb.x, part[2][0]); part[2][1] = fmaf(a.z, bb.y, part[2][1]);
                    part[2][2] = fmaf(a.z, bb.z, part[2][2]); part[2][3] = fmaf(a.z, bb.w, part[2][3]);
                    part[3][0] = fmaf(a.w, bb.x, part[3][0]); part[3][1] = fmaf(a.w, bb.y, part[3][1]);
                    part[3][2] = fmaf(a.w, bb.z, part[3][2]); part[3][3] = fmaf(a.w, bb.w, part[3][3]);
                }
#pragma unroll
                for (int i = 0; i < TM; ++i)
#pragma unroll
                    for (int j = 0; j < TN; ++j) acc[i][j] += part[i][j];
                __syncthreads();
            }
#pragma unroll
            for (int j = 0; j < TN; ++j) {
                const int cj = tx * TN + j;
                if (cj >= cols_v) break;
                const int gj = kc + cj;
                const float sj = (gj < k) ? S[gj] : 0.0f;
#pragma unroll
                for (int i = 0; i < TM; ++i) Ws[(size_t)gj * BM + ty * TM + i] = acc[i][j] * sj;
            }
        }
        __syncthreads();
        // ---------------- phase 2 -----------------------------------------------
        // U slab: 64 rows x 16 cols -> thread loads row tid/2, columns (tid%2)*8 .. +7
        const int ur = tid / 2, uc = (tid % 2) * 8;
        for (int64_t mt = mbeg; mt < mend; mt += BN) {
            float acc[TM][TN] = {};
            float uv[8];
            load8(U, ldk, mt + ur, mend, uc, k, uv);
            for (int k0 = 0; k0 < kp16; k0 += BK2) {
#pragma unroll
                for (int j = 0; j < 8; ++j) Bs[(uc + j) * LDB + ur] = uv[j];
                __syncthreads();
                if (k0 + BK2 < kp16) load8(U, ldk, mt + ur, mend, k0 + BK2 + uc, k, uv);
#pragma unroll
                for (int c = 0; c < BK2; ++c) {
                    const float4 a = ld4(Ws + (size_t)(k0 + c) * BM + ty * TM);
                    const float4 bb = ld4(Bs + c * LDB + tx * TN);
                    acc[0][0] = fmaf(a.x, bb.x, acc[0][0]); acc[0][1] = fmaf(a.x, bb.y, acc[0][1]);
                    acc[0][2] = fmaf(a.x, bb.z, acc[0][2]); acc[0][3] = fmaf(a.x, bb.w, acc[0][3]);
                    acc[1][0] = fmaf(a.y, bb.x, acc[1][0]); acc[1][1] = fmaf(a.y, bb.y, acc[1][1]);
                    acc[1][2] = fmaf(a.y, bb.z, acc[1][2]); acc[1][3] = fmaf(a.y, bb.w, acc[1][3]);
                    acc[2][0] = fmaf(a.z, bb.x, acc[2][0]); acc[2][1] = fmaf(a.z, bb.y, acc[2][1]);
                    acc[2][2] = fmaf(a.z, bb.z, acc[2][2]); acc[2][3] = fmaf(a.z, bb.w, acc[2][3]);
                    acc[3][0] = fmaf(a.w, bb.x, acc[3][0]); acc[3][1] = fmaf(a.w, bb.y, acc[3][1]);
                    acc[3][2] = fmaf(a.w, bb.z, acc[3][2]); acc[3][3] = fmaf(a.w, bb.w, acc[3][3]);
                }
                __syncthreads();
            }
#pragma unroll
            for (int i = 0; i < TM; ++i) {
                const int64_t gr = row0 + ty * TM + i;
                if (gr >= b) continue;
                const int64_t gm = mt + tx * TN;
                float* yp = Y + gr * m + gm;
                if (gm + TN <= mend && (m % 4) == 0) {
                    *reinterpret_cast<float4*>(yp) = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
                } else {
#pragma unroll
                    for (int j = 0; j < TN; ++j)
                        if (gm + j < mend) yp[j] = acc[i][j];
                }
            }
        }
        __syncthreads();
    }
}

template <typename T, int TN1>
lrc_status launch_apply_cc_n(const T* U, const T* S, const T* Vt, const T* X, T* Y, int64_t m, int64_t n,
                             int64_t k, int64_t b, int kp16, int passes, cudaStream_t s, const char* name) {
    using P = Cfg<T>;
    constexpr int LDB = 16 * (TN1 > P::TN2 ? TN1 : P::TN2) + 1;
    const int kw = passes * 16 * TN1;                 // rank columns covered by the passes
    const size_t smem = ((size_t)kw * P::BM + P::BK1 * (P::BM + 1) +
                         (size_t)(P::BK1 > P::BK2 ? P::BK1 : P::BK2) * LDB) * sizeof(T);
    if (smem > 227 * 1024) {
        set_error("%s: rank %lld needs %zu bytes of shared memory", name, (long long)k, smem);
        return LRC_ERR_UNSUPPORTED;
    }
    cudaError_t e = cudaFuncSetAttribute(apply_cc_kernel<T, TN1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, name);
    const int64_t ntiles = (b + P::BM - 1) / P::BM;
    const int64_t m_tiles = (m + 16 * P::TN2 - 1) / (16 * P::TN2);
    const int sms = sm_count();
    int ctas_per_sm = P::kCtasPerSm;
    while (ctas_per_sm > 1 && (size_t)ctas_per_sm * (smem + 1024) > 228 * 1024) --ctas_per_sm;
    const int64_t slots = (int64_t)sms * ctas_per_sm;
    // split Y's columns only when the row tiles alone leave most of the GPU idle
    // (each split recomputes phase 1)
    int64_t splits = 1;
    if (ntiles * 2 < sms) splits = (sms + ntiles - 1) / ntiles;
    if (splits > m_tiles) splits = m_tiles;
    if (splits > 65535) splits = 65535;
    const int64_t tiles_per_split = (m_tiles + splits - 1) / splits;
    const int64_t m_chunk = tiles_per_split * 16 * P::TN2;
    splits = (m + m_chunk - 1) / m_chunk;
    int64_t gx = ntiles < slots ? ntiles : slots;
    if (gx > 0x7fffffff) gx = 0x7fffffff;
    dim3 grid((unsigned)gx, (unsigned)splits);
    // the kernel's phase 1 walks kw rank columns (k rounded up to 16, then to the passes)
    apply_cc_kernel<T, TN1><<<grid, P::THREADS, smem, s>>>(U, S, Vt, X, Y, m, n, (int)k, b, lrc_packed_ld(k),
                                                            lrc_packed_ld(n), kw, ntiles, m_chunk);
    (void)kp16;
    return after_launch(name);
}

template <typename T>
lrc_status launch_apply_cc(const T* U, const T* S, const T* Vt, const T* X, T* Y, int64_t m,
                           int64_t n, int64_t k, int64_t b, cudaStream_t s, const char* name) {
    using P = Cfg<T>;
    if (k > 4096) {
        set_error("%s: rank %lld above the supported 4096", name, (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    const int kp16 = (int)((k + 15) / 16 * 16);
    const int groups = kp16 / 16;
    const int passes = (groups + P::kMaxTN1 - 1) / P::kMaxTN1;
    const int tn1 = (groups + passes - 1) / passes;   // passes * tn1 >= groups, tn1 <= kMaxTN1
    switch (tn1) {
        case 1: return launch_apply_cc_n<T, 1>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 2: return launch_apply_cc_n<T, 2>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 3: return launch_apply_cc_n<T, 3>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 4: return launch_apply_cc_n<T, 4>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 5: return launch_apply_cc_n<T, 5>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 6: return launch_apply_cc_n<T, 6>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 7: return launch_apply_cc_n<T, 7>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 8: return launch_apply_cc_n<T, 8>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 9: return launch_apply_cc_n<T, 9>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 10: return launch_apply_cc_n<T, 10>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        case 11: return launch_apply_cc_n<T, 11>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
        default: return launch_apply_cc_n<T, 12>(U, S, Vt, X, Y, m, n, k, b, kp16, passes, s, name);
    }
}

}  // namespace

// Batches below these sizes leave the fused kernels' row tiles too few to
// fill the GPU; they take the split path of apply_split.cu (ranks up to 1024).
constexpr int64_t kSplitMaxBatchF64 = 2048, kSplitMaxBatchF32 = 256, kSplitMaxRank = 1024;

lrc_status launch_apply_f64(const double* U, const double* S, const double* Vt, const double* X,
                            double* Y, int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s) {
    if (b <= kSplitMaxBatchF64 && k <= kSplitMaxRank) return launch_apply_split_f64(U, S, Vt, X, Y, m, n, k, b, s);
    return launch_apply_cc<double>(U, S, Vt, X, Y, m, n, k, b, s, "apply_cc_kernel<f64>");
}

lrc_status launch_apply_f32(const float* U, const float* S, const float* Vt, const float* X,
                            float* Y, int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s) {
    using namespace f32k;
    if (b <= kSplitMaxBatchF32 && k <= kSplitMaxRank) return launch_apply_split_f32(U, S, Vt, X, Y, m, n, k, b, s);
    const char* name = "apply_f32_kernel";
    if (k > 4096) {
        set_error("%s: rank %lld above the supported 4096", name, (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    const int kp16 = (int)((k + 15) / 16 * 16);
    const size_t smem = ((size_t)kp16 * BM + BK1 * LDA + BK1 * LDB) * sizeof(float);
    if (smem > 227 * 1024) {
        set_error("%s: rank %lld needs %zu bytes of shared memory", name, (long long)k, smem);
        return LRC_ERR_UNSUPPORTED;
    }
    cudaError_t e = cudaFuncSetAttribute(apply_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, name);
    const int64_t ntiles = (b + BM - 1) / BM;
    const int64_t m_tiles = (m + BN - 1) / BN;
    const int sms = sm_count();
    int per_sm = (int)((228 * 1024) / (smem + 1024));
    if (per_sm > 8) per_sm = 8;
    if (per_sm < 1) per_sm = 1;
    int64_t splits = 1;
    if (ntiles * 2 < sms) splits = (sms + ntiles - 1) / ntiles;
    if (splits > m_tiles) splits = m_tiles;
    if (splits > 65535) splits = 65535;
    const int64_t tiles_per_split = (m_tiles + splits - 1) / splits;
    const int64_t m_chunk = tiles_per_split * BN;
    splits = (m + m_chunk - 1) / m_chunk;
    const int64_t slots = (int64_t)sms * per_sm;
    int64_t gx = ntiles < slots ? ntiles : slots;
    dim3 grid((unsigned)gx, (unsigned)splits);
    apply_f32_kernel<<<grid, NT, smem, s>>>(U, S, Vt, X, Y, m, n, (int)k, b, lrc_packed_ld(k), lrc_packed_ld(n),
                                            kp16, ntiles, m_chunk);
    return after_launch(name);
}

}  // namespace lrc
