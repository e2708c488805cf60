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
// this kernel with thin 8-row tiles and many CTAs per SM, so the work spreads
// evenly over the SMs.  binary32 (FFMA-bound) runs the two products on the
// register-tiled kernel of gemm_cc.cu instead: phase 1 split over n (partial
// sums of at most 1024 terms, added in split order by
// reduce_scale_f32_kernel, which also applies diag(s)), phase 2 over
// 128 x 128 tiles of Y.  W (b x k') passes through the stream's workspace.
//
// LRC_F32_TC (a variant): phase 2 on the tensor cores.  W (per row: queries
// may differ in magnitude by any factor) and U (per 32 rows) are scaled by
// powers of two that bring each group's largest magnitude into [2^14, 2^15)
// and split into binary16 parts hi = fp16(x), lo = fp16(x - hi)
// laid side by side along the reduction, W as [W_hi | W_lo | W_hi] in the
// product's 128-row operand image and U as [U_hi | U_hi | U_lo] rows, so
// that one binary16 product with binary32 accumulation (apply_tc.cu) forms
// W U^T ~ W_hi U_hi + W_lo U_hi + W_hi U_lo; its epilogue multiplies each
// entry by the inverse scales (exact).
#include <cuda_fp16.h>

#include "common.cuh"
#include "tc.cuh"

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

// W[r][c] = (sum of the splits' partial products, in split order) * s[c] for
// c < k, zero for k <= c < ldw; one thread per four columns.
__global__ void __launch_bounds__(256)
reduce_scale_f32_kernel(const float* __restrict__ part, int splits, int64_t split_stride, int64_t rows, int64_t k,
                        int64_t ldw, const float* __restrict__ S, float* __restrict__ W) {
    const int64_t q = ldw / 4;
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= rows * q) return;
    const int64_t r = e / q, c = (e - r * q) * 4;
    float4 acc = __ldcs(reinterpret_cast<const float4*>(part + r * ldw + c));
    for (int z = 1; z < splits; ++z) {
        const float4 v = __ldcs(reinterpret_cast<const float4*>(part + (int64_t)z * split_stride + r * ldw + c));
        acc.x = __fadd_rn(acc.x, v.x);
        acc.y = __fadd_rn(acc.y, v.y);
        acc.z = __fadd_rn(acc.z, v.z);
        acc.w = __fadd_rn(acc.w, v.w);
    }
    acc.x = c + 0 < k ? __fmul_rn(acc.x, S[c + 0]) : 0.0f;
    acc.y = c + 1 < k ? __fmul_rn(acc.y, S[c + 1]) : 0.0f;
    acc.z = c + 2 < k ? __fmul_rn(acc.z, S[c + 2]) : 0.0f;
    acc.w = c + 3 < k ? __fmul_rn(acc.w, S[c + 3]) : 0.0f;
    *reinterpret_cast<float4*>(W + r * ldw + c) = acc;
}

lrc_status launch_reduce_scale_f32(const float* part, int splits, int64_t split_stride, int64_t rows, int64_t k,
                                   int64_t ldw, const float* S, float* W, cudaStream_t s) {
    const int64_t items = rows * (ldw / 4);
    reduce_scale_f32_kernel<<<(unsigned)((items + 255) / 256), 256, 0, s>>>(part, splits, split_stride, rows, k, ldw,
                                                                           S, W);
    return after_launch("reduce_scale_f32_kernel");
}

// ---------------------------------------------------------------- LRC_F32_TC
constexpr int kSplitRows = 32;     // rows per scale group (one CTA)

// e with max * 2^e in [2^14, 2^15), clamped to [-60, 60] (the product's
// epilogue factor 2^-(e_w + e_u) stays a normal binary32 number); 0 for a
// zero or non-finite group
__device__ __forceinline__ int group_exp(float maxabs) {
    if (!(maxabs > 0.0f) || !(maxabs <= 3.0e38f)) return 0;
    const int e = 14 - (((__float_as_int(maxabs) >> 23) & 0xff) - 127);
    return e < -60 ? -60 : (e > 60 ? 60 : e);
}

// A CTA per 32 rows of a binary32 matrix whose entry (row, c) is
// src[row * rs + c * cs] (columns from cols on read as zero; TRANS: the
// matrix is the transpose of a row-major one, cs its row pitch, so threads
// take consecutive rows for coalesced reads): scales the rows by powers of two
// -- one per row when PER_ROW (the queries of W may differ in magnitude by any
// factor), else one for the 32 rows -- writes the exponents to esc (index =
// row, or group) and three binary16 parts of every row, part p at columns
// [p kq, (p + 1) kq), the lo half where bit p of lomask is set, else the hi
// half.  IMG: the output is the canonical 128-row operand image of the
// tensor-core product (tile_bytes per tile, rows up to the end of the last
// tile written, zero past `rows`); else row-major with row pitch ldo (rows <
// `rows` only).  A thread converts eight consecutive columns of one row and
// stores each part with one 16-byte store.
template <bool IMG, bool PER_ROW, bool TRANS>
__device__ __forceinline__ void split_parts_block(int64_t blk, const float* __restrict__ src, int64_t rows, int cols,
                                                  int64_t rs, int64_t cs, int kq, int lomask,
                                                  unsigned char* __restrict__ dst, int64_t ldo, uint32_t tile_bytes,
                                                  int* __restrict__ esc) {
    __shared__ float wmax[8];
    __shared__ int rexp[kSplitRows];
    __shared__ int rmax[kSplitRows];    // row maxima as bits (|x| >= 0 orders as an integer)
    const int64_t r0 = blk * kSplitRows;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto at = [&](int64_t row, int c) { return src[row * rs + (int64_t)c * cs]; };
    if (PER_ROW) {
        // one coalesced pass over the 32 rows, maxima gathered by shared atomics
        if (tid < kSplitRows) rmax[tid] = 0;
        __syncthreads();
        for (int e = tid; e < kSplitRows * cols; e += 256) {
            const int r = TRANS ? e % kSplitRows : e / cols, c = TRANS ? e / kSplitRows : e % cols;
            if (r0 + r < rows) atomicMax(&rmax[r], __float_as_int(fabsf(at(r0 + r, c))));
        }
        __syncthreads();
        if (tid < kSplitRows) {
            const int ex = group_exp(__int_as_float(rmax[tid]));
            rexp[tid] = ex;
            if (r0 + tid < rows) esc[r0 + tid] = ex;
        }
    } else {
        float mx = 0.0f;
        for (int e = tid; e < kSplitRows * cols; e += 256) {
            const int r = TRANS ? e % kSplitRows : e / cols, c = TRANS ? e / kSplitRows : e % cols;
            if (r0 + r < rows) mx = fmaxf(mx, fabsf(at(r0 + r, c)));
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        if (lane == 0) wmax[warp] = mx;
        __syncthreads();
        if (tid < kSplitRows) {
            float gm = 0.0f;
#pragma unroll
            for (int w = 0; w < 8; ++w) gm = fmaxf(gm, wmax[w]);
            rexp[tid] = group_exp(gm);
            if (tid == 0) esc[blk] = rexp[0];
        }
    }
    __syncthreads();
    const int g8 = kq / 8;
    for (int e = tid; e < kSplitRows * g8; e += 256) {
        const int r = TRANS ? e % kSplitRows : e / g8;
        const int c0 = (TRANS ? e / kSplitRows : e - r * g8) * 8;
        const int64_t row = r0 + r;
        if (!IMG && row >= rows) continue;
        const float f = __int_as_float((127 + rexp[r]) << 23);
        uint32_t hi[4], lo[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            float x[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int c = c0 + 2 * j + h;
                x[h] = (row < rows && c < cols) ? __fmul_rn(at(row, c), f) : 0.0f;
            }
            const __half h0 = __float2half_rn(x[0]), h1 = __float2half_rn(x[1]);
            const __half l0 = __float2half_rn(__fsub_rn(x[0], __half2float(h0)));
            const __half l1 = __float2half_rn(__fsub_rn(x[1], __half2float(h1)));
            hi[j] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
            lo[j] = (uint32_t)__half_as_ushort(l0) | ((uint32_t)__half_as_ushort(l1) << 16);
        }
        const uint4 vh = make_uint4(hi[0], hi[1], hi[2], hi[3]), vl = make_uint4(lo[0], lo[1], lo[2], lo[3]);
#pragma unroll
        for (int p = 0; p < 3; ++p) {
            const int col = p * kq + c0;
            unsigned char* q = IMG ? dst + (size_t)(row / 128) * tile_bytes +
                                         tc::w_image_off((uint32_t)(row % 128), (uint32_t)col)
                                   : dst + ((size_t)row * ldo + col) * 2;
            *reinterpret_cast<uint4*>(q) = ((lomask >> p) & 1) ? vl : vh;
        }
    }
}

// One launch splits both operands of a product: blocks [0, wblocks) form the
// W image (A: a scale per row, parts [hi | lo | hi]), the rest the U rows
// (B: a scale per 32 rows, parts [hi | hi | lo]).
struct SplitPair {
    const float* A;
    int64_t a_rows, a_rs, a_cs;
    const float* B;
    int64_t b_rows, b_rs, b_cs;
    int cols, kq;
    int64_t wblocks, ldu;
    uint32_t tile_bytes;
    unsigned char* wimg;
    unsigned char* uimg;
    int* esc_w;
    int* esc_u;
};

template <bool TA, bool TB>
__global__ void __launch_bounds__(256) split_pair_kernel(const SplitPair a) {
    if ((int64_t)blockIdx.x < a.wblocks)
        split_parts_block<true, true, TA>(blockIdx.x, a.A, a.a_rows, a.cols, a.a_rs, a.a_cs, a.kq, 0b010, a.wimg, 0,
                                          a.tile_bytes, a.esc_w);
    else
        split_parts_block<false, false, TB>(blockIdx.x - a.wblocks, a.B, a.b_rows, a.cols, a.b_rs, a.b_cs, a.kq,
                                            0b100, a.uimg, a.ldu, 0, a.esc_u);
}

}  // namespace

// Ranks for which the tensor-core second product of LRC_F32_TC applies: the
// three-part W image of a 128-row tile (128 x 3 k16 binary16) leaves room in
// shared memory for the product's U ring and epilogue staging.
constexpr int64_t kF32TcMaxRank = 192;

// C (P x Q, row pitch Q) = A B^T on the tensor cores through the scaled
// binary16 split: A(i, j) = A[i a_rs + j a_cs] (P x k, scaled per row), B(i, j)
// = B[i b_rs + j b_cs] (Q x k, scaled per 32 rows).
lrc_status launch_split_product(const float* A, int64_t a_rs, int64_t a_cs, const float* B, int64_t b_rs,
                                int64_t b_cs, int64_t P, int64_t Q, int64_t k, unsigned char* wimg,
                                unsigned char* uimg, int* esc_w, int* esc_u, float* C, cudaStream_t s) {
    const int64_t kp16 = (k + 15) / 16 * 16, kp3 = 3 * kp16;
    const int64_t ptiles = (P + 127) / 128;
    SplitPair sp{};
    sp.A = A;
    sp.a_rows = P;
    sp.a_rs = a_rs;
    sp.a_cs = a_cs;
    sp.B = B;
    sp.b_rows = Q;
    sp.b_rs = b_rs;
    sp.b_cs = b_cs;
    sp.cols = (int)k;
    sp.kq = (int)kp16;
    sp.wblocks = ptiles * 4;
    sp.ldu = kp3;
    sp.tile_bytes = (uint32_t)(128 * kp3 * 2);
    sp.wimg = wimg;
    sp.uimg = uimg;
    sp.esc_w = esc_w;
    sp.esc_u = esc_u;
    const unsigned grid = (unsigned)(ptiles * 4 + (Q + kSplitRows - 1) / kSplitRows);
    if (a_cs == 1 && b_cs == 1) split_pair_kernel<false, false><<<grid, 256, 0, s>>>(sp);
    else if (a_cs == 1) split_pair_kernel<false, true><<<grid, 256, 0, s>>>(sp);
    else if (b_cs == 1) split_pair_kernel<true, false><<<grid, 256, 0, s>>>(sp);
    else split_pair_kernel<true, true><<<grid, 256, 0, s>>>(sp);
    lrc_status st = after_launch("split_pair_kernel");
    if (st != LRC_OK) return st;
    return launch_y_product(wimg, (int)kp3, uimg, kp3, Q, P, false, C, esc_w, esc_u, s, true);
}

size_t split_product_bytes(int64_t P, int64_t Q, int64_t k) {
    const int64_t kp3 = 3 * ((k + 15) / 16 * 16);
    const int64_t ptiles = (P + 127) / 128;
    return ((size_t)ptiles * 128 * kp3 * 2 + 255) / 256 * 256 + ((size_t)Q * kp3 * 2 + 255) / 256 * 256 +
           (size_t)(ptiles * 128 + (Q + kSplitRows - 1) / kSplitRows) * sizeof(int);
}

bool split_product_fits(int64_t P, int64_t Q, int64_t k) {
    int n2 = 0;
    return k <= kF32TcMaxRank && y_product_plan(Q, P, (int)(3 * ((k + 15) / 16 * 16)), false, &n2) == LRC_OK;
}

lrc_status launch_split_product(const float* A, int64_t a_rs, int64_t a_cs, const float* B, int64_t b_rs,
                                int64_t b_cs, int64_t P, int64_t Q, int64_t k, unsigned char* ws, float* C,
                                cudaStream_t s) {
    const int64_t kp16 = (k + 15) / 16 * 16, kp3 = 3 * kp16;
    const int64_t ptiles = (P + 127) / 128;
    unsigned char* wimg = ws;
    unsigned char* uimg = wimg + ((size_t)ptiles * 128 * kp3 * 2 + 255) / 256 * 256;
    int* esc_w = reinterpret_cast<int*>(uimg + ((size_t)Q * kp3 * 2 + 255) / 256 * 256);
    int* esc_u = esc_w + ptiles * 128;
    return launch_split_product(A, a_rs, a_cs, B, b_rs, b_cs, P, Q, k, wimg, uimg, esc_w, esc_u, C, s);
}


// Batches below these sizes leave the fused kernels' row tiles too few to
// fill the GPU; they take the split path of apply_split.cu (ranks up to 1024).
constexpr int64_t kSplitMaxBatchF64 = 2048, kSplitMaxBatchF32 = 32, kSplitMaxRank = 1024;

lrc_status launch_apply_f64(const double* U, const double* S, const double* Vt, const double* X,
                            double* Y, int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s) {
    if (b <= kSplitMaxBatchF64 && k <= kSplitMaxRank) return launch_apply_split_f64(U, S, Vt, X, Y, m, n, k, b, s);
    return launch_apply_cc<double>(U, S, Vt, X, Y, m, n, k, b, s, "apply_cc_kernel<f64>");
}

lrc_status launch_apply_f32(const float* U, const float* S, const float* Vt, const float* X,
                            float* Y, int64_t m, int64_t n, int64_t k, int64_t b, bool tc, cudaStream_t s) {
    if (b <= kSplitMaxBatchF32 && k <= kSplitMaxRank) return launch_apply_split_f32(U, S, Vt, X, Y, m, n, k, b, s);
    // phase 1: partial products of W = X V over n-splits, with V = (V^T)^T read
    // from the stored V^T rows; phase 2 after the ordered reduction and diag(s)
    const int64_t kp16 = (k + 15) / 16 * 16;
    const int64_t ldn = lrc_packed_ld(n), ldk = lrc_packed_ld(k);
    const int sms = sm_count();
    const int ex = gemm_cc_ex(k);
    const int64_t bn = 128 + 16 * ex;
    const int64_t tiles1 = ((b + 127) / 128) * ((k + bn - 1) / bn);
    const int64_t resident = (int64_t)sms * (ex ? 1 : 2);   // CTAs per SM of the two tile widths
    // at least two waves of CTAs; at most kMaxChunk terms of n per partial sum
    constexpr int64_t kMaxChunk = 1024;
    int64_t splits = (2 * resident + tiles1 - 1) / tiles1;
    const int64_t min_splits = (n + kMaxChunk - 1) / kMaxChunk;
    if (splits < min_splits) splits = min_splits;
    // at least 64 terms per partial: a product with few tiles (small b and k)
    // gets enough CTAs that no CTA walks a long serial chain of K slabs
    const int64_t max_splits = (n + 63) / 64;
    if (splits > max_splits) splits = max_splits > min_splits ? max_splits : min_splits;
    if (splits < 1) splits = 1;
    // the product rounds each split's K range up to its 16-wide slabs
    const int64_t kchunk = ((n + splits - 1) / splits + 15) / 16 * 16;
    splits = (n + kchunk - 1) / kchunk;
    int64_t part_elems, w_elems, t;
    if (!mul_ok(b, kp16, &w_elems) || !mul_ok(w_elems, splits, &part_elems) || !mul_ok(part_elems + w_elems, 4, &t)) {
        set_error("apply_f32: workspace size overflow");
        return LRC_ERR_INVALID_ARG;
    }
    // LRC_F32_TC: room for the binary16 parts of W and U (split_product_bytes)
    tc = tc && split_product_fits(b, m, k);
    const size_t base = ((size_t)(part_elems + w_elems) * sizeof(float) + 255) / 256 * 256;
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, base + (tc ? split_product_bytes(b, m, k) : 0), &ws);
    if (st != LRC_OK) return st;
    float* part = static_cast<float*>(ws);
    float* Wd = part + part_elems;
    if ((st = gemm_cc_f32(X, ldn, Vt, ldn, true, part, kp16, b, k, n, (int)splits, w_elems, s)) != LRC_OK) return st;
    if ((st = launch_reduce_scale_f32(part, (int)splits, w_elems, b, k, kp16, S, Wd, s)) != LRC_OK) return st;
    if (!tc) return gemm_cc_f32(Wd, kp16, U, ldk, true, Y, m, b, m, k, 1, 0, s);
    // Y (b x m) = W U^T with W = Wd (b x k, row pitch kp16) and U (m x k, row pitch ldk)
    return launch_split_product(Wd, kp16, 1, U, ldk, 1, b, m, k, static_cast<unsigned char*>(ws) + base, Y, s);
}

}  // namespace lrc
