// apply_cc.cu -- fused low-rank apply on the CUDA cores, binary64 and binary32
// (Sec. 4.4, Eq. gpu_matrix_apply: Y = [(X V) diag(s)] U^T).
//
// One CTA owns BM query rows and a range of output columns of Y.
//   phase 1: W = X[rows, :] V, reduced over n in BK-wide slabs staged in
//            shared memory, in BN-wide chunks of the rank dimension;
//            W <- W diag(s) is applied as each chunk finishes and the scaled
//            chunk is kept (transposed) in shared memory -- it never reaches
//            global memory;
//   phase 2: Y[rows, m-tile] = W U[m-tile, :]^T for every BN-wide m-tile of
//            the CTA's range, with U staged through shared memory.
// Each thread owns a TM x TN register tile of the current output tile, with
// rows strided by BM/TM and columns strided by BN/TN so that the shared-memory
// reads of a warp are conflict-free; staging buffers are padded by one
// element per row so that the transposing stores are conflict-free too.
// binary32 adds each BK slab's partial sums to the running sums separately
// (blocked accumulation) so the rounding error grows like sqrt(n / BK).
#include "common.cuh"

namespace lrc {
namespace {

constexpr int kThreads = 256;

template <typename T>
struct Tile;
template <>
struct Tile<double> {  // binary64: BM x BN = 32 x 64, 2 x 4 per thread
    static constexpr int BM = 32, BN = 64, BK = 16, TM = 2, TN = 4;
    static constexpr bool kBlocked = false;
};
template <>
struct Tile<float> {   // binary32: 64 x 64, 4 x 4 per thread
    static constexpr int BM = 64, BN = 64, BK = 32, TM = 4, TN = 4;
    static constexpr bool kBlocked = true;
};

template <typename T>
__global__ void __launch_bounds__(kThreads)
apply_cc_kernel(const T* __restrict__ U, const T* __restrict__ S, const T* __restrict__ Vt,
                const T* __restrict__ X, T* __restrict__ Y, int64_t m, int64_t n, int k, int64_t b,
                int64_t ldk, int64_t ldn, int kpad, int64_t m_chunk) {
    using P = Tile<T>;
    constexpr int BM = P::BM, BN = P::BN, BK = P::BK, TM = P::TM, TN = P::TN;
    constexpr int TX = BN / TN;            // threads along columns
    constexpr int TY = BM / TM;            // threads along rows
    constexpr int LDA = BM + 1, LDB = BN + 1;
    static_assert(TY * TX == kThreads, "thread tile");
    extern __shared__ __align__(16) unsigned char smem_raw[];
    T* Ws = reinterpret_cast<T*>(smem_raw);            // [kpad][BM]   scaled W, transposed
    T* As = Ws + (size_t)kpad * BM;                     // [BK][LDA]    X slab, transposed
    T* Bs = As + BK * LDA;                              // [BK][LDB]    Vt / U slab, transposed

    const int tid = threadIdx.x;
    const int tx = tid % TX, ty = tid / TX;
    const int64_t row0 = (int64_t)blockIdx.x * BM;
    const int64_t mbeg = (int64_t)blockIdx.y * m_chunk;
    const int64_t mend = (mbeg + m_chunk < m) ? mbeg + m_chunk : m;

    // ---------------- phase 1: W = X V, one BN-wide rank chunk at a time ----
    for (int kc = 0; kc < kpad; kc += BN) {
        T acc[TM][TN];
#pragma unroll
        for (int i = 0; i < TM; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) acc[i][j] = T(0);
        for (int64_t k0 = 0; k0 < n; k0 += BK) {
            // X slab: BM rows x BK cols -> As[c][r]
            for (int e = tid; e < BM * BK; e += kThreads) {
                const int r = e / BK, c = e % BK;
                const int64_t gr = row0 + r, gc = k0 + c;
                As[c * LDA + r] = (gr < b && gc < n) ? X[gr * ldn + gc] : T(0);
            }
            // Vt slab: BN rank rows x BK cols -> Bs[c][j]
            for (int e = tid; e < BN * BK; e += kThreads) {
                const int j = e / BK, c = e % BK;
                const int gj = kc + j;
                const int64_t gc = k0 + c;
                Bs[c * LDB + j] = (gj < k && gc < n) ? Vt[(int64_t)gj * ldn + gc] : T(0);
            }
            __syncthreads();
            T part[TM][TN];
#pragma unroll
            for (int i = 0; i < TM; ++i)
#pragma unroll
                for (int j = 0; j < TN; ++j) part[i][j] = P::kBlocked ? T(0) : acc[i][j];
#pragma unroll 4
            for (int c = 0; c < BK; ++c) {
                T a[TM], bb[TN];
#pragma unroll
                for (int i = 0; i < TM; ++i) a[i] = As[c * LDA + ty + i * TY];
#pragma unroll
                for (int j = 0; j < TN; ++j) bb[j] = Bs[c * LDB + tx + j * TX];
#pragma unroll
                for (int i = 0; i < TM; ++i)
#pragma unroll
                    for (int j = 0; j < TN; ++j) part[i][j] = fma(a[i], bb[j], part[i][j]);
            }
#pragma unroll
            for (int i = 0; i < TM; ++i)
#pragma unroll
                for (int j = 0; j < TN; ++j) acc[i][j] = P::kBlocked ? acc[i][j] + part[i][j] : part[i][j];
            __syncthreads();
        }
        // W <- W diag(s), kept transposed in shared memory
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int gj = kc + tx + j * TX;
            const T sj = (gj < k) ? S[gj] : T(0);
#pragma unroll
            for (int i = 0; i < TM; ++i) Ws[(size_t)gj * BM + ty + i * TY] = acc[i][j] * sj;
        }
    }
    __syncthreads();

    // ---------------- phase 2: Y[rows, m-tile] = W U[m-tile, :]^T -----------
    for (int64_t mt = mbeg; mt < mend; mt += BN) {
        T acc[TM][TN];
#pragma unroll
        for (int i = 0; i < TM; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) acc[i][j] = T(0);
        for (int k0 = 0; k0 < kpad; k0 += BK) {
            for (int e = tid; e < BN * BK; e += kThreads) {
                const int j = e / BK, c = e % BK;
                const int64_t gm = mt + j;
                const int gc = k0 + c;
                Bs[c * LDB + j] = (gm < mend && gc < k) ? U[gm * ldk + gc] : T(0);
            }
            __syncthreads();
#pragma unroll 4
            for (int c = 0; c < BK; ++c) {
                T a[TM], bb[TN];
#pragma unroll
                for (int i = 0; i < TM; ++i) a[i] = Ws[(size_t)(k0 + c) * BM + ty + i * TY];
#pragma unroll
                for (int j = 0; j < TN; ++j) bb[j] = Bs[c * LDB + tx + j * TX];
#pragma unroll
                for (int i = 0; i < TM; ++i)
#pragma unroll
                    for (int j = 0; j < TN; ++j) acc[i][j] = fma(a[i], bb[j], acc[i][j]);
            }
            __syncthreads();
        }
#pragma unroll
        for (int i = 0; i < TM; ++i) {
            const int64_t gr = row0 + ty + i * TY;
            if (gr >= b) continue;
#pragma unroll
            for (int j = 0; j < TN; ++j) {
                const int64_t gm = mt + tx + j * TX;
                if (gm < mend) Y[gr * m + gm] = acc[i][j];
            }
        }
    }
}

template <typename T>
lrc_status launch_apply_cc(const T* U, const T* S, const T* Vt, const T* X, T* Y, int64_t m,
                           int64_t n, int64_t k, int64_t b, cudaStream_t s, const char* name) {
    using P = Tile<T>;
    if (k > 4096) {
        set_error("%s: rank %lld above the supported 4096", name, (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    const int kpad = (int)((k + P::BN - 1) / P::BN * P::BN);
    const size_t smem = ((size_t)kpad * P::BM + P::BK * (P::BM + 1) + P::BK * (P::BN + 1)) * sizeof(T);
    if (smem > 227 * 1024) {
        set_error("%s: rank %lld needs %zu bytes of shared memory", name, (long long)k, smem);
        return LRC_ERR_UNSUPPORTED;
    }
    cudaError_t e = cudaFuncSetAttribute(apply_cc_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, name);
    const int64_t row_tiles = (b + P::BM - 1) / P::BM;
    const int64_t m_tiles = (m + P::BN - 1) / P::BN;
    // split the m range only when the batch alone cannot fill the GPU
    const int64_t target = 2 * (int64_t)sm_count();
    int64_t splits = 1;
    if (row_tiles < target) splits = (target + row_tiles - 1) / row_tiles;
    if (splits > m_tiles) splits = m_tiles;
    if (splits > 65535) splits = 65535;
    const int64_t tiles_per_split = (m_tiles + splits - 1) / splits;
    const int64_t m_chunk = tiles_per_split * P::BN;
    splits = (m + m_chunk - 1) / m_chunk;
    if (row_tiles > 0x7fffffff) {
        set_error("%s: batch too large", name);
        return LRC_ERR_UNSUPPORTED;
    }
    dim3 grid((unsigned)row_tiles, (unsigned)splits);
    apply_cc_kernel<T><<<grid, kThreads, smem, s>>>(U, S, Vt, X, Y, m, n, (int)k, b,
                                                    lrc_packed_ld(k), lrc_packed_ld(n), kpad, m_chunk);
    return after_launch(name);
}

}  // namespace

lrc_status launch_apply_f64(const double* U, const double* S, const double* Vt, const double* X,
                            double* Y, int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s) {
    return launch_apply_cc<double>(U, S, Vt, X, Y, m, n, k, b, s, "apply_cc_kernel<f64>");
}

lrc_status launch_apply_f32(const float* U, const float* S, const float* Vt, const float* X,
                            float* Y, int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s) {
    return launch_apply_cc<float>(U, S, Vt, X, Y, m, n, k, b, s, "apply_cc_kernel<f32>");
}

}  // namespace lrc
