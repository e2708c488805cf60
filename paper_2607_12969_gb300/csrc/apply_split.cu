// apply_split.cu -- low-rank apply for small batches on the CUDA cores,
// binary64 and binary32 (Sec. 4.4, Eq. gpu_matrix_apply:
// Y = [(X V) diag(s)] U^T).
//
// The fused kernels of apply_cc.cu give each CTA a tile of query rows; with
// few queries they leave most of the GPU idle.  Here the two products are
// separate launches, each spread over all SMs:
//   split_w1_kernel  grid (n-slice, row tile): partial W^T for BMS query rows
//                    (the batch rounded up to a power of two, at most 16)
//                    over one slice of n.  One thread per rank j keeps the
//                    BMS partial sums of its rank in registers; V^T slabs are
//                    staged in shared memory (rows padded by one element, so
//                    the threads' column reads do not conflict) and the X
//                    values are shared-memory broadcasts.  binary32 adds each
//                    slab's partial sums to the running sums separately
//                    (blocked accumulation).
//   split_w2_kernel  W = diag(s)-scaled sum of the slices' partials, added in
//                    slice order (deterministic).
//   split_y_kernel   grid (m-tile, row tile): one thread per column of Y keeps
//                    the BMS outputs of its column in registers; W of the row
//                    tile sits in shared memory (transposed, read as
//                    broadcasts) and U streams through padded slabs.
// W and the partials pass through the per-stream workspace.
#include "common.cuh"

namespace lrc {
namespace {

template <typename T>
struct SP;
template <>
struct SP<double> {
    static constexpr int BK = 16, BKJ = 16, YT = 128;
};
template <>
struct SP<float> {
    static constexpr int BK = 32, BKJ = 32, YT = 128;
};

constexpr int kMaxRanksPerThread = 2;     // phase 1: ranks j = tid, tid + blockDim

// The N consecutive values at p (16-byte aligned when they fill whole
// 16-byte words, which are then read as such).
template <typename T, int N>
__device__ __forceinline__ void load_row(const T* p, T (&v)[N]) {
    if constexpr (sizeof(T) == 4 && N % 4 == 0) {
#pragma unroll
        for (int i = 0; i < N / 4; ++i) {
            const float4 w = reinterpret_cast<const float4*>(p)[i];
            v[4 * i] = w.x;
            v[4 * i + 1] = w.y;
            v[4 * i + 2] = w.z;
            v[4 * i + 3] = w.w;
        }
    } else if constexpr (sizeof(T) == 8 && N % 2 == 0) {
#pragma unroll
        for (int i = 0; i < N / 2; ++i) {
            const double2 w = reinterpret_cast<const double2*>(p)[i];
            v[2 * i] = w.x;
            v[2 * i + 1] = w.y;
        }
    } else {
#pragma unroll
        for (int i = 0; i < N; ++i) v[i] = p[i];
    }
}

template <typename T, int BMS>
__global__ void __launch_bounds__(512)
split_w1_kernel(const T* __restrict__ X, const T* __restrict__ Vt, T* __restrict__ P, int64_t n, int64_t b, int k,
                int kp, int64_t ldn, int64_t slice) {
    constexpr int BK = SP<T>::BK, LDV = BK + 1;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    T* Vs = reinterpret_cast<T*>(smem_raw);          // [kp][LDV]   V^T slab
    T* Xs = Vs + (size_t)kp * LDV;                    // [BK][BMS]   X slab, transposed
    const int tid = threadIdx.x, nt = blockDim.x;
    const int64_t s = blockIdx.x;
    const int64_t row0 = (int64_t)blockIdx.y * BMS;
    const int64_t n0 = s * slice;
    const int64_t n1 = (n0 + slice < n) ? n0 + slice : n;
    T acc[kMaxRanksPerThread][BMS];
#pragma unroll
    for (int q = 0; q < kMaxRanksPerThread; ++q)
#pragma unroll
        for (int r = 0; r < BMS; ++r) acc[q][r] = T(0);
    for (int64_t c0 = n0; c0 < n1; c0 += BK) {
        for (int e = tid; e < kp * BK; e += nt) {
            const int j = e / BK, c = e - (e / BK) * BK;
            Vs[j * LDV + c] = (j < k && c0 + c < n1) ? Vt[(int64_t)j * ldn + c0 + c] : T(0);
        }
        for (int e = tid; e < BMS * BK; e += nt) {
            const int r = e / BK, c = e - (e / BK) * BK;
            Xs[c * BMS + r] = (row0 + r < b && c0 + c < n1) ? X[(row0 + r) * ldn + c0 + c] : T(0);
        }
        __syncthreads();
#pragma unroll
        for (int q = 0; q < kMaxRanksPerThread; ++q) {
            const int j = tid + q * nt;
            if (j >= kp) break;
            T part[BMS];
#pragma unroll
            for (int r = 0; r < BMS; ++r) part[r] = (sizeof(T) == 4) ? T(0) : acc[q][r];
#pragma unroll 4
            for (int c = 0; c < BK; ++c) {
                const T v = Vs[j * LDV + c];
                T xr[BMS];
                load_row(Xs + c * BMS, xr);          // the same address for every thread: a broadcast
#pragma unroll
                for (int r = 0; r < BMS; ++r) part[r] = fma(xr[r], v, part[r]);
            }
#pragma unroll
            for (int r = 0; r < BMS; ++r) acc[q][r] = (sizeof(T) == 4) ? acc[q][r] + part[r] : part[r];
        }
        __syncthreads();
    }
#pragma unroll
    for (int q = 0; q < kMaxRanksPerThread; ++q) {
        const int j = tid + q * nt;
        if (j >= kp) break;
#pragma unroll
        for (int r = 0; r < BMS; ++r)
            if (row0 + r < b) P[((size_t)s * b + row0 + r) * kp + j] = acc[q][r];
    }
}

// One thread per entry of W: the slices' partials in slice order.
template <typename T>
__global__ void __launch_bounds__(256)
split_w2_kernel(const T* __restrict__ P, const T* __restrict__ S, T* __restrict__ W, int64_t b, int k, int kp,
                int64_t slices) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= b * kp) return;
    const int j = (int)(e % kp);
    const size_t stride = (size_t)b * kp;
    T w = P[e];
#pragma unroll 8
    for (int64_t s = 1; s < slices; ++s) w += P[(size_t)s * stride + e];
    W[e] = (j < k) ? w * S[j] : T(0);
}

// One warp per entry of W, for many slices: lane l adds slices l, l + 32, ...
// in order, then a fixed butterfly combines the lanes (the same order on
// every run).
template <typename T>
__global__ void __launch_bounds__(256)
split_w2_warp_kernel(const T* __restrict__ P, const T* __restrict__ S, T* __restrict__ W, int64_t b, int k, int kp,
                     int64_t slices) {
    const int lane = threadIdx.x & 31;
    const int64_t e = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (e >= b * kp) return;
    const int j = (int)(e % kp);
    const size_t stride = (size_t)b * kp;
    T w = T(0);
    for (int64_t s = lane; s < slices; s += 32) w += P[(size_t)s * stride + e];
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) w += __shfl_xor_sync(0xffffffffu, w, off);
    if (lane == 0) W[e] = (j < k) ? w * S[j] : T(0);
}

template <typename T, int BMS>
__global__ void __launch_bounds__(SP<T>::YT)
split_y_kernel(const T* __restrict__ W, const T* __restrict__ U, T* __restrict__ Y, int64_t m, int64_t b, int k,
               int kp, int64_t ldk) {
    constexpr int BKJ = SP<T>::BKJ, LDU = BKJ + 1, kYThreads = SP<T>::YT;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    T* Ws = reinterpret_cast<T*>(smem_raw);          // [kp][BMS]   W rows of the tile, transposed
    T* Us = Ws + (size_t)(kp * BMS + 1) / 2 * 2;      // [kYThreads][LDU]   U slab (16-byte aligned)
    const int tid = threadIdx.x;
    const int64_t i0 = (int64_t)blockIdx.x * kYThreads;
    const int64_t row0 = (int64_t)blockIdx.y * BMS;
    for (int e = tid; e < BMS * kp; e += kYThreads) {
        const int r = e / kp, j = e - (e / kp) * kp;
        Ws[j * BMS + r] = (row0 + r < b) ? W[(row0 + r) * kp + j] : T(0);
    }
    T acc[BMS];
#pragma unroll
    for (int r = 0; r < BMS; ++r) acc[r] = T(0);
    for (int j0 = 0; j0 < kp; j0 += BKJ) {
        __syncthreads();
        for (int e = tid; e < kYThreads * BKJ; e += kYThreads) {
            const int i = e / BKJ, jj = e - (e / BKJ) * BKJ;
            Us[i * LDU + jj] = (i0 + i < m && j0 + jj < k) ? U[(i0 + i) * ldk + j0 + jj] : T(0);
        }
        __syncthreads();
        const int jn = (kp - j0 < BKJ) ? kp - j0 : BKJ;
#pragma unroll 4
        for (int jj = 0; jj < jn; ++jj) {
            const T u = Us[tid * LDU + jj];
            T wr[BMS];
            load_row(Ws + (j0 + jj) * BMS, wr);      // broadcast
#pragma unroll
            for (int r = 0; r < BMS; ++r) acc[r] = fma(wr[r], u, acc[r]);
        }
    }
    if (i0 + tid < m) {
#pragma unroll
        for (int r = 0; r < BMS; ++r)
            if (row0 + r < b) Y[(row0 + r) * m + i0 + tid] = acc[r];
    }
}

template <typename T, int BMS>
lrc_status launch_split_b(const T* U, const T* S, const T* Vt, const T* X, T* Y, int64_t m, int64_t n, int64_t k,
                          int64_t b, cudaStream_t s, const char* name) {
    constexpr int BK = SP<T>::BK, BKJ = SP<T>::BKJ, kYThreads = SP<T>::YT;
    const int kp = (int)((k + 15) / 16 * 16);
    const int threads1 = ((kp + kMaxRanksPerThread - 1) / kMaxRanksPerThread + 31) / 32 * 32;
    if (threads1 > 512) {
        set_error("%s: rank %lld above the small-batch path's 1024", name, (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    const size_t smem1 = ((size_t)kp * (BK + 1) + (size_t)BK * BMS) * sizeof(T);
    const size_t smem3 = ((size_t)(kp * BMS + 1) / 2 * 2 + (size_t)kYThreads * (BKJ + 1)) * sizeof(T);
    if (smem1 > 227 * 1024 || smem3 > 227 * 1024) {
        set_error("%s: rank %lld needs too much shared memory", name, (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    const int sms = sm_count();
    const int64_t btiles = (b + BMS - 1) / BMS;
    // n-slices: about four CTAs per SM in phase 1, slices a whole number of slabs
    int64_t slices = (4 * (int64_t)sms + btiles - 1) / btiles;
    const int64_t max_slices = (n + BK - 1) / BK;
    if (slices > max_slices) slices = max_slices;
    if (slices < 1) slices = 1;
    int64_t slice = (n + slices - 1) / slices;
    slice = (slice + BK - 1) / BK * BK;
    slices = (n + slice - 1) / slice;
    if (slices > 65535 || btiles > 65535) {
        set_error("%s: batch too large for the small-batch path", name);
        return LRC_ERR_UNSUPPORTED;
    }
    const size_t p_bytes = ((size_t)slices * b * kp * sizeof(T) + 255) / 256 * 256;
    const size_t w_bytes = (size_t)b * kp * sizeof(T);
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, p_bytes + w_bytes, &ws);
    if (st != LRC_OK) return st;
    T* P = static_cast<T*>(ws);
    T* W = reinterpret_cast<T*>(static_cast<unsigned char*>(ws) + p_bytes);

    cudaError_t e =
        cudaFuncSetAttribute(split_w1_kernel<T, BMS>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
    if (e != cudaSuccess) return cuda_fail(e, name);
    split_w1_kernel<T, BMS><<<dim3((unsigned)slices, (unsigned)btiles), threads1, smem1, s>>>(
        X, Vt, P, n, b, (int)k, kp, lrc_packed_ld(n), slice);
    if ((st = after_launch("split_w1_kernel")) != LRC_OK) return st;
    const int64_t nw = b * kp;
    if (slices >= 16) {
        split_w2_warp_kernel<T><<<(unsigned)((nw * 32 + 255) / 256), 256, 0, s>>>(P, S, W, b, (int)k, kp, slices);
        if ((st = after_launch("split_w2_warp_kernel")) != LRC_OK) return st;
    } else {
        split_w2_kernel<T><<<(unsigned)((nw + 255) / 256), 256, 0, s>>>(P, S, W, b, (int)k, kp, slices);
        if ((st = after_launch("split_w2_kernel")) != LRC_OK) return st;
    }
    e = cudaFuncSetAttribute(split_y_kernel<T, BMS>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem3);
    if (e != cudaSuccess) return cuda_fail(e, name);
    const int64_t mtiles = (m + kYThreads - 1) / kYThreads;
    if (mtiles > 0x7fffffff) {
        set_error("%s: m too large", name);
        return LRC_ERR_UNSUPPORTED;
    }
    split_y_kernel<T, BMS><<<dim3((unsigned)mtiles, (unsigned)btiles), kYThreads, smem3, s>>>(W, U, Y, m, b, (int)k,
                                                                                            kp, lrc_packed_ld(k));
    return after_launch("split_y_kernel");
}

// Row-tile height: the batch rounded up to a power of two, at most 16 (no
// arithmetic on absent rows for tiny batches).
template <typename T>
lrc_status launch_split(const T* U, const T* S, const T* Vt, const T* X, T* Y, int64_t m, int64_t n, int64_t k,
                        int64_t b, cudaStream_t s, const char* name) {
    if (b <= 1) return launch_split_b<T, 1>(U, S, Vt, X, Y, m, n, k, b, s, name);
    if (b <= 2) return launch_split_b<T, 2>(U, S, Vt, X, Y, m, n, k, b, s, name);
    if (b <= 4) return launch_split_b<T, 4>(U, S, Vt, X, Y, m, n, k, b, s, name);
    if (b <= 8) return launch_split_b<T, 8>(U, S, Vt, X, Y, m, n, k, b, s, name);
    return launch_split_b<T, 16>(U, S, Vt, X, Y, m, n, k, b, s, name);
}

}  // namespace

lrc_status launch_apply_split_f64(const double* U, const double* S, const double* Vt, const double* X, double* Y,
                                  int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s) {
    return launch_split<double>(U, S, Vt, X, Y, m, n, k, b, s, "small-batch apply (binary64)");
}

lrc_status launch_apply_split_f32(const float* U, const float* S, const float* Vt, const float* X, float* Y,
                                  int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s) {
    return launch_split<float>(U, S, Vt, X, Y, m, n, k, b, s, "small-batch apply (binary32)");
}

}  // namespace lrc
