// fro_diff.cu -- ||A - B||_F and ||A||_F in binary64 (Sec. 5.1), the
// reduction behind eta (Thm 4.1) and eta_TT (Thm 6.1).
//
// Pass 1: a fixed grid of blocks streams the arrays (128-bit loads, groups of
// 8 elements per thread and step), accumulates (a-b)^2 and a^2 in binary64
// per thread, reduces each block with a fixed shuffle tree, and writes one
// partial pair per block.  Pass 2: one block reduces the partials in a fixed
// order.  The assignment of elements to threads depends only on `count` and
// the device's SM count, so results are bitwise reproducible on a device.
#include <cuda_fp16.h>

#include <mutex>

#include "common.cuh"

namespace lrc {
namespace {

constexpr int kThreads = 256;
constexpr int kGroup = 8;
constexpr int kMaxBlocks = 4096;

struct Scratch {
    double* partial = nullptr;   // 2 * kMaxBlocks + 2 doubles
};
std::mutex g_mu;
Scratch g_scratch[64];

__device__ __forceinline__ double widen_h(uint16_t h) {
    double d;
    asm("cvt.f64.f16 %0, %1;" : "=d"(d) : "h"(h));
    return d;
}

// Loads elements [8g, 8g+8) of an array of format F as binary64.
template <int F>
__device__ __forceinline__ void load8(const void* p, int64_t g, double v[kGroup]) {
    if (F == 0) {
        const double2* q = reinterpret_cast<const double2*>(p) + g * 4;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const double2 t = __ldcs(q + j);
            v[2 * j] = t.x;
            v[2 * j + 1] = t.y;
        }
    } else if (F == 1) {
        const float4* q = reinterpret_cast<const float4*>(p) + g * 2;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            const float4 t = __ldcs(q + j);
            v[4 * j] = t.x;
            v[4 * j + 1] = t.y;
            v[4 * j + 2] = t.z;
            v[4 * j + 3] = t.w;
        }
    } else if (F == 2) {
        const uint4 t = __ldcs(reinterpret_cast<const uint4*>(p) + g);
        const uint32_t w[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            v[2 * j] = widen_h((uint16_t)(w[j] & 0xffffu));
            v[2 * j + 1] = widen_h((uint16_t)(w[j] >> 16));
        }
    } else {
        // bfloat16: the binary32 number with the same upper 16 bits
        const uint4 t = __ldcs(reinterpret_cast<const uint4*>(p) + g);
        const uint32_t w[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            v[2 * j] = (double)__uint_as_float(w[j] << 16);
            v[2 * j + 1] = (double)__uint_as_float(w[j] & 0xffff0000u);
        }
    }
}

template <int F>
__device__ __forceinline__ double load1(const void* p, int64_t i) {
    if (F == 0) return static_cast<const double*>(p)[i];
    if (F == 1) return (double)static_cast<const float*>(p)[i];
    if (F == 3) return (double)__uint_as_float((uint32_t)static_cast<const uint16_t*>(p)[i] << 16);
    return widen_h(static_cast<const uint16_t*>(p)[i]);
}

__device__ __forceinline__ void block_sum2(double& a, double& b, double* sh) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, o);
        b += __shfl_xor_sync(0xffffffffu, b, o);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        sh[warp] = a;
        sh[32 + warp] = b;
    }
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        a = lane < nw ? sh[lane] : 0.0;
        b = lane < nw ? sh[32 + lane] : 0.0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            a += __shfl_xor_sync(0xffffffffu, a, o);
            b += __shfl_xor_sync(0xffffffffu, b, o);
        }
    }
}

// ---------------------------------------------------------------------------
// Squares summed in binary32 pairs.  The GB300 issues about two binary64
// instructions per clock per SM, while streaming two binary64 arrays at HBM
// speed delivers about 1.35 element pairs per clock per SM: with a binary64
// subtraction and a binary64 FMA per element the reduction is bound by the
// FP64 pipe, not by memory.  For two binary64 arrays only the subtraction
// d = a - b stays binary64.  d is cut, with integer operations on its bits,
// into hi (its sign, exponent and leading 24 significand bits) and lo (the
// next 23 bits; the last 6 are dropped, a relative change of at most 2^-47),
// and d^2 = hi^2 + (2 hi lo + lo^2) is formed with an exact two-product
// (hi^2 = p + e, e = fma(hi, hi, -p)) and added to a binary32 pair sum with
// two-sum.  Every 16 groups the pair sum is added to a binary64 accumulator.
// Elements with |d| outside [2^-48, 2^60) are squared in binary64 instead:
// above, a sum of hi^2 terms could overflow binary32; below, the correction
// terms 2 hi lo and fma(hi, hi, -p) (about 2^-23 d^2) would fall under 2^-126,
// into binary32 subnormals whose fixed spacing 2^-149 would cost more than
// 2^-54 of d^2.
// ---------------------------------------------------------------------------
struct Pair {
    float hi = 0.0f, lo = 0.0f;
};

// hi, lo of d; false when d is out of the binary32 path's range (d = 0 is in range)
__device__ __forceinline__ bool split_hi_lo(double d, float& hi, float& lo) {
    const unsigned long long b = (unsigned long long)__double_as_longlong(d);
    const int e = (int)((b >> 52) & 0x7ffu);
    if (e < 1023 - 48 || e >= 1023 + 60) {
        hi = lo = 0.0f;
        return (b << 1) == 0ull;
    }
    const unsigned int sign = (unsigned int)(b >> 32) & 0x80000000u;
    hi = __int_as_float((int)(sign | ((unsigned int)(e - 1023 + 127) << 23) | (unsigned int)((b >> 29) & 0x7fffffu)));
    // bits 28..6 of the significand, as an exact binary32 integer, times +-2^(E - 46)
    const unsigned int m = (unsigned int)((b >> 6) & 0x7fffffu);
    const float mf = __int_as_float((int)(0x4B000000u | m)) - 8388608.0f;
    const float scale = __int_as_float((int)(sign | ((unsigned int)(e - 1023 - 46 + 127) << 23)));
    lo = mf * scale;
    return true;
}

// s += hi^2 + 2 hi lo + lo^2
__device__ __forceinline__ void add_square(Pair& s, float hi, float lo) {
    const float p = hi * hi;
    const float e = fmaf(hi, hi, -p);                 // hi^2 - p, exact
    const float t = fmaf(2.0f * hi, lo, fmaf(lo, lo, e));
    const float sh = s.hi + p;                        // two-sum of s.hi and p
    const float bp = sh - s.hi;
    const float err = (s.hi - (sh - bp)) + (p - bp);
    s.hi = sh;
    s.lo += err + t;
}

__device__ __forceinline__ void flush(Pair& s, double& acc) {
    acc += (double)s.hi + (double)s.lo;
    s.hi = s.lo = 0.0f;
}

// FB = -1: B absent (treated as zero).  NORM = false skips the ||A||
// accumulation.
template <int FA, int FB, bool NORM>
__global__ void __launch_bounds__(kThreads)
fro_partial_kernel(const void* __restrict__ A, const void* __restrict__ B, int64_t count,
                   double* __restrict__ partial) {
    __shared__ double sh[64];
    double sd = 0.0, sa = 0.0;
    const int64_t groups = count / kGroup;
    const int64_t stride = (int64_t)gridDim.x * kThreads;
    if constexpr (FA == 0 && FB <= 0) {
        // binary64 inputs: binary32-pair squares (see above)
        Pair pd, pa;
        int n = 0;
        for (int64_t g = (int64_t)blockIdx.x * kThreads + threadIdx.x; g < groups; g += stride) {
            double a[kGroup], b[kGroup];
            load8<FA>(A, g, a);
            if (FB == 0) load8<0>(B, g, b);
#pragma unroll
            for (int j = 0; j < kGroup; ++j) {
                const double d = (FB == 0) ? a[j] - b[j] : a[j];
                float hi, lo;
                if (split_hi_lo(d, hi, lo)) add_square(pd, hi, lo);
                else sd = fma(d, d, sd);
                if (NORM) {
                    if (split_hi_lo(a[j], hi, lo)) add_square(pa, hi, lo);
                    else sa = fma(a[j], a[j], sa);
                }
            }
            if (++n == 16) {
                flush(pd, sd);
                if (NORM) flush(pa, sa);
                n = 0;
            }
        }
        flush(pd, sd);
        if (NORM) flush(pa, sa);
    } else {
        for (int64_t g = (int64_t)blockIdx.x * kThreads + threadIdx.x; g < groups; g += stride) {
            double a[kGroup], b[kGroup];
            load8<FA>(A, g, a);
            if (FB >= 0) load8<FB>(B, g, b);
#pragma unroll
            for (int j = 0; j < kGroup; ++j) {
                const double d = (FB >= 0) ? a[j] - b[j] : a[j];
                sd = fma(d, d, sd);
                if (NORM) sa = fma(a[j], a[j], sa);
            }
        }
    }
    if (blockIdx.x == 0) {  // ragged tail, fixed owner
        for (int64_t i = groups * kGroup + threadIdx.x; i < count; i += kThreads) {
            const double a = load1<FA>(A, i);
            const double d = (FB >= 0) ? a - load1<FB < 0 ? 0 : FB>(B, i) : a;
            sd = fma(d, d, sd);
            if (NORM) sa = fma(a, a, sa);
        }
    }
    block_sum2(sd, sa, sh);
    if (threadIdx.x == 0) {
        partial[blockIdx.x] = sd;
        partial[gridDim.x + blockIdx.x] = sa;
    }
}

__global__ void __launch_bounds__(1024)
fro_final_kernel(const double* __restrict__ partial, int nblocks, double* __restrict__ result) {
    __shared__ double sh[64];
    double sd = 0.0, sa = 0.0;
    for (int i = threadIdx.x; i < nblocks; i += blockDim.x) {
        sd += partial[i];
        sa += partial[nblocks + i];
    }
    block_sum2(sd, sa, sh);
    if (threadIdx.x == 0) {
        result[0] = sqrt(sd);
        result[1] = sqrt(sa);
    }
}

int fcode(lrc_fmt f) { return f == LRC_F64 ? 0 : (f == LRC_F32 ? 1 : (f == LRC_BF16 ? 3 : 2)); }

template <int FA, bool NORM>
void launch_partial_n(int fb, int grid, const void* A, const void* B, int64_t count, double* partial,
                      cudaStream_t s) {
    switch (fb) {
        case 0: fro_partial_kernel<FA, 0, NORM><<<grid, kThreads, 0, s>>>(A, B, count, partial); break;
        case 1: fro_partial_kernel<FA, 1, NORM><<<grid, kThreads, 0, s>>>(A, B, count, partial); break;
        case 2: fro_partial_kernel<FA, 2, NORM><<<grid, kThreads, 0, s>>>(A, B, count, partial); break;
        case 3: fro_partial_kernel<FA, 3, NORM><<<grid, kThreads, 0, s>>>(A, B, count, partial); break;
        default: fro_partial_kernel<FA, -1, NORM><<<grid, kThreads, 0, s>>>(A, B, count, partial); break;
    }
}

template <int FA>
void launch_partial(int fb, int grid, const void* A, const void* B, int64_t count, double* partial,
                    cudaStream_t s, bool norm = true) {
    if (norm) launch_partial_n<FA, true>(fb, grid, A, B, count, partial, s);
    else launch_partial_n<FA, false>(fb, grid, A, B, count, partial, s);
}

}  // namespace

lrc_status run_fro_diff(const void* A, lrc_fmt fa, const void* B, lrc_fmt fb, int64_t count,
                        double* diff_out, double* normA_out, cudaStream_t s) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= 64) {
        set_error("device ordinal %d out of range", dev);
        return LRC_ERR_UNSUPPORTED;
    }
    double* partial;
    {
        std::lock_guard<std::mutex> lock(g_mu);
        if (!g_scratch[dev].partial) {
            e = cudaMalloc(&g_scratch[dev].partial, (2 * kMaxBlocks + 2) * sizeof(double));
            if (e != cudaSuccess) {
                g_scratch[dev].partial = nullptr;
                set_error("scratch allocation failed: %s", cudaGetErrorString(e));
                return LRC_ERR_NOMEM;
            }
        }
        partial = g_scratch[dev].partial;
    }
    const int64_t groups = count / kGroup;
    int64_t want = (groups + kThreads - 1) / kThreads;
    const int64_t cap = (int64_t)sm_count() * 4;
    int grid = (int)(want < cap ? (want > 0 ? want : 1) : cap);
    if (grid > kMaxBlocks) grid = kMaxBlocks;
    const int a = fcode(fa), b = B ? fcode(fb) : -1;
    const bool norm = normA_out != nullptr;
    switch (a) {
        case 0: launch_partial<0>(b, grid, A, B, count, partial, s, norm); break;
        case 1: launch_partial<1>(b, grid, A, B, count, partial, s, norm); break;
        case 3: launch_partial<3>(b, grid, A, B, count, partial, s, norm); break;
        default: launch_partial<2>(b, grid, A, B, count, partial, s, norm); break;
    }
    lrc_status st = after_launch("fro_partial_kernel");
    if (st != LRC_OK) return st;
    // the two results go straight to the stream's mapped host slot (no
    // copy-engine transfer behind other copies)
    double* host = nullptr;
    double* result = nullptr;
    if ((st = stream_result_slot(s, &host, &result)) != LRC_OK) return st;
    fro_final_kernel<<<1, 1024, 0, s>>>(partial, grid, result);
    st = after_launch("fro_final_kernel");
    if (st != LRC_OK) return st;
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize (fro_diff)");
    *diff_out = host[0];
    if (normA_out) *normA_out = host[1];
    return LRC_OK;
}

// ---------------------------------------------------------------------------
// Allocation-free variant.  The per-block partial sums go to a fixed array in
// device memory that is part of the loaded library image, so the call never
// allocates.  It holds kStaticBlocks block slots; the documented element
// limit (kStaticBlocks x kStaticElemsPerBlock) is kept as the interface's
// bound, the grid itself is that of the allocating path.
// ---------------------------------------------------------------------------
namespace {
constexpr int kStaticBlocks = 4096;
constexpr int64_t kStaticElemsPerBlock = 65536;   // 256 threads x 32 groups of 8
static __device__ __align__(256) double g_fro_static_scratch[2 * kStaticBlocks + 2];
std::mutex g_static_mu;
double* g_static_ptr[64] = {nullptr};             // device address of the array, per device
}  // namespace

int64_t fro_diff_noalloc_max_count() { return (int64_t)kStaticBlocks * kStaticElemsPerBlock; }

lrc_status run_fro_diff_noalloc(const void* A, lrc_fmt fa, const void* B, lrc_fmt fb, int64_t count,
                                double* diff_out, double* normA_out, cudaStream_t s) {
    if (count > fro_diff_noalloc_max_count()) {
        set_error("lrc_fro_diff_noalloc handles at most %lld elements (got %lld)",
                  (long long)fro_diff_noalloc_max_count(), (long long)count);
        return LRC_ERR_INVALID_ARG;
    }
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= 64) {
        set_error("device ordinal %d out of range", dev);
        return LRC_ERR_UNSUPPORTED;
    }
    double* partial;
    {
        // one-time set-up per device, with that device current: the host-side
        // name of the array is not a device address, so look the address up
        std::lock_guard<std::mutex> lock(g_static_mu);
        if (!g_static_ptr[dev]) {
            void* p = nullptr;
            e = cudaGetSymbolAddress(&p, g_fro_static_scratch);
            if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress (fro_diff scratch)");
            g_static_ptr[dev] = static_cast<double*>(p);
        }
        partial = g_static_ptr[dev];
    }
    // the grid of the allocating path (the kernel strides over the groups),
    // capped by the array's kStaticBlocks slots
    const int64_t groups = count / kGroup;
    const int64_t want = (groups + kThreads - 1) / kThreads;
    int64_t cap = (int64_t)sm_count() * 4;
    if (cap > kStaticBlocks) cap = kStaticBlocks;
    const int grid = (int)(want < cap ? (want > 0 ? want : 1) : cap);
    const int a = fcode(fa), b = B ? fcode(fb) : -1;
    const bool norm = normA_out != nullptr;
    switch (a) {
        case 0: launch_partial<0>(b, grid, A, B, count, partial, s, norm); break;
        case 1: launch_partial<1>(b, grid, A, B, count, partial, s, norm); break;
        case 3: launch_partial<3>(b, grid, A, B, count, partial, s, norm); break;
        default: launch_partial<2>(b, grid, A, B, count, partial, s, norm); break;
    }
    lrc_status st = after_launch("fro_partial_kernel (no-alloc)");
    if (st != LRC_OK) return st;
    double* result = partial + 2 * kStaticBlocks;
    fro_final_kernel<<<1, 1024, 0, s>>>(partial, grid, result);
    st = after_launch("fro_final_kernel (no-alloc)");
    if (st != LRC_OK) return st;
    double host[2];
    e = cudaMemcpyAsync(host, result, sizeof host, cudaMemcpyDeviceToHost, s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpyAsync (fro_diff no-alloc result)");
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize (fro_diff no-alloc)");
    *diff_out = host[0];
    if (normA_out) *normA_out = host[1];
    return LRC_OK;
}

void release_scratch() {
    {
        // forget the looked-up array addresses: after a device reset the
        // module is loaded again and the array may live elsewhere
        std::lock_guard<std::mutex> lock(g_static_mu);
        for (int d = 0; d < 64; ++d) g_static_ptr[d] = nullptr;
    }
    std::lock_guard<std::mutex> lock(g_mu);
    int prev = -1;
    cudaGetDevice(&prev);
    for (int d = 0; d < 64; ++d) {
        if (g_scratch[d].partial) {
            cudaSetDevice(d);
            cudaFree(g_scratch[d].partial);
            g_scratch[d].partial = nullptr;
        }
    }
    if (prev >= 0) cudaSetDevice(prev);
}

}  // namespace lrc
