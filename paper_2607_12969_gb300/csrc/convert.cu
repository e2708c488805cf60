// convert.cu -- factor rounding / packing (binary64 -> binary32 / binary16 /
// bfloat16) and exact widening back to binary64.
//
// Rounding is the hardware conversion cvt.rn.{f32,f16,bf16}.f64: IEEE 754
// round-to-nearest-even directly from binary64 (no intermediate format),
// subnormals kept (no .ftz), overflow to infinity.  The kernels are
// HBM-bound streams: each thread converts a group of 8 consecutive elements
// of one row with 128-bit loads and stores where the row pitch allows it.
#include <cuda_fp16.h>

#include "common.cuh"

namespace lrc {
namespace {

constexpr int kThreads = 256;
constexpr int kGroup = 8;

__device__ __forceinline__ uint16_t cvt_f16(double x) {
    uint16_t h;
    asm("cvt.rn.f16.f64 %0, %1;" : "=h"(h) : "d"(x));
    return h;
}
__device__ __forceinline__ uint16_t cvt_bf16(double x) {
    uint16_t h;
    asm("cvt.rn.bf16.f64 %0, %1;" : "=h"(h) : "d"(x));
    return h;
}
__device__ __forceinline__ float cvt_f32(double x) {
    float f;
    asm("cvt.rn.f32.f64 %0, %1;" : "=f"(f) : "d"(x));
    return f;
}
__device__ __forceinline__ double widen_f16(uint16_t h) {
    double d;
    asm("cvt.f64.f16 %0, %1;" : "=d"(d) : "h"(h));
    return d;
}

// FMT: 0 = binary64 copy, 1 = binary32, 2 = binary16, 3 = bfloat16
template <int FMT>
__global__ void __launch_bounds__(kThreads)
round_pack_kernel(const double* __restrict__ src, int64_t cols, int64_t ld_src,
                  void* __restrict__ dst, int64_t ld_dst, int64_t groups_per_row,
                  int64_t total_groups, bool vec_src, bool vec_dst) {
    const int64_t stride = (int64_t)gridDim.x * kThreads;
    for (int64_t g = (int64_t)blockIdx.x * kThreads + threadIdx.x; g < total_groups; g += stride) {
        const int64_t r = g / groups_per_row;
        const int64_t c0 = (g - r * groups_per_row) * kGroup;
        const double* srow = src + r * ld_src;
        double v[kGroup];
        if (vec_src && c0 + kGroup <= cols) {
#pragma unroll
            for (int j = 0; j < kGroup; j += 2) {
                const double2 p = __ldcs(reinterpret_cast<const double2*>(srow + c0 + j));
                v[j] = p.x;
                v[j + 1] = p.y;
            }
        } else {
#pragma unroll
            for (int j = 0; j < kGroup; ++j) v[j] = (c0 + j < cols) ? __ldcs(srow + c0 + j) : 0.0;
        }
        const bool full = vec_dst && (c0 + kGroup <= ld_dst);
        if (FMT == 2 || FMT == 3) {
            uint16_t* drow = static_cast<uint16_t*>(dst) + r * ld_dst;
            uint16_t h[kGroup];
#pragma unroll
            for (int j = 0; j < kGroup; ++j) h[j] = FMT == 2 ? cvt_f16(v[j]) : cvt_bf16(v[j]);
            if (full) {
                uint4 q;
                q.x = (uint32_t)h[0] | ((uint32_t)h[1] << 16);
                q.y = (uint32_t)h[2] | ((uint32_t)h[3] << 16);
                q.z = (uint32_t)h[4] | ((uint32_t)h[5] << 16);
                q.w = (uint32_t)h[6] | ((uint32_t)h[7] << 16);
                __stcs(reinterpret_cast<uint4*>(drow + c0), q);
            } else {
                for (int j = 0; j < kGroup; ++j)
                    if (c0 + j < ld_dst) drow[c0 + j] = h[j];
            }
        } else if (FMT == 1) {
            float* drow = static_cast<float*>(dst) + r * ld_dst;
            float f[kGroup];
#pragma unroll
            for (int j = 0; j < kGroup; ++j) f[j] = cvt_f32(v[j]);
            if (full) {
                __stcs(reinterpret_cast<float4*>(drow + c0), make_float4(f[0], f[1], f[2], f[3]));
                __stcs(reinterpret_cast<float4*>(drow + c0 + 4), make_float4(f[4], f[5], f[6], f[7]));
            } else {
                for (int j = 0; j < kGroup; ++j)
                    if (c0 + j < ld_dst) drow[c0 + j] = f[j];
            }
        } else {
            double* drow = static_cast<double*>(dst) + r * ld_dst;
            if (full) {
#pragma unroll
                for (int j = 0; j < kGroup; j += 2)
                    __stcs(reinterpret_cast<double2*>(drow + c0 + j), make_double2(v[j], v[j + 1]));
            } else {
                for (int j = 0; j < kGroup; ++j)
                    if (c0 + j < ld_dst) drow[c0 + j] = v[j];
            }
        }
    }
}

// Exact binary32 -> binary64 from the bit fields: normal numbers and zeros
// take integer operations only (the exponent rebias and significand shift of
// the IEEE 754 formats); subnormals, infinities and NaNs take the conversion
// instruction.
__device__ __forceinline__ double widen_f32(float f) {
    const uint32_t u = __float_as_uint(f);
    const uint32_t e = (u >> 23) & 0xffu;
    const unsigned long long sign = (unsigned long long)(u & 0x80000000u) << 32;
    if (e != 0u && e != 0xffu)
        return __longlong_as_double((long long)(sign | ((unsigned long long)(e + 896u) << 52) |
                                                ((unsigned long long)(u & 0x7fffffu) << 29)));
    if ((u & 0x7fffffffu) == 0u) return __longlong_as_double((long long)sign);
    return (double)f;
}

// FMT as above; dst is binary64.  Each thread widens a group of 8 elements of
// one row: one 16-byte (binary16) or two (binary32) loads, four 16-byte stores
// when the row pitches allow it.
template <int FMT>
__global__ void __launch_bounds__(kThreads)
widen_kernel(const void* __restrict__ src, int64_t cols, int64_t ld_src, double* __restrict__ dst,
             int64_t ld_dst, int64_t groups_per_row, int64_t total_groups, bool vec_src, bool vec_dst) {
    const int64_t stride = (int64_t)gridDim.x * kThreads;
    for (int64_t g = (int64_t)blockIdx.x * kThreads + threadIdx.x; g < total_groups; g += stride) {
        const int64_t r = g / groups_per_row;
        const int64_t c0 = (g - r * groups_per_row) * kGroup;
        double v[kGroup];
        if (vec_src && c0 + kGroup <= cols) {
            if (FMT == 2 || FMT == 3) {
                const uint4 q = __ldcs(reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(src) + r * ld_src + c0));
                const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    // a bfloat16 value is the binary32 number with the same upper 16 bits
                    const float2 f = FMT == 2 ? __half22float2(*reinterpret_cast<const __half2*>(&w[j]))
                                              : make_float2(__uint_as_float(w[j] << 16), __uint_as_float(w[j] & 0xffff0000u));
                    v[2 * j] = widen_f32(f.x);
                    v[2 * j + 1] = widen_f32(f.y);
                }
            } else if (FMT == 1) {
                const float4* p = reinterpret_cast<const float4*>(static_cast<const float*>(src) + r * ld_src + c0);
                const float4 a = __ldcs(p), b = __ldcs(p + 1);
                v[0] = widen_f32(a.x); v[1] = widen_f32(a.y); v[2] = widen_f32(a.z); v[3] = widen_f32(a.w);
                v[4] = widen_f32(b.x); v[5] = widen_f32(b.y); v[6] = widen_f32(b.z); v[7] = widen_f32(b.w);
            } else {
                const double2* p = reinterpret_cast<const double2*>(static_cast<const double*>(src) + r * ld_src + c0);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const double2 t = __ldcs(p + j);
                    v[2 * j] = t.x;
                    v[2 * j + 1] = t.y;
                }
            }
        } else {
#pragma unroll
            for (int j = 0; j < kGroup; ++j) {
                const int64_t c = c0 + j;
                double x = 0.0;
                if (c < cols) {
                    if (FMT == 2) x = widen_f16(static_cast<const uint16_t*>(src)[r * ld_src + c]);
                    else if (FMT == 3)
                        x = widen_f32(__uint_as_float((uint32_t)static_cast<const uint16_t*>(src)[r * ld_src + c] << 16));
                    else if (FMT == 1) x = (double)static_cast<const float*>(src)[r * ld_src + c];
                    else x = static_cast<const double*>(src)[r * ld_src + c];
                }
                v[j] = x;
            }
        }
        double* drow = dst + r * ld_dst;
        if (vec_dst && c0 + kGroup <= ld_dst) {
#pragma unroll
            for (int j = 0; j < kGroup; j += 2)
                __stcs(reinterpret_cast<double2*>(drow + c0 + j), make_double2(v[j], v[j + 1]));
        } else {
            for (int j = 0; j < kGroup; ++j)
                if (c0 + j < ld_dst) drow[c0 + j] = v[j];
        }
    }
}

int grid_for(int64_t groups) {
    const int64_t want = (groups + kThreads - 1) / kThreads;
    const int64_t cap = (int64_t)sm_count() * 8;
    return (int)(want < cap ? (want > 0 ? want : 1) : cap);
}

}  // namespace

lrc_status launch_round(const double* src, int64_t rows, int64_t cols, int64_t ld_src, void* dst,
                        int64_t ld_dst, lrc_fmt fmt, cudaStream_t s) {
    const int64_t gpr = (ld_dst + kGroup - 1) / kGroup;
    const int64_t total = rows * gpr;
    const bool vec_src = (ld_src % 2) == 0;
    const int grid = grid_for(total);
    switch (fmt) {
        case LRC_F64:
            round_pack_kernel<0><<<grid, kThreads, 0, s>>>(src, cols, ld_src, dst, ld_dst, gpr, total,
                                                            vec_src, (ld_dst % 2) == 0);
            break;
        case LRC_F32:
            round_pack_kernel<1><<<grid, kThreads, 0, s>>>(src, cols, ld_src, dst, ld_dst, gpr, total,
                                                            vec_src, (ld_dst % 4) == 0);
            break;
        case LRC_BF16:
            round_pack_kernel<3><<<grid, kThreads, 0, s>>>(src, cols, ld_src, dst, ld_dst, gpr, total,
                                                            vec_src, (ld_dst % 8) == 0);
            break;
        default:
            round_pack_kernel<2><<<grid, kThreads, 0, s>>>(src, cols, ld_src, dst, ld_dst, gpr, total,
                                                            vec_src, (ld_dst % 8) == 0);
            break;
    }
    return after_launch("round_pack_kernel");
}

lrc_status launch_widen(const void* src, lrc_fmt fmt, int64_t rows, int64_t cols, int64_t ld_src,
                        double* dst, int64_t ld_dst, cudaStream_t s) {
    const int64_t gpr = (ld_dst + kGroup - 1) / kGroup;
    const int64_t total = rows * gpr;
    const int grid = grid_for(total);
    const int64_t e = storage_bytes(fmt);
    // 16-byte vectors: row starts (base and pitch) on 16-byte boundaries
    const bool vec_src = (reinterpret_cast<uintptr_t>(src) % 16 == 0) && ((ld_src * e) % 16 == 0);
    const bool vec_dst = (reinterpret_cast<uintptr_t>(dst) % 16 == 0) && (ld_dst % 2 == 0);
    switch (fmt) {
        case LRC_F64:
            widen_kernel<0><<<grid, kThreads, 0, s>>>(src, cols, ld_src, dst, ld_dst, gpr, total, vec_src, vec_dst);
            break;
        case LRC_F32:
            widen_kernel<1><<<grid, kThreads, 0, s>>>(src, cols, ld_src, dst, ld_dst, gpr, total, vec_src, vec_dst);
            break;
        case LRC_BF16:
            widen_kernel<3><<<grid, kThreads, 0, s>>>(src, cols, ld_src, dst, ld_dst, gpr, total, vec_src, vec_dst);
            break;
        default:
            widen_kernel<2><<<grid, kThreads, 0, s>>>(src, cols, ld_src, dst, ld_dst, gpr, total, vec_src, vec_dst);
            break;
    }
    return after_launch("widen_kernel");
}

}  // namespace lrc
