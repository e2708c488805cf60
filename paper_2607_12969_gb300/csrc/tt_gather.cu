// tt_gather.cu -- sampled entries of a Tensor Train, T(i_1..i_d) =
// G_1(i_1) G_2(i_2) ... G_d(i_d) (Sec. 5.1), evaluated entry by entry: the
// independent check of a dense reconstruction on sampled entries.
//
// One warp per entry.  The running row vector v (length r_l) is spread over
// the lanes (lane j holds v_j, v_{j+32}, ...); one core slice G_l(i_l) is
// r_{l-1} x r_l with contiguous rows, so for every a the lanes read row a of
// the slice coalesced and add v_a (broadcast by a shuffle) times it.  The
// last core is a column, reduced across the warp with a fixed butterfly.
// Cores stay in L2; nothing but the indices and the outputs touches HBM.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <type_traits>

#include <algorithm>

#include "common.cuh"

namespace lrc {

namespace {

struct GatherArgs {
    const void* cores[16];
    int64_t dims[16];
    int64_t stride[16];     // prod_{j > l} dims[j]: i_l = (f / stride[l]) % dims[l]
    int ranks[17];
    int d;
    int64_t numel;
};

template <typename T>
__device__ __forceinline__ float ld_core(const T* p);
template <>
__device__ __forceinline__ float ld_core<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float ld_core<__half>(const __half* p) { return __half2float(__ldg(p)); }
template <>
__device__ __forceinline__ float ld_core<__nv_bfloat16>(const __nv_bfloat16* p) {
    return __uint_as_float((uint32_t)__ldg(reinterpret_cast<const unsigned short*>(p)) << 16);
}

__device__ __forceinline__ double ld_core64(const double* p) { return __ldg(p); }

template <typename T, typename A>
__device__ __forceinline__ A load_elem(const T* p) {
    if constexpr (sizeof(T) == 8) {
        return ld_core64(reinterpret_cast<const double*>(p));
    } else {
        return (A)ld_core<T>(p);
    }
}

template <typename O, typename A>
__device__ __forceinline__ O store_cast(A v) {
    if constexpr (std::is_same_v<O, __nv_bfloat16>) {
        return __float2bfloat16_rn((float)v);
    } else if constexpr (sizeof(O) == 2) {
        return __float2half_rn((float)v);
    } else {
        return (O)v;
    }
}

template <typename O>
__device__ __forceinline__ O quiet_nan();
template <>
__device__ __forceinline__ double quiet_nan<double>() { return __longlong_as_double(0x7ff8000000000000LL); }
template <>
__device__ __forceinline__ float quiet_nan<float>() { return __int_as_float(0x7fc00000); }
template <>
__device__ __forceinline__ __half quiet_nan<__half>() { return __ushort_as_half((unsigned short)0x7e00); }
template <>
__device__ __forceinline__ __nv_bfloat16 quiet_nan<__nv_bfloat16>() {
    return __ushort_as_bfloat16((unsigned short)0x7fc0);
}

// T: core element type, A: arithmetic type, O: output type, S: slots per lane
// (ranks up to 32 S).
template <typename T, typename A, typename O, int S>
__global__ void __launch_bounds__(256) tt_gather_kernel(const __grid_constant__ GatherArgs g,
                                                        const int64_t* __restrict__ idx, int64_t count,
                                                        O* __restrict__ out) {
    const int lane = threadIdx.x & 31;
    const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int d = g.d;
    for (int64_t e = warp; e < count; e += nwarps) {
        const int64_t f = idx[e];
        if (f < 0 || f >= g.numel) {
            if (lane == 0) out[e] = quiet_nan<O>();
            continue;
        }
        // multi-index: lane l < d decodes i_l (32-bit arithmetic when the
        // tensor has fewer than 2^32 entries), then the lanes share them
        int64_t my_i = 0;
        if (lane < d) {
            if (g.numel <= 0xffffffffLL) {
                const uint32_t fu = (uint32_t)f;
                my_i = (int64_t)((fu / (uint32_t)g.stride[lane]) % (uint32_t)g.dims[lane]);
            } else {
                my_i = (f / g.stride[lane]) % g.dims[lane];
            }
        }
        A v[S];
        // level 1: the row G_1(0, i_1, :)
        {
            const int64_t i = __shfl_sync(0xffffffffu, my_i, 0);
            const int r1 = g.ranks[1];
            const T* row = static_cast<const T*>(g.cores[0]) + i * r1;
#pragma unroll
            for (int s = 0; s < S; ++s) {
                const int b = lane + 32 * s;
                v[s] = b < r1 ? load_elem<T, A>(row + b) : (A)0;
            }
        }
        // interior levels: v <- v G_l(i_l)
        for (int l = 1; l < d - 1; ++l) {
            const int ra = g.ranks[l], rb = g.ranks[l + 1];
            const int64_t n = g.dims[l];
            const int64_t i = __shfl_sync(0xffffffffu, my_i, l);
            const T* base = static_cast<const T*>(g.cores[l]) + i * rb;
            const int64_t pitch = n * rb;
            A acc[S];
#pragma unroll
            for (int s = 0; s < S; ++s) acc[s] = (A)0;
#pragma unroll
            for (int sa = 0; sa < S; ++sa) {
                const int a0 = 32 * sa;
                if (a0 >= ra) break;
                const int na = min(32, ra - a0);
#pragma unroll 8
                for (int aa = 0; aa < na; ++aa) {
                    const A va = __shfl_sync(0xffffffffu, v[sa], aa);
                    const T* row = base + (int64_t)(a0 + aa) * pitch;
#pragma unroll
                    for (int s = 0; s < S; ++s) {
                        const int b = lane + 32 * s;
                        if (b < rb) acc[s] = fma(va, load_elem<T, A>(row + b), acc[s]);
                    }
                }
            }
#pragma unroll
            for (int s = 0; s < S; ++s) v[s] = acc[s];
        }
        // last level: T = v G_d(:, i_d), a column of length r_{d-1}
        {
            const int ra = g.ranks[d - 1];
            const int64_t n = g.dims[d - 1];
            const int64_t i = __shfl_sync(0xffffffffu, my_i, d - 1);
            const T* col = static_cast<const T*>(g.cores[d - 1]) + i;
            A part = (A)0;
#pragma unroll
            for (int s = 0; s < S; ++s) {
                const int a = lane + 32 * s;
                if (a < ra) part = fma(v[s], load_elem<T, A>(col + (int64_t)a * n), part);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
            if (lane == 0) out[e] = store_cast<O, A>(part);
        }
    }
}

template <typename T, typename A, typename O>
lrc_status launch_typed(const GatherArgs& g, int rmax, const int64_t* idx, int64_t count, void* out,
                        cudaStream_t s) {
    const int64_t warps_needed = count;
    const int64_t cap = (int64_t)sm_count() * 16;          // 16 CTAs of 8 warps per SM at most
    const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>((warps_needed + 7) / 8, cap));
    O* o = static_cast<O*>(out);
    if (rmax <= 32)
        tt_gather_kernel<T, A, O, 1><<<blocks, 256, 0, s>>>(g, idx, count, o);
    else if (rmax <= 64)
        tt_gather_kernel<T, A, O, 2><<<blocks, 256, 0, s>>>(g, idx, count, o);
    else if (rmax <= 128)
        tt_gather_kernel<T, A, O, 4><<<blocks, 256, 0, s>>>(g, idx, count, o);
    else
        tt_gather_kernel<T, A, O, 8><<<blocks, 256, 0, s>>>(g, idx, count, o);
    return after_launch("tt_gather_kernel");
}

}  // namespace

int tt_gather_max_rank() { return 256; }

lrc_status launch_tt_gather(const TTShape& sh, lrc_fmt fmt, const int64_t* idx, int64_t count, void* out,
                            cudaStream_t s) {
    GatherArgs g{};
    g.d = sh.d;
    g.numel = sh.numel;
    int rmax = 1;
    for (int l = 0; l < sh.d; ++l) {
        g.cores[l] = sh.cores[l];
        g.dims[l] = sh.dims[l];
    }
    for (int l = 0; l <= sh.d; ++l) {
        g.ranks[l] = (int)sh.ranks[l];
        rmax = std::max(rmax, (int)sh.ranks[l]);
    }
    int64_t st = 1;
    for (int l = sh.d - 1; l >= 0; --l) {
        g.stride[l] = st;
        st *= sh.dims[l];
    }
    switch (fmt) {
        case LRC_F64: return launch_typed<double, double, double>(g, rmax, idx, count, out, s);
        case LRC_F32: return launch_typed<float, float, float>(g, rmax, idx, count, out, s);
        case LRC_F16: return launch_typed<__half, float, float>(g, rmax, idx, count, out, s);
        case LRC_F16_O16: return launch_typed<__half, float, __half>(g, rmax, idx, count, out, s);
        case LRC_BF16: return launch_typed<__nv_bfloat16, float, __nv_bfloat16>(g, rmax, idx, count, out, s);
    }
    set_error("unknown format");
    return LRC_ERR_INVALID_ARG;
}

}  // namespace lrc
