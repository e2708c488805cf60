// apply_skinny.cu -- low-rank apply for batches of at most 16 queries, every
// format, on the CUDA cores (Sec. 4.4, Eq. gpu_matrix_apply:
// Y = [(X V) diag(s)] U^T).
//
// With a handful of queries the apply streams the two factors once and does
// b multiply-adds per factor element: two matrix-vector streams that must
// keep every SM's loads in flight.  Three launches on the caller's stream:
//   skinny_w1_kernel  grid (n-chunk, group of 32 rows of V^T): the chunk of X
//                     (at most 16 rows) is staged in shared memory; each warp
//                     takes 4 rows of V^T and streams them with 16-byte loads
//                     (four in flight per lane), each lane keeping the b
//                     partial dot products of every row, which a fixed
//                     butterfly then adds across the warp.  One partial W per
//                     chunk.
//   skinny_w2_kernel  W = (sum of the chunks' partials, in chunk order) diag(s);
//                     for binary16 output W is rounded to binary16 (the
//                     method-precision workspace of Sec. 3.4).
//   skinny_y_kernel   W (b x k) in shared memory; each warp takes 4 rows of U,
//                     streams them the same way and keeps the results of its
//                     rows so that Y's rows are written as contiguous runs.
// Arithmetic: binary64 FMAs for binary64, binary32 FMAs otherwise (binary16
// factors widened exactly; Sec. 3.4: FP16 products accumulate in FP32).  The
// summation order is fixed: results are reproducible on a device.
#include <cuda_fp16.h>

#include "common.cuh"
#include "tc.cuh"

namespace lrc {
namespace {

constexpr int kWarps = 8;
constexpr int kThreadsS = 32 * kWarps;
constexpr int kRows = 4;                      // factor rows per warp and pass

template <typename TS>
struct EVof {
    static constexpr int v = 16 / (int)sizeof(TS);     // elements per 16-byte vector
};

// 16 bytes of storage at p (16-byte aligned) as arithmetic values.
template <typename T, typename TS>
__device__ __forceinline__ void load_vec(const TS* p, T (&v)[EVof<TS>::v]) {
    if constexpr (sizeof(TS) == 2) {
        const uint4 q = __ldg(reinterpret_cast<const uint4*>(p));
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[i]));
            v[2 * i] = f.x;
            v[2 * i + 1] = f.y;
        }
    } else if constexpr (sizeof(TS) == 4) {
        const float4 q = __ldg(reinterpret_cast<const float4*>(p));
        v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
    } else {
        const double2 q = __ldg(reinterpret_cast<const double2*>(p));
        v[0] = q.x; v[1] = q.y;
    }
}

template <typename T>
__device__ __forceinline__ T to_t(__half x) { return (T)__half2float(x); }
template <typename T>
__device__ __forceinline__ T to_t(float x) { return (T)x; }
template <typename T>
__device__ __forceinline__ T to_t(double x) { return (T)x; }

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ void store_out(double* p, double v) { *p = v; }
__device__ __forceinline__ void store_out(float* p, float v) { *p = v; }
__device__ __forceinline__ void store_out(__half* p, float v) { *p = __float2half_rn(v); }

// ---------------------------------------------------------------- phase 1
template <typename TS, typename T, int B>
__global__ void __launch_bounds__(kThreadsS)
skinny_w1_kernel(const TS* __restrict__ X, const TS* __restrict__ Vt, int64_t n, int64_t ldn, int k, int b,
                 int64_t L, T* __restrict__ Wp) {
    constexpr int EV = EVof<TS>::v;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    T* xs = reinterpret_cast<T*>(smem_raw);      // [B][L], zero past the batch and the chunk
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t chunk = blockIdx.x;
    const int64_t i0 = chunk * L;
    const int64_t len = (n - i0) < L ? (n - i0) : L;
    // stage X: 16-byte vectors, four loads in flight per thread before their stores
    {
        const int64_t nv = (int64_t)B * (L / EV);
        for (int64_t v0 = threadIdx.x; v0 < nv; v0 += 4 * kThreadsS) {
            T val[4][EV];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int64_t v = v0 + (int64_t)u * kThreadsS;
                const int64_t c = v / (L / EV), i = (v - c * (L / EV)) * EV;
                if (v < nv && c < b && i + EV <= len) {
                    load_vec<T, TS>(X + c * ldn + i0 + i, val[u]);
                } else {
#pragma unroll
                    for (int e = 0; e < EV; ++e)
                        val[u][e] = (v < nv && c < b && i + e < len) ? to_t<T>(X[c * ldn + i0 + i + e]) : T(0);
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int64_t v = v0 + (int64_t)u * kThreadsS;
                if (v < nv) {
                    const int64_t c = v / (L / EV), i = (v - c * (L / EV)) * EV;
#pragma unroll
                    for (int e = 0; e < EV; ++e) xs[c * L + i + e] = val[u][e];
                }
            }
        }
    }
    __syncthreads();
    const int j0 = (blockIdx.y * kWarps + warp) * kRows;
    T acc[kRows][B];
#pragma unroll
    for (int r = 0; r < kRows; ++r)
#pragma unroll
        for (int c = 0; c < B; ++c) acc[r][c] = T(0);
    const int64_t nvec = len / EV;
    for (int64_t v = lane; v < nvec; v += 32) {
        T vv[kRows][EV];
#pragma unroll
        for (int r = 0; r < kRows; ++r) {
            if (j0 + r < k) load_vec<T, TS>(Vt + (int64_t)(j0 + r) * ldn + i0 + v * EV, vv[r]);
            else {
#pragma unroll
                for (int e = 0; e < EV; ++e) vv[r][e] = T(0);
            }
        }
#pragma unroll
        for (int c = 0; c < B; ++c) {
            T xv[EV];
#pragma unroll
            for (int e = 0; e < EV; ++e) xv[e] = xs[c * L + v * EV + e];
#pragma unroll
            for (int r = 0; r < kRows; ++r)
#pragma unroll
                for (int e = 0; e < EV; ++e) acc[r][c] = fma(xv[e], vv[r][e], acc[r][c]);
        }
    }
    // ragged end of the chunk: single elements
    for (int64_t i = nvec * EV + lane; i < len; i += 32) {
#pragma unroll
        for (int r = 0; r < kRows; ++r) {
            const T x = (j0 + r < k) ? to_t<T>(Vt[(int64_t)(j0 + r) * ldn + i0 + i]) : T(0);
#pragma unroll
            for (int c = 0; c < B; ++c) acc[r][c] = fma(xs[c * L + i], x, acc[r][c]);
        }
    }
    tc::pdl_trigger();
#pragma unroll
    for (int r = 0; r < kRows; ++r) {
#pragma unroll
        for (int c = 0; c < B; ++c) {
            const T sum = warp_sum(acc[r][c]);
            if (lane == c && c < b && j0 + r < k) Wp[(chunk * b + c) * k + j0 + r] = sum;
        }
    }
}

// ---------------------------------------------------------------- phase 1b
template <typename TS, typename T>
__global__ void __launch_bounds__(256)
skinny_w2_kernel(const T* __restrict__ Wp, int nchunks, int b, int k, const TS* __restrict__ S, int round16,
                 T* __restrict__ W) {
    tc::pdl_wait();                  // partials of the phase-1 grid
    tc::pdl_trigger();
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)b * k) return;
    const int j = (int)(e % k);
    T acc = Wp[e];
    for (int ch = 1; ch < nchunks; ++ch) acc += Wp[(int64_t)ch * b * k + e];
    acc *= to_t<T>(S[j]);
    if (round16) acc = (T)__half2float(__float2half_rn((float)acc));
    W[e] = acc;
}

// ---------------------------------------------------------------- phase 2
template <typename TS, typename T, typename TOut, int B>
__global__ void __launch_bounds__(kThreadsS)
skinny_y_kernel(const T* __restrict__ W, const TS* __restrict__ U, int64_t m, int k, int64_t ldk, int b,
                TOut* __restrict__ Y) {
    constexpr int EV = EVof<TS>::v;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    T* ws = reinterpret_cast<T*>(smem_raw);      // [B][kv], zero past the batch and the rank
    const int kv = (k + EV - 1) / EV * EV;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    tc::pdl_wait();                  // W of the reduction kernel
    for (int e = threadIdx.x; e < B * kv; e += kThreadsS) {
        const int c = e / kv, j = e - c * kv;
        ws[e] = (c < b && j < k) ? W[c * k + j] : T(0);
    }
    __syncthreads();
    const int64_t r0 = ((int64_t)blockIdx.x * kWarps + warp) * kRows;
    T acc[kRows][B];
#pragma unroll
    for (int r = 0; r < kRows; ++r)
#pragma unroll
        for (int c = 0; c < B; ++c) acc[r][c] = T(0);
    const int nvk = kv / EV;
    for (int v = lane; v < nvk; v += 32) {
        T uu[kRows][EV];
#pragma unroll
        for (int r = 0; r < kRows; ++r) {
            if (r0 + r < m) {
                load_vec<T, TS>(U + (r0 + r) * ldk + v * EV, uu[r]);
#pragma unroll
                for (int e = 0; e < EV; ++e)
                    if (v * EV + e >= k) uu[r][e] = T(0);    // pad columns of U are not read as numbers
            } else {
#pragma unroll
                for (int e = 0; e < EV; ++e) uu[r][e] = T(0);
            }
        }
#pragma unroll
        for (int c = 0; c < B; ++c) {
            T wv[EV];
#pragma unroll
            for (int e = 0; e < EV; ++e) wv[e] = ws[c * kv + v * EV + e];
#pragma unroll
            for (int r = 0; r < kRows; ++r)
#pragma unroll
                for (int e = 0; e < EV; ++e) acc[r][c] = fma(wv[e], uu[r][e], acc[r][c]);
        }
    }
    // output q = c * kRows + r (Y[c][r0 + r]) is kept by lane q % 32 in out[q / 32]
    constexpr int NOUT = (B * kRows + 31) / 32;
    T out[NOUT];
#pragma unroll
    for (int q = 0; q < NOUT; ++q) out[q] = T(0);
#pragma unroll
    for (int r = 0; r < kRows; ++r)
#pragma unroll
        for (int c = 0; c < B; ++c) {
            const T sum = warp_sum(acc[r][c]);
            const int q = c * kRows + r;
            if (lane == (q & 31)) out[q >> 5] = sum;
        }
#pragma unroll
    for (int q = 0; q < NOUT; ++q) {
        const int idx = q * 32 + lane;
        const int c = idx / kRows, r = idx % kRows;
        if (c < b && c < B && r0 + r < m) store_out(Y + (int64_t)c * m + r0 + r, out[q]);
    }
}

template <typename TS, typename T, typename TOut, int B>
lrc_status launch_skinny_b(const TS* U, const TS* S, const TS* Vt, const TS* X, TOut* Y, int64_t m, int64_t n,
                           int64_t k, int64_t b, bool round16, cudaStream_t s) {
    constexpr int EV = EVof<TS>::v;
    const int sms = sm_count();
    const int64_t ldn = lrc_packed_ld(n), ldk = lrc_packed_ld(k);
    // chunk length: a multiple of 256 elements with the staged X within 48 KB,
    // and enough chunks for two waves of CTAs
    const int64_t jblocks = (k + kWarps * kRows - 1) / (kWarps * kRows);
    int64_t L = (48 * 1024) / ((int64_t)B * (int64_t)sizeof(T)) / 256 * 256;
    if (L > 4096) L = 4096;
    const int64_t want = (2 * (int64_t)sms + jblocks - 1) / jblocks;
    int64_t Lw = (n + want - 1) / want;
    Lw = (Lw + 255) / 256 * 256;
    if (Lw < L) L = Lw;
    if (L < 256) L = 256;
    const int64_t nchunks = (n + L - 1) / L;
    int64_t t;
    if (!mul_ok(nchunks * b, k, &t) || nchunks > 65535 || jblocks > 65535) {
        set_error("small-batch apply: problem too large");
        return LRC_ERR_UNSUPPORTED;
    }
    const size_t part_bytes = ((size_t)nchunks * b * k * sizeof(T) + 255) / 256 * 256;
    const size_t w_bytes = (size_t)b * k * sizeof(T);
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, part_bytes + w_bytes, &ws);
    if (st != LRC_OK) return st;
    T* Wp = static_cast<T*>(ws);
    T* Wd = reinterpret_cast<T*>(static_cast<unsigned char*>(ws) + part_bytes);
    const size_t smem1 = (size_t)B * L * sizeof(T);
    skinny_w1_kernel<TS, T, B><<<dim3((unsigned)nchunks, (unsigned)jblocks), kThreadsS, smem1, s>>>(
        X, Vt, n, ldn, (int)k, (int)b, L, Wp);
    if ((st = after_launch("skinny_w1_kernel")) != LRC_OK) return st;
    cudaError_t e = launch_pdl(skinny_w2_kernel<TS, T>, dim3((unsigned)((b * k + 255) / 256)), dim3(256), 0, s,
                               (const T*)Wp, (int)nchunks, (int)b, (int)k, S, round16 ? 1 : 0, Wd);
    if (e != cudaSuccess) return cuda_fail(e, "skinny_w2_kernel launch");
    if ((st = after_launch("skinny_w2_kernel")) != LRC_OK) return st;
    const int kv = (int)((k + EV - 1) / EV * EV);
    const size_t smem3 = (size_t)B * kv * sizeof(T);
    if (smem3 > 48 * 1024) {
        e = cudaFuncSetAttribute(skinny_y_kernel<TS, T, TOut, B>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem3);
        if (e != cudaSuccess) return cuda_fail(e, "skinny_y_kernel smem attribute");
    }
    const int64_t yblocks = (m + kWarps * kRows - 1) / (kWarps * kRows);
    e = launch_pdl(skinny_y_kernel<TS, T, TOut, B>, dim3((unsigned)yblocks), dim3(kThreadsS), smem3, s,
                   (const T*)Wd, U, m, (int)k, ldk, (int)b, Y);
    if (e != cudaSuccess) return cuda_fail(e, "skinny_y_kernel launch");
    return after_launch("skinny_y_kernel");
}

template <typename TS, typename T, typename TOut>
lrc_status launch_skinny_t(const TS* U, const TS* S, const TS* Vt, const TS* X, TOut* Y, int64_t m, int64_t n,
                           int64_t k, int64_t b, bool round16, cudaStream_t s) {
    if (b <= 1) return launch_skinny_b<TS, T, TOut, 1>(U, S, Vt, X, Y, m, n, k, b, round16, s);
    if (b <= 4) return launch_skinny_b<TS, T, TOut, 4>(U, S, Vt, X, Y, m, n, k, b, round16, s);
    return launch_skinny_b<TS, T, TOut, 16>(U, S, Vt, X, Y, m, n, k, b, round16, s);
}

}  // namespace

// Largest batch this path takes per format: up to 16 queries for binary32;
// binary64 (DFMA-bound from a few queries on) and binary16 (whose tensor-core
// path is faster from 16 queries on) up to 4.
int64_t apply_skinny_max_batch(lrc_fmt fmt) { return fmt == LRC_F32 ? 16 : 4; }

lrc_status launch_apply_skinny(const void* U, const void* S, const void* Vt, const void* X, void* Y, int64_t m,
                               int64_t n, int64_t k, int64_t b, lrc_fmt fmt, cudaStream_t s) {
    if (b < 1 || b > apply_skinny_max_batch(fmt) || k > 1024) {
        set_error("small-batch apply: b = %lld, k = %lld outside the kernel", (long long)b, (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    switch (fmt) {
        case LRC_F64:
            return launch_skinny_t<double, double, double>((const double*)U, (const double*)S, (const double*)Vt,
                                                          (const double*)X, (double*)Y, m, n, k, b, false, s);
        case LRC_F32:
            return launch_skinny_t<float, float, float>((const float*)U, (const float*)S, (const float*)Vt,
                                                       (const float*)X, (float*)Y, m, n, k, b, false, s);
        case LRC_F16:
            return launch_skinny_t<__half, float, float>((const __half*)U, (const __half*)S, (const __half*)Vt,
                                                        (const __half*)X, (float*)Y, m, n, k, b, false, s);
        default:
            return launch_skinny_t<__half, float, __half>((const __half*)U, (const __half*)S, (const __half*)Vt,
                                                         (const __half*)X, (__half*)Y, m, n, k, b, true, s);
    }
}

}  // namespace lrc
