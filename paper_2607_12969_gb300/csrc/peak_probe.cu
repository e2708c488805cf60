// peak_probe.cu -- measured arithmetic rates of this GPU's units, the
// denominators of the roofline fractions of the binary32 and binary64 paths
// (the products of Sec. 3.4 run on the CUDA cores, or on the binary64 tensor
// cores, whichever is faster).
//
// Every thread runs kChains independent multiply-add chains for `iters`
// steps (no loads, no stores in the loop), so the unit's issue rate is the
// only bound; one final store per thread keeps the chains alive.  The grid
// fills every SM with 2048 threads.
#include "common.cuh"

namespace lrc {
namespace {

constexpr int kThreads = 256;
constexpr int kBlocksPerSm = 8;
constexpr int kChains = 8;

__global__ void __launch_bounds__(kThreads) probe_ffma_kernel(float* out, int64_t iters, float a, float b) {
    float x[kChains];
#pragma unroll
    for (int c = 0; c < kChains; ++c) x[c] = (float)(threadIdx.x + c);
    for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
        for (int c = 0; c < kChains; ++c) x[c] = fmaf(x[c], a, b);
    }
    float s = 0.0f;
#pragma unroll
    for (int c = 0; c < kChains; ++c) s += x[c];
    out[(int64_t)blockIdx.x * kThreads + threadIdx.x] = s;
}

__global__ void __launch_bounds__(kThreads) probe_ffma2_kernel(float* out, int64_t iters, float a, float b) {
    float2 x[kChains];
    const float2 a2 = make_float2(a, a), b2 = make_float2(b, b);
#pragma unroll
    for (int c = 0; c < kChains; ++c) x[c] = make_float2((float)(threadIdx.x + c), (float)c);
    for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
        for (int c = 0; c < kChains; ++c) x[c] = __ffma2_rn(x[c], a2, b2);
    }
    float s = 0.0f;
#pragma unroll
    for (int c = 0; c < kChains; ++c) s += x[c].x + x[c].y;
    out[(int64_t)blockIdx.x * kThreads + threadIdx.x] = s;
}

__global__ void __launch_bounds__(kThreads) probe_dfma_kernel(double* out, int64_t iters, double a, double b) {
    double x[kChains];
#pragma unroll
    for (int c = 0; c < kChains; ++c) x[c] = (double)(threadIdx.x + c);
    for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
        for (int c = 0; c < kChains; ++c) x[c] = fma(x[c], a, b);
    }
    double s = 0.0;
#pragma unroll
    for (int c = 0; c < kChains; ++c) s += x[c];
    out[(int64_t)blockIdx.x * kThreads + threadIdx.x] = s;
}

// binary64 tensor-core MMA, m8n8k4 (one 8 x 8 x 4 product per warp and
// instruction: 512 flops); kChains / 2 independent accumulator tiles
__global__ void __launch_bounds__(kThreads) probe_dmma_kernel(double* out, int64_t iters, double a, double b) {
    constexpr int T = kChains / 2;
    double c0[T], c1[T];
#pragma unroll
    for (int t = 0; t < T; ++t) {
        c0[t] = (double)(threadIdx.x + t);
        c1[t] = (double)t;
    }
    const double av = a * (double)(threadIdx.x & 3), bv = b;
    for (int64_t i = 0; i < iters; ++i) {
#pragma unroll
        for (int t = 0; t < T; ++t) {
            asm volatile("mma.sync.aligned.m8n8k4.row.col.f64.f64.f64.f64 {%0, %1}, {%2}, {%3}, {%0, %1};"
                         : "+d"(c0[t]), "+d"(c1[t])
                         : "d"(av), "d"(bv));
        }
    }
    double s = 0.0;
#pragma unroll
    for (int t = 0; t < T; ++t) s += c0[t] + c1[t];
    out[(int64_t)blockIdx.x * kThreads + threadIdx.x] = s;
}

}  // namespace

lrc_status run_probe_peak(int kind, int64_t iters, double* flops_out, cudaStream_t s) {
    const int grid = sm_count() * kBlocksPerSm;
    const int64_t threads = (int64_t)grid * kThreads;
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, (size_t)threads * sizeof(double), &ws);
    if (st != LRC_OK) return st;
    cudaEvent_t e0, e1;
    cudaError_t e = cudaEventCreate(&e0);
    if (e != cudaSuccess) return cuda_fail(e, "cudaEventCreate");
    e = cudaEventCreate(&e1);
    if (e != cudaSuccess) {
        cudaEventDestroy(e0);
        return cuda_fail(e, "cudaEventCreate");
    }
    // factors that keep the chains finite and away from subnormals
    const float af = 0.999999f, bf = 1.0e-3f;
    const double ad = 0.9999999999, bd = 1.0e-3;
    double per_thread_step = 0.0;   // flops per thread and loop step
    auto launch = [&](int64_t n) {
        switch (kind) {
            case 0: probe_ffma_kernel<<<grid, kThreads, 0, s>>>((float*)ws, n, af, bf); break;
            case 1: probe_ffma2_kernel<<<grid, kThreads, 0, s>>>((float*)ws, n, af, bf); break;
            case 2: probe_dfma_kernel<<<grid, kThreads, 0, s>>>((double*)ws, n, ad, bd); break;
            default: probe_dmma_kernel<<<grid, kThreads, 0, s>>>((double*)ws, n, ad, bd); break;
        }
    };
    switch (kind) {
        case 0: per_thread_step = 2.0 * kChains; break;
        case 1: per_thread_step = 4.0 * kChains; break;
        case 2: per_thread_step = 2.0 * kChains; break;
        default: per_thread_step = (512.0 / 32.0) * (kChains / 2); break;
    }
    launch(iters / 16 + 1);   // warm-up
    st = after_launch("probe kernel (warm-up)");
    if (st == LRC_OK) {
        cudaEventRecord(e0, s);
        launch(iters);
        st = after_launch("probe kernel");
        cudaEventRecord(e1, s);
    }
    if (st == LRC_OK) {
        e = cudaEventSynchronize(e1);
        if (e != cudaSuccess) {
            st = cuda_fail(e, "cudaEventSynchronize (probe)");
        } else {
            float ms = 0.0f;
            cudaEventElapsedTime(&ms, e0, e1);
            *flops_out = per_thread_step * (double)threads * (double)iters / ((double)ms * 1e-3);
        }
    }
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    return st;
}

}  // namespace lrc
