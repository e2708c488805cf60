// apply_skinny.cu -- low-rank apply for batches of at most 16 queries, every
// format, on the CUDA cores (Sec. 4.4, Eq. gpu_matrix_apply:
// Y = [(X V) diag(s)] U^T).
//
// With a handful of queries the apply streams the two factors once and does
// b multiply-adds per factor element: two matrix-vector streams whose speed
// is set by how many bytes each SM has in flight.  Every operand tile is
// therefore one set of TMA copies issued at the start of its CTA (2-D boxes,
// zero-filled outside the arrays, so the arithmetic needs no bounds tests).
// Two launches on the caller's stream, chained by programmatic dependent
// launch:
//   skinny_w1_kernel  grid (n-chunk, block of 32 rows of V^T): the chunk of X
//                     (at most 16 rows) and of the 32 rows of V^T land in
//                     shared memory; each warp takes 4 rows of V^T, each lane
//                     keeps the b partial dot products of every row over its
//                     16-byte columns, a recursive halving adds them across
//                     the warp.  One partial W per chunk.  The last CTA of a
//                     row block to finish (an arrival counter) adds the
//                     chunks' partials in chunk order, scales by diag(s) and
//                     writes that block of W; for binary16 output W is
//                     rounded to binary16 (the method-precision workspace of
//                     Sec. 3.4).  The CTAs let the second kernel start as
//                     soon as their copies are issued.
//   skinny_y_kernel   a CTA per 64 rows of U (32 for binary64): the rows are
//                     requested at once, so they stream while the first
//                     kernel still runs; after the wait for it W (b x k)
//                     follows as one bulk copy; groups of G lanes (8, or 32
//                     for at most 4 queries in 2- and 4-byte formats) take 4
//                     rows (2) each, a lane every G-th 16-byte column.
// Arithmetic: binary64 FMAs for binary64, binary32 FMAs otherwise (binary16
// factors widened exactly; Sec. 3.4: FP16 products accumulate in FP32).  The
// summation order is fixed: results are reproducible on a device.
#include <cuda_fp16.h>

#include "common.cuh"
#include "tc.cuh"

namespace lrc {

__device__ unsigned int g_err_skinny;

namespace {

constexpr int kWarps = 8;
constexpr int kThreadsS = 32 * kWarps;
constexpr int kRows = 4;                      // factor rows per warp (first product: 2 for 16 binary64 queries)
constexpr int kBox = 256;                     // columns per TMA box of the first product
constexpr size_t kSmemW1 = 100 * 1024;        // shared-memory budget of a first-product CTA
constexpr size_t kSmemMaxS = 220 * 1024;      // largest dynamic shared memory a CTA asks for

template <typename TS>
struct EVof {
    static constexpr int v = 16 / (int)sizeof(TS);     // elements per 16-byte vector
};

// 16 bytes of storage at p (16-byte aligned, shared memory) as arithmetic values.
template <typename T, typename TS>
__device__ __forceinline__ void load_vec(const TS* p, T (&v)[EVof<TS>::v]) {
    if constexpr (sizeof(TS) == 2) {
        const uint4 q = *reinterpret_cast<const uint4*>(p);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[i]));
            v[2 * i] = f.x;
            v[2 * i + 1] = f.y;
        }
    } else if constexpr (sizeof(TS) == 4) {
        const float4 q = *reinterpret_cast<const float4*>(p);
        v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
    } else {
        const double2 q = *reinterpret_cast<const double2*>(p);
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

// Sums each of the N values v[] over the aligned groups of G lanes (G a
// power of two <= 32) by recursive halving: at the step with lane offset o
// (G/2, G/4, ...) a lane keeps one half of its values -- the upper half when
// lane & o -- and adds the partner's copy of that half.  After
// min(log2 G, log2 N) steps a butterfly over the remaining offsets finishes:
// lane L then holds, in v[0 .. max(N/G, 1) - 1], the group totals of the
// values halving_index<N, G>(L) + t.  Fixed order: the same result on every
// run.  About N shuffles instead of N log2 G.
template <int N, int G>
__device__ __forceinline__ constexpr int halving_steps() {
    int s = 0;
    while ((1 << s) < G && (2 << s) <= N) ++s;
    return s;
}
template <int N, int G>
__device__ __forceinline__ int halving_index(int lane) {
    int base = 0;
#pragma unroll
    for (int s = 0; s < halving_steps<N, G>(); ++s)
        if (lane & ((G / 2) >> s)) base += N >> (s + 1);
    return base;
}
template <int N, int G>
__device__ __forceinline__ bool halving_writer(int lane) {
    return (lane & ((G >> halving_steps<N, G>()) - 1)) == 0;
}
template <typename T, int N, int G>
__device__ __forceinline__ void halving_sum(T (&v)[N], int lane) {
    static_assert((N & (N - 1)) == 0 && (G & (G - 1)) == 0 && G <= 32, "powers of two");
#pragma unroll
    for (int s = 0; s < halving_steps<N, G>(); ++s) {
        const int o = (G / 2) >> s, h = N >> (s + 1);
        const bool up = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < h; ++i) {
            const T send = up ? v[i] : v[i + h];
            const T keep = up ? v[i + h] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
#pragma unroll
    for (int o = (G / 2) >> halving_steps<N, G>(); o > 0; o >>= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
}

__device__ __forceinline__ void store_out(double* p, double v) { *p = v; }
__device__ __forceinline__ void store_out(float* p, float v) { *p = v; }
__device__ __forceinline__ void store_out(__half* p, float v) { *p = __float2half_rn(v); }

// The dynamic shared-memory base rounded up to 128 bytes by an offset (not
// through an integer), so that the compiler still sees a shared-memory
// pointer and emits shared loads rather than generic ones.
__device__ __forceinline__ unsigned char* align128(unsigned char* p) {
    return p + ((128u - (tc::smem_u32(p) & 127u)) & 127u);
}

// Waits for copy group q of the CTA's nq (all threads).  On a timeout thread
// 0 waits a little longer for every group still in flight before the CTA may
// exit.
__device__ __forceinline__ bool wait_tiles(uint64_t* bar, int q, int nq, volatile int* abort, unsigned int code) {
    if (tc::mbar_wait(&bar[q], 0, abort, &g_err_skinny, code)) return true;
    if (threadIdx.x == 0) {
        volatile int no_abort = 0;
        for (int i = 0; i < nq; ++i) tc::mbar_wait(&bar[i], 0, &no_abort, &g_err_skinny, code, 100000000ull);
    }
    return false;
}

// EV consecutive entries of W in shared memory (16-byte aligned when T is
// the storage type, 32-byte aligned when binary16 storage is widened to
// binary32) as 16-byte loads.
template <typename T, int EV>
__device__ __forceinline__ void load_w(const T* p, T (&v)[EV]) {
    if constexpr (sizeof(T) == 8) {
        static_assert(EV % 2 == 0, "binary64 vectors hold two entries");
#pragma unroll
        for (int e = 0; e < EV; e += 2) {
            const double2 q = *reinterpret_cast<const double2*>(p + e);
            v[e] = q.x; v[e + 1] = q.y;
        }
    } else {
        static_assert(EV % 4 == 0, "binary32 vectors hold four entries");
#pragma unroll
        for (int e = 0; e < EV; e += 4) {
            const float4 q = *reinterpret_cast<const float4*>(p + e);
            v[e] = q.x; v[e + 1] = q.y; v[e + 2] = q.z; v[e + 3] = q.w;
        }
    }
}

// 1-D bulk copy global -> shared (both 16-byte aligned, size a multiple of 16).
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(tc::smem_u32(dst)), "l"(src), "r"(bytes), "r"(tc::smem_u32(bar))
                 : "memory");
}

// ---------------------------------------------------------------- phase 1
// The fold of the last CTA of a row block: W[c][j] = s_j * sum over chunks ch
// of Wp[ch][c][j] for the block's rows j (BR of them) and every query c.
// Each entry takes G lanes (G = 256 / entries, a power of two, at most 32);
// lane g adds the chunks of its contiguous G-th of the range in chunk order,
// with 16 loads in flight, and a butterfly over the G lanes adds the G sums
// (every lane ends with the same value, in an order fixed by G: the result
// does not depend on which CTA finished last).
template <typename T, int BR>
__device__ __forceinline__ void fold_chunks(const T* __restrict__ Wp, int nchunks, int b, int k, int jb,
                                            const T* s_blk, int round16, int kv, T* __restrict__ W) {
    constexpr int kBatch = 16;
    const int E = BR * b;
    int G = 1;
    while (G < 32 && 2 * G * E <= kThreadsS) G *= 2;
    const int64_t bk = (int64_t)b * k;
    for (int t = threadIdx.x; t < ((E * G + 31) & ~31); t += kThreadsS) {
        const int e = t / G, g = t - e * G;
        const int c = e / BR, j = jb + (e - c * BR);
        const bool live = e < E && j < k;
        const int ch0 = (int)((int64_t)nchunks * g / G), ch1 = (int)((int64_t)nchunks * (g + 1) / G);
        const T* src = Wp + (int64_t)c * k + j;
        T sum = T(0);
        if (live) {
            for (int ch = ch0; ch < ch1; ch += kBatch) {
                T v[kBatch];
#pragma unroll
                for (int i = 0; i < kBatch; ++i) v[i] = (ch + i < ch1) ? __ldcg(src + (ch + i) * bk) : T(0);
#pragma unroll
                for (int i = 0; i < kBatch; ++i) sum += v[i];
            }
        }
        for (int o = G / 2; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (live && g == 0) {
            sum *= s_blk[j - jb];
            if (round16) sum = (T)__half2float(__float2half_rn((float)sum));
            W[(int64_t)c * kv + j] = sum;
        }
    }
}

// Arrival at a counter: release of this thread's (and, after a CTA barrier,
// the CTA's) earlier writes, acquire of the writes released by the earlier
// arrivals.
__device__ __forceinline__ unsigned int arrive_acq_rel(unsigned int* p) {
    unsigned int old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(p) : "memory");
    return old;
}

// Shared memory: [X boxes: nbox x B x kBox][V^T boxes: nbox x 8 RW x kBox]
// [a barrier per box pair][abort flag]; column i of the chunk is box i / kBox,
// offset i % kBox.  The boxes are multiplied in order as they land.  RW rows
// of V^T per warp.
template <typename TS, typename T, int B, int RW>
__global__ void __launch_bounds__(kThreadsS, 2)
skinny_w1_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_v, int k, int b,
                 int L, T* __restrict__ Wp, unsigned int* __restrict__ cnt, const TS* __restrict__ S, int kv,
                 int round16, T* __restrict__ W) {
    constexpr int EV = EVof<TS>::v;
    constexpr int BR = kWarps * RW;              // rows of V^T per CTA
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = align128(smem_raw);
    const int nbox = L / kBox;
    TS* xs = reinterpret_cast<TS*>(smem);
    TS* vs = xs + (size_t)nbox * B * kBox;
    uint64_t* bar = reinterpret_cast<uint64_t*>(vs + (size_t)nbox * BR * kBox);
    volatile int* abort = reinterpret_cast<volatile int*>(bar + nbox);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t chunk = blockIdx.x;
    const int32_t i0 = (int32_t)(chunk * L);
    const int jb = (int)blockIdx.y * BR;
    __shared__ int last_cta;
    __shared__ T s_blk[BR];          // s_j of the block's rows, for the fold
    tc::pdl_wait();                  // X, V^T, s and the workspace are the previous kernels'
    if (threadIdx.x < BR) s_blk[threadIdx.x] = jb + (int)threadIdx.x < k ? to_t<T>(S[jb + threadIdx.x]) : T(0);
    if (threadIdx.x == 0) {
        for (int q = 0; q < nbox; ++q) tc::mbar_init(&bar[q], 1);
        *abort = 0;
        tc::fence_barrier_init();
        for (int q = 0; q < nbox; ++q) {
            tc::mbar_arrive_expect_tx(&bar[q], (uint32_t)((B + BR) * kBox * (int)sizeof(TS)));
            tc::tma_load_2d(vs + (size_t)q * BR * kBox, &tm_v, i0 + q * kBox, jb, &bar[q]);
            tc::tma_load_2d(xs + (size_t)q * B * kBox, &tm_x, i0 + q * kBox, 0, &bar[q]);
        }
    }
    tc::pdl_trigger();               // the second product streams U meanwhile
    __syncthreads();
    const int jl = warp * RW;                 // first local row of the warp
    T acc[RW * B];                            // acc[r * B + c]: row jl + r, query c
#pragma unroll
    for (int i = 0; i < RW * B; ++i) acc[i] = T(0);
    for (int q = 0; q < nbox; ++q) {
        if (!wait_tiles(bar, q, nbox, abort, 1u)) return;
        const TS* vq = vs + ((size_t)q * BR + jl) * kBox;
        const TS* xq = xs + (size_t)q * B * kBox;
        for (int o = lane * EV; o < kBox; o += 32 * EV) {
            T vv[RW][EV];
#pragma unroll
            for (int r = 0; r < RW; ++r) load_vec<T, TS>(vq + (size_t)r * kBox + o, vv[r]);
#pragma unroll
            for (int c = 0; c < B; ++c) {
                T xv[EV];
                load_vec<T, TS>(xq + (size_t)c * kBox + o, xv);
#pragma unroll
                for (int r = 0; r < RW; ++r)
#pragma unroll
                    for (int e = 0; e < EV; ++e) acc[r * B + c] = fma(xv[e], vv[r][e], acc[r * B + c]);
            }
        }
    }
    constexpr int N = RW * B;
    halving_sum<T, N, 32>(acc, lane);
    if (halving_writer<N, 32>(lane)) {
        const int base = halving_index<N, 32>(lane);
#pragma unroll
        for (int t = 0; t < (N >= 32 ? N / 32 : 1); ++t) {
            const int idx = base + t, r = idx / B, c = idx - r * B;
            const int j = jb + jl + r;
            if (c < b && j < k) Wp[(chunk * b + c) * k + j] = acc[t];
        }
    }
    // the last CTA of this row block adds the partials of every chunk
    __syncthreads();
    if (threadIdx.x == 0) last_cta = arrive_acq_rel(&cnt[blockIdx.y]) == gridDim.x - 1;
    __syncthreads();
    if (!last_cta) return;
    fold_chunks<T, BR>(Wp, (int)gridDim.x, b, k, jb, s_blk, round16, kv, W);
    if (blockIdx.y == gridDim.y - 1)             // the zero columns k .. kv-1 of W
        for (int e = threadIdx.x; e < b * (kv - k); e += kThreadsS) {
            const int c = e / (kv - k);
            W[(int64_t)c * kv + k + (e - c * (kv - k))] = T(0);
        }
    if (threadIdx.x == 0) cnt[blockIdx.y] = 0u;
}

// ---------------------------------------------------------------- phase 2
// A CTA owns 16 RPG rows of U, in groups of G lanes (G = 8, or 32 for at
// most 4 queries, where the work per row is short and a longer reduction
// across lanes costs less than a longer loop): each group takes RPG rows, a
// lane covers every G-th 16-byte column of its rows (the rank is only a few
// hundred); G / 2 warps.  Shared memory: [U: nkb boxes of 16 RPG rows x kbw]
// [W: B x kv][barrier of U][barrier of W][abort flag]; column j of U is box
// j / kbw, offset j % kbw; kv = nkb * kbw.  One thread waits for the copies
// (the CTA may be resident while the first kernel still runs: the other
// warps sleep at the CTA barrier instead of polling).
template <int G>
constexpr int y_warps() { return G / 2; }
template <typename TS, typename T, typename TOut, int B, int RPG, int G>
__global__ void __launch_bounds__(32 * y_warps<G>())
skinny_y_kernel(const __grid_constant__ CUtensorMap tm_u, const T* __restrict__ W, int64_t m, int b, int nkb,
                int kbw, unsigned int* __restrict__ cnt, int ncnt, TOut* __restrict__ Y) {
    constexpr int EV = EVof<TS>::v;
    constexpr int NT = 32 * y_warps<G>();
    constexpr int RC = y_warps<G>() * (32 / G) * RPG;       // rows of the CTA (16 RPG)
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = align128(smem_raw);
    const int kv = nkb * kbw;
    TS* us = reinterpret_cast<TS*>(smem);
    T* ws = reinterpret_cast<T*>(us + (size_t)nkb * RC * kbw);
    uint64_t* bar = reinterpret_cast<uint64_t*>(ws + (size_t)B * kv);
    volatile int* abort = reinterpret_cast<volatile int*>(bar + 2);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t rb = (int64_t)blockIdx.x * RC;
    const uint32_t w_bytes = (uint32_t)((size_t)b * kv * sizeof(T));
    // rows b..B-1 of W are zero (disjoint from the bulk copy of rows 0..b-1)
    for (int e = b * kv + threadIdx.x; e < B * kv; e += NT) ws[e] = T(0);
    if (threadIdx.x == 0) {
        tc::mbar_init(&bar[0], 1);
        tc::mbar_init(&bar[1], 1);
        *abort = 0;
        tc::fence_barrier_init();
        tc::mbar_arrive_expect_tx(&bar[0], (uint32_t)(nkb * RC * kbw * (int)sizeof(TS)));
        for (int q = 0; q < nkb; ++q)
            tc::tma_load_2d(us + (size_t)q * RC * kbw, &tm_u, q * kbw, (int32_t)rb, &bar[0]);
        tc::pdl_wait();              // W of the first kernel
        // leave the first kernel's counters at zero for the next call, also
        // after an aborted first kernel whose CTAs did not all arrive
        if (blockIdx.x == 0)
            for (int i = 0; i < ncnt; ++i) cnt[i] = 0u;
        tc::mbar_arrive_expect_tx(&bar[1], w_bytes);
        bulk_load(ws, W, w_bytes, &bar[1]);
        if (!(tc::mbar_wait(&bar[1], 0, abort, &g_err_skinny, 2u) &&
              tc::mbar_wait(&bar[0], 0, abort, &g_err_skinny, 2u))) {
            // no copy may still be landing when the CTA exits
            volatile int no_abort = 0;
            for (int i = 0; i < 2; ++i) tc::mbar_wait(&bar[i], 0, &no_abort, &g_err_skinny, 2u, 100000000ull);
            *abort = 1;
        }
    }
    tc::pdl_trigger();               // the next call's first kernel may set up
    __syncthreads();
    if (*abort) return;
    const int sl = lane & (G - 1);
    const int rl = (warp * (32 / G) + (lane / G)) * RPG;
    constexpr int N = RPG * B;
    T acc[N];                                    // acc[r * B + c]: row rl + r, query c
#pragma unroll
    for (int i = 0; i < N; ++i) acc[i] = T(0);
    for (int v = sl; v < kv / EV; v += G) {
        const int j = v * EV, q = j / kbw, o = j - q * kbw;
        T uu[RPG][EV];
#pragma unroll
        for (int r = 0; r < RPG; ++r) load_vec<T, TS>(us + ((size_t)q * RC + rl + r) * kbw + o, uu[r]);
#pragma unroll
        for (int c = 0; c < B; ++c) {
            T wv[EV];
            load_w(ws + (size_t)c * kv + j, wv);
#pragma unroll
            for (int r = 0; r < RPG; ++r)
#pragma unroll
                for (int e = 0; e < EV; ++e) acc[r * B + c] = fma(wv[e], uu[r][e], acc[r * B + c]);
        }
    }
    halving_sum<T, N, G>(acc, lane);
    const int64_t r0 = rb + rl;
    if (halving_writer<N, G>(lane)) {
        const int base = halving_index<N, G>(lane);
#pragma unroll
        for (int t = 0; t < (N >= G ? N / G : 1); ++t) {
            const int idx = base + t, r = idx / B, c = idx - r * B;
            if (c < b && r0 + r < m) store_out(Y + (int64_t)c * m + r0 + r, acc[t]);
        }
    }
}

// lanes per row group of the second product (binary64 stays at 8: its
// multiply-adds, not the latency of the chain, bound it)
constexpr int y_group(int B, int64_t e) { return (B <= 4 && e < 8) ? 32 : 8; }

template <typename TS>
constexpr int y_rpg() { return sizeof(TS) == 8 ? 2 : 4; }

// rows of V^T per warp in the first product: 4, or 2 for 16 binary64 queries
// (64 binary64 accumulators a thread would spill)
constexpr int w1_rows(int B, int64_t e) { return (B == 16 && e == 8) ? 2 : kRows; }

template <typename TS>
CUtensorMapDataType map_type() {
    if constexpr (sizeof(TS) == 2) return CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
    else if constexpr (sizeof(TS) == 4) return CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    else return CU_TENSOR_MAP_DATA_TYPE_FLOAT64;
}

// Launch plan of one size: chunk length of the first product, boxes of the
// second, shared memory of both.
struct SkinnyPlan {
    int64_t L, nchunks, jblocks, nkb, kbw, kv, yblocks;
    size_t smem1, smem3;
};

SkinnyPlan plan_skinny(int64_t m, int64_t n, int64_t k, int B, int64_t e, int64_t et) {
    const int64_t br = kWarps * (int64_t)w1_rows(B, e);
    SkinnyPlan p{};
    const int64_t ev = 16 / e;
    // chunk length: a multiple of kBox with the CTA's tiles within the
    // shared-memory budget (two CTAs per SM), and enough chunks for two CTAs
    // per SM
    p.jblocks = (k + br - 1) / br;
    int64_t L = (int64_t)(kSmemW1 / (size_t)((B + br) * e)) / kBox * kBox;
    if (L < kBox) L = kBox;
    const int64_t want = (2 * (int64_t)sm_count() + p.jblocks - 1) / p.jblocks;
    int64_t Lw = (n + want - 1) / want;
    Lw = (Lw + kBox - 1) / kBox * kBox;
    if (Lw < L) L = Lw;
    p.L = L;
    p.nchunks = (n + L - 1) / L;
    // second product: U in nkb boxes of kbw columns (kbw a multiple of the
    // 16-byte vector, at most 256)
    p.nkb = (k + 255) / 256;
    p.kbw = ((k + p.nkb - 1) / p.nkb + ev - 1) / ev * ev;
    p.kv = p.nkb * p.kbw;
    p.smem1 = (size_t)(L / kBox) * (B + br) * kBox * e + 8 * (size_t)(L / kBox + 1) + 128;
    // second product: CTAs of 16 RPG rows of U
    const int64_t rc = 16 * (int64_t)(e == 8 ? 2 : 4);
    p.yblocks = (m + rc - 1) / rc;
    p.smem3 = (size_t)p.nkb * rc * p.kbw * e + (size_t)B * p.kv * et + 24 + 128;
    return p;
}

template <typename TS, typename T, typename TOut, int B>
lrc_status launch_skinny_b(const TS* U, const TS* S, const TS* Vt, const TS* X, TOut* Y, int64_t m, int64_t n,
                           int64_t k, int64_t b, bool round16, cudaStream_t s) {
    const int64_t ldn = lrc_packed_ld(n), ldk = lrc_packed_ld(k);
    const int64_t e = (int64_t)sizeof(TS);
    const SkinnyPlan p = plan_skinny(m, n, k, B, e, (int64_t)sizeof(T));
    int64_t t;
    if (!mul_ok(p.nchunks * b, k, &t) || p.nchunks > 65535 || p.jblocks > kStreamCounters || n > INT32_MAX ||
        m > INT32_MAX || p.smem1 > kSmemMaxS || p.smem3 > kSmemMaxS) {
        set_error("small-batch apply: problem outside the kernel");
        return LRC_ERR_UNSUPPORTED;
    }
    const size_t part_bytes = ((size_t)p.nchunks * b * k * sizeof(T) + 255) / 256 * 256;
    const size_t w_bytes = (size_t)b * p.kv * sizeof(T);
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, part_bytes + w_bytes, &ws);
    if (st != LRC_OK) return st;
    unsigned int* cnt = nullptr;
    if ((st = stream_counters(s, &cnt)) != LRC_OK) return st;
    T* Wp = static_cast<T*>(ws);
    T* Wd = reinterpret_cast<T*>(static_cast<unsigned char*>(ws) + part_bytes);

    CUtensorMap tx, tv, tu;
    if ((st = encode_map_2d(&tx, map_type<TS>(), X, n, b, ldn * e, kBox, B, false, "X")) != LRC_OK) return st;
    constexpr int RW = w1_rows(B, (int64_t)sizeof(TS));
    if ((st = encode_map_2d(&tv, map_type<TS>(), Vt, n, k, ldn * e, kBox, kWarps * RW, false, "Vt")) != LRC_OK)
        return st;
    constexpr int kRowsY = 16 * y_rpg<TS>();
    if ((st = encode_map_2d(&tu, map_type<TS>(), U, k, m, ldk * e, (uint32_t)p.kbw, kRowsY, false, "U")) != LRC_OK)
        return st;

    cudaError_t ce = cudaFuncSetAttribute(skinny_w1_kernel<TS, T, B, RW>,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem1);
    if (ce != cudaSuccess) return cuda_fail(ce, "skinny_w1_kernel smem attribute");
    ce = launch_pdl(skinny_w1_kernel<TS, T, B, RW>, dim3((unsigned)p.nchunks, (unsigned)p.jblocks), dim3(kThreadsS),
                    p.smem1, s, tx, tv, (int)k, (int)b, (int)p.L, Wp, cnt, S, (int)p.kv, round16 ? 1 : 0, Wd);
    if (ce != cudaSuccess) return cuda_fail(ce, "skinny_w1_kernel launch");
    if ((st = after_launch("skinny_w1_kernel")) != LRC_OK) return st;
    constexpr int G = y_group(B, (int64_t)sizeof(TS));
    auto ykernel = skinny_y_kernel<TS, T, TOut, B, y_rpg<TS>(), G>;
    ce = cudaFuncSetAttribute(ykernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem3);
    if (ce != cudaSuccess) return cuda_fail(ce, "skinny_y_kernel smem attribute");
    ce = launch_pdl(ykernel, dim3((unsigned)p.yblocks), dim3(32 * y_warps<G>()), p.smem3, s, tu, (const T*)Wd, m, (int)b,
                    (int)p.nkb, (int)p.kbw, cnt, (int)p.jblocks, Y);
    if (ce != cudaSuccess) return cuda_fail(ce, "skinny_y_kernel launch");
    return after_launch("skinny_y_kernel");
}

template <typename TS, typename T, typename TOut>
lrc_status launch_skinny_t(const TS* U, const TS* S, const TS* Vt, const TS* X, TOut* Y, int64_t m, int64_t n,
                           int64_t k, int64_t b, bool round16, cudaStream_t s) {
    if (b <= 1) return launch_skinny_b<TS, T, TOut, 1>(U, S, Vt, X, Y, m, n, k, b, round16, s);
    if (b <= 4) return launch_skinny_b<TS, T, TOut, 4>(U, S, Vt, X, Y, m, n, k, b, round16, s);
    if constexpr (sizeof(TS) != 2)
        if (b <= 8) return launch_skinny_b<TS, T, TOut, 8>(U, S, Vt, X, Y, m, n, k, b, round16, s);
    if constexpr (sizeof(TS) != 2) return launch_skinny_b<TS, T, TOut, 16>(U, S, Vt, X, Y, m, n, k, b, round16, s);
    set_error("small-batch apply: b = %lld above the kernel's batch", (long long)b);
    return LRC_ERR_UNSUPPORTED;
}

int64_t max_batch(lrc_fmt fmt) { return fmt == LRC_F16 || fmt == LRC_F16_O16 ? 4 : 16; }

}  // namespace

// Batches this path takes: up to 16 queries for binary32 and binary64, up
// to 4 for binary16 (whose tensor-core path is faster from 16 queries on);
// ranks whose tiles fit in shared memory.
bool apply_skinny_takes(lrc_fmt fmt, int64_t b, int64_t k) {
    if (fmt == LRC_BF16) return false;    // bfloat16 takes the tensor-core path at every batch size
    if (b < 1 || b > max_batch(fmt) || k < 1 || k > 1024) return false;
    const int B = b <= 1 ? 1 : (b <= 4 ? 4 : (b <= 8 ? 8 : 16));
    const int64_t e = storage_bytes(fmt);
    const SkinnyPlan p = plan_skinny(1, 1, k, B, e, fmt == LRC_F64 ? 8 : 4);
    return p.smem1 <= kSmemMaxS && p.smem3 <= kSmemMaxS;
}

lrc_status launch_apply_skinny(const void* U, const void* S, const void* Vt, const void* X, void* Y, int64_t m,
                               int64_t n, int64_t k, int64_t b, lrc_fmt fmt, cudaStream_t s) {
    if (!apply_skinny_takes(fmt, b, k)) {
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

uint32_t take_skinny_error() {
    unsigned int v = 0;
    if (cudaMemcpyFromSymbol(&v, g_err_skinny, sizeof v) != cudaSuccess) return 0xffffffffu;
    if (v) {
        const unsigned int z = 0;
        cudaMemcpyToSymbol(g_err_skinny, &z, sizeof z);
    }
    return v;
}

}  // namespace lrc
