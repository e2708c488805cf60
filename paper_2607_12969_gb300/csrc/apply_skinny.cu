// apply_skinny.cu -- low-rank apply for small batches (Sec. 4.4, Eq.
// gpu_matrix_apply: Y = [(X V) diag(s)] U^T): at most 16 queries in every
// format on the CUDA cores, and up to 64 queries in binary16 and bfloat16 on
// the tensor cores (the second half of the file).
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

#include <algorithm>

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

// ---------------------------------------------------------------- 16-bit storage on the tensor cores
// Batches of at most 64 queries in binary16 and bfloat16: the b
// multiply-adds per factor element would bound the CUDA-core loops, so both
// products run as tcgen05 MMAs whose N is the query
// count padded to NB (16, 32 or 64; twice that in the second product for
// FP32 output, whose hi and lo planes of W sit side by side along N) and
// whose M is 128 ranks (first product) or 128 rows of U (second).
//   skinny_tc_w_kernel  grid (chunk of n, tile of 128 ranks) in clusters of
//                       kTcCluster chunks.  The CTA copies its chunk of V^T
//                       (128 ranks x cb k-blocks) and of X (the b rows,
//                       zero-filled to NB) at once, multiplies
//                       W^T = V^T X^T into one tensor-memory accumulator
//                       (at most 8 k-blocks: the accumulation length of the
//                       chunked FP32 accumulation) and stages it in shared
//                       memory; every CTA of the cluster then adds, for an
//                       eighth of the entries, the kTcCluster partials in
//                       rank order through distributed shared memory and
//                       writes that part of the cluster partial (W itself
//                       when a rank tile has one cluster).  The last
//                       cluster of a rank tile to arrive (a counter) adds
//                       the cluster partials in cluster order, scales by
//                       diag(s) and writes W as the second product's operand
//                       planes: hi and lo binary16 for FP32 output (w = hi +
//                       lo to about 22 bits), one rounding for 16-bit
//                       output, laid out as the second product's shared
//                       memory image (k-blocks of NB rows x 128 bytes in the
//                       128-byte swizzle, the lo box after the hi box).
//   skinny_tc_y_kernel  a CTA per 128 rows of U: the U tile is requested
//                       before the wait for the first kernel (U is an input
//                       of the call), W after it (one bulk copy of the
//                       image); D = U_tile W^T holds the
//                       tile's outputs for every query (FP32 output: the hi
//                       and lo halves of D added in binary32), and each
//                       query's 128 outputs are one coalesced run of stores.
// Fixed summation orders (tensor core within a chunk, cluster rank, cluster
// index): results are reproducible on a device.
constexpr int kTcK = 64;                         // 16-bit elements per 128-byte swizzled row
constexpr int kTcM = 128;                        // MMA rows
constexpr int kTcCluster = 8;                    // chunks of n per cluster
constexpr int kTcMaxChunks = 64;                 // chunks of n per rank tile, at most
constexpr int kTcMaxBatch = 64;                  // queries, at most
constexpr int kTcThreadsW = 512;
constexpr int kTcThreadsY = 128;
constexpr uint32_t kTcABytes = kTcM * kTcK * 2;  // one 128-row operand box

__device__ __forceinline__ unsigned char* align1024(unsigned char* p) {
    return p + ((1024u - (tc::smem_u32(p) & 1023u)) & 1023u);
}

__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Every thread of every CTA of the cluster: shared-memory writes before it
// are visible to the cluster's reads after it.
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// 16 bytes of the shared memory of cluster CTA `rank` at the offset of the
// local shared address `addr`.
__device__ __forceinline__ float4 ld_cluster4(uint32_t addr, uint32_t rank) {
    uint32_t ra;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(addr), "r"(rank));
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(ra)
                 : "memory");
    return v;
}

__device__ __forceinline__ float4 add4(float4 a, float4 b) {
    return make_float4(__fadd_rn(a.x, b.x), __fadd_rn(a.y, b.y), __fadd_rn(a.z, b.z), __fadd_rn(a.w, b.w));
}

// W entries (q, j0..j0+3) = s_j * sum, rounded (hi and lo binary16 for FP32
// output, one rounding otherwise) into the second product's swizzled image:
// the 4 ranks lie in 16-byte chunk (j0 % 64) / 8 of a 128-byte row of
// k-block j0 / 64, the lo box right after the hi box.
template <int NB>
__device__ __forceinline__ void emit_w(unsigned char* W, int planes, int bf16, int q, int j0, float4 sum,
                                       const float (&sj)[4]) {
    const float w[4] = {__fmul_rn(sum.x, sj[0]), __fmul_rn(sum.y, sj[1]), __fmul_rn(sum.z, sj[2]),
                        __fmul_rn(sum.w, sj[3])};
    uint16_t hi[4], lo[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        if (bf16) {
            hi[i] = tc::to_bf16_bits(w[i]);
        } else {
            const __half h = __float2half_rn(w[i]);
            hi[i] = __half_as_ushort(h);
            lo[i] = __half_as_ushort(__float2half_rn(w[i] - __half2float(h)));
        }
    }
    const int kblk = j0 >> 6, ch = (j0 & 63) >> 3, within = (j0 & 7) * 2;
    unsigned char* dst = W + ((size_t)kblk * planes * NB + q) * 128 + ((ch ^ (q & 7)) << 4) + within;
    *reinterpret_cast<uint2*>(dst) = make_uint2(hi[0] | ((uint32_t)hi[1] << 16), hi[2] | ((uint32_t)hi[3] << 16));
    if (planes == 2)
        *reinterpret_cast<uint2*>(dst + NB * 128) =
            make_uint2(lo[0] | ((uint32_t)lo[1] << 16), lo[2] | ((uint32_t)lo[3] << 16));
}

// s_j for the 4 ranks j0..j0+3 (0 from rank k on)
__device__ __forceinline__ void load_s4(const uint16_t* S, int k, int bf16, int j0, float (&sj)[4]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int j = j0 + i;
        sj[i] = 0.0f;
        if (j < k) sj[i] = bf16 ? tc::bf16_bits_to_float(S[j]) : __half2float(__ushort_as_half(S[j]));
    }
}

struct TcWArgs {
    int k, kp, b, nkb, cb, nclusters;
    int planes;               // W planes: 2 (hi and lo, FP32 output) or 1
    int bf16;                 // bfloat16 storage and W
    uint32_t idesc;           // MMA instruction descriptor
    uint32_t bar_off;         // barriers after the tile / fold region
    const uint16_t* S;
    float* P;                 // cluster partials [rank tile][cluster][NB queries][128 ranks]
    unsigned char* W;         // W image: [k-block][plane][NB rows x 128 bytes, 128-byte swizzle]
    unsigned int* cnt;        // an arrival counter per rank tile
};

// Shared memory: [region: cb V^T boxes, cb X boxes; later the staged partial
// (NB x 128 binary32, [query][rank])][cb + 1 barriers][tensor-memory address]
// [abort flag].
template <int NB>
__global__ void __launch_bounds__(kTcThreadsW, 1)
skinny_tc_w_kernel(const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_x, const TcWArgs a) {
    constexpr uint32_t kXBytes = NB * kTcK * 2;
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = align1024(smem_raw);
    unsigned char* vs = smem;
    unsigned char* xs = smem + (size_t)a.cb * kTcABytes;
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + a.bar_off);
    uint64_t* mma_done = full + a.cb;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
    __shared__ int last_cluster;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int chunk = blockIdx.x, rt = blockIdx.y;
    const int kb0 = chunk * a.cb;
    const int nb = a.nkb - kb0 < a.cb ? (a.nkb - kb0 > 0 ? a.nkb - kb0 : 0) : a.cb;
    if (threadIdx.x == 0) {
        for (int i = 0; i < a.cb + 1; ++i) tc::mbar_init(&full[i], 1);
        *abort = 0;
        tc::fence_barrier_init();
        tc::tma_prefetch_desc(&tm_v);
        tc::tma_prefetch_desc(&tm_x);
    }
    constexpr uint32_t kCols = NB < 32 ? 32u : (uint32_t)NB;
    if (warp == 1) tc::tmem_alloc(tmem_slot, kCols);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    tc::pdl_wait();                  // X, V^T, s and the workspace are the previous kernels'
    if (threadIdx.x == 0)
        for (int i = 0; i < nb; ++i) {
            tc::mbar_arrive_expect_tx(&full[i], kTcABytes + kXBytes);
            const int32_t x = (kb0 + i) * kTcK;
            tc::tma_load_2d(vs + (size_t)i * kTcABytes, &tm_v, x, rt * kTcM, &full[i]);
            tc::tma_load_2d(xs + (size_t)i * kXBytes, &tm_x, x, 0, &full[i]);
        }
    tc::pdl_trigger();               // the second product streams U meanwhile
    if (threadIdx.x == 0) {
        int i = 0;
        for (; i < nb; ++i) {
            if (!tc::mbar_wait(&full[i], 0, abort, &g_err_skinny, 8u)) break;
            tc::tc_fence_after();
            const uint64_t dv = tc::desc_sw128(tc::smem_u32(vs + (size_t)i * kTcABytes));
            const uint64_t dx = tc::desc_sw128(tc::smem_u32(xs + (size_t)i * kXBytes));
#pragma unroll
            for (int kk = 0; kk < kTcK / 16; ++kk)
                tc::mma_f16(tmem, dv + 2 * kk, dx + 2 * kk, a.idesc, (i | kk) != 0 ? 1u : 0u);
        }
        tc::mma_commit(mma_done);    // also after a give-up: the MMAs issued finish first
        volatile int no_abort = 0;
        tc::mbar_wait(mma_done, 0, &no_abort, &g_err_skinny, 8u, 100000000ull);
        for (int j = i; j < nb; ++j)  // copies still landing
            tc::mbar_wait(&full[j], 0, &no_abort, &g_err_skinny, 8u, 100000000ull);
    }
    __syncwarp();
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    // the partial, staged as [query][rank] (the operand boxes are no longer read)
    float* stage = reinterpret_cast<float*>(smem);
    if (warp < 4) {
        const int r = warp * 32 + lane;
#pragma unroll
        for (int c0 = 0; c0 < NB; c0 += 32) {
            uint32_t v[32];
            tc::tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c0, v);
            tc::tmem_ld_wait();
#pragma unroll
            for (int q = 0; q < (NB < 32 ? NB : 32); ++q)
                stage[(c0 + q) * kTcM + r] = nb > 0 ? __uint_as_float(v[q]) : 0.0f;
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, kCols);
    }
    __syncwarp();
    cluster_sync();                  // every partial of the cluster is staged
    // The cluster partial: CTA j of the cluster adds, for its eighth of the
    // (query, 4 ranks) entries, the kTcCluster staged partials in rank order.
    // With a single cluster a rank tile (n up to 8 chunks) that sum is the
    // whole reduction: the CTAs write their W entries themselves.
    const int cl = chunk / kTcCluster;
    const int crank = (int)cluster_ctarank();
    const int n4 = a.b * (kTcM / 4);
    const int ranks = a.kp - rt * kTcM < kTcM ? a.kp - rt * kTcM : kTcM;
    float4* cp = reinterpret_cast<float4*>(a.P + ((size_t)rt * a.nclusters + cl) * NB * kTcM);
    for (int e = n4 * crank / kTcCluster + (int)threadIdx.x; e < n4 * (crank + 1) / kTcCluster;
         e += kTcThreadsW) {
        const uint32_t addr = tc::smem_u32(stage) + 16u * (uint32_t)e;
        float4 v[kTcCluster];
#pragma unroll
        for (int r = 0; r < kTcCluster; ++r) v[r] = ld_cluster4(addr, (uint32_t)r);
        float4 sum = v[0];
#pragma unroll
        for (int r = 1; r < kTcCluster; ++r) sum = add4(sum, v[r]);
        if (a.nclusters > 1) {
            cp[e] = sum;
        } else {
            const int q = e / (kTcM / 4), r4 = (e - q * (kTcM / 4)) * 4;
            if (r4 < ranks) {
                float sj[4];
                load_s4(a.S, a.k, a.bf16, rt * kTcM + r4, sj);
                emit_w<NB>(a.W, a.planes, a.bf16, q, rt * kTcM + r4, sum, sj);
            }
        }
    }
    __syncwarp();
    cluster_sync();                  // the staged partials stay until every CTA has read them
    if (crank != 0 || a.nclusters == 1) return;
    // the cluster's first CTA arrives for the cluster (the cluster barrier
    // ordered the other CTAs' partial stores before this release)
    if (threadIdx.x == 0) last_cluster = arrive_acq_rel(&a.cnt[rt]) == (unsigned)(a.nclusters - 1);
    __syncthreads();
    if (!last_cluster) return;
    // The rank tile's cluster partials added in cluster order, scaled by
    // diag(s), written as W.  Thread t takes ranks 4 (t % 32) .. + 3 of
    // queries t / 32, t / 32 + 16, ...
    const int r4 = (int)(threadIdx.x & 31) * 4;
    if (r4 >= ranks) return;                       // ranks is a multiple of 16
    const int j0 = rt * kTcM + r4;
    float sj[4];
    load_s4(a.S, a.k, a.bf16, j0, sj);
    const float4* src = reinterpret_cast<const float4*>(a.P + (size_t)rt * a.nclusters * NB * kTcM);
    constexpr int kC4 = NB * kTcM / 4;             // float4 per cluster partial
    auto emit = [&](int q, float4 sum) { emit_w<NB>(a.W, a.planes, a.bf16, q, j0, sum, sj); };
    constexpr int kQStep = kTcThreadsW / 32;       // queries a pass of the CTA takes
    const int q0 = (int)(threadIdx.x >> 5);
    if (NB > kQStep && a.nclusters <= 4) {
        // several queries a thread: every load of the thread in flight at once
        constexpr int kQ = NB > kQStep ? NB / kQStep : 1;
        float4 v[kQ][4];
#pragma unroll
        for (int i = 0; i < kQ; ++i)
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int q = q0 + i * kQStep;
                v[i][c] = (q < a.b && c < a.nclusters)
                              ? __ldcg(src + (size_t)c * kC4 + q * (kTcM / 4) + (r4 >> 2))
                              : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
        for (int i = 0; i < kQ; ++i) {
            const int q = q0 + i * kQStep;
            if (q >= a.b) break;
            float4 sum = v[i][0];
#pragma unroll
            for (int c = 1; c < 4; ++c)
                if (c < a.nclusters) sum = add4(sum, v[i][c]);
            emit(q, sum);
        }
        return;
    }
    for (int q = q0; q < a.b; q += kQStep) {
        const int e = q * (kTcM / 4) + (r4 >> 2);
        float4 v[kTcMaxChunks / kTcCluster];
#pragma unroll
        for (int c = 0; c < kTcMaxChunks / kTcCluster; ++c)
            v[c] = c < a.nclusters ? __ldcg(src + (size_t)c * kC4 + e) : make_float4(0.f, 0.f, 0.f, 0.f);
        float4 sum = v[0];
#pragma unroll
        for (int c = 1; c < kTcMaxChunks / kTcCluster; ++c)
            if (c < a.nclusters) sum = add4(sum, v[c]);
        emit(q, sum);
    }
}

struct TcYArgs {
    int64_t m;
    int b, kp, kc, planes, rtiles;
    int out16, bf16;          // 16-bit output (bfloat16 when bf16)
    uint32_t idesc;
    unsigned int* cnt;        // the first kernel's counters, left at zero for the next call
    const unsigned char* W;   // the first kernel's W image (rows b..NB-1 unused: their D columns are not stored)
    void* Y;
};

// Shared memory: [U: kc boxes of 128 rows][W: kc x planes boxes of NB rows,
// the lo box of a k-block right after its hi box, so that the two form one
// B operand of planes x NB rows: D = [U W_hi^T | U W_lo^T]]
// [3 barriers][tensor-memory address][abort flag].
template <int NB>
__global__ void __launch_bounds__(kTcThreadsY, 1)
skinny_tc_y_kernel(const __grid_constant__ CUtensorMap tm_u, const TcYArgs a) {
    constexpr uint32_t kWBytes = NB * kTcK * 2;
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = align1024(smem_raw);
    unsigned char* us = smem;
    unsigned char* ws = smem + (size_t)a.kc * kTcABytes;
    uint64_t* bar = reinterpret_cast<uint64_t*>(ws + (size_t)a.planes * a.kc * kWBytes);   // U, W, MMA
    const uint32_t tcols = a.planes * NB <= 32 ? 32u : (uint32_t)(a.planes * NB);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bar + 3);
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t row0 = (int64_t)blockIdx.x * kTcM;
    if (threadIdx.x == 0) {
        for (int i = 0; i < 3; ++i) tc::mbar_init(&bar[i], 1);
        *abort = 0;
        tc::fence_barrier_init();
        tc::tma_prefetch_desc(&tm_u);
        tc::mbar_arrive_expect_tx(&bar[0], (uint32_t)a.kc * kTcABytes);
        for (int i = 0; i < a.kc; ++i) tc::tma_load_2d(us + (size_t)i * kTcABytes, &tm_u, i * kTcK, (int32_t)row0, &bar[0]);
    }
    if (warp == 1) tc::tmem_alloc(tmem_slot, tcols);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    tc::pdl_trigger();               // the next call's first kernel may set up
    if (threadIdx.x == 0) {
        tc::pdl_wait();              // W of the first kernel
        if (blockIdx.x == 0)         // also after an aborted first kernel
            for (int i = 0; i < a.rtiles; ++i) a.cnt[i] = 0u;
        const uint32_t w_bytes = (uint32_t)(a.planes * a.kc) * kWBytes;
        tc::mbar_arrive_expect_tx(&bar[1], w_bytes);
        tc::bulk_load(ws, a.W, w_bytes, &bar[1]);
        const bool ok = tc::mbar_wait(&bar[0], 0, abort, &g_err_skinny, 32u) &&
                        tc::mbar_wait(&bar[1], 0, abort, &g_err_skinny, 32u);
        if (ok) {
            tc::tc_fence_after();
            for (int i = 0; i < a.kc; ++i) {
                const uint64_t du = tc::desc_sw128(tc::smem_u32(us + (size_t)i * kTcABytes));
                const uint64_t dw = tc::desc_sw128(tc::smem_u32(ws + (size_t)i * a.planes * kWBytes));
#pragma unroll
                for (int kk = 0; kk < kTcK / 16; ++kk) {
                    if ((i * kTcK + kk * 16) >= a.kp) break;
                    tc::mma_f16(tmem, du + 2 * kk, dw + 2 * kk, a.idesc, (i | kk) != 0 ? 1u : 0u);
                }
            }
        }
        tc::mma_commit(&bar[2]);
        volatile int no_abort = 0;
        tc::mbar_wait(&bar[2], 0, &no_abort, &g_err_skinny, 32u, 100000000ull);
        if (!ok)                     // no copy may still be landing when the CTA exits
            for (int i = 0; i < 2; ++i) tc::mbar_wait(&bar[i], 0, &no_abort, &g_err_skinny, 32u, 100000000ull);
    }
    __syncwarp();
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    if (!*abort) {
        // columns 0..NB-1: U W_hi^T (or U W^T); NB..2 NB-1: U W_lo^T; 32 queries at a time
        const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
        const int64_t row = row0 + warp * 32 + lane;
#pragma unroll 1
        for (int c0 = 0; c0 < NB && c0 < a.b; c0 += 32) {
        uint32_t v[32], vl[32];
        tc::tmem_ld32(tl + (uint32_t)c0, v);
        if constexpr (NB >= 32)
            if (a.planes == 2) tc::tmem_ld32(tl + (uint32_t)(NB + c0), vl);
        tc::tmem_ld_wait();
        if (row < a.m) {
#pragma unroll
            for (int qq = 0; qq < (NB < 32 ? NB : 32); ++qq) {
                const int q = c0 + qq;
                if (q >= a.b) break;
                float y = __uint_as_float(v[qq]);
                if (a.planes == 2) {
                    if constexpr (NB >= 32) y = __fadd_rn(y, __uint_as_float(vl[qq]));
                    else y = __fadd_rn(y, __uint_as_float(v[NB + qq]));
                }
                if (!a.out16) {
                    static_cast<float*>(a.Y)[(int64_t)q * a.m + row] = y;
                } else {
                    const uint16_t h = a.bf16 ? tc::to_bf16_bits(y) : __half_as_ushort(__float2half_rn(y));
                    static_cast<uint16_t*>(a.Y)[(int64_t)q * a.m + row] = h;
                }
            }
        }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, tcols);
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

// Plan of the tensor-core variant: k-blocks per chunk (at most 8, at most
// kTcMaxChunks chunks), clusters, shared memory of both kernels.
struct TcPlan {
    int kp, kc, rtiles, nkb, cb, nchunks, nclusters, planes;
    size_t region, smem1, smem3;
};

TcPlan plan_skinny_tc(int64_t n, int64_t k, int64_t b, int NB, bool fp32_out) {
    TcPlan p{};
    p.kp = (int)((k + 15) / 16 * 16);
    p.kc = (p.kp + kTcK - 1) / kTcK;
    p.rtiles = (p.kp + kTcM - 1) / kTcM;
    p.nkb = (int)((n + kTcK - 1) / kTcK);
    // fewer, longer chunks above 4 queries: the folds read chunks x b x 128
    // entries a rank tile (m = n = 16384, k' = 272: b = 64 17.4 -> 15.3 us
    // with 32 chunks instead of 64; b = 1 10.4 against 10.6 us)
    const int want = b <= 4 ? kTcMaxChunks : kTcMaxChunks / 2;
    p.cb = (p.nkb + want - 1) / want;
    if (p.cb < 1) p.cb = 1;
    if (p.cb > 8) p.cb = (p.nkb + kTcMaxChunks - 1) / kTcMaxChunks;   // at most 8 k-blocks a chunk
    p.nchunks = (p.nkb + p.cb - 1) / p.cb;
    p.nclusters = (p.nchunks + kTcCluster - 1) / kTcCluster;
    p.planes = fp32_out ? 2 : 1;
    size_t region = (size_t)p.cb * (kTcABytes + (size_t)NB * kTcK * 2);
    region = std::max(region, (size_t)NB * kTcM * 4);                       // the staged partial
    p.region = (region + 15) / 16 * 16;
    p.smem1 = 1024 + p.region + 8 * (size_t)(p.cb + 1) + 16;
    p.smem3 = 1024 + (size_t)p.kc * kTcABytes + (size_t)p.planes * p.kc * NB * kTcK * 2 + 3 * 8 + 16;
    return p;
}

// MMA width (queries) for b queries
int tc_width(int64_t b) { return b <= 16 ? 16 : (b <= 32 ? 32 : 64); }

bool skinny_tc_takes(lrc_fmt fmt, int64_t m, int64_t n, int64_t k, int64_t b) {
    if (fmt != LRC_F16 && fmt != LRC_F16_O16 && fmt != LRC_BF16) return false;
    if (b < 1 || b > kTcMaxBatch || k < 1 || k > 512 || n < 1 || m < 1 || m > INT32_MAX) return false;
    if ((n + kTcK - 1) / kTcK > 8 * kTcMaxChunks) return false;     // at most 8 k-blocks per chunk
    const TcPlan p = plan_skinny_tc(n, k, b, tc_width(b), fmt == LRC_F16);
    return p.smem1 <= kSmemMaxS && p.smem3 <= kSmemMaxS;
}

template <int NB>
lrc_status launch_skinny_tc_nb(const void* U, const void* S, const void* Vt, const void* X, void* Y, int64_t m,
                               int64_t n, int64_t k, int64_t b, lrc_fmt fmt, cudaStream_t s) {
    const bool bf16 = fmt == LRC_BF16;
    const TcPlan p = plan_skinny_tc(n, k, b, NB, fmt == LRC_F16);
    const size_t part_bytes = ((size_t)p.rtiles * p.nclusters * NB * kTcM * 4 + 255) / 256 * 256;
    const size_t w_bytes = (size_t)p.planes * p.kc * NB * 128;     // the W image
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, part_bytes + w_bytes, &ws);
    if (st != LRC_OK) return st;
    unsigned int* cnt = nullptr;
    if ((st = stream_counters(s, &cnt)) != LRC_OK) return st;
    float* P = static_cast<float*>(ws);
    unsigned char* W = static_cast<unsigned char*>(ws) + part_bytes;

    const CUtensorMapDataType dt = bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
    const int64_t ldn = lrc_packed_ld(n), ldk = lrc_packed_ld(k);
    CUtensorMap tv, tx, tu;
    if ((st = encode_map_2d(&tv, dt, Vt, n, k, ldn * 2, kTcK, kTcM, true, "Vt")) != LRC_OK) return st;
    if ((st = encode_map_2d(&tx, dt, X, n, b, ldn * 2, kTcK, NB, true, "X")) != LRC_OK) return st;
    if ((st = encode_map_2d(&tu, dt, U, k, m, ldk * 2, kTcK, kTcM, true, "U")) != LRC_OK) return st;
    const uint32_t ab = bf16 ? tc::kIdescBF16 : 0u;

    TcWArgs a1{};
    a1.k = (int)k;
    a1.kp = p.kp;
    a1.b = (int)b;
    a1.nkb = p.nkb;
    a1.cb = p.cb;
    a1.nclusters = p.nclusters;
    a1.planes = p.planes;
    a1.bf16 = bf16 ? 1 : 0;
    a1.idesc = tc::idesc_f16_f32(kTcM, NB) | ab;
    a1.bar_off = (uint32_t)p.region;
    a1.S = static_cast<const uint16_t*>(S);
    a1.P = P;
    a1.W = W;
    a1.cnt = cnt;
    cudaError_t ce = cudaFuncSetAttribute(skinny_tc_w_kernel<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)p.smem1);
    if (ce != cudaSuccess) return cuda_fail(ce, "skinny_tc_w_kernel smem attribute");
    {
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3((unsigned)(p.nclusters * kTcCluster), (unsigned)p.rtiles);
        cfg.blockDim = dim3(kTcThreadsW);
        cfg.dynamicSmemBytes = p.smem1;
        cfg.stream = s;
        cudaLaunchAttribute attr[2];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = kTcCluster;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 2;
        ce = cudaLaunchKernelEx(&cfg, skinny_tc_w_kernel<NB>, tv, tx, a1);
    }
    if (ce != cudaSuccess) return cuda_fail(ce, "skinny_tc_w_kernel launch");
    if ((st = after_launch("skinny_tc_w_kernel")) != LRC_OK) return st;

    TcYArgs a3{};
    a3.m = m;
    a3.b = (int)b;
    a3.kp = p.kp;
    a3.kc = p.kc;
    a3.planes = p.planes;
    a3.rtiles = p.rtiles;
    a3.out16 = fmt == LRC_F16 ? 0 : 1;
    a3.bf16 = bf16 ? 1 : 0;
    a3.idesc = tc::idesc_f16_f32(kTcM, (uint32_t)(p.planes * NB)) | ab;
    a3.cnt = cnt;
    a3.W = W;
    a3.Y = Y;
    ce = cudaFuncSetAttribute(skinny_tc_y_kernel<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem3);
    if (ce != cudaSuccess) return cuda_fail(ce, "skinny_tc_y_kernel smem attribute");
    ce = launch_pdl(skinny_tc_y_kernel<NB>, dim3((unsigned)((m + kTcM - 1) / kTcM)), dim3(kTcThreadsY), p.smem3, s, tu,
                    a3);
    if (ce != cudaSuccess) return cuda_fail(ce, "skinny_tc_y_kernel launch");
    return after_launch("skinny_tc_y_kernel");
}

int64_t max_batch(lrc_fmt fmt) { return fmt == LRC_F16 || fmt == LRC_F16_O16 ? 4 : 16; }

}  // namespace

// Batches this path takes: up to 64 queries in binary16 and bfloat16 on the
// tensor cores (rank at most 512, n at most 32768); otherwise up to 16
// queries for binary32 and binary64 and up to 4 for binary16 on the CUDA
// cores, ranks whose tiles fit in shared memory.
bool apply_skinny_takes(lrc_fmt fmt, int64_t m, int64_t n, int64_t k, int64_t b) {
    if (skinny_tc_takes(fmt, m, n, k, b)) return true;
    if (fmt == LRC_BF16) return false;
    if (b < 1 || b > max_batch(fmt) || k < 1 || k > 1024) return false;
    const int B = b <= 1 ? 1 : (b <= 4 ? 4 : (b <= 8 ? 8 : 16));
    const int64_t e = storage_bytes(fmt);
    const SkinnyPlan p = plan_skinny(1, 1, k, B, e, fmt == LRC_F64 ? 8 : 4);
    return p.smem1 <= kSmemMaxS && p.smem3 <= kSmemMaxS;
}

lrc_status launch_apply_skinny(const void* U, const void* S, const void* Vt, const void* X, void* Y, int64_t m,
                               int64_t n, int64_t k, int64_t b, lrc_fmt fmt, cudaStream_t s) {
    if (!apply_skinny_takes(fmt, m, n, k, b)) {
        set_error("small-batch apply: b = %lld, k = %lld outside the kernel", (long long)b, (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    if (skinny_tc_takes(fmt, m, n, k, b)) {
        switch (tc_width(b)) {
            case 16: return launch_skinny_tc_nb<16>(U, S, Vt, X, Y, m, n, k, b, fmt, s);
            case 32: return launch_skinny_tc_nb<32>(U, S, Vt, X, Y, m, n, k, b, fmt, s);
            default: return launch_skinny_tc_nb<64>(U, S, Vt, X, Y, m, n, k, b, fmt, s);
        }
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
