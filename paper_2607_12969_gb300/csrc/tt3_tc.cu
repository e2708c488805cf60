// tt3_tc.cu -- 3-way TT reconstruction from binary16 cores with both chain
// stages on the tensor cores (Sec. 7.5, Eq. gpu_tt_reconstruction with d = 3:
// B_2 = Z_1 K_2, Z_2 = reshape(B_2), out = Z_2 K_3; Sec. 3.4: FP32
// accumulation).
//
// Work unit: 128 consecutive values of i_1 (the MMA M) and one i_2, and a
// slice of the n_3 outputs (n_3 is split in S parts when that balances the
// units over the SMs better).  Per unit:
//   stage 1  D1 (128 x r_2, TMEM) = G_1[i_1 tile, :] (128 x r_1) G_2(i_2)
//            (r_1 x r_2)  -- A = G_1 rows, B = G_2(i_2)^T, both binary16;
//   convert  D1 -> Z_2 rows as binary16 (hi/lo pair for FP32 output, one
//            rounding for FP16 output, the method-precision workspace);
//   stage 2  D2 (128 x n_3 slice, TMEM) = Z_2 rows G_3 (B = G_3^T);
//   store    D2 -> registers -> 128-byte-swizzled staging -> 3-D TMA stores
//            of out[i_1 tile, i_2, slice] (rows n_2 n_3 elements apart), each
//            epilogue warp storing its own 32 rows.
// D1 lives in the first columns of the unit's own D2 accumulator, so two
// units are in flight within 2 x slice <= 512 TMEM columns.  Warp roles:
//   0..3 epilogue, 4..7 converters, 8 MMA issuer (one thread), 9..12 loaders
//   (G_1 tile, G_2(i_2)^T per unit through an asynchronous-copy ring).  G_3^T
//   and the zero operand padding are written once by all threads before the
//   roles split.
// Intermediates never reach global memory.
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "tc.cuh"

namespace lrc {

__device__ unsigned int g_err_tt3_tc;

namespace {

using namespace tc;

constexpr int BM = 128;
constexpr int kThreads = 416;
constexpr int kLoadThreads = 128;
constexpr int kBatch = 8;                  // words per loader thread per round (synchronous paths)
constexpr int kRaw = 4;                    // raw G_2 slices in flight (asynchronous copies)

struct T3Args {
    int64_t n1, n2;
    int nd, r1, r2, r1p, r2p;      // n_3, ranks, ranks rounded up to 16
    int n2h, sn;                   // n_3 slice per unit, number of slices
    int64_t units;                 // (i_1 tile, i_2, n_3 slice) units
    int cw, out16;
    uint32_t tmem_cols;
    uint32_t off_a1, off_b1, off_a2, off_b2, off_stage, off_bar;
    uint32_t b1_bytes, a2_bytes;
    uint32_t off_raw, raw_bytes;   // ring of kRaw raw G_2(i_2) slices
    const __half* G1;
    const __half* G2;
    const __half* G3;
    int g1_words, g2_words;        // rows of G_1 / G_2 loadable as 4-byte words
};

struct Bars {
    uint64_t *a1_full, *a1_empty;
    uint64_t *b1_full, *b1_empty;      // [2]
    uint64_t *d1_full;                 // [2]
    uint64_t *a2_full, *a2_empty;      // [2]
    uint64_t *d2_full, *acc_empty;     // [2]
    uint64_t *mma_done;
    uint32_t* tmem_slot;
    int* abort;
};

__device__ __forceinline__ Bars carve(unsigned char* smem, const T3Args& a) {
    uint64_t* p = reinterpret_cast<uint64_t*>(smem + a.off_bar);
    Bars B;
    B.a1_full = p + 0;
    B.a1_empty = p + 1;
    B.b1_full = p + 3;
    B.b1_empty = p + 5;
    B.d1_full = p + 7;
    B.a2_full = p + 9;
    B.a2_empty = p + 11;
    B.d2_full = p + 13;
    B.acc_empty = p + 15;
    B.mma_done = p + 17;
    B.tmem_slot = reinterpret_cast<uint32_t*>(p + 18);
    B.abort = reinterpret_cast<int*>(B.tmem_slot + 1);
    return B;
}

// Byte offset of element (row, k) in a canonical no-swizzle K-major operand
// with `rows` rows: 8-row x 16-byte core matrices, K-direction core stride
// rows*16 bytes (the LBO), row-group stride 128 bytes (the SBO).
__device__ __forceinline__ uint32_t canon_off(uint32_t row, uint32_t k, uint32_t rows) {
    return (k >> 3) * rows * 16u + (row >> 3) * 128u + (row & 7u) * 16u + (k & 7u) * 2u;
}

__device__ __forceinline__ void unit_coords(const T3Args& a, int64_t u, int64_t& qt, int64_t& i, int& h) {
    const int64_t per_qt = a.n2 * a.sn;
    qt = u / per_qt;
    const int64_t rest = u - qt * per_qt;
    i = rest / a.sn;
    h = (int)(rest - i * a.sn);
}

__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Issues the asynchronous copy of G_2(i_2) (r_1 rows of r_2 ranks, 4-byte
// words) into a raw slot laid out [a][b-pair], row pitch r_2/2 words.  Each
// loader warp copies whole rows (lane = word; r_2 <= 64, so one pass).
__device__ __forceinline__ void raw_issue(const T3Args& a, int64_t i, int lwarp, int lane, uint32_t* raw) {
    const int wpr = a.r2 / 2;                           // r_2 is even on this path
    if (lane < wpr) {
        for (int k = lwarp; k < a.r1; k += kLoadThreads / 32)
            cp_async4(raw + k * wpr + lane, a.G2 + ((int64_t)k * a.n2 + i) * a.r2 + 2 * lane);
    }
}

// G_2(i_2)^T into B1 (row b, column a) from a raw slot, shared to shared:
// a thread takes ranks a, a+1 and b, b+1 (two raw words) and writes them as
// two 4-byte words, one per row b and b+1 of the K-major layout.
__device__ __forceinline__ void raw_transpose(const T3Args& a, int lwarp, int lane, const uint32_t* raw,
                                              unsigned char* b1) {
    const int wpr = a.r2 / 2;
    if (lane < wpr) {
        for (int k = 2 * lwarp; k < a.r1; k += 2 * (kLoadThreads / 32)) {
            const uint32_t w0 = raw[k * wpr + lane];                          // a = k:   (b, b+1)
            const uint32_t w1 = (k + 1 < a.r1) ? raw[(k + 1) * wpr + lane] : 0u;  // a = k+1: (b, b+1)
            const uint32_t rb0 = (w0 & 0xffffu) | (w1 << 16);                 // row b:   (a, a+1)
            const uint32_t rb1 = (w0 >> 16) | (w1 & 0xffff0000u);             // row b+1: (a, a+1)
            *reinterpret_cast<uint32_t*>(b1 + canon_off(2 * lane, k, a.r2p)) = rb0;
            *reinterpret_cast<uint32_t*>(b1 + canon_off(2 * lane + 1, k, a.r2p)) = rb1;
        }
    }
}

// Synchronous path (odd rank or misaligned core): G_2(i_2)^T straight from
// global memory, eight loads in flight per thread.
__device__ __forceinline__ void b1_direct(const T3Args& a, int64_t i, int lt, unsigned char* b1) {
    const int wpr = (a.r2 + 1) / 2;
    const int total = a.r1 * wpr;
    for (int e0 = lt; e0 < total; e0 += kLoadThreads * kBatch) {
        uint32_t w[kBatch];
#pragma unroll
        for (int t = 0; t < kBatch; ++t) {
            const int e = e0 + t * kLoadThreads;
            w[t] = 0;
            if (e < total) {
                const int k = e / wpr, bw = e % wpr;
                const __half* src = a.G2 + ((int64_t)k * a.n2 + i) * a.r2 + 2 * bw;
                const uint32_t lo16 = __half_as_ushort(src[0]);
                const uint32_t hi16 = (2 * bw + 1 < a.r2) ? __half_as_ushort(src[1]) : 0u;
                w[t] = lo16 | (hi16 << 16);
            }
        }
#pragma unroll
        for (int t = 0; t < kBatch; ++t) {
            const int e = e0 + t * kLoadThreads;
            if (e < total) {
                const int k = e / wpr, bw = e % wpr;
                *reinterpret_cast<unsigned short*>(b1 + canon_off(2 * bw, k, a.r2p)) = (unsigned short)(w[t] & 0xffffu);
                if (2 * bw + 1 < a.r2)
                    *reinterpret_cast<unsigned short*>(b1 + canon_off(2 * bw + 1, k, a.r2p)) =
                        (unsigned short)(w[t] >> 16);
            }
        }
    }
}

// Shared prologue, all threads: zero A1 and both B1 buffers (their padding
// rows and columns stay zero), then write G_3^T (n_3 rows, r2p ranks,
// K-major) into B2.  A thread takes a 2 x 2 block -- ranks k, k+1 of
// outputs c, c+1 -- as two 4-byte loads along n_3 and writes it as two 4-byte
// words, one per B2 row; eight blocks per thread are in flight.
__device__ __forceinline__ void build_g3t(const T3Args& a, unsigned char* smem) {
    const int nt = blockDim.x;
    uint4* z = reinterpret_cast<uint4*>(smem + a.off_a1);
    const uint32_t zbytes = a.off_b2 - a.off_a1;
    for (uint32_t e = threadIdx.x; e < zbytes / 16; e += nt) z[e] = make_uint4(0, 0, 0, 0);
    unsigned char* b2 = smem + a.off_b2;
    const int cpairs = a.nd / 2;                              // n_3 is a multiple of 16
    const int total = cpairs * (a.r2p / 2);
    const bool words = (reinterpret_cast<uintptr_t>(a.G3) & 3u) == 0;
    for (int e0 = threadIdx.x; e0 < total; e0 += nt * kBatch) {
        uint32_t w0[kBatch], w1[kBatch];
#pragma unroll
        for (int t = 0; t < kBatch; ++t) {
            const int e = e0 + t * nt;
            const int k = 2 * (e / cpairs), c = 2 * (e % cpairs);
            w0[t] = 0;
            w1[t] = 0;
            if (e < total) {
                const __half* p0 = a.G3 + (int64_t)k * a.nd + c;
                if (k < a.r2)
                    w0[t] = words ? __ldg(reinterpret_cast<const unsigned int*>(p0))
                                  : (uint32_t)__half_as_ushort(p0[0]) | ((uint32_t)__half_as_ushort(p0[1]) << 16);
                if (k + 1 < a.r2) {
                    const __half* p1 = p0 + a.nd;
                    w1[t] = words ? __ldg(reinterpret_cast<const unsigned int*>(p1))
                                  : (uint32_t)__half_as_ushort(p1[0]) | ((uint32_t)__half_as_ushort(p1[1]) << 16);
                }
            }
        }
#pragma unroll
        for (int t = 0; t < kBatch; ++t) {
            const int e = e0 + t * nt;
            if (e < total) {
                const int k = 2 * (e / cpairs), c = 2 * (e % cpairs);
                *reinterpret_cast<uint32_t*>(b2 + canon_off(c, k, a.nd)) = (w0[t] & 0xffffu) | (w1[t] << 16);
                *reinterpret_cast<uint32_t*>(b2 + canon_off(c + 1, k, a.nd)) = (w0[t] >> 16) | (w1[t] & 0xffff0000u);
            }
        }
    }
}

__global__ void __launch_bounds__(kThreads, 1)
tt3_f16_tc_kernel(const __grid_constant__ CUtensorMap tm_out, const T3Args a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                           ~static_cast<uintptr_t>(1023));
    const Bars B = carve(smem, a);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort = B.abort;
    unsigned int* err = &g_err_tt3_tc;
    // contiguous unit range of this CTA
    const int64_t ubeg = a.units * blockIdx.x / gridDim.x;
    const int64_t uend = a.units * (blockIdx.x + 1) / gridDim.x;
    const int64_t nunits = uend - ubeg;

    if (threadIdx.x == 0) {
        mbar_init(B.a1_full, 1);
        mbar_init(B.a1_empty, 1);
        for (int q = 0; q < 2; ++q) {
            mbar_init(&B.b1_full[q], 1);
            mbar_init(&B.b1_empty[q], 1);
            mbar_init(&B.d1_full[q], 1);
            mbar_init(&B.a2_full[q], 128);
            mbar_init(&B.a2_empty[q], 1);
            mbar_init(&B.d2_full[q], 1);
            mbar_init(&B.acc_empty[q], 128);
        }
        mbar_init(B.mma_done, 1);
        *B.abort = 0;
        fence_barrier_init();
    }
    if (warp == 8) tmem_alloc(B.tmem_slot, a.tmem_cols);
    uint32_t* raw = reinterpret_cast<uint32_t*>(smem + a.off_raw);
    const uint32_t raw_words = a.raw_bytes / 4;
    if (warp >= 9 && a.g2_words) {
        // start the first kRaw - 1 G_2 slices before the shared prologue
        for (int64_t p = 0; p < kRaw - 1; ++p) {
            if (p < nunits) {
                int64_t qp, ip;
                int hp;
                unit_coords(a, ubeg + p, qp, ip, hp);
                raw_issue(a, ip, warp - 9, lane, raw + (uint32_t)(p % kRaw) * raw_words);
            }
            cp_async_commit();
        }
    }
    build_g3t(a, smem);          // every thread: operand padding and G_3^T
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *B.tmem_slot;

    if (warp >= 9) {
        // ------------------------------------------------------------ loaders
        const int lt = threadIdx.x - 288;                      // 0..127
        const bool leader = (lt == 0);
        int64_t prev_qt = -1;
        int builds = 0;
        for (int64_t j = 0; j < nunits; ++j) {
            int64_t qt, i;
            int h;
            unit_coords(a, ubeg + j, qt, i, h);
            if (qt != prev_qt) {
                if (builds > 0 &&
                    !group_wait(B.a1_empty, (uint32_t)((builds - 1) & 1), abort, err, 1u, 3, kLoadThreads))
                    break;
                // G_1 rows of this i_1 tile: 128 x r_1 (words of two ranks)
                unsigned char* a1 = smem + a.off_a1;
                const int wpr = (a.r1 + 1) / 2;                 // words per row
                const int total = BM * wpr;
                for (int e0 = lt; e0 < total; e0 += kLoadThreads * kBatch) {
                    uint32_t w[kBatch];
#pragma unroll
                    for (int t = 0; t < kBatch; ++t) {
                        const int e = e0 + t * kLoadThreads;
                        const int row = e / wpr, kw = e % wpr;
                        const int64_t q = qt * BM + row;
                        w[t] = 0;
                        if (e < total && q < a.n1) {
                            const __half* src = a.G1 + q * a.r1 + 2 * kw;
                            if (a.g1_words) w[t] = __ldg(reinterpret_cast<const unsigned int*>(src));
                            else {
                                const uint32_t lo16 = __half_as_ushort(src[0]);
                                const uint32_t hi16 = (2 * kw + 1 < a.r1) ? __half_as_ushort(src[1]) : 0u;
                                w[t] = lo16 | (hi16 << 16);
                            }
                        }
                    }
#pragma unroll
                    for (int t = 0; t < kBatch; ++t) {
                        const int e = e0 + t * kLoadThreads;
                        if (e < total) {
                            const int row = e / wpr, kw = e % wpr;
                            // ranks 2kw and 2kw+1 are adjacent in a row of the K-major layout
                            *reinterpret_cast<uint32_t*>(a1 + canon_off(row, 2 * kw, BM)) = w[t];
                        }
                    }
                }
                fence_proxy_async_smem();
                named_bar_sync(3, kLoadThreads);
                if (leader) mbar_arrive(B.a1_full);
                prev_qt = qt;
                ++builds;
            }
            const int slot = (int)(j & 1);
            if (a.g2_words) {
                {   // issue unit j + kRaw - 1, then wait for unit j's slice (in-order groups)
                    const int64_t p = j + kRaw - 1;
                    if (p < nunits) {
                        int64_t qp, ip;
                        int hp;
                        unit_coords(a, ubeg + p, qp, ip, hp);
                        raw_issue(a, ip, lt >> 5, lane, raw + (uint32_t)(p % kRaw) * raw_words);
                    }
                    cp_async_commit();
                    cp_async_wait<kRaw - 1>();
                }
                named_bar_sync(3, kLoadThreads);             // every thread's part of slice j has landed
            }
            if (!group_wait(&B.b1_empty[slot], (uint32_t)((j >> 1) & 1) ^ 1u, abort, err, 1u, 3, kLoadThreads)) break;
            // G_2(i_2)^T: row b (r_2), column a (r_1): element G_2[a, i_2, b]
            unsigned char* b1 = smem + a.off_b1 + (size_t)slot * a.b1_bytes;
            if (a.g2_words) raw_transpose(a, lt >> 5, lane, raw + (uint32_t)(j % kRaw) * raw_words, b1);
            else b1_direct(a, i, lt, b1);
            fence_proxy_async_smem();
            named_bar_sync(3, kLoadThreads);
            if (leader) mbar_arrive(&B.b1_full[slot]);
        }
        cp_async_wait<0>();                                // no copy in flight when the CTA exits
    } else if (warp == 8) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            bool ok = true;
            const uint32_t idesc1 = idesc_f16_f32(BM, (uint32_t)a.r2p);
            const uint32_t idesc2 = idesc_f16_f32(BM, (uint32_t)a.n2h);
            const uint32_t a1s = smem_u32(smem + a.off_a1);
            const uint32_t b2s = smem_u32(smem + a.off_b2);
            int64_t cur_qt = -1;
            int qcount = 0;
            auto stage1 = [&](int64_t j) -> bool {
                int64_t qt, i;
                int h;
                unit_coords(a, ubeg + j, qt, i, h);
                const int buf = (int)(j & 1);
                if (qt != cur_qt) {
                    if (!mbar_wait(B.a1_full, (uint32_t)(qcount & 1), abort, err, 2u)) return false;
                    cur_qt = qt;
                    ++qcount;
                }
                if (!mbar_wait(&B.acc_empty[buf], (uint32_t)((j >> 1) & 1) ^ 1u, abort, err, 2u)) return false;
                if (!mbar_wait(&B.b1_full[buf], (uint32_t)((j >> 1) & 1), abort, err, 2u)) return false;
                tc_fence_after();
                const uint32_t b1s = smem_u32(smem + a.off_b1 + (size_t)buf * a.b1_bytes);
                const uint32_t lbo1 = (uint32_t)a.r2p * 16u;
                // descriptors stepped by adds: 16 ranks = 4096 B of A, 2 x lbo1 B of B
                const uint64_t ad = smem_desc(a1s, 2048, 128, 0), bd = smem_desc(b1s, lbo1, 128, 0);
                const uint64_t bstep = (uint64_t)(2u * lbo1) >> 4;
                for (int ks = 0; ks < a.r1p / 16; ++ks)
                    mma_f16(tmem + (uint32_t)buf * a.n2h, ad + (uint64_t)ks * 256u, bd + (uint64_t)ks * bstep, idesc1,
                            ks > 0);
                mma_commit(&B.b1_empty[buf]);
                mma_commit(&B.d1_full[buf]);
                // last unit of this i_1 tile: G_1 tile may be replaced once these MMAs finish
                bool last = (j + 1 == nunits);
                if (!last) {
                    int64_t qn, in;
                    int hn;
                    unit_coords(a, ubeg + j + 1, qn, in, hn);
                    last = (qn != qt);
                }
                if (last) mma_commit(B.a1_empty);
                return true;
            };
            auto stage2 = [&](int64_t j) -> bool {
                int64_t qt, i;
                int h;
                unit_coords(a, ubeg + j, qt, i, h);
                const int buf = (int)(j & 1);
                if (!mbar_wait(&B.a2_full[buf], (uint32_t)((j >> 1) & 1), abort, err, 2u)) return false;
                tc_fence_after();
                const uint32_t ahi = smem_u32(smem + a.off_a2 + (size_t)buf * 2 * a.a2_bytes);
                const uint32_t alo = ahi + a.a2_bytes;
                const uint32_t lbo2 = (uint32_t)a.nd * 16u;
                const uint32_t bslice = b2s + (uint32_t)h * (uint32_t)a.n2h * 16u;   // rows h*n2h..
                const uint64_t bd = smem_desc(bslice, lbo2, 128, 0);
                const uint64_t hd = smem_desc(ahi, 2048, 128, 0), ld = smem_desc(alo, 2048, 128, 0);
                const uint64_t bstep = (uint64_t)(2u * lbo2) >> 4;
                for (int ks = 0; ks < a.r2p / 16; ++ks) {
                    const uint64_t bdesc = bd + (uint64_t)ks * bstep;
                    mma_f16(tmem + (uint32_t)buf * a.n2h, hd + (uint64_t)ks * 256u, bdesc, idesc2, ks > 0);
                    if (!a.out16) mma_f16(tmem + (uint32_t)buf * a.n2h, ld + (uint64_t)ks * 256u, bdesc, idesc2, 1u);
                }
                mma_commit(&B.a2_empty[buf]);
                mma_commit(&B.d2_full[buf]);
                return true;
            };
            // stage 2 of unit j goes before stage 1 of unit j+1: stage 1 needs the
            // TMEM buffer the epilogue is still draining, stage 2 does not
            if (ok && nunits > 0) ok = stage1(0);
            for (int64_t j = 0; j < nunits && ok; ++j) {
                if (!(ok = stage2(j))) break;
                if (j + 1 < nunits) ok = stage1(j + 1);
            }
            mma_commit(B.mma_done);
            volatile int no_abort = 0;
            mbar_wait(B.mma_done, 0, &no_abort, err, 2u, 100000000ull);
        }
    } else if (warp >= 4) {
        // ------------------------------------------------------------ converters (warps 4..7)
        const int g = warp & 3;
        const int r = g * 32 + lane;
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        for (int64_t j = 0; j < nunits; ++j) {
            const int buf = (int)(j & 1);
            if (!group_wait(&B.d1_full[buf], (uint32_t)((j >> 1) & 1), abort, err, 4u, 2, 128)) break;
            tc_fence_after();
            uint32_t v[64];
            const uint32_t tcol = tmem + lane_base + (uint32_t)buf * a.n2h;
            tmem_ld32(tcol, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
            if (a.r2p > 32) tmem_ld32(tcol + 32, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
            tmem_ld_wait();
            if (!group_wait(&B.a2_empty[buf], (uint32_t)((j >> 1) & 1) ^ 1u, abort, err, 4u, 2, 128)) break;
            unsigned char* ahi = smem + a.off_a2 + (size_t)buf * 2 * a.a2_bytes;
            unsigned char* alo = ahi + a.a2_bytes;
#pragma unroll
            for (int c0 = 0; c0 < 64; c0 += 8) {
                if (c0 >= a.r2p) break;
                uint32_t hi[4], lo[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float w0 = __uint_as_float(v[c0 + 2 * q]), w1 = __uint_as_float(v[c0 + 2 * q + 1]);
                    const __half h0 = __float2half_rn(w0), h1 = __float2half_rn(w1);
                    hi[q] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
                    lo[q] = pack_half2(w0 - __half2float(h0), w1 - __half2float(h1));
                }
                const uint32_t off = (uint32_t)(c0 >> 3) * 2048u + (uint32_t)(r >> 3) * 128u + (uint32_t)(r & 7) * 16u;
                *reinterpret_cast<uint4*>(ahi + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                if (!a.out16) *reinterpret_cast<uint4*>(alo + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(&B.a2_full[buf]);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        // each warp drains its own 32 rows through its own staging pair and
        // issues its own 32-row TMA stores: no barrier across the four warps
        const int g = warp & 3;
        const int r = g * 32 + lane;
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        unsigned char* wstage = smem + a.off_stage + (size_t)g * (2 * 32 * 128);
        int chunk = 0;
        for (int64_t j = 0; j < nunits; ++j) {
            int64_t qt, i;
            int h;
            unit_coords(a, ubeg + j, qt, i, h);
            const int buf = (int)(j & 1);
            if (!group_wait(&B.d2_full[buf], (uint32_t)((j >> 1) & 1), abort, err, 8u, 1, 128)) break;
            tc_fence_after();
            for (int cc = 0; cc < a.n2h; cc += a.cw, ++chunk) {
                uint32_t v[64];
                const uint32_t tcol = tmem + lane_base + (uint32_t)buf * a.n2h + (uint32_t)cc;
                tmem_ld32(tcol, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
                if (a.out16) tmem_ld32(tcol + 32, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
                tmem_ld_wait();
                uint32_t packed[32];
                if (a.out16) {
#pragma unroll
                    for (int q = 0; q < 32; ++q)
                        packed[q] = pack_half2(__uint_as_float(v[2 * q]), __uint_as_float(v[2 * q + 1]));
                } else {
#pragma unroll
                    for (int q = 0; q < 32; ++q) packed[q] = v[q];
                }
                unsigned char* sb = wstage + (size_t)(chunk & 1) * (32 * 128);
                if (chunk >= 2) {
                    if (lane == 0) bulk_wait_read<1>();
                    __syncwarp();
                }
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const uint32_t off = (uint32_t)lane * 128u + (uint32_t)((q ^ (lane & 7)) * 16);
                    *reinterpret_cast<uint4*>(sb + off) =
                        make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_3d(&tm_out, h * a.n2h + cc, (int32_t)i, (int32_t)(qt * BM + g * 32), sb);
                    bulk_commit();
                }
            }
            tc_fence_before();
            mbar_arrive(&B.acc_empty[buf]);
        }
        if (lane == 0) bulk_wait<0>();
        (void)r;
    }
    // single-lane roles rejoin their warps first: the CTA barrier is an aligned one
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 8) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, a.tmem_cols);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode3 = nullptr;
std::once_flag g_encode3_once;

uint32_t pow2_cols(uint32_t c) {
    uint32_t p = 32;
    while (p < c) p <<= 1;
    return p;
}

// Plans the 3-way kernel; returns false when the shape is outside it.
bool tt3_f16_tc_plan(const TTShape& sh, bool out16, T3Args* out_args, size_t* smem_out, int64_t* grid_out) {
    if (sh.d != 3) return false;
    T3Args a{};
    a.n1 = sh.dims[0];
    a.n2 = sh.dims[1];
    a.nd = (int)sh.dims[2];
    a.r1 = (int)sh.ranks[1];
    a.r2 = (int)sh.ranks[2];
    if (sh.dims[2] > 256 || a.nd % 16 != 0) return false;
    if (a.r1 > 128 || a.r2 > 64) return false;
    const int eo = out16 ? 2 : 4;
    if (a.nd * eo < 128) return false;
    a.r1p = (a.r1 + 15) / 16 * 16;
    a.r2p = (a.r2 + 15) / 16 * 16;
    a.cw = 128 / eo;
    a.out16 = out16 ? 1 : 0;
    const int sms = sm_count();
    const int64_t qtiles = (a.n1 + BM - 1) / BM;
    // choose the n_3 split that balances units over the SMs best
    double best = -1.0;
    int best_sn = 1;
    for (int sn : {1, 2, 4}) {
        const int n2h = a.nd / sn;
        if (a.nd % sn != 0 || n2h % 16 != 0 || n2h < a.r2p) continue;
        if (sn > 1 && n2h % a.cw != 0) continue;       // slices must not overlap in the store
        const int64_t units = qtiles * a.n2 * sn;
        const int64_t per = (units + sms - 1) / sms;
        const double bal = (double)units / ((double)per * (double)(units < sms ? units : sms));
        if (bal > best + 1e-9) {
            best = bal;
            best_sn = sn;
        }
    }
    a.sn = best_sn;
    a.n2h = a.nd / a.sn;
    if (a.n2h < a.r2p) return false;
    a.units = qtiles * a.n2 * a.sn;
    a.tmem_cols = pow2_cols(2u * (uint32_t)a.n2h);
    const uint32_t chunks = (uint32_t)((a.n2h + a.cw - 1) / a.cw * a.cw);
    if ((uint32_t)a.n2h + chunks > a.tmem_cols || a.tmem_cols > 512) return false;
    a.b1_bytes = (uint32_t)a.r2p * a.r1p * 2;
    a.a2_bytes = (uint32_t)BM * a.r2p * 2;
    uint32_t off = 0;
    a.off_a1 = off;
    off += (uint32_t)BM * a.r1p * 2;
    a.off_b1 = off;
    off += 2 * a.b1_bytes;
    a.off_a2 = off;
    off += 4 * a.a2_bytes;
    a.off_b2 = off;
    off += (uint32_t)a.nd * a.r2p * 2;
    off = (off + 15) / 16 * 16;
    a.raw_bytes = (uint32_t)a.r1 * (uint32_t)((a.r2 + 1) / 2) * 4u;
    a.raw_bytes = (a.raw_bytes + 15) / 16 * 16;
    a.off_raw = off;
    off += kRaw * a.raw_bytes;
    off = (off + 1023) / 1024 * 1024;
    a.off_stage = off;
    off += 2 * BM * 128;
    off = (off + 7) / 8 * 8;
    a.off_bar = off;
    off += 18 * 8 + 16;
    const size_t smem = (size_t)off + 1024;
    if (smem > 227 * 1024) return false;
    a.G1 = static_cast<const __half*>(sh.cores[0]);
    a.G2 = static_cast<const __half*>(sh.cores[1]);
    a.G3 = static_cast<const __half*>(sh.cores[2]);
    // 4-byte loads need an even rank and a 4-byte aligned core
    a.g1_words = ((a.r1 & 1) == 0 && (reinterpret_cast<uintptr_t>(a.G1) & 3u) == 0) ? 1 : 0;
    a.g2_words = ((a.r2 & 1) == 0 && (reinterpret_cast<uintptr_t>(a.G2) & 3u) == 0) ? 1 : 0;
    *out_args = a;
    *smem_out = smem;
    *grid_out = a.units < sms ? a.units : sms;
    return true;
}

}  // namespace

lrc_status launch_tt3_f16_tc(const TTShape& sh, bool out16, void* out, cudaStream_t s, bool* handled) {
    T3Args a;
    size_t smem = 0;
    int64_t grid = 0;
    *handled = false;
    if (!tt3_f16_tc_plan(sh, out16, &a, &smem, &grid)) return LRC_OK;
    *handled = true;
    std::call_once(g_encode3_once, [] {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode3 = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    });
    if (!g_encode3) {
        set_error("cuTensorMapEncodeTiled is not available from the driver");
        return LRC_ERR_CUDA;
    }
    const int eo = out16 ? 2 : 4;
    CUtensorMap tm;
    cuuint64_t dims[3] = {(cuuint64_t)a.nd, (cuuint64_t)a.n2, (cuuint64_t)a.n1};
    cuuint64_t strides[2] = {(cuuint64_t)a.nd * eo, (cuuint64_t)a.nd * (cuuint64_t)a.n2 * eo};
    cuuint32_t box[3] = {(cuuint32_t)a.cw, 1, 32};      // one epilogue warp's 32 rows
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult cr = g_encode3(&tm, out16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, out,
                            dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (cr != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled failed for the 3-way TT output (CUresult %d)", (int)cr);
        return LRC_ERR_CUDA;
    }
    cudaError_t e = cudaFuncSetAttribute(tt3_f16_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "tt3_f16_tc_kernel smem attribute");
    tt3_f16_tc_kernel<<<(unsigned)grid, kThreads, smem, s>>>(tm, a);
    return after_launch("tt3_f16_tc_kernel");
}

uint32_t take_tt3_tc_error() {
    unsigned int v = 0;
    if (cudaMemcpyFromSymbol(&v, g_err_tt3_tc, sizeof v) != cudaSuccess) return 0xffffffffu;
    if (v) {
        const unsigned int z = 0;
        cudaMemcpyToSymbol(g_err_tt3_tc, &z, sizeof z);
    }
    return v;
}

}  // namespace lrc
