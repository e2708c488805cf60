// apply_tc.cu -- low-rank apply on the 5th-generation tensor cores, binary16
// storage with binary32 accumulation (Sec. 4.4, Eq. gpu_matrix_apply:
// Y = [(X V) diag(s)] U^T; Sec. 3.4: FP16 products accumulate in FP32).
//
// Three launches on the caller's stream:
//  1. apply_w1_kernel -- W = X V in FP32 partials.  For every 128-row tile of
//     X and every column group of W (at most 160 ranks for FP32 output, so that
//     two accumulators and a running sum fit in tensor memory) the reduction
//     over n is a row of 64-wide k-blocks.  The rows are laid end to end and
//     cut into equal contiguous ranges, one per CTA of a persistent grid:
//     every SM gets the same share of the product whatever b is (one row tile
//     or hundreds).  A CTA's range crosses a few rows; each piece (segment)
//     accumulates in tensor memory -- for FP32 output in chunks of at most
//     kChunkBlocks k-blocks whose results the epilogue adds with IEEE
//     binary32 additions into a running sum kept in tensor memory (the tensor
//     core's own accumulation error grows with the number of accumulation
//     steps) -- and is written to the workspace as an FP32 partial.  Column
//     groups are the slower index of the rows, so the CTAs working on the two
//     groups of one row tile run side by side and the second read of an X
//     tile hits L2.
//     The same kernels take bfloat16 storage (LRC_BF16): bfloat16 tensor-core
//     operands (the instruction descriptor's A/B format), bfloat16 W and output.
//  2. apply_w2_kernel -- every W entry adds its tile's partials in a fixed
//     order (deterministic), is scaled by diag(s) in FP32 and written as
//     binary16: a hi/lo pair (hi = fp16(w), lo = fp16(w - hi)) for FP32
//     output, which keeps about 22 significand bits through the second
//     product, or one rounding for FP16 output (the method-precision
//     workspace of Sec. 3.4).  The layout is the shared-memory image of the
//     second product's A operand, so it is loaded with one bulk copy.  With
//     many partials per row (small b) apply_w2_slice_kernel spreads each
//     entry's partials over 16 warps.
//  3. apply_y_kernel -- Y tiles = W U^T.  A persistent grid takes equal
//     contiguous ranges of (row tile, column tile) pairs; W of the current
//     row tile sits in shared memory, U streams through a TMA ring, and two
//     tensor-memory accumulators let the epilogue drain one tile (TMEM ->
//     registers -> swizzled shared memory -> TMA stores of 128-row boxes, two
//     warps per lane quarter on alternate column chunks) while the next is
//     multiplied.
// Warp roles: warp 0 TMA producer, warp 1 tensor-memory owner and MMA issuer
// (one thread), then the epilogue warps (one TMEM lane = one row per thread;
// four in kernel 1, eight in kernel 3).  W is b x k' values, a few percent of
// the traffic.
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "tc.cuh"

namespace lrc {

__device__ unsigned int g_err_apply_tc;

namespace {

using namespace tc;

constexpr int BM = 128;
constexpr int BK = 64;                       // FP16 elements per 128-byte swizzled row
constexpr int kThreads = 192;
// the second product: warp 0 producer, warp 1 MMA, warps 2..9 epilogue -- two
// warps per tensor-memory lane quarter, taking alternate column chunks (the
// epilogue is bound by the latency of each chunk's load / stage / fence /
// store sequence, not by bandwidth)
constexpr int kEpiWarpsY = 8;
constexpr int kThreadsY = 64 + 32 * kEpiWarpsY;
constexpr uint32_t kXBytes = BM * BK * 2;    // one X box
constexpr int kChunkBlocks = 8;              // k-blocks per accumulation chunk (FP32 output)
constexpr int kStageBlocks = 2;              // k-blocks per phase-1 ring stage

__device__ __forceinline__ unsigned char* align1024(unsigned char* p) {
    return reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~static_cast<uintptr_t>(1023));
}

// ================================================================ phase 1
struct W1Args {
    int64_t b;
    int64_t btiles;
    int64_t nkb;              // k-blocks per row, ceil(n / 64)
    int64_t Q;                // rows x nkb
    int G;                    // column groups; row = group * btiles + row tile
    int kgp;                  // group width (ranks, multiple of 16); group g starts at g * kgp
    int kp;                   // the last group ends at kp
    int chunk_blocks;
    int stages;
    uint32_t slot_bytes;
    uint32_t bar_off;
    uint32_t sum_col;         // tensor-memory column of the running sum (FP32 output)
    uint32_t tmem_cols;
    uint32_t idesc_ab;        // operand-format bits of the MMA descriptor (0: binary16)
    float* P;                 // partials: [segment id][kgp columns][128 rows]
};

// Next accumulation chunk of the k-block range [qbeg, qend): a chunk lies in
// one row, starts a new chunk every `cb` k-blocks from the start of its
// segment (the part of the row inside the range) and ends with the segment.
__device__ __forceinline__ bool next_chunk(int64_t& q, int64_t qbeg, int64_t qend, int64_t nkb, int64_t cb,
                                           int64_t& q0, int64_t& q1, int64_t& row, bool& first, bool& last) {
    if (q >= qend) return false;
    row = q / nkb;
    const int64_t re = (row + 1) * nkb;
    const int64_t seg_end = re < qend ? re : qend;
    q0 = q;
    q1 = (q + cb < seg_end) ? q + cb : seg_end;
    first = (q == qbeg) || (q == row * nkb);
    last = (q1 == seg_end);
    q = q1;
    return true;
}

// Phase 1 of one problem, run by CTA `cta` of the `ncta` CTAs given to it.
__device__ __forceinline__ void w1_body(const CUtensorMap* tm_x, const CUtensorMap* tm_v, const W1Args& a, int64_t cta,
                                        int64_t ncta) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = align1024(smem_raw);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + a.bar_off);
    uint64_t* empty = full + a.stages;
    uint64_t* acc_full = empty + a.stages;     // [2]
    uint64_t* acc_empty = acc_full + 2;        // [2]
    uint64_t* mma_done = acc_empty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort = reinterpret_cast<int*>(tmem_slot + 1);
    unsigned int* err = &g_err_apply_tc;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t qbeg = a.Q * cta / ncta;
    const int64_t qend = a.Q * (cta + 1) / ncta;
    pdl_trigger();                 // the reduction kernel may be scheduled now; it waits for this grid

    if (threadIdx.x == 0) {
        for (int i = 0; i < a.stages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 128);
        }
        mbar_init(mma_done, 1);
        *abort = 0;
        fence_barrier_init();
        tma_prefetch_desc(tm_x);
        tma_prefetch_desc(tm_v);
    }
    if (warp == 1) tmem_alloc(tmem_slot, a.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // a ring stage carries kStageBlocks k-blocks of one chunk: slot layout
    // [X k-block 0][X k-block 1][V^T k-block 0][V^T k-block 1]
    const uint32_t vbox = (uint32_t)a.kgp * 128u;
    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int it = 0;
            bool ok = true;
            int64_t q = qbeg, q0, q1, row;
            bool first, last;
            while (ok && next_chunk(q, qbeg, qend, a.nkb, a.chunk_blocks, q0, q1, row, first, last)) {
                const int grp = (int)(row / a.btiles);
                const int64_t bt = row - (int64_t)grp * a.btiles;
                const int64_t rbase = row * a.nkb;
                for (int64_t qs = q0; qs < q1; qs += kStageBlocks, ++it) {
                    const int nb = (q1 - qs >= kStageBlocks) ? kStageBlocks : (int)(q1 - qs);
                    const int slot = it % a.stages;
                    if (!(ok = mbar_wait(&empty[slot], ((it / a.stages) & 1) ^ 1, abort, err, 1u))) break;
                    unsigned char* sp = smem + (size_t)slot * a.slot_bytes;
                    mbar_arrive_expect_tx(&full[slot], (uint32_t)nb * (kXBytes + vbox));
                    for (int u = 0; u < nb; ++u) {
                        const int32_t kx = (int32_t)((qs + u - rbase) * BK);
                        tma_load_2d(sp + (size_t)u * kXBytes, tm_x, kx, (int32_t)(bt * BM), &full[slot]);
                        tma_load_2d(sp + (size_t)kStageBlocks * kXBytes + (size_t)u * vbox, tm_v, kx, grp * a.kgp,
                                    &full[slot]);
                    }
                }
            }
            if (!ok) {
                // let copies already in flight land before the CTA can exit
                const int first_it = it - a.stages > 0 ? it - a.stages : 0;
                for (int j = first_it; j < it; ++j) {
                    volatile int no_abort = 0;
                    mbar_wait(&full[j % a.stages], (j / a.stages) & 1, &no_abort, err, 0u, 100000000ull);
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        // Descriptors are built once per stage and stepped by plain adds (32
        // bytes = 2 in the address field): a single issuing thread is the
        // bottleneck, so every instruction between MMAs counts.
        if (lane == 0) {
            int it = 0, ci = 0;
            bool ok = true;
            int64_t q = qbeg, q0, q1, row;
            bool first, last;
            while (ok && next_chunk(q, qbeg, qend, a.nkb, a.chunk_blocks, q0, q1, row, first, last)) {
                const int buf = ci & 1;
                if (!(ok = mbar_wait(&acc_empty[buf], ((ci >> 1) & 1) ^ 1, abort, err, 2u))) break;
                tc_fence_after();
                const int grp = (int)(row / a.btiles);
                const int kgw = min(a.kgp, a.kp - grp * a.kgp);
                const uint32_t idesc = idesc_f16_f32(BM, (uint32_t)kgw) | a.idesc_ab;
                const uint32_t dacc = tmem + (uint32_t)(buf * a.kgp);
                uint32_t accf = 0;
                for (int64_t qs = q0; qs < q1; qs += kStageBlocks, ++it) {
                    const int nb = (q1 - qs >= kStageBlocks) ? kStageBlocks : (int)(q1 - qs);
                    const int slot = it % a.stages;
                    if (!(ok = mbar_wait(&full[slot], (it / a.stages) & 1, abort, err, 2u))) break;
                    tc_fence_after();
                    const uint32_t base = smem_u32(smem + (size_t)slot * a.slot_bytes);
                    const uint64_t dx = desc_sw128(base);
                    const uint64_t dv = desc_sw128(base + (uint32_t)kStageBlocks * kXBytes);
                    for (int u = 0; u < nb; ++u) {
                        const uint64_t dxu = dx + (uint64_t)u * (kXBytes >> 4);
                        const uint64_t dvu = dv + (uint64_t)u * (vbox >> 4);
#pragma unroll
                        for (int kk = 0; kk < BK / 16; ++kk) {
                            mma_f16(dacc, dxu + 2 * kk, dvu + 2 * kk, idesc, accf);
                            accf = 1u;
                        }
                    }
                    mma_commit(&empty[slot]);
                }
                if (ok) mma_commit(&acc_full[buf]);
                ++ci;
            }
            // every MMA issued by this thread has finished before TMEM is released
            mma_commit(mma_done);
            volatile int no_abort = 0;
            mbar_wait(mma_done, 0, &no_abort, err, 2u, 100000000ull);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int g = warp & 3;
        const int r = g * 32 + lane;
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        int ci = 0;
        int64_t q = qbeg, q0, q1, row;
        bool first, last;
        while (next_chunk(q, qbeg, qend, a.nkb, a.chunk_blocks, q0, q1, row, first, last)) {
            const int buf = ci & 1;
            if (!group_wait(&acc_full[buf], (ci >> 1) & 1, abort, err, 4u, 1, 128)) break;
            tc_fence_after();
            const int grp = (int)(row / a.btiles);
            const int64_t bt = row - (int64_t)grp * a.btiles;
            const int kgw = min(a.kgp, a.kp - grp * a.kgp);
            const bool valid = bt * BM + r < a.b;
            float* prow = a.P + ((size_t)(cta + row) * a.kgp) * BM + r;
            // every condition is decided once per 32 columns: the stores below
            // are straight-line code (a branch per element costs far more than
            // the store itself)
            for (int c0 = 0; c0 < kgw; c0 += 32) {
                uint32_t v[32];
                tmem_ld32(tmem + lane_base + (uint32_t)(buf * a.kgp + c0), v);
                const int nj = (c0 + 32 <= kgw) ? 32 : 16;     // group widths are multiples of 16
                // running sum of the segment's chunks: 32 tensor-memory columns per
                // 32 accumulator columns (the region is a whole number of 32-column
                // pieces, so the pieces past the group width are scratch)
                const uint32_t sp = tmem + lane_base + a.sum_col + (uint32_t)c0;
                if (!first) {
                    uint32_t sv[32];
                    tmem_ld32(sp, sv);
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        v[j] = __float_as_uint(__fadd_rn(__uint_as_float(sv[j]), __uint_as_float(v[j])));
                } else {
                    tmem_ld_wait();
                }
                if (!last) {
                    tmem_st32(sp, v);
                } else if (valid) {
                    float* pp = prow + (size_t)c0 * BM;
#pragma unroll
                    for (int j = 0; j < 16; ++j) pp[(size_t)j * BM] = __uint_as_float(v[j]);
                    if (nj == 32) {
#pragma unroll
                        for (int j = 16; j < 32; ++j) pp[(size_t)j * BM] = __uint_as_float(v[j]);
                    }
                }
            }
            tmem_st_wait();
            tc_fence_before();
            mbar_arrive(&acc_empty[buf]);
            ++ci;
        }
    }
    // single-lane roles rejoin their warps first: the CTA barrier is an aligned one
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, a.tmem_cols);
    }
}

__global__ void __launch_bounds__(kThreads, 1)
apply_w1_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_v,
                const W1Args a) {
    w1_body(&tm_x, &tm_v, a, blockIdx.x, gridDim.x);
}

// Several problems in one launch: CTA blocks [cta_off[p], cta_off[p + 1]) run
// problem p with its own arguments and tensor maps.
constexpr int kMaxGroup = 16;
struct GroupW1 {
    CUtensorMap tm[kMaxGroup][2];    // X, V^T
    W1Args args[kMaxGroup];
    int cta_off[kMaxGroup + 1];
    int count;
};

__device__ __forceinline__ int group_of(const int* off, int count, int64_t blk) {
    int p = 0;
    while (p + 1 < count && blk >= off[p + 1]) ++p;
    return p;
}

__global__ void __launch_bounds__(kThreads, 1) apply_w1_group_kernel(const __grid_constant__ GroupW1 g) {
    const int p = group_of(g.cta_off, g.count, blockIdx.x);
    w1_body(&g.tm[p][0], &g.tm[p][1], g.args[p], blockIdx.x - g.cta_off[p], g.cta_off[p + 1] - g.cta_off[p]);
}

// ================================================================ reduction
struct W2Args {
    int64_t b, btiles, nkb, Q;
    int P1;                   // phase-1 grid size
    int G, kgp, kp, k, planes;
    uint32_t tile_bytes;      // one plane of one row tile: 128 x kp x 2
    const float* P;
    const uint16_t* S;        // binary16 or bfloat16 encodings
    int bf16;                 // operands, W and output are bfloat16 (one plane)
    unsigned char* W;         // [row tile][plane][tile_bytes]
};

__device__ __forceinline__ float s_value(const W2Args& a, int j) {
    const uint16_t h = a.S[j];
    return a.bf16 ? bf16_bits_to_float(h) : __half2float(__ushort_as_half(h));
}

// CTA of the phase-1 grid whose range [floor(c Q / P1), floor((c+1) Q / P1))
// holds k-block q.
__device__ __forceinline__ int64_t cta_of(int64_t q, int64_t Q, int64_t P1) { return ((q + 1) * P1 + Q - 1) / Q - 1; }

// Writes the eight entries of W (row r, columns col0..col0+7) of row tile bt
// into the operand image(s).
__device__ __forceinline__ void put_w8(const W2Args& a, int64_t bt, int r, int col0, const float (&w)[8]) {
    uint32_t hi[4], lo[4];
    if (a.bf16) {
#pragma unroll
        for (int j = 0; j < 4; ++j) hi[j] = lo[j] = pack_bf162(w[2 * j], w[2 * j + 1]);
    } else {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const __half h0 = __float2half_rn(w[2 * j]), h1 = __float2half_rn(w[2 * j + 1]);
            hi[j] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
            lo[j] = pack_half2(w[2 * j] - __half2float(h0), w[2 * j + 1] - __half2float(h1));
        }
    }
    unsigned char* base = a.W + (size_t)bt * a.planes * a.tile_bytes + w_image_off((uint32_t)r, (uint32_t)col0);
    *reinterpret_cast<uint4*>(base) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
    if (a.planes == 2) *reinterpret_cast<uint4*>(base + a.tile_bytes) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
}

// One thread per (row tile, 8 columns, row): the partials of the entry are
// added in CTA order, kBatch partials' loads in flight at a time.
__device__ __forceinline__ void w2_body(const W2Args& a, int64_t blk) {
    const int cg8 = a.kp / 8;
    const int64_t e = blk * blockDim.x + threadIdx.x;
    if (e >= a.btiles * cg8 * BM) return;
    const int r = (int)(e % BM);
    const int64_t t = e / BM;
    const int cg = (int)(t % cg8);
    const int64_t bt = t / cg8;
    const int col0 = cg * 8;
    const int grp = col0 / a.kgp;               // group widths are multiples of 16
    const int j0 = col0 - grp * a.kgp;
    float w[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) w[i] = 0.0f;
    if (bt * BM + r < a.b) {
        const int64_t ur = (int64_t)grp * a.btiles + bt;
        const int64_t cf = cta_of(ur * a.nkb, a.Q, a.P1);
        const int64_t cl = cta_of(ur * a.nkb + a.nkb - 1, a.Q, a.P1);
        constexpr int kBatch = 4;
        const size_t pstride = (size_t)a.kgp * BM;
        const float* p0 = a.P + ((size_t)(cf + ur) * a.kgp + j0) * BM + r;
        const int64_t np = cl - cf + 1;
        for (int64_t c0 = 0; c0 < np; c0 += kBatch) {
            float t8[kBatch][8];
#pragma unroll
            for (int u = 0; u < kBatch; ++u)
                if (c0 + u < np) {
#pragma unroll
                    for (int i = 0; i < 8; ++i) t8[u][i] = __ldg(p0 + (size_t)(c0 + u) * pstride + (size_t)i * BM);
                }
#pragma unroll
            for (int u = 0; u < kBatch; ++u)
                if (c0 + u < np) {
#pragma unroll
                    for (int i = 0; i < 8; ++i) w[i] = (c0 + u == 0) ? t8[u][i] : __fadd_rn(w[i], t8[u][i]);
                }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) w[i] = __fmul_rn(w[i], col0 + i < a.k ? s_value(a, col0 + i) : 0.0f);
    }
    put_w8(a, bt, r, col0, w);
}

// For rows with many partials (small b): a CTA per (row tile, block of 32
// rows, 8 columns) with 16 warps.  Lane = row (coalesced loads of the
// partials' row runs), warp w adds partials w, w + 16, ... in order, several
// partials' loads in flight at a time; warp 0 then adds the 16 warp sums in
// warp order -- the same order on every run.
constexpr int kW2Slices = 16;
__device__ __forceinline__ void w2_slice_body(const W2Args& a, int64_t blk) {
    __shared__ float red[kW2Slices][8][33];
    const int cg8 = a.kp / 8;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t cg = blk % cg8;
    const int64_t t = blk / cg8;
    const int rb = (int)(t & 3);
    const int64_t bt = t >> 2;
    const int col0 = (int)cg * 8;
    const int r = rb * 32 + lane;
    const bool any = bt * BM + rb * 32 < a.b;
    float w[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) w[i] = 0.0f;
    if (any) {
        const int grp = col0 / a.kgp;               // group widths are multiples of 16
        const int j0 = col0 - grp * a.kgp;
        const int64_t ur = (int64_t)grp * a.btiles + bt;
        const int64_t cf = cta_of(ur * a.nkb, a.Q, a.P1);
        const int64_t cl = cta_of(ur * a.nkb + a.nkb - 1, a.Q, a.P1);
        const int64_t np = cl - cf + 1;
        const size_t pstride = (size_t)a.kgp * BM;
        const float* p0 = a.P + ((size_t)(cf + ur) * a.kgp + j0) * BM + r;
        if (bt * BM + r < a.b) {
            constexpr int kBatch = 4;
            for (int64_t c0 = warp; c0 < np; c0 += kW2Slices * kBatch) {
                float t8[kBatch][8];
#pragma unroll
                for (int u = 0; u < kBatch; ++u) {
                    const int64_t c = c0 + (int64_t)u * kW2Slices;
                    if (c < np) {
#pragma unroll
                        for (int i = 0; i < 8; ++i) t8[u][i] = __ldg(p0 + (size_t)c * pstride + (size_t)i * BM);
                    }
                }
#pragma unroll
                for (int u = 0; u < kBatch; ++u) {
                    if (c0 + (int64_t)u * kW2Slices < np) {
#pragma unroll
                        for (int i = 0; i < 8; ++i) w[i] = __fadd_rn(w[i], t8[u][i]);
                    }
                }
            }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) red[warp][i][lane] = w[i];
        __syncthreads();
        if (warp != 0) return;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            float v = red[0][i][lane];
#pragma unroll
            for (int q = 1; q < kW2Slices; ++q) v = __fadd_rn(v, red[q][i][lane]);
            w[i] = __fmul_rn(v, col0 + i < a.k ? s_value(a, col0 + i) : 0.0f);
        }
        if (bt * BM + r >= a.b) {
#pragma unroll
            for (int i = 0; i < 8; ++i) w[i] = 0.0f;
        }
    } else if (warp != 0) {
        return;
    }
    put_w8(a, bt, r, col0, w);
}

// Four CTAs a SM (at most 64 registers a thread): the 576 CTAs of a
// b = 8192, k' = 144 reduction run in one wave.
__global__ void __launch_bounds__(256, 4)
apply_w2_kernel(const W2Args a) {
    pdl_trigger();
    pdl_wait();                    // partials of the phase-1 grid
    w2_body(a, blockIdx.x);
}

__global__ void __launch_bounds__(32 * kW2Slices)
apply_w2_slice_kernel(const W2Args a) {
    pdl_trigger();
    pdl_wait();
    w2_slice_body(a, blockIdx.x);
}

struct GroupW2 {
    W2Args args[kMaxGroup];
    int blk_off[kMaxGroup + 1];
    int count;
};

// SLICE: the sliced reduction (many partials per entry) for every problem of
// the launch, else the plain one
template <bool SLICE>
__global__ void __launch_bounds__(SLICE ? 32 * kW2Slices : 256) apply_w2_group_kernel(const __grid_constant__ GroupW2 g) {
    pdl_trigger();
    pdl_wait();
    const int p = group_of(g.blk_off, g.count, blockIdx.x);
    if constexpr (SLICE) w2_slice_body(g.args[p], blockIdx.x - g.blk_off[p]);
    else w2_body(g.args[p], blockIdx.x - g.blk_off[p]);
}

// ================================================================ phase 2
struct YArgs {
    int64_t m, b, T, btiles;
    int kp, n2, kc2, mtiles, planes, stages;
    uint32_t u_bytes, slot_bytes, tile_bytes;
    uint32_t w_off, ystage_off, bar_off, tmem_cols;
    int out16, tma_store;
    int bf16;                 // bfloat16 operands and output
    uint32_t idesc_ab;        // operand-format bits of the MMA descriptor
    int ydepth;               // staging buffers per epilogue warp (1 or 2): TMA stores in flight
    // U resident (one plane of W): the CTA's units run column tile by column
    // tile; the U tile of a column tile is loaded once and W streams through
    // two buffers (the barriers full/empty[0..1]), so that each output tile
    // reads a W tile (128 x k') instead of a U tile (n2 x k') from L2
    int ures;
    const unsigned char* W;
    void* Y;
    // optional power-of-two scales of the operands, in groups of 32 rows of W
    // and 32 rows of U: entry (i, j) of the product is multiplied by
    // 2^-(esc_w[i / 32] + esc_u[j / 32]) (exact in binary32); esc_w[i] when
    // esc_w_rows is set
    const int* esc_w;
    int esc_w_rows;
    const int* esc_u;
};

// Phase 2 of one problem, run by CTA `cta` of the `ncta` CTAs given to it.
__device__ __forceinline__ void y_body(const CUtensorMap* tm_u, const CUtensorMap* tm_y, const YArgs& a, int64_t cta,
                                       int64_t ncta) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = align1024(smem_raw);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + a.bar_off);
    uint64_t* empty = full + a.stages;
    uint64_t* w_full = empty + a.stages;
    uint64_t* w_empty = w_full + 1;
    uint64_t* acc_full = w_empty + 1;          // [2]
    uint64_t* acc_empty = acc_full + 2;        // [2]
    uint64_t* mma_done = acc_empty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
    volatile int* abort = reinterpret_cast<int*>(tmem_slot + 1);
    unsigned int* err = &g_err_apply_tc;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t tbeg = a.T * cta / ncta;
    const int64_t tend = a.T * (cta + 1) / ncta;

    if (threadIdx.x == 0) {
        for (int i = 0; i < a.stages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        mbar_init(w_full, 1);
        mbar_init(w_empty, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 32 * kEpiWarpsY);
        }
        mbar_init(mma_done, 1);
        *abort = 0;
        fence_barrier_init();
        tma_prefetch_desc(tm_u);
        tma_prefetch_desc(tm_y);
    }
    if (warp == 1) tmem_alloc(tmem_slot, a.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    pdl_wait();                    // W images of the reduction kernel (the prologue above overlapped it)

    if (warp == 0 && a.ures) {
        // ------------------------------------------------------------ producer, U resident
        if (lane == 0) {
            int wl = 0, ul = 0;
            int64_t cur_mt = -1;
            bool ok = true;
            for (int64_t t = tbeg; t < tend && ok; ++t) {
                const int64_t mt = t / a.btiles;
                const int64_t bt = t - mt * a.btiles;
                if (mt != cur_mt) {
                    // U of the new column tile, once the MMAs on the previous one are done
                    if (!(ok = mbar_wait(w_empty, (ul & 1) ^ 1, abort, err, 1u))) break;
                    mbar_arrive_expect_tx(w_full, (uint32_t)a.kc2 * a.u_bytes);
                    for (int kc = 0; kc < a.kc2; ++kc)
                        tma_load_2d(smem + (size_t)kc * a.u_bytes, tm_u, kc * BK, (int32_t)(mt * a.n2), w_full);
                    ++ul;
                    cur_mt = mt;
                }
                const int slot = wl & 1;
                if (!(ok = mbar_wait(&empty[slot], ((wl >> 1) & 1) ^ 1, abort, err, 1u))) break;
                mbar_arrive_expect_tx(&full[slot], a.tile_bytes);
                bulk_load(smem + a.w_off + (size_t)slot * a.tile_bytes, a.W + (size_t)bt * a.tile_bytes, a.tile_bytes,
                          &full[slot]);
                ++wl;
            }
            if (!ok) {
                volatile int no_abort = 0;
                for (int j = wl - 2 > 0 ? wl - 2 : 0; j < wl; ++j)
                    mbar_wait(&full[j & 1], (j >> 1) & 1, &no_abort, err, 0u, 100000000ull);
                if (ul > 0) mbar_wait(w_full, (ul - 1) & 1, &no_abort, err, 0u, 100000000ull);
            }
        }
    } else if (warp == 1 && a.ures) {
        // ------------------------------------------------------------ MMA issuer, U resident
        if (lane == 0) {
            int wl = 0, ul = 0, tl = 0;
            int64_t cur_mt = -1;
            bool ok = true;
            const uint32_t idesc2 = idesc_f16_f32(BM, (uint32_t)a.n2) | a.idesc_ab;
            for (int64_t t = tbeg; t < tend && ok; ++t, ++tl) {
                const int64_t mt = t / a.btiles;
                if (mt != cur_mt) {
                    if (ul > 0) mma_commit(w_empty);        // the previous U is free once these MMAs finish
                    if (!(ok = mbar_wait(w_full, ul & 1, abort, err, 2u))) break;
                    tc_fence_after();
                    ++ul;
                    cur_mt = mt;
                }
                const int ab = tl & 1;
                if (!(ok = mbar_wait(&acc_empty[ab], ((tl >> 1) & 1) ^ 1, abort, err, 2u))) break;
                const int slot = wl & 1;
                if (!(ok = mbar_wait(&full[slot], (wl >> 1) & 1, abort, err, 2u))) break;
                tc_fence_after();
                const uint64_t whd = smem_desc(smem_u32(smem + a.w_off + (size_t)slot * a.tile_bytes), 2048, 128, 0);
                const uint32_t dcol = tmem + (uint32_t)(ab * a.n2);
                for (int kc = 0; kc < a.kc2; ++kc) {
                    const uint64_t ud = desc_sw128(smem_u32(smem + (size_t)kc * a.u_bytes));
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const int ks = kc * (BK / 16) + kk;
                        if (ks * 16 >= a.kp) break;
                        mma_f16(dcol, whd + (uint64_t)ks * 256u, ud + 2 * kk, idesc2, (kc | kk) != 0);
                    }
                }
                mma_commit(&empty[slot]);
                mma_commit(&acc_full[ab]);
                ++wl;
            }
            mma_commit(mma_done);
            volatile int no_abort = 0;
            mbar_wait(mma_done, 0, &no_abort, err, 2u, 100000000ull);
        }
    } else if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int it = 0, wl = 0;
            int64_t cur_bt = -1;
            bool ok = true;
            for (int64_t t = tbeg; t < tend && ok; ++t) {
                const int64_t bt = t / a.mtiles;
                const int mt = (int)(t - bt * a.mtiles);
                if (bt != cur_bt) {
                    // W of the new row tile, once the MMAs on the previous one are done
                    if (!(ok = mbar_wait(w_empty, (wl & 1) ^ 1, abort, err, 1u))) break;
                    mbar_arrive_expect_tx(w_full, (uint32_t)a.planes * a.tile_bytes);
                    for (int p = 0; p < a.planes; ++p)
                        bulk_load(smem + a.w_off + (size_t)p * a.tile_bytes,
                                  a.W + ((size_t)bt * a.planes + p) * a.tile_bytes, a.tile_bytes, w_full);
                    ++wl;
                    cur_bt = bt;
                }
                for (int kc = 0; kc < a.kc2; ++kc, ++it) {
                    const int slot = it % a.stages;
                    if (!(ok = mbar_wait(&empty[slot], ((it / a.stages) & 1) ^ 1, abort, err, 1u))) break;
                    mbar_arrive_expect_tx(&full[slot], a.u_bytes);
                    tma_load_2d(smem + (size_t)slot * a.slot_bytes, tm_u, kc * BK, (int32_t)(mt * a.n2),
                                &full[slot]);
                }
            }
            if (!ok) {
                volatile int no_abort = 0;
                const int first = it - a.stages > 0 ? it - a.stages : 0;
                for (int j = first; j < it; ++j)
                    mbar_wait(&full[j % a.stages], (j / a.stages) & 1, &no_abort, err, 0u, 100000000ull);
                if (wl > 0) mbar_wait(w_full, (wl - 1) & 1, &no_abort, err, 0u, 100000000ull);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            int it = 0, wl = 0, tl = 0;
            int64_t cur_bt = -1;
            bool ok = true;
            const uint32_t whi = smem_u32(smem + a.w_off);
            const uint64_t whd = smem_desc(whi, 2048, 128, 0);
            const uint64_t wld = smem_desc(whi + a.tile_bytes, 2048, 128, 0);
            const uint32_t idesc2 = idesc_f16_f32(BM, (uint32_t)a.n2) | a.idesc_ab;
            for (int64_t t = tbeg; t < tend && ok; ++t, ++tl) {
                const int64_t bt = t / a.mtiles;
                if (bt != cur_bt) {
                    if (wl > 0) mma_commit(w_empty);        // the previous W is free once these MMAs finish
                    if (!(ok = mbar_wait(w_full, wl & 1, abort, err, 2u))) break;
                    tc_fence_after();
                    ++wl;
                    cur_bt = bt;
                }
                const int ab = tl & 1;
                if (!(ok = mbar_wait(&acc_empty[ab], ((tl >> 1) & 1) ^ 1, abort, err, 2u))) break;
                tc_fence_after();
                const uint32_t dcol = tmem + (uint32_t)(ab * a.n2);
                for (int kc = 0; kc < a.kc2; ++kc, ++it) {
                    const int slot = it % a.stages;
                    if (!(ok = mbar_wait(&full[slot], (it / a.stages) & 1, abort, err, 2u))) break;
                    tc_fence_after();
                    const uint64_t ud = desc_sw128(smem_u32(smem + (size_t)slot * a.slot_bytes));
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const int ks = kc * (BK / 16) + kk;
                        if (ks * 16 >= a.kp) break;
                        // W in the canonical layout: K-direction core matrices 2048 B apart,
                        // so 16 ranks = 4096 B = 256 in the address field
                        mma_f16(dcol, whd + (uint64_t)ks * 256u, ud + 2 * kk, idesc2, (kc | kk) != 0);
                        if (a.planes == 2) mma_f16(dcol, wld + (uint64_t)ks * 256u, ud + 2 * kk, idesc2, 1u);
                    }
                    mma_commit(&empty[slot]);
                }
                if (ok) mma_commit(&acc_full[ab]);
            }
            mma_commit(mma_done);
            volatile int no_abort = 0;
            mbar_wait(mma_done, 0, &no_abort, err, 2u, 100000000ull);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int g = warp & 3;
        const int r = g * 32 + lane;
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        const int ecols = a.out16 ? 64 : 32;       // columns per 128-byte staging row
        const int half = (warp - 2) >> 2;          // which of the two warps of this lane quarter
        // the four warps of a half stage one column chunk of all 128 rows (one
        // 32-row slice each, lane quarter g at g * 4 KB) and one of them stores it
        // with a single 128-row TMA box
        const bool issuer = (g == 0) && (lane == 0);
        unsigned char* hstage = smem + a.ystage_off + (size_t)half * a.ydepth * (128 * 128);
        int chunk = 0, tl = 0;
        for (int64_t t = tbeg; t < tend; ++t, ++tl) {
            int64_t bt;
            int mt;
            if (a.ures) {
                mt = (int)(t / a.btiles);
                bt = t - (int64_t)mt * a.btiles;
            } else {
                bt = t / a.mtiles;
                mt = (int)(t - bt * a.mtiles);
            }
            const int64_t row0 = bt * BM;
            const int ab = tl & 1;
            const bool scaled = a.esc_w != nullptr;
            // this warp's 32 rows are one scale group of W (or the thread's row
            // has its own scale); lane j holds the scale of the tile's j-th
            // group of 32 columns (read before the accumulator wait, so the
            // loads overlap it)
            int ew = 0, eu_lane = 0;
            if (scaled) {
                if (a.esc_w_rows) ew = row0 + r < a.b ? a.esc_w[row0 + r] : 0;
                else ew = row0 + g * 32 < a.b ? a.esc_w[(row0 >> 5) + g] : 0;
                const int64_t cl = (int64_t)mt * a.n2 + lane * 32;
                eu_lane = (lane < (a.n2 >> 5) && cl < a.m) ? a.esc_u[cl >> 5] : 0;
            }
            if (!group_wait(&acc_full[ab], (tl >> 1) & 1, abort, err, 4u, 1, 32 * kEpiWarpsY)) break;
            tc_fence_after();
            for (int cc = half * ecols; cc < a.n2; cc += 2 * ecols, ++chunk) {
                uint32_t v[64];
                const uint32_t tcol = tmem + lane_base + (uint32_t)(ab * a.n2 + cc);
                tmem_ld32(tcol, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
                if (a.out16) tmem_ld32(tcol + 32, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
                tmem_ld_wait();
                const int64_t col0 = (int64_t)mt * a.n2 + cc;
                if (scaled) {
                    // columns [col0, col0 + 32) and, for binary16 output, [col0 + 32, col0 + 64)
                    // are one scale group of U each
                    const int eu0 = __shfl_sync(0xffffffffu, eu_lane, cc >> 5);
                    const float f0 = __int_as_float((127 - ew - eu0) << 23);
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] = __float_as_uint(__fmul_rn(__uint_as_float(v[j]), f0));
                    if (a.out16) {
                        const int eu1 = __shfl_sync(0xffffffffu, eu_lane, (cc >> 5) + 1);
                        const float f1 = __int_as_float((127 - ew - eu1) << 23);
#pragma unroll
                        for (int j = 32; j < 64; ++j) v[j] = __float_as_uint(__fmul_rn(__uint_as_float(v[j]), f1));
                    }
                }
                {
                    uint32_t packed[32];
                    if (a.out16 && a.bf16) {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            packed[j] = pack_bf162(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    } else if (a.out16) {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            packed[j] = pack_half2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j) packed[j] = v[j];
                    }
                    unsigned char* box = hstage + (size_t)(chunk & (a.ydepth - 1)) * (128 * 128);
                    unsigned char* sb = box + (size_t)g * (32 * 128);
                    if (a.tma_store && chunk >= a.ydepth && issuer) {
                        if (a.ydepth == 2) bulk_wait_read<1>();
                        else bulk_wait_read<0>();
                    }
                    named_bar_sync(2 + half, 128);      // the buffer's previous store has read it
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const uint32_t off = (uint32_t)lane * 128u + (uint32_t)((j ^ (lane & 7)) * 16);
                        *reinterpret_cast<uint4*>(sb + off) =
                            make_uint4(packed[4 * j], packed[4 * j + 1], packed[4 * j + 2], packed[4 * j + 3]);
                    }
                    if (a.tma_store) {
                        fence_proxy_async_smem();
                        named_bar_sync(2 + half, 128);      // all four slices are written
                        if (issuer) {
                            if (col0 < a.m) tma_store_2d(tm_y, (int32_t)col0, (int32_t)row0, box);
                            bulk_commit();      // one group per chunk, even empty: the staging reuse counts on it
                        }
                    } else {
                        // Rows whose pitch is not a multiple of 16 bytes (no TMA store): the
                        // warp writes its own 32 staged rows, lane l the row's bytes
                        // 4l..4l+3 -- one coalesced 128-byte run per row.  The 32 shared
                        // loads come first, so that the stores do not each wait for one
                        // (a load-store chain per row ran the ten-matrix batch's product
                        // at about 1.2 TB/s).
                        __syncwarp();
                        const int nvalid = (int)(a.m - col0 < ecols ? a.m - col0 : ecols);   // columns inside Y
                        const int64_t rbase = row0 + g * 32;
                        const int nrows = a.b - rbase >= 32 ? 32 : (a.b - rbase > 0 ? (int)(a.b - rbase) : 0);
                        uint32_t wv[32];
#pragma unroll
                        for (int rr = 0; rr < 32; ++rr)
                            wv[rr] = *reinterpret_cast<const uint32_t*>(
                                sb + rr * 128 + (((lane >> 2) ^ (rr & 7)) * 16) + (lane & 3) * 4);
                        if (a.out16) {
                            const int c = 2 * lane;
#pragma unroll
                            for (int rr = 0; rr < 32; ++rr) {
                                if (rr >= nrows) break;
                                uint16_t* y = static_cast<uint16_t*>(a.Y) + (rbase + rr) * a.m + col0 + c;
                                const uint32_t w = wv[rr];
                                if (c + 1 < nvalid && ((reinterpret_cast<uintptr_t>(y) & 3u) == 0)) {
                                    *reinterpret_cast<uint32_t*>(y) = w;
                                } else {
                                    if (c < nvalid) y[0] = (uint16_t)(w & 0xffffu);
                                    if (c + 1 < nvalid) y[1] = (uint16_t)(w >> 16);
                                }
                            }
                        } else if (lane < nvalid) {
                            uint32_t* y = static_cast<uint32_t*>(a.Y) + rbase * a.m + col0 + lane;
#pragma unroll
                            for (int rr = 0; rr < 32; ++rr) {
                                if (rr >= nrows) break;
                                y[(int64_t)rr * a.m] = wv[rr];
                            }
                        }
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(&acc_empty[ab]);
        }
        if (lane == 0 && a.tma_store) bulk_wait<0>();
    }
    // single-lane roles rejoin their warps first: the CTA barrier is an aligned one
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, a.tmem_cols);
    }
}

__global__ void __launch_bounds__(kThreadsY, 1)
apply_y_kernel(const __grid_constant__ CUtensorMap tm_u, const __grid_constant__ CUtensorMap tm_y, const YArgs a) {
    y_body(&tm_u, &tm_y, a, blockIdx.x, gridDim.x);
}

struct GroupY {
    CUtensorMap tm[kMaxGroup][2];    // U, Y
    YArgs args[kMaxGroup];
    int cta_off[kMaxGroup + 1];
    int count;
};

__global__ void __launch_bounds__(kThreadsY, 1) apply_y_group_kernel(const __grid_constant__ GroupY g) {
    const int p = group_of(g.cta_off, g.count, blockIdx.x);
    y_body(&g.tm[p][0], &g.tm[p][1], g.args[p], blockIdx.x - g.cta_off[p], g.cta_off[p + 1] - g.cta_off[p]);
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

lrc_status get_encoder() {
    std::call_once(g_encode_once, [] {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    });
    if (!g_encode) {
        set_error("cuTensorMapEncodeTiled is not available from the driver");
        return LRC_ERR_CUDA;
    }
    return LRC_OK;
}

// 2-D map over a row-major [rows x cols] array with a row pitch of `pitch_bytes`
// (128-byte swizzled boxes unless stated).
lrc_status make_map(CUtensorMap* map, CUtensorMapDataType dt, const void* base, int64_t cols, int64_t rows,
                    int64_t pitch_bytes, uint32_t box_cols, uint32_t box_rows, const char* what,
                    CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)pitch_bytes};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled failed for %s (CUresult %d)", what, (int)r);
        return LRC_ERR_CUDA;
    }
    return LRC_OK;
}

uint32_t pow2_cols(uint32_t c) {
    uint32_t p = 32;
    while (p < c) p <<= 1;
    return p;
}

constexpr size_t kSmemMax = 227 * 1024;


size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Phase-2 plan for a b x m product with kp columns of W per plane: tile
// width n2, ring depth, shared-memory offsets.  `balance` picks the width
// that gives the CTAs the most even share (largest tiles per CTA x width);
// otherwise 256-wide tiles whenever there are at least two per SM.
lrc_status plan_y(YArgs& a3, size_t& smem3, int64_t m, int64_t b, int kp, int planes, bool out16, bool balance) {
    const int sms = sm_count();
    const int64_t btiles = (b + BM - 1) / BM;
    a3.m = m;
    a3.b = b;
    a3.kp = kp;
    a3.kc2 = (kp + BK - 1) / BK;
    a3.planes = planes;
    a3.out16 = out16 ? 1 : 0;
    const int e_out = out16 ? 2 : 4;
    a3.tma_store = ((m * e_out) % 16 == 0) ? 1 : 0;
    const uint32_t tile_bytes = (uint32_t)BM * (uint32_t)kp * 2u;
    int order[2] = {256, 128};
    if (balance) {
        const int64_t w256 = (btiles * ((m + 255) / 256) + sms - 1) / sms * 256;
        const int64_t w128 = (btiles * ((m + 127) / 128) + sms - 1) / sms * 128;
        if (w128 < w256) {
            order[0] = 128;
            order[1] = 256;
        }
    }
    smem3 = 0;
    for (int n2 : order) {
        if (!balance && n2 == 256 && btiles * ((m + 255) / 256) < 2 * (int64_t)sms) continue;   // too few tiles
        // two staging buffers per epilogue warp if they fit, else one; then the ring
        for (int depth = 2; depth >= 1 && !smem3; --depth) {
            for (int stages = 4; stages >= 2 && !smem3; --stages) {
                if (n2 == 256 && stages < 3) break;      // prefer a deeper ring with narrower tiles
                const uint32_t u_bytes = (uint32_t)n2 * 128;
                size_t off = (size_t)stages * u_bytes;
                const size_t w_off = off;
                off += (size_t)planes * tile_bytes;
                off = round_up(off, 1024);
                const size_t ystage_off = off;
                off += (size_t)kEpiWarpsY * depth * 32 * 128;
                const size_t bar_off = off;
                off += (size_t)(2 * stages + 7) * 8 + 16;
                if (off + 1024 > kSmemMax) continue;
                a3.n2 = n2;
                a3.stages = stages;
                a3.ydepth = depth;
                a3.u_bytes = u_bytes;
                a3.slot_bytes = u_bytes;
                a3.w_off = (uint32_t)w_off;
                a3.ystage_off = (uint32_t)ystage_off;
                a3.bar_off = (uint32_t)bar_off;
                smem3 = off + 1024;
            }
        }
        if (smem3) break;
    }
    if (!smem3) {
        set_error("binary16 product: %d columns of W do not fit in shared memory", kp);
        return LRC_ERR_UNSUPPORTED;
    }
    a3.mtiles = (int)((m + a3.n2 - 1) / a3.n2);
    a3.btiles = btiles;
    a3.T = btiles * a3.mtiles;
    a3.tmem_cols = pow2_cols(2u * (uint32_t)a3.n2);
    a3.ures = 0;
    return LRC_OK;
}

// The U-resident layout of the product (one plane of W): U tile of kc2 boxes,
// two W buffers, staging; false when it does not fit in shared memory, and
// for a single k-block, where the U ring streams one box per output tile and
// the per-tile W copy would only add latency (measured: k' = 48 and 64 were
// 2-9 % slower U-resident, k' = 144 7 % faster).
bool plan_y_ures(YArgs& a3, size_t& smem3, uint32_t tile_bytes) {
    if (a3.planes != 1 || a3.kc2 < 2) return false;
    for (int depth = 2; depth >= 1; --depth) {
        size_t off = (size_t)a3.kc2 * a3.u_bytes;
        const size_t w_off = off;
        off += 2 * (size_t)tile_bytes;
        off = round_up(off, 1024);
        const size_t ystage_off = off;
        off += (size_t)kEpiWarpsY * depth * 32 * 128;
        const size_t bar_off = off;
        off += (size_t)(2 * 2 + 7) * 8 + 16;
        if (off + 1024 > kSmemMax) continue;
        a3.ures = 1;
        a3.stages = 2;
        a3.ydepth = depth;
        a3.w_off = (uint32_t)w_off;
        a3.ystage_off = (uint32_t)ystage_off;
        a3.bar_off = (uint32_t)bar_off;
        smem3 = off + 1024;
        return true;
    }
    return false;
}

CUtensorMapDataType t16(bool bf16) { return bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16; }

lrc_status make_y_map(CUtensorMap* ty, const YArgs& a3, void* Y, int64_t m, int64_t b, bool out16) {
    if (!a3.tma_store) return LRC_OK;   // unused by the kernel
    const int e_out = out16 ? 2 : 4;
    return make_map(ty, out16 ? t16(a3.bf16 != 0) : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, Y, m, b, m * e_out,
                    out16 ? 64 : 32, BM, "Y");
}

lrc_status launch_y(const CUtensorMap& tu, const CUtensorMap& ty, const YArgs& a3, size_t smem3, int64_t P3,
                    cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(apply_y_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem3);
    if (e != cudaSuccess) return cuda_fail(e, "apply_y_kernel smem attribute");
    e = launch_pdl(apply_y_kernel, dim3((unsigned)P3), dim3(kThreadsY), smem3, s, tu, a3.tma_store ? ty : tu, a3);
    if (e != cudaSuccess) return cuda_fail(e, "apply_y_kernel launch");
    return after_launch("apply_y_kernel");
}

}  // namespace

namespace {

// The three launches of one binary16 / bfloat16 apply, planned in two
// stages: the shapes (column groups, ring depths, tile widths), then -- once
// the phase-1 and phase-2 CTA counts and the workspace are known -- the
// pointers, the reduction's layout and the tensor maps.
struct F16Plan {
    W1Args a1{};
    W2Args a2{};
    YArgs a3{};
    size_t smem1 = 0, smem3 = 0;
    int64_t P1 = 0, P3 = 0, w2_blocks = 0;
    bool slice = false;
    CUtensorMap tx, tv, tu, ty;
};

lrc_status plan_f16_shape(int64_t m, int64_t n, int64_t k, int64_t b, bool out16, bool bf16, F16Plan& pl) {
    if (bf16 && !out16) {
        set_error("bfloat16 apply: the output is bfloat16");
        return LRC_ERR_UNSUPPORTED;
    }
    const int kp = (int)((k + 15) / 16 * 16);
    if (kp > 512) {
        set_error("binary16 apply supports rank up to 512 (got %lld)", (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    const int64_t btiles = (b + BM - 1) / BM;
    const int planes = out16 ? 1 : 2;
    const uint32_t tile_bytes = (uint32_t)BM * (uint32_t)kp * 2u;

    // ---- phase-1 plan: column groups, ring depth, running sum
    W1Args& a1 = pl.a1;
    a1.b = b;
    a1.btiles = btiles;
    a1.nkb = (n + BK - 1) / BK;
    const int kg_max = out16 ? 256 : 160;
    a1.G = (kp + kg_max - 1) / kg_max;
    a1.kgp = ((kp + a1.G - 1) / a1.G + 15) / 16 * 16;
    a1.kp = kp;
    a1.Q = btiles * a1.G * a1.nkb;
    a1.idesc_ab = bf16 ? kIdescBF16 : 0u;
    a1.chunk_blocks = out16 ? (int)(a1.nkb < 0x7fffffff ? a1.nkb : 0x7fffffff) : kChunkBlocks;
    const bool use_sum = a1.chunk_blocks < a1.nkb;
    a1.slot_bytes = (uint32_t)round_up((size_t)kStageBlocks * (kXBytes + (size_t)a1.kgp * 128), 1024);
    for (int stages = 6; stages >= 2; --stages) {
        size_t off = (size_t)stages * a1.slot_bytes;
        off = round_up(off, 8);
        const size_t bar_off = off;
        off += (size_t)(2 * stages + 5) * 8 + 16;
        if (off + 1024 <= kSmemMax) {
            a1.stages = stages;
            a1.bar_off = (uint32_t)bar_off;
            pl.smem1 = off + 1024;
            break;
        }
    }
    if (!pl.smem1) {
        set_error("binary16 apply: rank %lld does not fit in shared memory", (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    // two accumulators at columns 0 and kgp; the epilogue reads 32 columns at a
    // time; the running sum of FP32 output follows in whole 32-column pieces
    const uint32_t acc_cols = (uint32_t)a1.kgp + (uint32_t)round_up((size_t)a1.kgp, 32);
    a1.sum_col = (uint32_t)round_up(acc_cols, 32);
    a1.tmem_cols = pow2_cols(use_sum ? a1.sum_col + (uint32_t)round_up((size_t)a1.kgp, 32) : acc_cols);
    if (a1.tmem_cols > 512) {
        set_error("binary16 apply: rank %lld does not fit in tensor memory", (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }

    // ---- phase-2 plan: tile width, ring depth
    lrc_status st = plan_y(pl.a3, pl.smem3, m, b, kp, planes, out16, false);
    if (st != LRC_OK) return st;
    // 16-bit output: a W tile (128 x k') per output tile instead of a U tile
    // (n2 x k'), where the U tile fits in shared memory with two W buffers
    plan_y_ures(pl.a3, pl.smem3, tile_bytes);
    pl.a3.tile_bytes = tile_bytes;
    pl.a3.bf16 = bf16 ? 1 : 0;
    pl.a3.idesc_ab = bf16 ? kIdescBF16 : 0u;
    return LRC_OK;
}

// Workspace of the call for P1 phase-1 CTAs: W images, then the partials.
size_t f16_ws_images(const F16Plan& pl) {
    const int planes = pl.a3.planes;
    return round_up((size_t)pl.a1.btiles * planes * pl.a3.tile_bytes, 256);
}
size_t f16_ws_bytes(const F16Plan& pl, int64_t P1) {
    return f16_ws_images(pl) +
           round_up((size_t)(pl.a1.btiles * pl.a1.G + P1) * pl.a1.kgp * BM * sizeof(float), 256);
}

lrc_status plan_f16_finish(F16Plan& pl, const void* U, const void* S, const void* Vt, const void* X, void* Y,
                           int64_t m, int64_t n, int64_t k, int64_t b, bool out16, bool bf16, int64_t P1,
                           int64_t P3, unsigned char* ws) {
    W1Args& a1 = pl.a1;
    YArgs& a3 = pl.a3;
    pl.P1 = P1;
    pl.P3 = P3;
    a1.P = reinterpret_cast<float*>(ws + f16_ws_images(pl));
    a3.W = ws;
    a3.Y = Y;
    W2Args& a2 = pl.a2;
    a2.b = b;
    a2.btiles = a1.btiles;
    a2.nkb = a1.nkb;
    a2.Q = a1.Q;
    a2.P1 = (int)P1;
    a2.G = a1.G;
    a2.kgp = a1.kgp;
    a2.kp = a1.kp;
    a2.k = (int)k;
    a2.planes = a3.planes;
    a2.tile_bytes = a3.tile_bytes;
    a2.P = a1.P;
    a2.S = static_cast<const uint16_t*>(S);
    a2.bf16 = bf16 ? 1 : 0;
    a2.W = ws;
    const int kp = a1.kp;
    const int64_t max_parts = (a1.nkb * P1 + a1.Q - 1) / a1.Q + 1;     // CTAs sharing one row, at most
    pl.slice = max_parts >= 16;
    pl.w2_blocks = pl.slice ? a1.btiles * 4 * (kp / 8) : (a1.btiles * (kp / 8) * BM + 255) / 256;

    const int64_t ldn = lrc_packed_ld(n), ldk = lrc_packed_ld(k);
    const CUtensorMapDataType dt = t16(bf16);
    lrc_status st;
    if ((st = make_map(&pl.tx, dt, X, n, b, ldn * 2, BK, BM, "X")) != LRC_OK) return st;
    if ((st = make_map(&pl.tv, dt, Vt, n, k, ldn * 2, BK, (uint32_t)a1.kgp, "Vt")) != LRC_OK) return st;
    if ((st = make_map(&pl.tu, dt, U, k, m, ldk * 2, BK, (uint32_t)a3.n2, "U")) != LRC_OK) return st;
    if ((st = make_y_map(&pl.ty, a3, Y, m, b, out16)) != LRC_OK) return st;
    if (!a3.tma_store) pl.ty = pl.tu;          // unused by the kernel
    return LRC_OK;
}

}  // namespace

lrc_status launch_apply_f16(const void* U, const void* S, const void* Vt, const void* X, void* Y, int64_t m,
                            int64_t n, int64_t k, int64_t b, bool out16, cudaStream_t s, bool bf16) {
    lrc_status st = get_encoder();
    if (st != LRC_OK) return st;
    F16Plan pl;
    if ((st = plan_f16_shape(m, n, k, b, out16, bf16, pl)) != LRC_OK) return st;
    const int sms = sm_count();
    const int64_t P1 = pl.a1.Q < sms ? pl.a1.Q : sms;
    const int64_t P3 = pl.a3.T < sms ? pl.a3.T : sms;
    void* ws = nullptr;
    if ((st = stream_workspace(s, f16_ws_bytes(pl, P1), &ws)) != LRC_OK) return st;
    if ((st = plan_f16_finish(pl, U, S, Vt, X, Y, m, n, k, b, out16, bf16, P1, P3, static_cast<unsigned char*>(ws))) !=
        LRC_OK)
        return st;

    cudaError_t e = cudaFuncSetAttribute(apply_w1_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl.smem1);
    if (e != cudaSuccess) return cuda_fail(e, "apply_w1_kernel smem attribute");
    apply_w1_kernel<<<(unsigned)P1, kThreads, pl.smem1, s>>>(pl.tx, pl.tv, pl.a1);
    if ((st = after_launch("apply_w1_kernel")) != LRC_OK) return st;
    if (pl.slice) {
        e = launch_pdl(apply_w2_slice_kernel, dim3((unsigned)pl.w2_blocks), dim3(32 * kW2Slices), 0, s, pl.a2);
        if (e != cudaSuccess) return cuda_fail(e, "apply_w2_slice_kernel launch");
        if ((st = after_launch("apply_w2_slice_kernel")) != LRC_OK) return st;
    } else {
        e = launch_pdl(apply_w2_kernel, dim3((unsigned)pl.w2_blocks), dim3(256), 0, s, pl.a2);
        if (e != cudaSuccess) return cuda_fail(e, "apply_w2_kernel launch");
        if ((st = after_launch("apply_w2_kernel")) != LRC_OK) return st;
    }
    return launch_y(pl.tu, pl.ty, pl.a3, pl.smem3, P3, s);
}

int apply_f16_group_max() { return kMaxGroup; }

lrc_status launch_apply_f16_group(const ApplyProblem* pr, int count, bool out16, bool bf16, cudaStream_t s) {
    if (count < 1 || count > kMaxGroup) {
        set_error("grouped binary16 apply: 1 to %d problems per launch (got %d)", kMaxGroup, count);
        return LRC_ERR_INVALID_ARG;
    }
    lrc_status st = get_encoder();
    if (st != LRC_OK) return st;
    static thread_local F16Plan pls[kMaxGroup];
    int64_t qsum = 0, tsum = 0;
    for (int p = 0; p < count; ++p) {
        pls[p] = F16Plan{};
        if ((st = plan_f16_shape(pr[p].m, pr[p].n, pr[p].k, pr[p].b, out16, bf16, pls[p])) != LRC_OK) return st;
        qsum += pls[p].a1.Q;
        tsum += pls[p].a3.T;
    }
    // CTAs in proportion to each problem's share of the units (at least one,
    // at most one per unit), about one SM's worth in all
    const int sms = sm_count();
    int64_t P1[kMaxGroup], P3[kMaxGroup];
    size_t ws_bytes = 0;
    for (int p = 0; p < count; ++p) {
        int64_t c1 = sms * pls[p].a1.Q / qsum, c3 = sms * pls[p].a3.T / tsum;
        c1 = c1 < 1 ? 1 : (c1 > pls[p].a1.Q ? pls[p].a1.Q : c1);
        c3 = c3 < 1 ? 1 : (c3 > pls[p].a3.T ? pls[p].a3.T : c3);
        P1[p] = c1;
        P3[p] = c3;
        ws_bytes += f16_ws_bytes(pls[p], c1);
    }
    void* wsp = nullptr;
    if ((st = stream_workspace(s, ws_bytes, &wsp)) != LRC_OK) return st;
    unsigned char* ws = static_cast<unsigned char*>(wsp);
    static thread_local GroupW1 g1;
    static thread_local GroupW2 g2[2];
    static thread_local GroupY g3;
    g1.count = g3.count = count;
    g1.cta_off[0] = g3.cta_off[0] = 0;
    g2[0].count = g2[1].count = 0;
    g2[0].blk_off[0] = g2[1].blk_off[0] = 0;
    size_t smem1 = 0, smem3 = 0;
    for (int p = 0; p < count; ++p) {
        F16Plan& pl = pls[p];
        if ((st = plan_f16_finish(pl, pr[p].U, pr[p].S, pr[p].Vt, pr[p].X, pr[p].Y, pr[p].m, pr[p].n, pr[p].k, pr[p].b,
                                  out16, bf16, P1[p], P3[p], ws)) != LRC_OK)
            return st;
        ws += f16_ws_bytes(pl, P1[p]);
        g1.tm[p][0] = pl.tx;
        g1.tm[p][1] = pl.tv;
        g1.args[p] = pl.a1;
        g1.cta_off[p + 1] = g1.cta_off[p] + (int)P1[p];
        GroupW2& w = g2[pl.slice ? 1 : 0];
        w.args[w.count] = pl.a2;
        w.blk_off[w.count + 1] = w.blk_off[w.count] + (int)pl.w2_blocks;
        ++w.count;
        g3.tm[p][0] = pl.tu;
        g3.tm[p][1] = pl.ty;
        g3.args[p] = pl.a3;
        g3.cta_off[p + 1] = g3.cta_off[p] + (int)P3[p];
        smem1 = pl.smem1 > smem1 ? pl.smem1 : smem1;
        smem3 = pl.smem3 > smem3 ? pl.smem3 : smem3;
    }
    cudaError_t e = cudaFuncSetAttribute(apply_w1_group_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
    if (e != cudaSuccess) return cuda_fail(e, "apply_w1_group_kernel smem attribute");
    apply_w1_group_kernel<<<(unsigned)g1.cta_off[count], kThreads, smem1, s>>>(g1);
    if ((st = after_launch("apply_w1_group_kernel")) != LRC_OK) return st;
    if (g2[0].count) {
        e = launch_pdl(apply_w2_group_kernel<false>, dim3((unsigned)g2[0].blk_off[g2[0].count]), dim3(256), 0, s, g2[0]);
        if (e != cudaSuccess) return cuda_fail(e, "apply_w2_group_kernel launch");
        if ((st = after_launch("apply_w2_group_kernel")) != LRC_OK) return st;
    }
    if (g2[1].count) {
        e = launch_pdl(apply_w2_group_kernel<true>, dim3((unsigned)g2[1].blk_off[g2[1].count]), dim3(32 * kW2Slices), 0,
                       s, g2[1]);
        if (e != cudaSuccess) return cuda_fail(e, "apply_w2_group_kernel launch");
        if ((st = after_launch("apply_w2_group_kernel")) != LRC_OK) return st;
    }
    e = cudaFuncSetAttribute(apply_y_group_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem3);
    if (e != cudaSuccess) return cuda_fail(e, "apply_y_group_kernel smem attribute");
    e = launch_pdl(apply_y_group_kernel, dim3((unsigned)g3.cta_off[count]), dim3(kThreadsY), smem3, s, g3);
    if (e != cudaSuccess) return cuda_fail(e, "apply_y_group_kernel launch");
    return after_launch("apply_y_group_kernel");
}

lrc_status encode_map_2d(CUtensorMap* map, CUtensorMapDataType dt, const void* base, int64_t cols, int64_t rows,
                         int64_t pitch_bytes, uint32_t box_cols, uint32_t box_rows, bool swizzle128,
                         const char* what) {
    lrc_status st = get_encoder();
    if (st != LRC_OK) return st;
    return make_map(map, dt, base, cols, rows, pitch_bytes, box_cols, box_rows, what,
                    swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE);
}

lrc_status y_product_plan(int64_t m, int64_t b, int kp, bool out16, int* n2) {
    YArgs a{};
    size_t smem = 0;
    lrc_status st = plan_y(a, smem, m, b, kp, 1, out16, false);
    if (st == LRC_OK) *n2 = a.n2;
    return st;
}

lrc_status launch_y_product(const unsigned char* Wimg, int kp, const void* U, int64_t ldu, int64_t m, int64_t b,
                            bool out16, void* Y, const int* esc_w, const int* esc_u, cudaStream_t s,
                            bool w_per_row, bool bf16) {
    lrc_status st = get_encoder();
    if (st != LRC_OK) return st;
    YArgs a3{};
    size_t smem3 = 0;
    if ((st = plan_y(a3, smem3, m, b, kp, 1, out16, false)) != LRC_OK) return st;
    a3.tile_bytes = (uint32_t)BM * (uint32_t)kp * 2u;
    a3.W = Wimg;
    a3.Y = Y;
    a3.esc_w = esc_w;
    a3.esc_w_rows = w_per_row ? 1 : 0;
    a3.esc_u = esc_u;
    a3.bf16 = bf16 ? 1 : 0;
    a3.idesc_ab = bf16 ? kIdescBF16 : 0u;
    CUtensorMap tu, ty;
    if ((st = make_map(&tu, t16(bf16), U, kp, m, ldu * 2, BK, (uint32_t)a3.n2, "U")) != LRC_OK) return st;
    if ((st = make_y_map(&ty, a3, Y, m, b, out16)) != LRC_OK) return st;
    const int sms = sm_count();
    const int64_t P3 = a3.T < sms ? a3.T : sms;
    return launch_y(tu, ty, a3, smem3, P3, s);
}

namespace {
__global__ void wait_timeout_probe_kernel(uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        tc::mbar_init(&bar, 1);        // nothing ever arrives on it
        abort_flag = 0;
        tc::fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) tc::mbar_wait(&bar, 0, &abort_flag, &g_err_apply_tc, 8u, limit_ns);
}
}  // namespace

lrc_status launch_wait_timeout_probe(int64_t limit_ns, cudaStream_t s) {
    wait_timeout_probe_kernel<<<1, 32, 0, s>>>((uint64_t)limit_ns);
    return after_launch("wait_timeout_probe_kernel");
}

uint32_t take_apply_tc_error() {
    unsigned int v = 0;
    if (cudaMemcpyFromSymbol(&v, g_err_apply_tc, sizeof v) != cudaSuccess) return 0xffffffffu;
    if (v) {
        const unsigned int z = 0;
        cudaMemcpyToSymbol(g_err_apply_tc, &z, sizeof z);
    }
    return v;
}

}  // namespace lrc
