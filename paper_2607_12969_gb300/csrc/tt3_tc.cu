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
// TMEM holds two D2 accumulators (slice columns each) and one or two D1
// buffers after them; the converters release D1 as soon as it is in their
// registers, so stage 1 of the next unit overlaps this unit's conversion and
// stage 2.  Warp roles:
//   0..3 epilogue, and 11..14 too when the plan takes two epilogue warps per
//   tensor-memory lane quarter (alternate 128-byte column chunks; otherwise
//   they idle), 4..7 converters, 8 stage-2 MMA issuer
//   (one thread; it also
//   owns the tensor memory), 9 loader (one thread), 10 stage-1 MMA issuer (one
//   thread).  The two stages' MMAs are issued from two threads: their chains
//   are independent (stage 1 waits for a free D1 and its operands, stage 2
//   for A2 and a free accumulator), and a single issuer spent more time on
//   instruction issue and commits than the epilogue takes to drain a unit.  A small image kernel first writes every operand the tensor
//   cores read from the cores -- the G_1 rows of each i_1 tile, G_2(i_2)^T
//   for every i_2, G_3^T -- in its shared-memory layout; the loader moves
//   them with bulk copies (the main kernel is launched dependent on the
//   image kernel and overlaps its set-up with it).
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
constexpr int kThreads = 480;
constexpr int kEpiWarpsMax = 8;    // warps 0..3 and 11..14

struct T3Args {
    int64_t n1, n2;
    int nd, r1, r2, r1p, r2p;      // n_3, ranks, ranks rounded up to 16
    int n2h, sn;                   // n_3 slice per unit, number of slices
    int64_t units;                 // (i_1 tile, i_2, n_3 slice) units
    int cw, out16;
    int nep;                       // epilogue warps per lane quarter (1 or 2)
    int nd1;                       // D1 buffers (TMEM columns 2 n2h .. 2 n2h + nd1 r2p)
    uint32_t tmem_cols;
    uint32_t off_a1, off_b1, off_a2, off_b2, off_stage, off_bar;
    uint32_t a1_bytes, b1_bytes, a2_bytes, b2_bytes;
    const __half* G1;
    const __half* G2;
    const __half* G3;
    // operand images written by the image kernel (canonical K-major layouts)
    const unsigned char* a1img;    // [i_1 tile][128 x r1p]   rows of G_1
    const unsigned char* b1img;    // [i_2][r2p x r1p]        G_2(i_2)^T
    const unsigned char* b2img;    // [n_3 x r2p]             G_3^T
};

struct Bars {
    uint64_t *a1_full, *a1_empty;
    uint64_t *b1_full, *b1_empty;      // [2]
    uint64_t *d1_full, *d1_empty;      // [2]
    uint64_t *a2_full, *mma_done1;     // [2], [1]: stage-1 issuer's MMAs complete
    uint64_t *d2_full, *acc_empty;     // [2]
    uint64_t *mma_done;
    uint64_t *b2_full;
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
    B.mma_done1 = p + 11;
    B.d2_full = p + 13;
    B.acc_empty = p + 15;
    B.mma_done = p + 17;
    B.b2_full = p + 18;
    B.d1_empty = p + 19;
    B.tmem_slot = reinterpret_cast<uint32_t*>(p + 21);
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

// Coordinates of consecutive units without divisions (the single-thread
// roles walk their units in order; a 64-bit division costs them hundreds of
// cycles a unit).
struct UnitWalk {
    int64_t qt, i;
    int h;
    __device__ __forceinline__ void start(const T3Args& a, int64_t u) { unit_coords(a, u, qt, i, h); }
    // does the unit after this one start another i_1 tile?
    __device__ __forceinline__ bool last_of_tile(const T3Args& a) const { return h + 1 == a.sn && i + 1 == a.n2; }
    __device__ __forceinline__ void next(const T3Args& a) {
        if (++h == a.sn) {
            h = 0;
            if (++i == a.n2) {
                i = 0;
                ++qt;
            }
        }
    }
};

// Operand images: the rows of G_1 of every 128-row i_1 tile, G_2(i_2)^T for
// every i_2 (row b, column a = G_2[a, i_2, b]) and G_3^T (row c, column
// b = G_3[b, c]), each in the canonical K-major layout with zero padding, so
// the main kernel moves each with one bulk copy.  A thread writes one
// 16-byte chunk (one row, eight consecutive ranks); neighbouring threads take
// neighbouring rows, so the reads of the cores stay coalesced.
__global__ void __launch_bounds__(256)
tt3_img_kernel(const __grid_constant__ T3Args a, unsigned char* a1img, unsigned char* b1img, unsigned char* b2img) {
    const int64_t qtiles = (a.n1 + BM - 1) / BM;
    const int g1 = a.r1p / 8, g2 = a.r2p / 8;
    const int64_t na1 = qtiles * g1 * BM;                 // (tile, k-group, row)
    const int64_t nb1 = a.n2 * g1 * a.r2p;                // (i_2, k-group, row b)
    const int64_t nb2 = (int64_t)g2 * a.nd;               // (k-group, row c)
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < na1 + nb1 + nb2;
         e += (int64_t)gridDim.x * blockDim.x) {
        __half v[8];
        unsigned char* dst;
        if (e < na1) {
            const int row = (int)(e % BM);
            const int64_t t2 = e / BM;
            const int kg = (int)(t2 % g1);
            const int64_t t = t2 / g1;
            const int64_t q = t * BM + row;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int k = kg * 8 + u;
                v[u] = (q < a.n1 && k < a.r1) ? a.G1[q * a.r1 + k] : __float2half_rn(0.0f);
            }
            dst = a1img + t * a.a1_bytes + canon_off((uint32_t)row, (uint32_t)(kg * 8), BM);
        } else if (e < na1 + nb1) {
            const int64_t e1 = e - na1;
            const int bb = (int)(e1 % a.r2p);
            const int64_t t2 = e1 / a.r2p;
            const int kg = (int)(t2 % g1);
            const int64_t i = t2 / g1;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int k = kg * 8 + u;
                v[u] = (bb < a.r2 && k < a.r1) ? a.G2[((int64_t)k * a.n2 + i) * a.r2 + bb] : __float2half_rn(0.0f);
            }
            dst = b1img + i * a.b1_bytes + canon_off((uint32_t)bb, (uint32_t)(kg * 8), (uint32_t)a.r2p);
        } else {
            const int64_t e2 = e - na1 - nb1;
            const int c = (int)(e2 % a.nd);
            const int kg = (int)(e2 / a.nd);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int k = kg * 8 + u;
                v[u] = k < a.r2 ? a.G3[(int64_t)k * a.nd + c] : __float2half_rn(0.0f);
            }
            dst = b2img + canon_off((uint32_t)c, (uint32_t)(kg * 8), (uint32_t)a.nd);
        }
        uint4 w;
        w.x = (uint32_t)__half_as_ushort(v[0]) | ((uint32_t)__half_as_ushort(v[1]) << 16);
        w.y = (uint32_t)__half_as_ushort(v[2]) | ((uint32_t)__half_as_ushort(v[3]) << 16);
        w.z = (uint32_t)__half_as_ushort(v[4]) | ((uint32_t)__half_as_ushort(v[5]) << 16);
        w.w = (uint32_t)__half_as_ushort(v[6]) | ((uint32_t)__half_as_ushort(v[7]) << 16);
        *reinterpret_cast<uint4*>(dst) = w;
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
            mbar_init(&B.d2_full[q], 1);
            mbar_init(&B.acc_empty[q], 128 * a.nep);
        }
        mbar_init(B.mma_done, 1);
        mbar_init(B.mma_done1, 1);
        mbar_init(B.b2_full, 1);
        for (int q = 0; q < 2; ++q) mbar_init(&B.d1_empty[q], 128);
        *B.abort = 0;
        fence_barrier_init();
    }
    if (warp == 8) tmem_alloc(B.tmem_slot, a.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *B.tmem_slot;

    if (warp == 9) {
        // ------------------------------------------------------------ loader
        // one thread: bulk copies of the operand images (G_3^T once, the G_1
        // tile per i_1 tile, G_2(i_2)^T per unit through two slots)
        if (lane == 0) {
            pdl_wait();                // the image kernel's writes are complete and visible
            mbar_arrive_expect_tx(B.b2_full, a.b2_bytes);
            bulk_load(smem + a.off_b2, a.b2img, a.b2_bytes, B.b2_full);
            int64_t prev_qt = -1;
            int builds = 0;
            int64_t j = 0;
            UnitWalk w;
            w.start(a, ubeg);
            for (; j < nunits; ++j, w.next(a)) {
                const int64_t qt = w.qt, i = w.i;
                if (qt != prev_qt) {
                    if (builds > 0 && !mbar_wait(B.a1_empty, (uint32_t)((builds - 1) & 1), abort, err, 1u)) break;
                    mbar_arrive_expect_tx(B.a1_full, a.a1_bytes);
                    bulk_load(smem + a.off_a1, a.a1img + (size_t)qt * a.a1_bytes, a.a1_bytes, B.a1_full);
                    prev_qt = qt;
                    ++builds;
                }
                const int slot = (int)(j & 1);
                // slot free once stage 1 of unit j - 2 has read it: with two D1
                // buffers that is D1's own completion (one commit less a unit)
                uint64_t* freed = a.nd1 == 2 ? &B.d1_full[slot] : &B.b1_empty[slot];
                if (!mbar_wait(freed, (uint32_t)((j >> 1) & 1) ^ 1u, abort, err, 1u)) break;
                mbar_arrive_expect_tx(&B.b1_full[slot], a.b1_bytes);
                bulk_load(smem + a.off_b1 + (size_t)slot * a.b1_bytes, a.b1img + (size_t)i * a.b1_bytes, a.b1_bytes,
                          &B.b1_full[slot]);
            }
            // copies in flight land before the CTA can exit
            volatile int no_abort = 0;
            mbar_wait(B.b2_full, 0, &no_abort, err, 0u, 100000000ull);
            if (builds > 0) mbar_wait(B.a1_full, (uint32_t)((builds - 1) & 1), &no_abort, err, 0u, 100000000ull);
            for (int64_t q = (j - 2 > 0 ? j - 2 : 0); q < j && q < nunits; ++q)
                mbar_wait(&B.b1_full[q & 1], (uint32_t)((q >> 1) & 1), &no_abort, err, 0u, 100000000ull);
        }
    } else if (warp == 8 || warp == 10) {
        // ------------------------------------------------------------ MMA issuers
        // warp 10: stage 1 of every unit; warp 8: stage 2 of every unit
        if (lane == 0) {
            bool ok = true;
            const uint32_t idesc1 = idesc_f16_f32(BM, (uint32_t)a.r2p);
            const uint32_t idesc2 = idesc_f16_f32(BM, (uint32_t)a.n2h);
            const uint32_t a1s = smem_u32(smem + a.off_a1);
            const uint32_t b2s = smem_u32(smem + a.off_b2);
            int64_t cur_qt = -1;
            int qcount = 0;
            UnitWalk w1, w2;          // units of the next stage 1 and stage 2 (both in order)
            w1.start(a, ubeg);
            w2.start(a, ubeg);
            auto stage1 = [&](int64_t j) -> bool {
                const int64_t qt = w1.qt;
                const bool last = (j + 1 == nunits) || w1.last_of_tile(a);
                w1.next(a);
                const int buf = (int)(j & 1);
                if (qt != cur_qt) {
                    if (!mbar_wait(B.a1_full, (uint32_t)(qcount & 1), abort, err, 2u)) return false;
                    cur_qt = qt;
                    ++qcount;
                }
                // D1 has its own columns: it waits only for the converters of unit j - nd1
                const int db = a.nd1 == 2 ? (int)(j & 1) : 0;
                const int64_t dphase = a.nd1 == 2 ? (j >> 1) : j;
                if (j >= a.nd1 && !mbar_wait(&B.d1_empty[db], (uint32_t)((dphase - 1) & 1), abort, err, 2u))
                    return false;
                if (!mbar_wait(&B.b1_full[buf], (uint32_t)((j >> 1) & 1), abort, err, 2u)) return false;
                tc_fence_after();
                const uint32_t b1s = smem_u32(smem + a.off_b1 + (size_t)buf * a.b1_bytes);
                const uint32_t lbo1 = (uint32_t)a.r2p * 16u;
                // descriptors stepped by adds: 16 ranks = 4096 B of A, 2 x lbo1 B of B
                const uint64_t ad = smem_desc(a1s, 2048, 128, 0), bd = smem_desc(b1s, lbo1, 128, 0);
                const uint64_t bstep = (uint64_t)(2u * lbo1) >> 4;
                const uint32_t d1col = tmem + 2u * (uint32_t)a.n2h + (uint32_t)(db * a.r2p);
                for (int ks = 0; ks < a.r1p / 16; ++ks)
                    mma_f16(d1col, ad + (uint64_t)ks * 256u, bd + (uint64_t)ks * bstep, idesc1, ks > 0);
                if (a.nd1 == 1) mma_commit(&B.b1_empty[buf]);
                mma_commit(&B.d1_full[db]);
                // last unit of this i_1 tile: G_1 tile may be replaced once these MMAs finish
                if (last) mma_commit(B.a1_empty);
                return true;
            };
            auto stage2 = [&](int64_t j) -> bool {
                const int h = w2.h;
                w2.next(a);
                const int buf = (int)(j & 1);
                if (!mbar_wait(&B.a2_full[buf], (uint32_t)((j >> 1) & 1), abort, err, 2u)) return false;
                if (!mbar_wait(&B.acc_empty[buf], (uint32_t)((j >> 1) & 1) ^ 1u, abort, err, 2u)) return false;
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
                mma_commit(&B.d2_full[buf]);          // also frees the A2 slot for unit j + 2
                return true;
            };
            uint64_t* done = B.mma_done;
            if (warp == 10) {
                // stage 1 runs up to nd1 units ahead of the converters
                for (int64_t j = 0; j < nunits && ok; ++j) ok = stage1(j);
                done = B.mma_done1;
            } else {
                ok = mbar_wait(B.b2_full, 0, abort, err, 2u);
                for (int64_t j = 0; j < nunits && ok; ++j) ok = stage2(j);
            }
            // this thread's MMAs complete before the tensor memory is released
            mma_commit(done);
            volatile int no_abort = 0;
            mbar_wait(done, 0, &no_abort, err, 2u, 100000000ull);
        }
    } else if (warp >= 4 && warp < 8) {
        // ------------------------------------------------------------ converters (warps 4..7)
        const int g = warp & 3;
        const int r = g * 32 + lane;
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        for (int64_t j = 0; j < nunits; ++j) {
            const int buf = (int)(j & 1);
            const int db = a.nd1 == 2 ? (int)(j & 1) : 0;
            const int64_t dphase = a.nd1 == 2 ? (j >> 1) : j;
            if (!group_wait(&B.d1_full[db], (uint32_t)(dphase & 1), abort, err, 4u, 2, 128)) break;
            tc_fence_after();
            uint32_t v[64];
            const uint32_t tcol = tmem + lane_base + 2u * (uint32_t)a.n2h + (uint32_t)(db * a.r2p);
            tmem_ld32(tcol, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
            if (a.r2p > 32) tmem_ld32(tcol + 32, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
            tmem_ld_wait();
            tc_fence_before();
            mbar_arrive(&B.d1_empty[db]);          // D1 is in registers: the next stage 1 may overwrite it
            // A2 slot free once stage 2 of unit j - 2 has completed
            if (!group_wait(&B.d2_full[buf], (uint32_t)((j >> 1) & 1) ^ 1u, abort, err, 4u, 2, 128)) break;
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
    } else if (warp < 4 || a.nep == 2) {
        // ------------------------------------------------------------ epilogue
        // each warp drains its own 32 rows (its lane quarter) on every other
        // column chunk through its own staging pair and issues its own 32-row
        // TMA stores: no barrier across the eight warps
        const int g = warp & 3;
        const int hh = warp >= 11 ? 1 : 0;
        const int r = g * 32 + lane;
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        unsigned char* wstage = smem + a.off_stage + (size_t)(hh * 4 + g) * (2 * 32 * 128);
        int chunk = 0;
        UnitWalk w;
        w.start(a, ubeg);
        for (int64_t j = 0; j < nunits; ++j, w.next(a)) {
            const int64_t qt = w.qt, i = w.i;
            const int h = w.h;
            const int buf = (int)(j & 1);
            if (!group_wait(&B.d2_full[buf], (uint32_t)((j >> 1) & 1), abort, err, 8u, 1, 128 * a.nep)) break;
            tc_fence_after();
            for (int cc = hh * a.cw; cc < a.n2h; cc += a.nep * a.cw, ++chunk) {
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
    // TMEM: two D2 accumulators of n2h columns, then nd1 D1 buffers of r2p
    // columns (two when they fit, so stage 1 runs a unit ahead)
    a.nd1 = (2 * a.n2h + 2 * a.r2p <= 512) ? 2 : 1;
    const uint32_t need = 2u * (uint32_t)a.n2h + (uint32_t)(a.nd1 * a.r2p);
    const uint32_t d1_read_end = 2u * (uint32_t)a.n2h + (uint32_t)((a.nd1 - 1) * a.r2p) + (a.r2p > 32 ? 64u : 32u);
    a.tmem_cols = pow2_cols(need > d1_read_end ? need : d1_read_end);
    const uint32_t chunks = (uint32_t)((a.n2h + a.cw - 1) / a.cw * a.cw);
    if ((uint32_t)a.n2h + chunks > 2u * (uint32_t)a.n2h + (uint32_t)a.r2p || a.tmem_cols > 512) return false;
    a.a1_bytes = (uint32_t)BM * a.r1p * 2;
    a.b1_bytes = (uint32_t)a.r2p * a.r1p * 2;
    a.a2_bytes = (uint32_t)BM * a.r2p * 2;
    a.b2_bytes = (uint32_t)a.nd * a.r2p * 2;
    uint32_t off = 0;
    a.off_a1 = off;
    off += a.a1_bytes;
    a.off_b1 = off;
    off += 2 * a.b1_bytes;
    a.off_a2 = off;
    off += 4 * a.a2_bytes;
    a.off_b2 = off;
    off += a.b2_bytes;
    off = (off + 1023) / 1024 * 1024;
    // two epilogue warps per lane quarter when a unit has a chunk for each:
    // measured faster for binary16 output (the conversion bounds that
    // epilogue: 512^2 x 224 37.4 -> 32.1 us) and for binary32 units of at
    // most 128 columns (256^3: 20.7 -> 19.5 us); binary32 units of 224
    // columns, already at the store rate, measured slower (49.5 -> 52.0 us)
    a.nep = (a.n2h >= 2 * a.cw && (out16 || a.n2h <= 128)) ? 2 : 1;
    a.off_stage = off;
    off += (uint32_t)(4 * a.nep) * 2 * 32 * 128;
    off = (off + 7) / 8 * 8;
    a.off_bar = off;
    off += 21 * 8 + 16;
    const size_t smem = (size_t)off + 1024;
    if (smem > 227 * 1024) return false;
    a.G1 = static_cast<const __half*>(sh.cores[0]);
    a.G2 = static_cast<const __half*>(sh.cores[1]);
    a.G3 = static_cast<const __half*>(sh.cores[2]);
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
    // operand images in the stream workspace
    const int64_t qtiles = (a.n1 + BM - 1) / BM;
    auto r256 = [](size_t v) { return (v + 255) / 256 * 256; };
    const size_t a1_total = r256((size_t)qtiles * a.a1_bytes), b1_total = r256((size_t)a.n2 * a.b1_bytes);
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, a1_total + b1_total + a.b2_bytes, &ws);
    if (st != LRC_OK) return st;
    unsigned char* wb = static_cast<unsigned char*>(ws);
    a.a1img = wb;
    a.b1img = wb + a1_total;
    a.b2img = wb + a1_total + b1_total;
    const int64_t nel = (qtiles * BM * a.r1p + a.n2 * a.r2p * a.r1p + (int64_t)a.nd * a.r2p) / 8;   // 16-byte chunks
    const int64_t iblocks = (nel + 255) / 256;
    const int sms = sm_count();
    tt3_img_kernel<<<(unsigned)(iblocks < 8 * sms ? iblocks : 8 * sms), 256, 0, s>>>(a, wb, wb + a1_total,
                                                                                     wb + a1_total + b1_total);
    if ((st = after_launch("tt3_img_kernel")) != LRC_OK) return st;
    cudaError_t e = cudaFuncSetAttribute(tt3_f16_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "tt3_f16_tc_kernel smem attribute");
    e = launch_pdl(tt3_f16_tc_kernel, dim3((unsigned)grid), dim3(kThreads), smem, s, tm, a);
    if (e != cudaSuccess) return cuda_fail(e, "tt3_f16_tc_kernel launch");
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
