// apply_tc.cu -- fused low-rank apply on the 5th-generation tensor cores,
// binary16 storage with binary32 accumulation (Sec. 4.4, Eq. gpu_matrix_apply:
// Y = [(X V) diag(s)] U^T; Sec. 3.4: FP16 products accumulate in FP32).
//
// One CTA owns BM = 128 query rows (the MMA M) and a contiguous range of
// N2-wide tiles of Y's columns.  Warp roles:
//   warp 0      TMA producer: streams X / V^T boxes (phase 1) and U boxes
//               (phase 2) through a ring of shared-memory slots;
//   warp 1      tensor-memory owner and MMA issuer (one thread);
//   warps 2..5  epilogue (one TMEM lane = one query row per thread).
// Phase 1 accumulates W = X V (128 x k', FP32) in tensor memory.  For FP32
// output the reduction over n is split into chunks of kChunkBlocks x 64
// elements accumulated in two ping-pong tensor-memory buffers; the epilogue
// adds each chunk's partial sums with IEEE binary32 additions into a running
// sum.  (The tensor core's own accumulation error grows with the number of
// accumulation steps; chunking bounds it by the chunk length.)  The running
// sum lives in the shared-memory region that later holds W's hi/lo halves,
// laid out so that every thread only ever touches the bytes of its own row.
// The epilogue scales W by diag(s) in FP32 and writes it to shared memory
// as binary16 -- for the FP32-output variant as a hi/lo pair
// (hi = fp16(w), lo = fp16(w - hi)) so that the second product keeps about
// 22 significand bits; the FP16-output variant rounds W once to binary16,
// the method-precision workspace of Sec. 3.4.  W never reaches global memory.
// Phase 2 computes Y tiles = W U^T with two tensor-memory accumulators in
// flight, so the epilogue drains one tile (TMEM -> registers -> swizzled
// shared memory -> TMA store) while the next is being multiplied; each
// epilogue warp stages and stores its own 32 rows, without barriers across
// the four warps.
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
constexpr uint32_t kXBytes = BM * BK * 2;    // one X box
constexpr int kChunkBlocks = 8;              // 64-wide k-blocks per accumulation chunk (FP32 output)

struct Args {
    int64_t m, b;
    int k, kp;                 // rank and rank rounded up to 16
    int n2;                    // phase-2 tile width (MMA N)
    int nkb;                   // phase-1 k-blocks, ceil(n / 64)
    int kc2;                   // phase-2 k-chunks, ceil(kp / 64)
    int mtiles;                // ceil(m / n2)
    int mt_per_cta;
    int chunk_blocks;          // k-blocks per phase-1 accumulation chunk
    int nchunk;                // ceil(nkb / chunk_blocks)
    int acc1_bufs;             // 2 = ping-pong, 1 = single phase-1 accumulator
    int stages;
    uint32_t slot_bytes;
    uint32_t v_bytes;          // kp rows x 128 bytes
    uint32_t u_bytes;          // n2 rows x 128 bytes
    int v_boxes, v_box_rows;
    uint32_t tmem_cols;
    uint32_t w_off, wlo_off, ystage_off, s_off, bar_off;   // shared-memory carve-up
    int out16;
    int tma_store;
    const __half* S;
    void* Y;
};

struct Bars {
    uint64_t* full;
    uint64_t* empty;
    uint64_t* acc1_full;    // [2]
    uint64_t* acc1_empty;   // [2]
    uint64_t* w_ready;
    uint64_t* acc2_full;    // [2]
    uint64_t* acc2_empty;   // [2]
    uint64_t* mma_done;
    uint32_t* tmem_slot;
    int* abort;
};

__device__ __forceinline__ Bars carve_bars(unsigned char* smem, const Args& a) {
    Bars B;
    uint64_t* p = reinterpret_cast<uint64_t*>(smem + a.bar_off);
    B.full = p;
    B.empty = p + a.stages;
    B.acc1_full = p + 2 * a.stages;
    B.acc1_empty = B.acc1_full + 2;
    B.w_ready = B.acc1_empty + 2;
    B.acc2_full = B.w_ready + 1;
    B.acc2_empty = B.acc2_full + 2;
    B.mma_done = B.acc2_empty + 2;
    B.tmem_slot = reinterpret_cast<uint32_t*>(B.mma_done + 1);
    B.abort = reinterpret_cast<int*>(B.tmem_slot + 1);
    return B;
}

__global__ void __launch_bounds__(kThreads, 1)
apply_f16_tc_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_v,
                    const __grid_constant__ CUtensorMap tm_u, const __grid_constant__ CUtensorMap tm_y,
                    const Args a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                           ~static_cast<uintptr_t>(1023));
    const Bars B = carve_bars(smem, a);
    float* s_f = reinterpret_cast<float*>(smem + a.s_off);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t row0 = (int64_t)blockIdx.x * BM;
    const int mt_begin = blockIdx.y * a.mt_per_cta;
    const int mt_end = min(mt_begin + a.mt_per_cta, a.mtiles);
    volatile int* abort = B.abort;
    unsigned int* err = &g_err_apply_tc;

    if (threadIdx.x == 0) {
        for (int i = 0; i < a.stages; ++i) {
            mbar_init(&B.full[i], 1);
            mbar_init(&B.empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&B.acc1_full[i], 1);
            mbar_init(&B.acc1_empty[i], 128);
        }
        mbar_init(B.w_ready, 128);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&B.acc2_full[i], 1);
            mbar_init(&B.acc2_empty[i], 128);
        }
        mbar_init(B.mma_done, 1);
        *B.abort = 0;
        fence_barrier_init();
        tma_prefetch_desc(&tm_x);
        tma_prefetch_desc(&tm_v);
        tma_prefetch_desc(&tm_u);
        tma_prefetch_desc(&tm_y);
    }
    for (int j = threadIdx.x; j < a.kp; j += kThreads) s_f[j] = j < a.k ? __half2float(a.S[j]) : 0.0f;
    if (warp == 1) tmem_alloc(B.tmem_slot, a.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *B.tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int it = 0;
            bool ok = true;
            for (int kb = 0; kb < a.nkb && ok; ++kb, ++it) {
                const int slot = it % a.stages;
                if (!(ok = mbar_wait(&B.empty[slot], ((it / a.stages) & 1) ^ 1, abort, err, 1u))) break;
                unsigned char* sp = smem + (size_t)slot * a.slot_bytes;
                mbar_arrive_expect_tx(&B.full[slot], kXBytes + a.v_bytes);
                tma_load_2d(sp, &tm_x, kb * BK, (int32_t)row0, &B.full[slot]);
                for (int vb = 0; vb < a.v_boxes; ++vb)
                    tma_load_2d(sp + kXBytes + (size_t)vb * a.v_box_rows * 128, &tm_v, kb * BK, vb * a.v_box_rows,
                                &B.full[slot]);
            }
            for (int mt = mt_begin; mt < mt_end && ok; ++mt) {
                for (int kc = 0; kc < a.kc2 && ok; ++kc, ++it) {
                    const int slot = it % a.stages;
                    if (!(ok = mbar_wait(&B.empty[slot], ((it / a.stages) & 1) ^ 1, abort, err, 1u))) break;
                    mbar_arrive_expect_tx(&B.full[slot], a.u_bytes);
                    tma_load_2d(smem + (size_t)slot * a.slot_bytes, &tm_u, kc * BK, mt * a.n2, &B.full[slot]);
                }
            }
            if (!ok) {
                // let copies already in flight land before the CTA can exit
                const int first = it - a.stages > 0 ? it - a.stages : 0;
                for (int j = first; j < it; ++j) {
                    volatile int no_abort = 0;
                    mbar_wait(&B.full[j % a.stages], (j / a.stages) & 1, &no_abort, err, 0u, 100000000ull);
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            int it = 0;
            bool ok = true;
            const int nchunks = a.kp > 256 ? 2 : 1;
            for (int kb = 0; kb < a.nkb && ok; ++kb, ++it) {
                const int c = kb / a.chunk_blocks;                 // accumulation chunk
                const int kin = kb - c * a.chunk_blocks;           // k-block within the chunk
                const int buf = c % a.acc1_bufs;
                if (kin == 0) {
                    if (!(ok = mbar_wait(&B.acc1_empty[buf], ((c / a.acc1_bufs) & 1) ^ 1, abort, err, 2u))) break;
                    tc_fence_after();
                }
                const int slot = it % a.stages;
                if (!(ok = mbar_wait(&B.full[slot], (it / a.stages) & 1, abort, err, 2u))) break;
                tc_fence_after();
                const uint32_t xa = smem_u32(smem + (size_t)slot * a.slot_bytes);
                const uint32_t va = xa + kXBytes;
                const uint32_t dacc = tmem + buf * a.kp;
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk) {
                    const uint64_t adesc = desc_sw128(xa + kk * 32);
                    for (int q = 0; q < nchunks; ++q) {
                        const int r0 = q * 256;
                        const int nn = (q == 0) ? (a.kp > 256 ? 256 : a.kp) : a.kp - 256;
                        mma_f16(dacc + r0, adesc, desc_sw128(va + r0 * 128 + kk * 32), idesc_f16_f32(BM, nn),
                                (kin | kk) != 0);
                    }
                }
                mma_commit(&B.empty[slot]);
                if (kin == a.chunk_blocks - 1 || kb == a.nkb - 1) mma_commit(&B.acc1_full[buf]);
            }
            if (ok) ok = mbar_wait(B.w_ready, 0, abort, err, 2u);
            tc_fence_after();
            const uint32_t whi = smem_u32(smem + a.w_off);
            const uint32_t wlo = smem_u32(smem + a.wlo_off);
            const uint32_t idesc2 = idesc_f16_f32(BM, a.n2);
            for (int mt = mt_begin, t = 0; mt < mt_end && ok; ++mt, ++t) {
                const int ab = t & 1;
                if (!(ok = mbar_wait(&B.acc2_empty[ab], ((t >> 1) & 1) ^ 1, abort, err, 2u))) break;
                tc_fence_after();
                const uint32_t dcol = tmem + ab * a.n2;
                for (int kc = 0; kc < a.kc2 && ok; ++kc, ++it) {
                    const int slot = it % a.stages;
                    if (!(ok = mbar_wait(&B.full[slot], (it / a.stages) & 1, abort, err, 2u))) break;
                    tc_fence_after();
                    const uint32_t ua = smem_u32(smem + (size_t)slot * a.slot_bytes);
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const int ks = kc * (BK / 16) + kk;
                        if (ks * 16 >= a.kp) break;
                        const uint64_t bdesc = desc_sw128(ua + kk * 32);
                        // W in the canonical layout: K-direction core matrices 2048 B apart,
                        // M-direction core matrices 128 B apart
                        mma_f16(dcol, smem_desc(whi + ks * 4096, 2048, 128, 0), bdesc, idesc2, (kc | kk) != 0);
                        if (!a.out16)
                            mma_f16(dcol, smem_desc(wlo + ks * 4096, 2048, 128, 0), bdesc, idesc2, 1u);
                    }
                    mma_commit(&B.empty[slot]);
                }
                if (ok) mma_commit(&B.acc2_full[ab]);
            }
            // every MMA issued by this thread has finished before TMEM is released
            mma_commit(B.mma_done);
            volatile int no_abort = 0;
            mbar_wait(B.mma_done, 0, &no_abort, err, 2u, 100000000ull);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int g = warp & 3;                 // TMEM lane quarter of this warp
        const int r = g * 32 + lane;            // tile row of this thread
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        bool ok = true;
        unsigned char* whi = smem + a.w_off;
        unsigned char* wlo = smem + a.wlo_off;
        for (int c = 0; c < a.nchunk && ok; ++c) {
            const int buf = c % a.acc1_bufs;
            if (!(ok = group_wait(&B.acc1_full[buf], (c / a.acc1_bufs) & 1, abort, err, 4u, 1, 128))) break;
            tc_fence_after();
            const bool first = (c == 0), last = (c == a.nchunk - 1);
            for (int c0 = 0; c0 < a.kp; c0 += 32) {
                uint32_t v[32];
                tmem_ld32(tmem + lane_base + buf * a.kp + c0, v);
                tmem_ld_wait();
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int col = c0 + q * 8;
                    if (col >= a.kp) continue;
                    // bytes of row r, columns col..col+7, in the core-matrix layout of W
                    const uint32_t off = (uint32_t)(col >> 3) * 2048u + (uint32_t)(r >> 3) * 128u +
                                         (uint32_t)(r & 7) * 16u;
                    float w[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) w[j] = __uint_as_float(v[q * 8 + j]);
                    if (!first) {   // running sum: w[0..3] at the hi position, w[4..7] at the lo position
                        const float4 r0 = *reinterpret_cast<const float4*>(whi + off);
                        const float4 r1 = *reinterpret_cast<const float4*>(wlo + off);
                        w[0] = __fadd_rn(r0.x, w[0]);
                        w[1] = __fadd_rn(r0.y, w[1]);
                        w[2] = __fadd_rn(r0.z, w[2]);
                        w[3] = __fadd_rn(r0.w, w[3]);
                        w[4] = __fadd_rn(r1.x, w[4]);
                        w[5] = __fadd_rn(r1.y, w[5]);
                        w[6] = __fadd_rn(r1.z, w[6]);
                        w[7] = __fadd_rn(r1.w, w[7]);
                    }
                    if (!last) {
                        *reinterpret_cast<float4*>(whi + off) = make_float4(w[0], w[1], w[2], w[3]);
                        *reinterpret_cast<float4*>(wlo + off) = make_float4(w[4], w[5], w[6], w[7]);
                        continue;
                    }
                    uint32_t hi[4], lo[4];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float w0 = w[2 * j] * s_f[col + 2 * j];
                        const float w1 = w[2 * j + 1] * s_f[col + 2 * j + 1];
                        const __half h0 = __float2half_rn(w0), h1 = __float2half_rn(w1);
                        hi[j] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
                        lo[j] = pack_half2(w0 - __half2float(h0), w1 - __half2float(h1));
                    }
                    *reinterpret_cast<uint4*>(whi + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                    if (!a.out16) *reinterpret_cast<uint4*>(wlo + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
                }
            }
            tc_fence_before();
            mbar_arrive(&B.acc1_empty[buf]);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(B.w_ready);

        const int ecols = a.out16 ? 64 : 32;       // columns per 128-byte staging row
        int chunk = 0;
        for (int mt = mt_begin, t = 0; mt < mt_end && ok; ++mt, ++t) {
            const int ab = t & 1;
            if (!(ok = group_wait(&B.acc2_full[ab], (t >> 1) & 1, abort, err, 4u, 1, 128))) break;
            tc_fence_after();
            for (int cc = 0; cc < a.n2; cc += ecols, ++chunk) {
                uint32_t v[64];
                tmem_ld32(tmem + lane_base + ab * a.n2 + cc, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
                if (a.out16)
                    tmem_ld32(tmem + lane_base + ab * a.n2 + cc + 32, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
                tmem_ld_wait();
                uint32_t packed[32];
                if (a.out16) {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        packed[j] = pack_half2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j) packed[j] = v[j];
                }
                const int64_t col0 = (int64_t)mt * a.n2 + cc;
                if (a.tma_store) {
                    // this warp's 32 rows: own staging pair, own TMA store, no
                    // barrier across the four epilogue warps
                    unsigned char* sb = smem + a.ystage_off + (size_t)g * (2 * 32 * 128) + (chunk & 1) * (32 * 128);
                    if (chunk >= 2) {
                        if (lane == 0) bulk_wait_read<1>();
                        __syncwarp();
                    }
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const uint32_t off = (uint32_t)lane * 128u + (uint32_t)((j ^ (lane & 7)) * 16);
                        *reinterpret_cast<uint4*>(sb + off) =
                            make_uint4(packed[4 * j], packed[4 * j + 1], packed[4 * j + 2], packed[4 * j + 3]);
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0 && col0 < a.m) {
                        tma_store_2d(&tm_y, (int32_t)col0, (int32_t)(row0 + g * 32), sb);
                        bulk_commit();
                    }
                } else {
                    const int64_t grow = row0 + r;
                    if (grow < a.b) {
                        if (a.out16) {
                            __half* yrow = static_cast<__half*>(a.Y) + grow * a.m;
                            for (int j = 0; j < 64; ++j)
                                if (col0 + j < a.m) yrow[col0 + j] = __float2half_rn(__uint_as_float(v[j]));
                        } else {
                            float* yrow = static_cast<float*>(a.Y) + grow * a.m;
                            for (int j = 0; j < 32; ++j)
                                if (col0 + j < a.m) yrow[col0 + j] = __uint_as_float(v[j]);
                        }
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(&B.acc2_empty[ab]);
        }
        if (lane == 0 && a.tma_store) bulk_wait<0>();
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, a.tmem_cols);
    }
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

// 2-D map over a row-major [rows x cols] array with a row pitch of `pitch_bytes`.
lrc_status make_map(CUtensorMap* map, CUtensorMapDataType dt, int esize, const void* base, int64_t cols,
                    int64_t rows, int64_t pitch_bytes, uint32_t box_cols, uint32_t box_rows, const char* what) {
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)pitch_bytes};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    (void)esize;
    CUresult r = g_encode(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
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

}  // namespace

lrc_status launch_apply_f16(const void* U, const void* S, const void* Vt, const void* X, void* Y, int64_t m,
                            int64_t n, int64_t k, int64_t b, bool out16, cudaStream_t s) {
    lrc_status st = get_encoder();
    if (st != LRC_OK) return st;
    Args a{};
    a.m = m;
    a.b = b;
    a.k = (int)k;
    a.kp = (int)((k + 15) / 16 * 16);
    if (a.kp > 512) {
        set_error("binary16 apply supports rank up to 512 (got %lld)", (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    a.out16 = out16 ? 1 : 0;
    a.nkb = (int)((n + BK - 1) / BK);
    a.kc2 = (a.kp + BK - 1) / BK;
    a.v_boxes = a.kp > 256 ? 2 : 1;
    a.v_box_rows = a.kp / a.v_boxes;
    a.v_bytes = (uint32_t)a.kp * 128;
    const int e_out = out16 ? 2 : 4;
    a.tma_store = ((m * e_out) % 16 == 0) ? 1 : 0;
    a.S = static_cast<const __half*>(S);
    a.Y = Y;

    // shared memory plan: widest phase-2 tile and deepest ring that fit
    const uint32_t w_bytes = (uint32_t)BM * a.kp * 2;
    size_t smem = 0;
    bool chosen = false;
    for (int n2 : {256, 128}) {
        for (int stages = 4; stages >= 1 && !chosen; --stages) {
            if (n2 == 256 && stages < 2) break;      // prefer a 2-deep ring with narrower tiles
            const uint32_t u_bytes = (uint32_t)n2 * 128;
            uint32_t slot = kXBytes + a.v_bytes > u_bytes ? kXBytes + a.v_bytes : u_bytes;
            slot = (slot + 1023) / 1024 * 1024;
            uint32_t off = (uint32_t)stages * slot;
            const uint32_t w_off = off;
            off += w_bytes;
            const uint32_t wlo_off = out16 ? w_off : off;
            if (!out16) off += w_bytes;
            off = (off + 1023) / 1024 * 1024;
            const uint32_t ystage_off = off;
            off += 2 * 16384;
            const uint32_t s_off = off;
            off += (uint32_t)a.kp * 4;
            off = (off + 7) / 8 * 8;
            const uint32_t bar_off = off;
            off += (uint32_t)(2 * stages + 10) * 8 + 16;
            const size_t total = (size_t)off + 1024;    // base alignment slack
            if (total > 227 * 1024) continue;
            a.n2 = n2;
            a.u_bytes = u_bytes;
            a.slot_bytes = slot;
            a.stages = stages;
            a.w_off = w_off;
            a.wlo_off = wlo_off;
            a.ystage_off = ystage_off;
            a.s_off = s_off;
            a.bar_off = bar_off;
            smem = total;
            chosen = true;
        }
        if (chosen) break;
    }
    if (!chosen) {
        set_error("binary16 apply: rank %lld does not fit in shared memory", (long long)k);
        return LRC_ERR_UNSUPPORTED;
    }
    // chunked phase-1 accumulation for FP32 output; one chunk for FP16 output
    a.chunk_blocks = out16 ? a.nkb : kChunkBlocks;
    a.nchunk = (a.nkb + a.chunk_blocks - 1) / a.chunk_blocks;
    a.acc1_bufs = (a.nchunk > 1 && 2 * a.kp <= 512) ? 2 : 1;
    const uint32_t acc1_cols = (uint32_t)(a.acc1_bufs * a.kp);
    a.tmem_cols = pow2_cols(acc1_cols > (uint32_t)(2 * a.n2) ? acc1_cols : (uint32_t)(2 * a.n2));
    a.mtiles = (int)((m + a.n2 - 1) / a.n2);

    const int64_t btiles = (b + BM - 1) / BM;
    if (btiles > 0x7fffffff) {
        set_error("binary16 apply: batch too large");
        return LRC_ERR_UNSUPPORTED;
    }
    const int sms = sm_count();
    int64_t splits = btiles >= sms ? 1 : sms / btiles;
    if (splits < 1) splits = 1;
    if (splits > a.mtiles) splits = a.mtiles;
    a.mt_per_cta = (int)((a.mtiles + splits - 1) / splits);
    const int gy = (a.mtiles + a.mt_per_cta - 1) / a.mt_per_cta;
    if (gy > 65535) {
        set_error("binary16 apply: too many column tiles");
        return LRC_ERR_UNSUPPORTED;
    }

    const int64_t ldn = lrc_packed_ld(n), ldk = lrc_packed_ld(k);
    CUtensorMap tx, tv, tu, ty;
    if ((st = make_map(&tx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, X, n, b, ldn * 2, BK, BM, "X")) != LRC_OK) return st;
    if ((st = make_map(&tv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, Vt, n, k, ldn * 2, BK, (uint32_t)a.v_box_rows, "Vt")) !=
        LRC_OK)
        return st;
    if ((st = make_map(&tu, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, U, k, m, ldk * 2, BK, (uint32_t)a.n2, "U")) != LRC_OK)
        return st;
    if (a.tma_store) {
        if ((st = make_map(&ty, out16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, e_out, Y, m,
                           b, m * e_out, out16 ? 64 : 32, 32, "Y")) != LRC_OK)
            return st;
    } else {
        ty = tu;   // unused by the kernel
    }
    cudaError_t e = cudaFuncSetAttribute(apply_f16_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "apply_f16_tc_kernel smem attribute");
    dim3 grid((unsigned)btiles, (unsigned)gy);
    apply_f16_tc_kernel<<<grid, kThreads, smem, s>>>(tx, tv, tu, ty, a);
    return after_launch("apply_f16_tc_kernel");
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
