// tt_tc.cu -- dense TT reconstruction from binary16 cores on the tensor cores
// (Sec. 5.1: T(i_1..i_d) = G_1(i_1)...G_d(i_d); Sec. 7.5,
// Eq. gpu_tt_reconstruction: B_l = Z_{l-1} K_l, Z_l = reshape(B_l); Sec. 3.4:
// FP16 products accumulate in FP32).
//
// T is viewed as P prefix rows (i_1..i_{d-1}) x n_d columns.  A persistent
// CTA walks tiles of 128 consecutive prefix rows:
//   warps 4..7  builders: compute, in FP32, the few rows of Z_1..Z_{d-2} the
//               tile's prefixes pass through (shared memory), then each
//               builder thread forms one row of Z_{d-1} (= Z_{d-2}[parent]
//               G_{d-1}(i_{d-1})) and writes it as the binary16 A operand of
//               the final product -- a hi/lo pair for FP32 output, one
//               rounding for FP16 output (the method-precision workspace);
//               A is double-buffered so the next tile is built while the
//               current one is multiplied;
//   warp 8      tensor-memory owner and MMA issuer: out_tile (128 x n_d) =
//               Z_{d-1} G_d with G_d^T (n_d x r) kept in shared memory;
//   warps 0..3  epilogue: tensor memory -> registers -> shared staging ->
//               TMA store, with two accumulators in flight.
// The chain's intermediates never reach global memory.  The kernel covers
// n_d a multiple of 16 up to 256 whose output rows are at least 128 bytes,
// and a last rank up to 64; other shapes use the CUDA-core chain kernel.
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "tc.cuh"

namespace lrc {

__device__ unsigned int g_err_tt_tc;

namespace {

using namespace tc;

constexpr int BM = 128;
constexpr int kThreads = 288;          // 4 epilogue + 4 builder + 1 MMA warp
constexpr int kMaxLevelRank = 128;

struct TTArgs {
    int d;
    int64_t dims[16];
    int64_t ranks[17];
    int64_t div[16];                   // level-l row of prefix p is p / div[l]
    const __half* cores[16];
    int64_t nprefix;
    int64_t ntiles;
    int nd, rlast, rprev, rp;          // n_d, r_{d-1}, r_{d-2} (0 if d == 2), rlast rounded up to 16
    int lvl_rows, lvl_ld;              // level buffers: rows and row pitch (floats)
    int cw;                            // output columns per 128-byte staging row
    int out16;
    uint32_t tmem_cols;
    uint32_t a_bytes;                  // one A operand (128 x rp binary16)
    uint32_t off_a, off_b, off_stage, off_lvl, off_bar;
    void* out;
};

struct Bars {
    uint64_t* a_full;    // [2]
    uint64_t* a_empty;   // [2]
    uint64_t* acc_full;  // [2]
    uint64_t* acc_empty; // [2]
    uint64_t* b_ready;
    uint64_t* mma_done;
    uint32_t* tmem_slot;
    int* abort;
};

__device__ __forceinline__ Bars carve(unsigned char* smem, const TTArgs& a) {
    Bars B;
    uint64_t* p = reinterpret_cast<uint64_t*>(smem + a.off_bar);
    B.a_full = p;
    B.a_empty = p + 2;
    B.acc_full = p + 4;
    B.acc_empty = p + 6;
    B.b_ready = p + 8;
    B.mma_done = p + 9;
    B.tmem_slot = reinterpret_cast<uint32_t*>(p + 10);
    B.abort = reinterpret_cast<int*>(B.tmem_slot + 1);
    return B;
}

// Builds the tile's Z_{d-1} rows into the A operand buffers (hi, lo).
template <int RMAX>
__device__ __forceinline__ void build_tile(const TTArgs& a, int64_t p0, int64_t pend, int bt, float* lvl0,
                                           float* lvl1, unsigned char* ahi, unsigned char* alo) {
    const int d = a.d;
    // ---- levels Z_1 .. Z_{d-2}: only the rows the tile passes through
    int64_t lo = 0;
    float* zin = lvl0;
    if (d >= 3) {
        lo = p0 / a.div[0];
        const int64_t hi = (pend - 1) / a.div[0];
        const int r1 = (int)a.ranks[1];
        const int cnt = (int)(hi - lo + 1);
        const __half* G = a.cores[0];
        for (int e = bt; e < cnt * r1; e += 128) {
            const int q = e / r1, c = e % r1;
            lvl0[q * a.lvl_ld + c] = __half2float(G[(lo + q) * r1 + c]);
        }
        named_bar_sync(2, 128);
        float* zout = lvl1;
        for (int l = 1; l <= d - 3; ++l) {
            const int r0 = (int)a.ranks[l], r1b = (int)a.ranks[l + 1];
            const int64_t nl = a.dims[l];
            const int64_t nlo = p0 / a.div[l];
            const int64_t nhi = (pend - 1) / a.div[l];
            const int c2 = (int)(nhi - nlo + 1);
            const __half* Gl = a.cores[l];
            for (int e = bt; e < c2 * r1b; e += 128) {
                const int q = e / r1b, c = e % r1b;
                const int64_t gq = nlo + q;
                const int64_t parent = gq / nl, i = gq - parent * nl;
                const float* zr = zin + (parent - lo) * a.lvl_ld;
                float acc = 0.0f;
                for (int t = 0; t < r0; ++t)
                    acc = fmaf(zr[t], __half2float(Gl[((int64_t)t * nl + i) * r1b + c]), acc);
                zout[q * a.lvl_ld + c] = acc;
            }
            named_bar_sync(2, 128);
            float* tmp = zin;
            zin = zout;
            zout = tmp;
            lo = nlo;
        }
    }
    // ---- last level: one row of Z_{d-1} per builder thread
    float acc[RMAX];
#pragma unroll
    for (int c = 0; c < RMAX; ++c) acc[c] = 0.0f;
    const int64_t p = p0 + bt;
    if (p < pend) {
        if (d == 2) {
            const __half* G = a.cores[0];
#pragma unroll
            for (int c = 0; c < RMAX; ++c)
                if (c < a.rlast) acc[c] = __half2float(G[p * a.rlast + c]);
        } else {
            const int64_t nl = a.dims[d - 2];
            const int64_t parent = p / nl, i = p - parent * nl;
            const float* zr = zin + (parent - lo) * a.lvl_ld;
            const __half* G = a.cores[d - 2];
            for (int t = 0; t < a.rprev; ++t) {
                const float z = zr[t];
                const __half* g = G + ((int64_t)t * nl + i) * a.rlast;
#pragma unroll
                for (int c = 0; c < RMAX; ++c)
                    if (c < a.rlast) acc[c] = fmaf(z, __half2float(g[c]), acc[c]);
            }
        }
    }
    // ---- A operand, canonical K-major layout: core (row group, 8-column group)
#pragma unroll
    for (int c0 = 0; c0 < RMAX; c0 += 8) {
        if (c0 >= a.rp) break;
        uint32_t hi[4], lo4[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float w0 = acc[c0 + 2 * j], w1 = acc[c0 + 2 * j + 1];
            const __half h0 = __float2half_rn(w0), h1 = __float2half_rn(w1);
            hi[j] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
            lo4[j] = pack_half2(w0 - __half2float(h0), w1 - __half2float(h1));
        }
        const uint32_t off = (uint32_t)(c0 >> 3) * 2048u + (uint32_t)(bt >> 3) * 128u + (uint32_t)(bt & 7) * 16u;
        *reinterpret_cast<uint4*>(ahi + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        if (!a.out16) *reinterpret_cast<uint4*>(alo + off) = make_uint4(lo4[0], lo4[1], lo4[2], lo4[3]);
    }
}

template <int RMAX>
__global__ void __launch_bounds__(kThreads, 1)
tt_f16_tc_kernel(const __grid_constant__ CUtensorMap tm_out, const TTArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                           ~static_cast<uintptr_t>(1023));
    const Bars B = carve(smem, a);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort = B.abort;
    unsigned int* err = &g_err_tt_tc;
    const int64_t my_tiles = (a.ntiles - blockIdx.x + gridDim.x - 1) / gridDim.x;

    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&B.a_full[i], 128);
            mbar_init(&B.a_empty[i], 1);
            mbar_init(&B.acc_full[i], 1);
            mbar_init(&B.acc_empty[i], 128);
        }
        mbar_init(B.b_ready, 128);
        mbar_init(B.mma_done, 1);
        *B.abort = 0;
        fence_barrier_init();
    }
    if (warp == 8) tmem_alloc(B.tmem_slot, a.tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *B.tmem_slot;

    if (warp >= 4 && warp < 8) {
        // ------------------------------------------------------------ builders
        const int bt = threadIdx.x - 128;
        // G_d^T (n_d x rp) in the canonical K-major layout, once per CTA
        {
            unsigned char* bsm = smem + a.off_b;
            const __half* Gd = a.cores[a.d - 1];
            const uint32_t lbo = (uint32_t)a.nd * 16u;
            for (int e = bt; e < a.nd * a.rp; e += 128) {
                const int i = e / a.rp, c = e % a.rp;
                const __half v = c < a.rlast ? Gd[(int64_t)c * a.nd + i] : __float2half_rn(0.0f);
                const uint32_t off = (uint32_t)(c >> 3) * lbo + (uint32_t)(i >> 3) * 128u + (uint32_t)(i & 7) * 16u +
                                     (uint32_t)(c & 7) * 2u;
                *reinterpret_cast<__half*>(bsm + off) = v;
            }
            fence_proxy_async_smem();
            mbar_arrive(B.b_ready);
        }
        float* lvl0 = reinterpret_cast<float*>(smem + a.off_lvl);
        float* lvl1 = lvl0 + (size_t)a.lvl_rows * a.lvl_ld;
        bool ok = true;
        for (int64_t j = 0; j < my_tiles && ok; ++j) {
            const int buf = (int)(j & 1);
            if (!(ok = group_wait(&B.a_empty[buf], (uint32_t)((j >> 1) & 1) ^ 1u, abort, err, 1u, 2, 128))) break;
            const int64_t tile = blockIdx.x + j * gridDim.x;
            const int64_t p0 = tile * BM;
            const int64_t pend = (p0 + BM < a.nprefix) ? p0 + BM : a.nprefix;
            unsigned char* ahi = smem + a.off_a + (size_t)buf * 2 * a.a_bytes;
            build_tile<RMAX>(a, p0, pend, bt, lvl0, lvl1, ahi, ahi + a.a_bytes);
            fence_proxy_async_smem();
            mbar_arrive(&B.a_full[buf]);
            named_bar_sync(2, 128);   // level buffers are reused by the next tile
        }
    } else if (warp == 8) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            bool ok = mbar_wait(B.b_ready, 0, abort, err, 2u);
            tc_fence_after();
            const uint32_t bsm = smem_u32(smem + a.off_b);
            const uint32_t idesc = idesc_f16_f32(BM, (uint32_t)a.nd);
            const uint32_t lbo_b = (uint32_t)a.nd * 16u;
            const uint64_t bd = smem_desc(bsm, lbo_b, 128, 0);
            const uint64_t bstep = (uint64_t)(2u * lbo_b) >> 4;
            for (int64_t j = 0; j < my_tiles && ok; ++j) {
                const int buf = (int)(j & 1);
                const uint32_t par = (uint32_t)((j >> 1) & 1);
                if (!(ok = mbar_wait(&B.a_full[buf], par, abort, err, 2u))) break;
                if (!(ok = mbar_wait(&B.acc_empty[buf], par ^ 1u, abort, err, 2u))) break;
                tc_fence_after();
                const uint32_t ahi = smem_u32(smem + a.off_a + (size_t)buf * 2 * a.a_bytes);
                const uint32_t alo = ahi + a.a_bytes;
                const uint32_t dcol = tmem + (uint32_t)buf * (uint32_t)a.nd;
                // descriptors stepped by adds (16 ranks = 4096 B of A, 2 x lbo_b B of B)
                const uint64_t hd = smem_desc(ahi, 2048, 128, 0), ld = smem_desc(alo, 2048, 128, 0);
                for (int ks = 0; ks < a.rp / 16; ++ks) {
                    const uint64_t bdesc = bd + (uint64_t)ks * bstep;
                    mma_f16(dcol, hd + (uint64_t)ks * 256u, bdesc, idesc, ks > 0);
                    if (!a.out16) mma_f16(dcol, ld + (uint64_t)ks * 256u, bdesc, idesc, 1u);
                }
                mma_commit(&B.a_empty[buf]);
                mma_commit(&B.acc_full[buf]);
            }
            mma_commit(B.mma_done);
            volatile int no_abort = 0;
            mbar_wait(B.mma_done, 0, &no_abort, err, 2u, 100000000ull);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int g = warp & 3;
        const int r = g * 32 + lane;
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        const bool issuer = (threadIdx.x == 0);
        bool ok = true;
        int chunk = 0;
        for (int64_t j = 0; j < my_tiles && ok; ++j) {
            const int buf = (int)(j & 1);
            if (!(ok = group_wait(&B.acc_full[buf], (uint32_t)((j >> 1) & 1), abort, err, 4u, 1, 128))) break;
            tc_fence_after();
            const int64_t tile = blockIdx.x + j * gridDim.x;
            const int64_t p0 = tile * BM;
            // 128-byte staging rows (32 FP32 or 64 FP16 columns); a last chunk
            // reaching past n_d is clipped by the TMA store
            for (int cc = 0; cc < a.nd; cc += a.cw, ++chunk) {
                uint32_t v[64];
                const uint32_t tcol = tmem + lane_base + (uint32_t)buf * (uint32_t)a.nd + (uint32_t)cc;
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
                unsigned char* sb = smem + a.off_stage + (size_t)(chunk & 1) * (BM * 128);
                if (chunk >= 2) {
                    if (issuer) bulk_wait_read<1>();
                    named_bar_sync(1, 128);
                }
                // 128-byte swizzle: 16-byte chunk q of row r sits at chunk q ^ (r mod 8)
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const uint32_t off = (uint32_t)r * 128u + (uint32_t)((q ^ (r & 7)) * 16);
                    *reinterpret_cast<uint4*>(sb + off) =
                        make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
                }
                fence_proxy_async_smem();
                named_bar_sync(1, 128);
                if (issuer) {
                    tma_store_2d(&tm_out, cc, (int32_t)p0, sb);
                    bulk_commit();
                }
            }
            tc_fence_before();
            mbar_arrive(&B.acc_empty[buf]);
        }
        if (issuer) bulk_wait<0>();
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

PFN_cuTensorMapEncodeTiled_v12000 g_encode_tt = nullptr;
std::once_flag g_encode_tt_once;

uint32_t pow2_cols(uint32_t c) {
    uint32_t p = 32;
    while (p < c) p <<= 1;
    return p;
}

}  // namespace

// True when the tensor-core kernel covers this shape.
bool tt_f16_tc_supported(const TTShape& sh, bool out16) {
    const int d = sh.d;
    const int64_t nd = sh.dims[d - 1];
    if (nd % 16 != 0 || nd > 256) return false;
    if (nd * (out16 ? 2 : 4) < 128) return false;      // output rows narrower than one staging row
    if (sh.ranks[d - 1] > 64) return false;
    for (int l = 1; l < d - 1; ++l)
        if (sh.ranks[l] > kMaxLevelRank) return false;
    return true;
}

lrc_status launch_tt_f16_tc(const TTShape& sh, bool out16, void* out, cudaStream_t s) {
    std::call_once(g_encode_tt_once, [] {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode_tt = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    });
    if (!g_encode_tt) {
        set_error("cuTensorMapEncodeTiled is not available from the driver");
        return LRC_ERR_CUDA;
    }
    TTArgs a{};
    const int d = sh.d;
    a.d = d;
    for (int l = 0; l < d; ++l) {
        a.dims[l] = sh.dims[l];
        a.ranks[l] = sh.ranks[l];
        a.cores[l] = static_cast<const __half*>(sh.cores[l]);
    }
    a.ranks[d] = 1;
    a.nprefix = 1;
    for (int l = 0; l < d - 1; ++l) a.nprefix *= sh.dims[l];
    for (int l = 0; l < d - 1; ++l) {
        int64_t v = 1;
        for (int j = l + 1; j <= d - 2; ++j) v *= sh.dims[j];
        a.div[l] = v;
    }
    a.nd = (int)sh.dims[d - 1];
    a.rlast = (int)sh.ranks[d - 1];
    a.rprev = d >= 3 ? (int)sh.ranks[d - 2] : 0;
    a.rp = (a.rlast + 15) / 16 * 16;
    a.out16 = out16 ? 1 : 0;
    a.out = out;
    // level buffers: rows the parent levels can span within one 128-prefix tile
    int lvl_rows = 1, lvl_ld = 1;
    for (int l = 0; l <= d - 3; ++l) {
        const int64_t rows = (BM - 1) / a.div[l] + 2;
        if (rows > lvl_rows) lvl_rows = (int)(rows < BM + 1 ? rows : BM + 1);
        if (sh.ranks[l + 1] > lvl_ld) lvl_ld = (int)sh.ranks[l + 1];
    }
    a.lvl_rows = lvl_rows;
    a.lvl_ld = lvl_ld | 1;
    const int eo = out16 ? 2 : 4;
    a.cw = 128 / eo;                                   // columns per 128-byte staging row
    a.a_bytes = (uint32_t)BM * a.rp * 2;
    uint32_t off = 0;
    a.off_a = off;
    off += 4 * a.a_bytes;                                   // 2 buffers x (hi, lo)
    off = (off + 127) / 128 * 128;
    a.off_b = off;
    off += (uint32_t)a.nd * a.rp * 2;
    off = (off + 1023) / 1024 * 1024;
    a.off_stage = off;
    off += 2 * BM * 128;
    a.off_lvl = off;
    off += 2u * (uint32_t)a.lvl_rows * (uint32_t)a.lvl_ld * 4u;
    off = (off + 7) / 8 * 8;
    a.off_bar = off;
    off += 10 * 8 + 16;
    const size_t smem = (size_t)off + 1024;
    if (smem > 227 * 1024) {
        set_error("tt_f16_tc_kernel: shape needs %zu bytes of shared memory", smem);
        return LRC_ERR_UNSUPPORTED;
    }
    a.tmem_cols = pow2_cols(2u * (uint32_t)a.nd);
    // the second accumulator's last staging chunk must stay inside the allocation
    const uint32_t last_col = (uint32_t)a.nd + (uint32_t)((a.nd + a.cw - 1) / a.cw * a.cw);
    if (last_col > a.tmem_cols) {
        set_error("tt_f16_tc_kernel: n_d = %d does not fit the tensor-memory plan", a.nd);
        return LRC_ERR_UNSUPPORTED;
    }
    a.ntiles = (a.nprefix + BM - 1) / BM;
    const int sms = sm_count();
    const int64_t grid = a.ntiles < sms ? a.ntiles : sms;

    CUtensorMap tm;
    cuuint64_t dims[2] = {(cuuint64_t)a.nd, (cuuint64_t)a.nprefix};
    cuuint64_t strides[1] = {(cuuint64_t)a.nd * eo};
    cuuint32_t box[2] = {(cuuint32_t)a.cw, (cuuint32_t)BM};
    cuuint32_t estr[2] = {1, 1};
    CUresult cr = g_encode_tt(&tm, out16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, out,
                              dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (cr != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled failed for the TT output (CUresult %d)", (int)cr);
        return LRC_ERR_CUDA;
    }
    cudaError_t e;
    const int rmax = a.rlast <= 16 ? 16 : (a.rlast <= 32 ? 32 : (a.rlast <= 48 ? 48 : 64));
    switch (rmax) {
        case 16:
            e = cudaFuncSetAttribute(tt_f16_tc_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return cuda_fail(e, "tt_f16_tc_kernel smem attribute");
            tt_f16_tc_kernel<16><<<(unsigned)grid, kThreads, smem, s>>>(tm, a);
            break;
        case 32:
            e = cudaFuncSetAttribute(tt_f16_tc_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return cuda_fail(e, "tt_f16_tc_kernel smem attribute");
            tt_f16_tc_kernel<32><<<(unsigned)grid, kThreads, smem, s>>>(tm, a);
            break;
        case 48:
            e = cudaFuncSetAttribute(tt_f16_tc_kernel<48>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return cuda_fail(e, "tt_f16_tc_kernel smem attribute");
            tt_f16_tc_kernel<48><<<(unsigned)grid, kThreads, smem, s>>>(tm, a);
            break;
        default:
            e = cudaFuncSetAttribute(tt_f16_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return cuda_fail(e, "tt_f16_tc_kernel smem attribute");
            tt_f16_tc_kernel<64><<<(unsigned)grid, kThreads, smem, s>>>(tm, a);
            break;
    }
    return after_launch("tt_f16_tc_kernel");
}

lrc_status launch_tt_f16(const TTShape& sh, bool out16, void* out, cudaStream_t s) {
    bool handled = false;
    lrc_status st = launch_tt3_f16_tc(sh, out16, out, s, &handled);
    if (handled) return st;
    st = launch_tt_split_f16(sh, out16, out, s, &handled);
    if (handled) return st;
    st = launch_ttn_f16_tc(sh, out16, out, s, &handled);
    if (handled) return st;
    if (tt_f16_tc_supported(sh, out16)) return launch_tt_f16_tc(sh, out16, out, s);
    return launch_tt_cc(sh, out16 ? LRC_F16_O16 : LRC_F16, out, s);
}

uint32_t take_tt_tc_error() {
    unsigned int v = 0;
    if (cudaMemcpyFromSymbol(&v, g_err_tt_tc, sizeof v) != cudaSuccess) return 0xffffffffu;
    if (v) {
        const unsigned int z = 0;
        cudaMemcpyToSymbol(g_err_tt_tc, &z, sizeof z);
    }
    return v;
}

}  // namespace lrc
