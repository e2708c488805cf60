// tt_narrow_tc.cu -- dense TT reconstruction from binary16 cores on the
// tensor cores when the last two modes are narrow (Sec. 5.1:
// T(i_1..i_d) = G_1(i_1)...G_d(i_d); Sec. 7.5, Eq. gpu_tt_reconstruction:
// B_l = Z_{l-1} K_l, Z_l = reshape(B_l); Sec. 3.4: FP32 accumulation).
//
// T is viewed as P prefix rows (i_1..i_{d-2}) x n_{d-1} n_d columns (C order:
// every row is contiguous).  A work unit is a tile of 128 consecutive
// prefixes:
//   build    a chain kernel (one 128-thread CTA per tile, many per SM, so
//            the global-memory latency of the small irregular chain
//            overlaps) computes the tile's rows of Z_{d-2} on the CUDA cores
//            in FP32 and writes them as the binary16 A-operand image -- a
//            hi/lo pair for FP32 output, one rounding for FP16 output (the
//            method-precision workspace) -- to the stream workspace; the
//            main kernel's loader copies each image into shared memory
//            (double-buffered, one bulk copy per plane);
//   stage 1  D1 (128 x n_{d-1} r_{d-1}, TMEM) = Z_{d-2} K_{d-1}: all i_{d-1}
//            at once, B = K_{d-1}^T kept in shared memory (rows (i, b));
//   convert  converter warps split each D1 row into n_{d-1} binary16 rows of
//            Z_{d-1} = reshape(B_{d-1}) (hi/lo or one rounding), one operand
//            tile per i_{d-1};
//   stage 2  D2[:, i n_d .. (i+1) n_d) = Z_{d-1}(i) G_d for every i_{d-1} = i
//            (B = G_d^T in shared memory);
//   store    epilogue warps drain D2 (TMEM -> registers -> swizzled shared
//            memory -> TMA stores of whole 32-row boxes, each warp its own
//            rows).
// Stage 1 of the next unit runs while the epilogue drains this one.  Warp
// roles of the main kernel: 0..3 epilogue, 4..7 converters, 8 MMA issuer
// (one thread), 9 loader (one thread).  Z_{d-1} = reshape(B_{d-1}), the large
// intermediate, never reaches global memory; the Z_{d-2} images are a few
// percent of the output and stay in L2.
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "tc.cuh"

namespace lrc {

__device__ unsigned int g_err_ttn_tc;

namespace {

using namespace tc;

constexpr int BM = 128;
constexpr int kThreads = 320;
constexpr int kMaxD = 16;

struct TNArgs {
    int d;
    int64_t np;                       // prefix rows, prod_{l <= d-3} n_l (0-based modes)
    int64_t units;                    // ceil(np / 128)
    int ra, rap;                      // rank into the last two modes, padded to 16
    int nb, rb, rbp;                  // mode d-2: size, rank after it, padded
    int nc;                           // mode d-1 size
    int n1w;                          // nb * rbp: stage-1 N
    int out16;
    uint32_t a1_bytes, tile2_bytes;   // one A1 plane; one A2 tile plane (128 x rbp)
    uint32_t off_a1, off_b1, off_a2, off_b2, off_exp, off_stage, off_bar;
    int64_t dims[kMaxD];
    int ranks[kMaxD + 1];
    int64_t div[kMaxD];               // div[l] = prod_{j=l+1}^{d-3} n_j
    const __half* cores[kMaxD];
    const unsigned char* img;          // Z_{d-2} operand images: [unit][plane][a1_bytes]
    const int* exps;                   // their row exponents: [unit][128]
    const unsigned char* b1img;        // K_{d-1}^T and G_d^T operand images
    const unsigned char* b2img;
    uint32_t b1_bytes, b2_bytes;
};

struct Bars {
    uint64_t *a1_full, *a1_empty;     // [2]
    uint64_t *d1_full, *cv_done, *a2_empty, *d2_full, *d2_free, *mma_done;
    uint64_t *sc_full, *sc_empty;     // [2] stage-1 row exponents, loaders -> converters
    uint64_t *t_full, *t_empty;       // [2] total row exponents, converters -> epilogue
    uint64_t* b_full;                 // the B operand images
    uint32_t* tmem_slot;
    int* abort;
};

__device__ __forceinline__ Bars carve(unsigned char* smem, const TNArgs& a) {
    uint64_t* p = reinterpret_cast<uint64_t*>(smem + a.off_bar);
    Bars B;
    B.a1_full = p + 0;
    B.a1_empty = p + 2;
    B.d1_full = p + 4;
    B.cv_done = p + 5;
    B.a2_empty = p + 6;
    B.d2_full = p + 7;
    B.d2_free = p + 8;
    B.mma_done = p + 9;
    B.sc_full = p + 10;
    B.sc_empty = p + 12;
    B.t_full = p + 14;
    B.t_empty = p + 16;
    B.b_full = p + 18;
    B.tmem_slot = reinterpret_cast<uint32_t*>(p + 19);
    B.abort = reinterpret_cast<int*>(B.tmem_slot + 1);
    return B;
}

// Byte offset of element (row, k) in a canonical no-swizzle K-major operand
// with `rows` rows: 8-row x 16-byte core matrices, K-direction stride
// rows * 16 bytes, row-group stride 128 bytes.
__device__ __forceinline__ uint32_t canon_off(uint32_t row, uint32_t k, uint32_t rows) {
    return (k >> 3) * rows * 16u + (row >> 3) * 128u + (row & 7u) * 16u + (k & 7u) * 2u;
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi) { return pack_half2(lo, hi); }

// Row scaling for the hi/lo split (FP32 output): a row whose largest
// magnitude is x is multiplied by 2^s with x 2^s in [2^14, 2^15), so that
// the lo parts stay clear of the binary16 subnormals (which would cap the
// pair's accuracy at an absolute 2^-24); powers of two scale exactly.
__device__ __forceinline__ int row_exp(float maxabs) {
    if (!(maxabs > 0.0f)) return 0;
    const int e = (int)((__float_as_uint(maxabs) >> 23) & 0xffu) - 127;
    const int sc = 14 - e;
    return sc < -60 ? -60 : (sc > 60 ? 60 : sc);
}
__device__ __forceinline__ float pow2f(int s) { return __int_as_float((s + 127) << 23); }



// ---------------------------------------------------------------- pre-kernels
// B operands as shared-memory images: K_{d-1}^T (row i * rbp + b, column a =
// G_{d-2}[a, i, b]) and G_d^T (row c, column b = G_{d-1}[b, c]), canonical
// K-major layouts with zero padding.
__global__ void __launch_bounds__(256)
ttn_bimg_kernel(const __grid_constant__ TNArgs a, unsigned char* b1img, unsigned char* b2img) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int total1 = a.n1w * a.rap, total2 = a.nc * a.rbp;
    if (e < total1) {
        const int row = (int)(e / a.rap), k = (int)(e % a.rap);
        const int i = row / a.rbp, bb = row - (row / a.rbp) * a.rbp;
        const __half* G = a.cores[a.d - 2];
        const __half v = (k < a.ra && bb < a.rb) ? G[((int64_t)k * a.nb + i) * a.rb + bb] : __float2half_rn(0.0f);
        *reinterpret_cast<__half*>(b1img + canon_off((uint32_t)row, (uint32_t)k, (uint32_t)a.n1w)) = v;
    } else if (e < total1 + total2) {
        const int e2 = (int)(e - total1);
        const int c = e2 / a.rbp, k = e2 - (e2 / a.rbp) * a.rbp;
        const __half* H = a.cores[a.d - 1];
        const __half v = k < a.rb ? H[(int64_t)k * a.nc + c] : __float2half_rn(0.0f);
        *reinterpret_cast<__half*>(b2img + canon_off((uint32_t)c, (uint32_t)k, (uint32_t)a.nc)) = v;
    }
}

// The chain up to Z_{d-2} (Eq. gpu_tt_reconstruction: B_l = Z_{l-1} K_l,
// Z_l = reshape(B_l)) for every tile of 128 prefixes, persistent CTAs (two
// per SM when they fit).  The cores G_1 .. G_{d-2} (binary16) are bulk-copied into shared memory
// once, so the chain's small irregular products run on shared-memory
// operands: for each tile the few ancestor rows of Z_1 .. Z_{d-3} in FP32,
// then the tile's rows of Z_{d-2} as tasks (one i, four columns, up to
// kPar parents: each core value loaded serves kPar rows).  The rows are
// written as the binary16 A-operand images of the main kernel (hi/lo with a
// power-of-two row scale for FP32 output, one rounding for FP16 output, zero
// padding) plus their row exponents.
constexpr int kChThreads = 256, kPar = 8;

struct ChArgs {
    uint32_t core_off[kMaxD];      // shared-memory byte offset of core l (l <= d-3)
    uint32_t core_bytes[kMaxD];
    uint32_t cores_total;          // bytes of the copied cores, rounded up to 16
    uint32_t off_lv, off_stg, off_rmx, off_bar;
    int lvrows, lvw;               // FP32 level buffer: rows x width (each of two)
};

__global__ void __launch_bounds__(kChThreads, 2)
ttn_chain_kernel(const __grid_constant__ TNArgs a, const __grid_constant__ ChArgs c, unsigned char* img, int* exps) {
    pdl_trigger();                 // the main kernel may set up meanwhile; it waits for this grid
    extern __shared__ __align__(16) unsigned char csm[];
    const int tid = threadIdx.x;
    uint64_t* bar = reinterpret_cast<uint64_t*>(csm + c.off_bar);
    const int last = a.d - 3;
    // ---- the cores into shared memory: 16-byte-aligned bodies by bulk copy,
    // the tails (under 16 bytes) by plain loads
    if (tid == 0) {
        mbar_init(bar, 1);
        fence_barrier_init();
        uint32_t tx = 0;
        for (int l = 0; l <= last; ++l) tx += c.core_bytes[l] / 16 * 16;
        mbar_arrive_expect_tx(bar, tx);
        for (int l = 0; l <= last; ++l) {
            const uint32_t body = c.core_bytes[l] / 16 * 16;
            if (body) bulk_load(csm + c.core_off[l], a.cores[l], body, bar);
        }
    }
    for (int l = 0; l <= last; ++l) {
        const uint32_t body = c.core_bytes[l] / 16 * 16;
        const uint32_t tail = c.core_bytes[l] - body;
        if ((uint32_t)tid < tail / 2)
            reinterpret_cast<__half*>(csm + c.core_off[l] + body)[tid] =
                __ldg(reinterpret_cast<const __half*>(reinterpret_cast<const unsigned char*>(a.cores[l]) + body) + tid);
    }
    __syncthreads();
    {
        volatile int no_abort = 0;
        if (!mbar_wait(bar, 0, &no_abort, &g_err_ttn_tc, 16u)) return;
    }
    float* const lv0 = reinterpret_cast<float*>(csm + c.off_lv);
    float* const lv1 = lv0 + c.lvrows * c.lvw;
    float* stg = reinterpret_cast<float*>(csm + c.off_stg);          // [128][rap + 4] unscaled rows
    const int planes = a.out16 ? 1 : 2;

    for (int64_t u = blockIdx.x; u < a.units; u += gridDim.x) {
        const int64_t p0 = u * BM;
        const int64_t pend = (p0 + BM < a.np) ? p0 + BM : a.np;
        // ancestors: levels 0 .. last-1 (contiguous row ranges), FP32
        int cur = 0;
        int64_t lo = 0;
        for (int l = 0; l < last; ++l) {
            const int64_t nlo = p0 / a.div[l], nhi = (pend - 1) / a.div[l];
            const int cnt = (int)(nhi - nlo + 1);
            const int r0 = a.ranks[l], r1 = a.ranks[l + 1];
            const int64_t nl = a.dims[l];
            const __half* G = reinterpret_cast<const __half*>(csm + c.core_off[l]);
            float* zo = (l == 0 || cur) ? lv0 : lv1;          // level 0 -> buffer 0, then alternate
            const float* zi = cur ? lv1 : lv0;
            for (int e = tid; e < cnt * r1; e += kChThreads) {
                const int q = e / r1, cc = e - (e / r1) * r1;
                const int64_t gq = nlo + q;
                float acc;
                if (l == 0) {
                    acc = __half2float(G[gq * r1 + cc]);
                } else {
                    const int64_t parent = gq / nl, i = gq - (gq / nl) * nl;
                    const float* zr = zi + (parent - lo) * c.lvw;
                    acc = 0.0f;
                    for (int k = 0; k < r0; ++k) acc = fmaf(zr[k], __half2float(G[(k * nl + i) * r1 + cc]), acc);
                }
                zo[q * c.lvw + cc] = acc;
            }
            __syncthreads();
            if (l > 0) cur ^= 1;
            lo = nlo;
        }
        // the tile's rows of Z_{d-2}: tasks (i, four columns) over parent chunks
        const float* zp = cur ? lv1 : lv0;
        const int64_t nl = a.dims[last];
        const int r0 = a.ranks[last];
        const __half* G = reinterpret_cast<const __half*>(csm + c.core_off[last]);
        const int64_t qlo = (last == 0) ? 0 : lo, qhi = (last == 0) ? 0 : (pend - 1) / nl;
        const int nq = (int)(qhi - qlo + 1);
        const int ncg = a.rap / 4;                      // the zero padding columns too
        // i values this tile touches: all of [0, nl), or a sub-range when the tile
        // lies inside a single parent
        const int64_t ibeg = (nq == 1) ? p0 - qlo * nl : 0;
        const int64_t iend = (nq == 1) ? pend - qlo * nl : nl;
        const int ntask = (int)(iend - ibeg) * ncg;
        for (int qc = 0; qc < nq; qc += kPar) {
            for (int task = tid; task < ntask; task += kChThreads) {
                const int i = (int)ibeg + task / ncg;
                const int c0 = (task - (task / ncg) * ncg) * 4;
                float acc[kPar][4];
#pragma unroll
                for (int pp = 0; pp < kPar; ++pp)
#pragma unroll
                    for (int q = 0; q < 4; ++q) acc[pp][q] = 0.0f;
                bool any = false;
#pragma unroll
                for (int pp = 0; pp < kPar; ++pp) {
                    const int64_t pr = (qlo + qc + pp) * nl + i;
                    any |= (qc + pp < nq && pr >= p0 && pr < pend);
                }
                if (!any) continue;
                for (int k = 0; k < r0; ++k) {
                    float g[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        g[q] = (c0 + q < a.ra) ? __half2float(G[((int64_t)k * nl + i) * a.ra + c0 + q]) : 0.0f;
#pragma unroll
                    for (int pp = 0; pp < kPar; ++pp) {
                        const float z = (last == 0) ? 1.0f : ((qc + pp < nq) ? zp[(qc + pp) * c.lvw + k] : 0.0f);
#pragma unroll
                        for (int q = 0; q < 4; ++q) acc[pp][q] = fmaf(z, g[q], acc[pp][q]);
                    }
                }
#pragma unroll
                for (int pp = 0; pp < kPar; ++pp) {
                    const int64_t pr = (qlo + qc + pp) * nl + i;
                    if (qc + pp < nq && pr >= p0 && pr < pend)
                        *reinterpret_cast<float4*>(stg + (size_t)(pr - p0) * (a.rap + 4) + c0) =
                            make_float4(acc[pp][0], acc[pp][1], acc[pp][2], acc[pp][3]);
                }
            }
        }
        __syncthreads();
        // one thread per row: scale, round to binary16 (hi / lo), store the image
        unsigned char* base = img + (size_t)u * planes * a.a1_bytes;
        for (int r = tid; r < BM; r += kChThreads) {
            const bool valid = p0 + r < pend;
            const float* zr = stg + (size_t)r * (a.rap + 4);   // padded rows: no bank conflicts
            float f = 1.0f;
            int sc = 0;
            if (!a.out16 && valid) {
                float mx = 0.0f;
                for (int q = 0; q < a.rap; ++q) mx = fmaxf(mx, fabsf(zr[q]));
                sc = row_exp(mx);
                f = pow2f(sc);
            }
            for (int c0 = 0; c0 < a.rap; c0 += 8) {
                uint32_t hi[4], lw[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float w0 = valid ? zr[c0 + 2 * q] * f : 0.0f, w1 = valid ? zr[c0 + 2 * q + 1] * f : 0.0f;
                    const __half h0 = __float2half_rn(w0), h1 = __float2half_rn(w1);
                    hi[q] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
                    lw[q] = pack2(w0 - __half2float(h0), w1 - __half2float(h1));
                }
                const uint32_t off = canon_off((uint32_t)r, (uint32_t)c0, BM);
                *reinterpret_cast<uint4*>(base + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                if (!a.out16) *reinterpret_cast<uint4*>(base + a.a1_bytes + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
            }
            exps[u * BM + r] = sc;
        }
        __syncthreads();               // stg and the level buffers are reused by the next tile
    }
}

__global__ void __launch_bounds__(kThreads, 1)
ttn_f16_tc_kernel(const __grid_constant__ CUtensorMap tm_out, const TNArgs a) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                           ~static_cast<uintptr_t>(1023));
    const Bars B = carve(smem, a);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort = B.abort;
    unsigned int* err = &g_err_ttn_tc;
    const int planes = a.out16 ? 1 : 2;
    const int64_t ubeg = a.units * blockIdx.x / gridDim.x;
    const int64_t uend = a.units * (blockIdx.x + 1) / gridDim.x;
    const int64_t nunits = uend - ubeg;

    if (threadIdx.x == 0) {
        for (int q = 0; q < 2; ++q) {
            mbar_init(&B.a1_full[q], 1);
            mbar_init(&B.a1_empty[q], 1);
        }
        mbar_init(B.d1_full, 1);
        mbar_init(B.cv_done, 128);
        mbar_init(B.a2_empty, 1);
        mbar_init(B.d2_full, 1);
        mbar_init(B.d2_free, 128);
        mbar_init(B.mma_done, 1);
        for (int q = 0; q < 2; ++q) {
            mbar_init(&B.sc_full[q], 1);
            mbar_init(&B.sc_empty[q], 128);
            mbar_init(&B.t_full[q], 128);
            mbar_init(&B.t_empty[q], 128);
        }
        mbar_init(B.b_full, 1);
        *B.abort = 0;
        fence_barrier_init();
        tma_prefetch_desc(&tm_out);
        // the B operand images written by the pre-kernels
        pdl_wait();
        mbar_arrive_expect_tx(B.b_full, a.b1_bytes + a.b2_bytes);
        bulk_load(smem + a.off_b1, a.b1img, a.b1_bytes, B.b_full);
        bulk_load(smem + a.off_b2, a.b2img, a.b2_bytes, B.b_full);
    }
    if (warp == 8) tmem_alloc(B.tmem_slot, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *B.tmem_slot;
    const uint32_t d1col = tmem, d2col = tmem + 256;
    int* s1x = reinterpret_cast<int*>(smem + a.off_exp);     // [2][128] stage-1 row exponents
    int* tx = s1x + 2 * BM;                                  // [2][128] total row exponents

    if (warp == 9) {
        // ------------------------------------------------------------ loader
        // operand images of Z_{d-2} (and their row exponents) made by the
        // chain kernel, one bulk copy per plane
        if (lane == 0) {
            pdl_wait();                // the chain kernel's images are complete and visible
            bool ok = true;
            int64_t j = 0;
            for (; j < nunits; ++j) {
                const int buf = (int)(j & 1);
                if (j >= 2 && !(ok = mbar_wait(&B.a1_empty[buf], (uint32_t)(((j >> 1) - 1) & 1), abort, err, 1u)))
                    break;
                unsigned char* a1 = smem + a.off_a1 + (size_t)buf * planes * a.a1_bytes;
                mbar_arrive_expect_tx(&B.a1_full[buf], (uint32_t)planes * a.a1_bytes);
                for (int pl = 0; pl < planes; ++pl)
                    bulk_load(a1 + (size_t)pl * a.a1_bytes, a.img + ((size_t)(ubeg + j) * planes + pl) * a.a1_bytes,
                              a.a1_bytes, &B.a1_full[buf]);
                if (!a.out16) {
                    if (j >= 2 &&
                        !(ok = mbar_wait(&B.sc_empty[buf], (uint32_t)(((j >> 1) - 1) & 1), abort, err, 1u)))
                        break;
                    mbar_arrive_expect_tx(&B.sc_full[buf], BM * 4u);
                    bulk_load(s1x + buf * BM, a.exps + (size_t)(ubeg + j) * BM, BM * 4u, &B.sc_full[buf]);
                }
            }
            if (!ok) {
                // copies already in flight land before the CTA can exit
                volatile int no_abort = 0;
                for (int64_t q = (j - 2 > 0 ? j - 2 : 0); q <= j && q < nunits; ++q) {
                    mbar_wait(&B.a1_full[q & 1], (uint32_t)((q >> 1) & 1), &no_abort, err, 0u, 100000000ull);
                    if (!a.out16)
                        mbar_wait(&B.sc_full[q & 1], (uint32_t)((q >> 1) & 1), &no_abort, err, 0u, 100000000ull);
                }
            }
        }
    } else if (warp == 8) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            bool ok = true;
            const uint32_t idesc1 = idesc_f16_f32(BM, (uint32_t)a.n1w);
            const uint32_t idesc2 = idesc_f16_f32(BM, (uint32_t)a.nc);
            const uint64_t b1d = smem_desc(smem_u32(smem + a.off_b1), (uint32_t)a.n1w * 16u, 128, 0);
            const uint64_t b1step = (uint64_t)(2u * (uint32_t)a.n1w * 16u) >> 4;
            const uint64_t b2d = smem_desc(smem_u32(smem + a.off_b2), (uint32_t)a.nc * 16u, 128, 0);
            const uint64_t b2step = (uint64_t)(2u * (uint32_t)a.nc * 16u) >> 4;
            const uint32_t a2s = smem_u32(smem + a.off_a2);
            ok = mbar_wait(B.b_full, 0, abort, err, 2u);
            auto stage1 = [&](int64_t j) -> bool {
                const int buf = (int)(j & 1);
                if (!mbar_wait(&B.a1_full[buf], (uint32_t)((j >> 1) & 1), abort, err, 2u)) return false;
                tc_fence_after();
                const uint32_t a1s = smem_u32(smem + a.off_a1 + (size_t)buf * planes * a.a1_bytes);
                const uint64_t hd = smem_desc(a1s, 2048, 128, 0), ld = smem_desc(a1s + a.a1_bytes, 2048, 128, 0);
                for (int ks = 0; ks < a.rap / 16; ++ks) {
                    mma_f16(d1col, hd + (uint64_t)ks * 256u, b1d + (uint64_t)ks * b1step, idesc1, ks > 0);
                    if (!a.out16) mma_f16(d1col, ld + (uint64_t)ks * 256u, b1d + (uint64_t)ks * b1step, idesc1, 1u);
                }
                mma_commit(&B.a1_empty[buf]);
                mma_commit(B.d1_full);
                return true;
            };
            auto stage2 = [&](int64_t j) -> bool {
                if (!mbar_wait(B.cv_done, (uint32_t)(j & 1), abort, err, 2u)) return false;
                if (j >= 1 && !mbar_wait(B.d2_free, (uint32_t)((j - 1) & 1), abort, err, 2u)) return false;
                tc_fence_after();
                for (int i = 0; i < a.nb; ++i) {
                    const uint32_t t0 = a2s + (uint32_t)i * a.tile2_bytes;
                    const uint64_t hd = smem_desc(t0, 2048, 128, 0);
                    const uint64_t ld = smem_desc(t0 + (uint32_t)a.nb * a.tile2_bytes, 2048, 128, 0);
                    const uint32_t dc = d2col + (uint32_t)(i * a.nc);
                    for (int ks = 0; ks < a.rbp / 16; ++ks) {
                        mma_f16(dc, hd + (uint64_t)ks * 256u, b2d + (uint64_t)ks * b2step, idesc2, ks > 0);
                        if (!a.out16) mma_f16(dc, ld + (uint64_t)ks * 256u, b2d + (uint64_t)ks * b2step, idesc2, 1u);
                    }
                }
                mma_commit(B.a2_empty);
                mma_commit(B.d2_full);
                return true;
            };
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
        // ------------------------------------------------------------ converters
        const int g = warp & 3;
        const int r = g * 32 + lane;
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        unsigned char* a2 = smem + a.off_a2;
        for (int64_t j = 0; j < nunits; ++j) {
            const int eb = (int)(j & 1);
            if (!group_wait(B.d1_full, (uint32_t)(j & 1), abort, err, 4u, 2, 128)) break;
            if (j >= 1 && !group_wait(B.a2_empty, (uint32_t)((j - 1) & 1), abort, err, 4u, 2, 128)) break;
            tc_fence_after();
            float f2 = 1.0f;
            if (!a.out16) {
                // this row's stage-1 exponent, then the exponent for stage 2
                if (!group_wait(&B.sc_full[eb], (uint32_t)((j >> 1) & 1), abort, err, 4u, 2, 128)) break;
                const int s1 = s1x[eb * BM + r];
                mbar_arrive(&B.sc_empty[eb]);
                float mx = 0.0f;
                for (int c0 = 0; c0 < a.n1w; c0 += 32) {
                    uint32_t v[32];
                    tmem_ld32(d1col + lane_base + (uint32_t)c0, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int q = 0; q < 32; ++q) mx = fmaxf(mx, fabsf(__uint_as_float(v[q])));
                }
                const int s2 = row_exp(mx);
                f2 = pow2f(s2);
                if (j >= 2 && !group_wait(&B.t_empty[eb], (uint32_t)(((j >> 1) - 1) & 1), abort, err, 4u, 2, 128))
                    break;
                tx[eb * BM + r] = s1 + s2;
                mbar_arrive(&B.t_full[eb]);
            }
            for (int c0 = 0; c0 < a.n1w; c0 += 32) {
                uint32_t v[32];
                tmem_ld32(d1col + lane_base + (uint32_t)c0, v);
                tmem_ld_wait();
                if (!a.out16) {
#pragma unroll
                    for (int q = 0; q < 32; ++q) v[q] = __float_as_uint(__uint_as_float(v[q]) * f2);
                }
                // columns c0 .. c0+31 of D1: rank groups of 8 within tiles i
#pragma unroll
                for (int q8 = 0; q8 < 4; ++q8) {
                    const int col = c0 + q8 * 8;
                    if (col >= a.n1w) break;            // n1w is a multiple of 16, not always of 32
                    const int i = col / a.rbp, k = col - (col / a.rbp) * a.rbp;
                    uint32_t hi[4], lw[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const float w0 = __uint_as_float(v[q8 * 8 + 2 * q]), w1 = __uint_as_float(v[q8 * 8 + 2 * q + 1]);
                        const __half h0 = __float2half_rn(w0), h1 = __float2half_rn(w1);
                        hi[q] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
                        lw[q] = pack2(w0 - __half2float(h0), w1 - __half2float(h1));
                    }
                    const uint32_t off = (uint32_t)i * a.tile2_bytes + canon_off((uint32_t)r, (uint32_t)k, BM);
                    *reinterpret_cast<uint4*>(a2 + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                    if (!a.out16)
                        *reinterpret_cast<uint4*>(a2 + (size_t)a.nb * a.tile2_bytes + off) =
                            make_uint4(lw[0], lw[1], lw[2], lw[3]);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(B.cv_done);
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int g = warp & 3;
        const uint32_t lane_base = (uint32_t)(g * 32) << 16;
        unsigned char* wstage = smem + a.off_stage + (size_t)g * (2 * 32 * 128);
        const int ecols = a.out16 ? 64 : 32;
        const int w2 = a.nb * a.nc;
        int chunk = 0;
        const int r = g * 32 + lane;
        for (int64_t j = 0; j < nunits; ++j) {
            if (!group_wait(B.d2_full, (uint32_t)(j & 1), abort, err, 8u, 1, 128)) break;
            tc_fence_after();
            float fo = 1.0f;
            if (!a.out16) {
                const int eb = (int)(j & 1);
                if (!group_wait(&B.t_full[eb], (uint32_t)((j >> 1) & 1), abort, err, 8u, 1, 128)) break;
                fo = pow2f(-tx[eb * BM + r]);
                mbar_arrive(&B.t_empty[eb]);
            }
            const int64_t row0 = (ubeg + j) * BM + g * 32;
            for (int cc = 0; cc < w2; cc += ecols, ++chunk) {
                uint32_t v[64];
                tmem_ld32(d2col + lane_base + (uint32_t)cc, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
                if (a.out16) tmem_ld32(d2col + lane_base + (uint32_t)cc + 32, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
                tmem_ld_wait();
                uint32_t packed[32];
                if (a.out16) {
#pragma unroll
                    for (int q = 0; q < 32; ++q)
                        packed[q] = pack_half2(__uint_as_float(v[2 * q]), __uint_as_float(v[2 * q + 1]));
                } else {
#pragma unroll
                    for (int q = 0; q < 32; ++q) packed[q] = __float_as_uint(__uint_as_float(v[q]) * fo);
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
                    if (row0 < a.np) tma_store_2d(&tm_out, cc, (int32_t)row0, sb);
                    bulk_commit();      // one group per chunk, even empty: the staging reuse counts on it
                }
            }
            tc_fence_before();
            mbar_arrive(B.d2_free);
        }
        if (lane == 0) bulk_wait<0>();
    }
    // single-lane roles rejoin their warps first: the CTA barrier is an aligned one
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 8) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode_n = nullptr;
std::once_flag g_encode_n_once;

bool ttn_plan(const TTShape& sh, bool out16, TNArgs* out_args, size_t* smem_out, int64_t* grid_out) {
    TNArgs a{};
    const int d = sh.d;
    if (d < 3 || d > kMaxD) return false;
    a.d = d;
    for (int l = 0; l < d; ++l) {
        a.dims[l] = sh.dims[l];
        a.ranks[l] = (int)sh.ranks[l];
        a.cores[l] = static_cast<const __half*>(sh.cores[l]);
    }
    a.ranks[d] = 1;
    a.np = 1;
    for (int l = 0; l <= d - 3; ++l) a.np *= sh.dims[l];
    for (int l = 0; l <= d - 3; ++l) {
        int64_t v = 1;
        for (int j = l + 1; j <= d - 3; ++j) v *= sh.dims[j];
        a.div[l] = v;
    }
    a.ra = (int)sh.ranks[d - 2];
    a.rap = (a.ra + 15) / 16 * 16;
    a.nb = (int)sh.dims[d - 2];
    a.rb = (int)sh.ranks[d - 1];
    a.rbp = (a.rb + 15) / 16 * 16;
    a.nc = (int)sh.dims[d - 1];
    a.n1w = a.nb * a.rbp;
    a.out16 = out16 ? 1 : 0;
    const int eo = out16 ? 2 : 4;
    // the kernel's shape: stage-1 and stage-2 widths within one MMA / 256 TMEM columns
    if (a.rap > 64 || a.n1w > 256 || a.n1w % 16 != 0 || a.nc % 16 != 0 || a.nb * a.nc > 256) return false;
    if ((int64_t)a.nb * a.nc * eo % 128 != 0) return false;     // whole 128-byte staging rows
    // the chain levels keep parent rows of at most 64 ranks in shared memory
    for (int l = 0; l <= d - 2; ++l)
        if (sh.ranks[l] > 64) return false;
    const int planes = out16 ? 1 : 2;
    a.a1_bytes = (uint32_t)BM * a.rap * 2;
    a.tile2_bytes = (uint32_t)BM * a.rbp * 2;
    uint32_t off = 0;
    a.off_a1 = off;
    off += 2u * planes * a.a1_bytes;
    a.off_b1 = off;
    off += (uint32_t)a.n1w * a.rap * 2;
    off = (off + 1023) / 1024 * 1024;
    a.off_a2 = off;
    off += (uint32_t)planes * a.nb * a.tile2_bytes;
    a.off_b2 = off;
    off += (uint32_t)a.nc * a.rbp * 2;
    off = (off + 15) / 16 * 16;
    a.off_exp = off;
    off += 4 * BM * 4;                 // two exponent rings of 2 x 128
    off = (off + 1023) / 1024 * 1024;
    a.off_stage = off;
    off += 4 * 2 * 32 * 128;
    a.off_bar = off;
    off += 19 * 8 + 16;
    const size_t smem = (size_t)off + 1024;
    if (smem > 227 * 1024) return false;
    a.units = (a.np + BM - 1) / BM;
    const int sms = sm_count();
    *out_args = a;
    *smem_out = smem;
    *grid_out = a.units < sms ? a.units : sms;
    return true;
}

}  // namespace

lrc_status launch_ttn_f16_tc(const TTShape& sh, bool out16, void* out, cudaStream_t s, bool* handled) {
    TNArgs a;
    size_t smem = 0;
    int64_t grid = 0;
    *handled = false;
    if (!ttn_plan(sh, out16, &a, &smem, &grid)) return LRC_OK;
    *handled = true;
    std::call_once(g_encode_n_once, [] {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode_n = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    });
    if (!g_encode_n) {
        set_error("cuTensorMapEncodeTiled is not available from the driver");
        return LRC_ERR_CUDA;
    }
    const int eo = out16 ? 2 : 4;
    CUtensorMap tm;
    const int64_t w = (int64_t)a.nb * a.nc;
    cuuint64_t dims[2] = {(cuuint64_t)w, (cuuint64_t)a.np};
    cuuint64_t strides[1] = {(cuuint64_t)w * eo};
    cuuint32_t box[2] = {(cuuint32_t)(128 / eo), 32};
    cuuint32_t estr[2] = {1, 1};
    CUresult cr = g_encode_n(&tm, out16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, out,
                             dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (cr != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled failed for the TT output (CUresult %d)", (int)cr);
        return LRC_ERR_CUDA;
    }
    // workspace: B images, two FP32 chain buffers, the Z_{d-2} images and
    // their row exponents
    const int d = sh.d;
    const int planes = out16 ? 1 : 2;
    auto r256 = [](size_t v) { return (v + 255) / 256 * 256; };
    a.b1_bytes = (uint32_t)a.n1w * a.rap * 2;
    a.b2_bytes = (uint32_t)a.nc * a.rbp * 2;
    size_t chain_bytes = 0;
    {
        int64_t rows = sh.dims[0];
        for (int l = 1; l < d - 3; ++l) {
            rows *= sh.dims[l];
            const size_t b = (size_t)rows * sh.ranks[l + 1] * 4;
            chain_bytes = b > chain_bytes ? b : chain_bytes;
        }
    }
    if (a.units > 0x7fffffff) {
        set_error("TT too large for the narrow-mode kernel");
        return LRC_ERR_UNSUPPORTED;
    }
    const size_t img_bytes = (size_t)a.units * planes * a.a1_bytes;
    const size_t off_b2 = r256(a.b1_bytes), off_c0 = off_b2 + r256(a.b2_bytes);
    const size_t off_c1 = off_c0 + r256(chain_bytes), off_img = off_c1 + r256(chain_bytes);
    const size_t off_exp = off_img + r256(img_bytes);
    void* ws = nullptr;
    lrc_status st = stream_workspace(s, off_exp + (size_t)a.units * BM * sizeof(int), &ws);
    if (st != LRC_OK) return st;
    unsigned char* wb = static_cast<unsigned char*>(ws);
    a.b1img = wb;
    a.b2img = wb + off_b2;
    a.img = wb + off_img;
    a.exps = reinterpret_cast<int*>(wb + off_exp);

    const int nb_el = a.n1w * a.rap + a.nc * a.rbp;
    ttn_bimg_kernel<<<(unsigned)((nb_el + 255) / 256), 256, 0, s>>>(a, wb, wb + off_b2);
    if ((st = after_launch("ttn_bimg_kernel")) != LRC_OK) return st;
    // the chain kernel: cores in shared memory, one CTA per SM
    cudaError_t e;
    {
        ChArgs c{};
        const int last = d - 3;
        uint32_t coff = 0;
        for (int l = 0; l <= last; ++l) {
            c.core_off[l] = coff;
            c.core_bytes[l] = (uint32_t)(sh.ranks[l] * sh.dims[l] * sh.ranks[l + 1] * 2);
            coff += (c.core_bytes[l] + 15) / 16 * 16;
        }
        c.cores_total = coff;
        // level buffers: the ancestors of one tile at levels 0 .. last-1
        int lvrows = 1, lvw = 1;
        for (int l = 0; l < last; ++l) {
            const int64_t rows = (BM - 1) / a.div[l] + 2;
            lvrows = rows > lvrows ? (int)rows : lvrows;
            lvw = sh.ranks[l + 1] > lvw ? (int)sh.ranks[l + 1] : lvw;
        }
        c.lvrows = lvrows;
        c.lvw = lvw;
        uint32_t off = (coff + 15) / 16 * 16;
        c.off_lv = off;
        off += (uint32_t)(2 * lvrows * lvw * 4);
        off = (off + 15) / 16 * 16;
        c.off_stg = off;
        off += (uint32_t)BM * (a.rap + 4) * 4;
        c.off_rmx = off;
        off = (off + 7) / 8 * 8;
        c.off_bar = off;
        off += 16;
        if (off > 227 * 1024) {
            set_error("TT cores too large for the narrow-mode chain kernel");
            return LRC_ERR_UNSUPPORTED;
        }
        // every core must start 16-byte aligned for the bulk copies
        for (int l = 0; l <= last; ++l)
            if (reinterpret_cast<uintptr_t>(sh.cores[l]) & 15u) {
                set_error("TT core %d is not 16-byte aligned", l);
                return LRC_ERR_ALIGNMENT;
            }
        e = cudaFuncSetAttribute(ttn_chain_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)off);
        if (e != cudaSuccess) return cuda_fail(e, "ttn_chain_kernel smem attribute");
        const int sms = sm_count();
        const int per_sm = (2 * ((size_t)off + 1024) <= 228 * 1024) ? 2 : 1;   // latency hiding
        const int64_t cgrid = a.units < (int64_t)sms * per_sm ? a.units : (int64_t)sms * per_sm;
        e = launch_pdl(ttn_chain_kernel, dim3((unsigned)cgrid), dim3(kChThreads), (size_t)off, s, a, c, wb + off_img,
                       reinterpret_cast<int*>(wb + off_exp));
        if (e != cudaSuccess) return cuda_fail(e, "ttn_chain_kernel launch");
        if ((st = after_launch("ttn_chain_kernel")) != LRC_OK) return st;
    }
    e = cudaFuncSetAttribute(ttn_f16_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "ttn_f16_tc_kernel smem attribute");
    e = launch_pdl(ttn_f16_tc_kernel, dim3((unsigned)grid), dim3(kThreads), smem, s, tm, a);
    if (e != cudaSuccess) return cuda_fail(e, "ttn_f16_tc_kernel launch");
    return after_launch("ttn_f16_tc_kernel");
}

uint32_t take_ttn_tc_error() {
    unsigned int v = 0;
    if (cudaMemcpyFromSymbol(&v, g_err_ttn_tc, sizeof v) != cudaSuccess) return 0xffffffffu;
    if (v) {
        const unsigned int z = 0;
        cudaMemcpyToSymbol(g_err_ttn_tc, &z, sizeof z);
    }
    return v;
}

}  // namespace lrc
