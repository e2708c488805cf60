// tt_split.cu -- binary16 TT reconstruction (Sec. 5.1; Sec. 7.5,
// Eq. gpu_tt_reconstruction) as the product chain of tt_chain.cu with the
// output product on the tensor cores.
//
// The chain meets at bond c (the bond with the fewest multiplies):
// Z = G_1...G_c is a P x r matrix and S = G_{c+1}...G_d an r x Q matrix
// (P = n_1...n_c, Q = n_{c+1}...n_d, r = r_c), and the C-order tensor is the
// P x Q product Z S.  One launch (tt_side_kernel) forms Z and S: each CTA
// walks the chain for 32 rows of Z or 32 columns of S in shared memory (binary16 cores widened exactly, binary32 arithmetic) and
// writes them into the tensor-core operand images; a second launch, the
// binary16 tensor-core product of apply_tc.cu, forms Z S with Z as its
// 128-row W tiles and S^T as its U rows -- nearly all of the work and all of
// the output traffic.
//
// Operands of that product are binary16 with binary32 accumulation (Sec. 3.4).
// An operand that is a stored binary16 core is exact in binary16; binary32
// cores (the LRC_F32_TC variant) take the hi/lo split below on both sides.  An operand the
// chain computed is binary32; for a binary32 output it enters the product as
// a pair hi = fp16(x), lo = fp16(x - hi) laid side by side along the
// reduction, so one product of concatenated operands forms
//     Z S ~ Z_hi S_hi + Z_lo S_hi + Z_hi S_lo
// (about 22 significand bits per operand); for a binary16 output it is
// rounded once (the method-precision workspace of Sec. 3.4).  Every tile of
// a computed operand is scaled, in groups of 32 rows of Z or 32 columns of
// S, by a power of two that brings the group's largest magnitude into
// [2^14, 2^15) before rounding, so lo stays a normal binary16 number; the
// product's epilogue multiplies each output entry by the inverse scales
// (exact).
// bfloat16 cores (LRC_BF16) take the same chain with bfloat16 operand images
// rounded once (the format's method-precision workspace) and a bfloat16
// tensor-core product.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <type_traits>

#include "common.cuh"
#include "tc.cuh"

namespace lrc {
namespace {

constexpr int BM = 128;
constexpr int kMaxParts = 3;
constexpr int kUnit = 32;      // rows of Z or columns of S per CTA of the side kernel (one scale group)

// Part kinds of an operand laid along the reduction: bit p of `lomask` set =
// part p is the lo half, otherwise the hi half (or the single rounding).
struct Parts {
    int n;
    int lomask;
};

// e with max * 2^e in [2^14, 2^15), clamped to [-60, 60] (so that the
// product's epilogue factor 2^-(e_w + e_u) stays a normal binary32 number);
// 0 when the tile is zero or not finite
__device__ __forceinline__ int scale_exp(float maxabs) {
    if (!(maxabs > 0.0f) || !(maxabs <= 3.0e38f)) return 0;
    const int ex = ((__float_as_int(maxabs) >> 23) & 0xff) - 127;   // floor(log2 max) for normal numbers
    const int e = 14 - ex;
    return e < -60 ? -60 : (e > 60 ? 60 : e);
}

// 2^e for |e| <= 126
__device__ __forceinline__ float pow2(int e) { return __int_as_float((127 + e) << 23); }

__device__ __forceinline__ __half part_value(float y, bool lo) {
    const __half hi = __float2half_rn(y);
    return lo ? __float2half_rn(y - __half2float(hi)) : hi;
}

// Encoding of one operand-image element: binary16 parts, or one bfloat16
// rounding (the bfloat16 chain has a single part).
template <bool BF>
__device__ __forceinline__ uint16_t image_bits(float y, bool lo) {
    if constexpr (BF) return tc::to_bf16_bits(y);
    else return __half_as_ushort(part_value(y, lo));
}

__device__ __forceinline__ float block_max(float v, float* sh) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) sh[warp] = v;
    __syncthreads();
    float m = 0.0f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) m = fmaxf(m, sh[w]);
    return m;
}

struct SideArgs {
    int d, c;                 // cores 0..c-1 form Z, cores c..d-1 form S (0-based)
    int r, rp, ldb;           // r = r_c; rp = r rounded up to 16; ldb: row pitch of the buffers
    int buf_rows;             // rows of each buffer
    int64_t P, Q, wunits;     // wunits: CTAs forming Z (kUnit rows each)
    int64_t dims[16];
    int ranks[17];
    int64_t D[16];            // D[l] = n_{l+1} ... n_{c-1}: prefix p passes through row p / D[l] of Z_{l+1}
    int64_t Qs[17];           // Qs[l] = n_l ... n_{d-1}: suffix counts of the right side
    const void* cores[16];    // binary16 (image mode) or binary32 cores
    Parts pw, pu;
    int scale_w, scale_u;
    unsigned char* Wimg;      // ceil(P / 128) images of 128 x kp
    uint16_t* Uimg;           // Q rows of kp
    float* Zout;              // binary32 mode: Z (P x r) and S (r x Q), row-major
    float* Sout;
    int* esc_w;               // [ceil(P / kUnit)]
    int* esc_u;               // [ceil(Q / kUnit)]
};

__device__ __forceinline__ float core_at(const __half* g, int64_t i) { return __half2float(__ldg(g + i)); }
__device__ __forceinline__ float core_at(const __nv_bfloat16* g, int64_t i) {
    return tc::bf16_bits_to_float(__ldg(reinterpret_cast<const unsigned short*>(g) + i));
}
__device__ __forceinline__ float core_at(const float* g, int64_t i) { return __ldg(g + i); }

// Copies count core elements to shared memory, dst[didx(e)] = G[sidx(e)],
// eight loads in flight per thread before their stores (a loop that stores to
// shared memory between global loads would wait out each load in turn).
template <typename TC, typename SI, typename DI>
__device__ __forceinline__ void copy_core(const TC* __restrict__ g, int64_t count, SI sidx, DI didx, float* dst) {
    for (int64_t e0 = 0; e0 < count; e0 += 8 * (int64_t)blockDim.x) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int64_t e = e0 + u * (int64_t)blockDim.x + threadIdx.x;
            v[u] = e < count ? core_at(g, sidx(e)) : 0.0f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int64_t e = e0 + u * (int64_t)blockDim.x + threadIdx.x;
            if (e < count) dst[didx(e)] = v[u];
        }
    }
}

// Core l widened to binary32 in shared memory (every interior core of a
// shape this path takes fits; gs is 16-byte aligned); the barriers retire
// the previous level and publish the core.
template <typename TC>
__device__ __forceinline__ const float* stage_core(const SideArgs& a, int l, float* gs) {
    constexpr int EV = 16 / (int)sizeof(TC);
    const int64_t n = (int64_t)a.ranks[l] * a.dims[l] * a.ranks[l + 1];
    const TC* g = static_cast<const TC*>(a.cores[l]);
    __syncthreads();
    const int64_t nv = ((reinterpret_cast<uintptr_t>(g) & 15u) == 0) ? n / EV : 0;   // 16-byte vectors
    for (int64_t v0 = 0; v0 < nv; v0 += 4 * (int64_t)blockDim.x) {
        uint4 w[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t i = v0 + u * (int64_t)blockDim.x + threadIdx.x;
            if (i < nv) w[u] = __ldg(reinterpret_cast<const uint4*>(g) + i);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t i = v0 + u * (int64_t)blockDim.x + threadIdx.x;
            if (i < nv) {
                if constexpr (std::is_same_v<TC, __nv_bfloat16>) {
                    const uint32_t q[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
                    float f[8];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        f[2 * j] = __uint_as_float(q[j] << 16);
                        f[2 * j + 1] = __uint_as_float(q[j] & 0xffff0000u);
                    }
                    reinterpret_cast<float4*>(gs + i * 8)[0] = make_float4(f[0], f[1], f[2], f[3]);
                    reinterpret_cast<float4*>(gs + i * 8)[1] = make_float4(f[4], f[5], f[6], f[7]);
                } else if constexpr (sizeof(TC) == 2) {
                    const __half2* h = reinterpret_cast<const __half2*>(&w[u]);
                    const float2 f0 = __half22float2(h[0]), f1 = __half22float2(h[1]);
                    const float2 f2 = __half22float2(h[2]), f3 = __half22float2(h[3]);
                    reinterpret_cast<float4*>(gs + i * 8)[0] = make_float4(f0.x, f0.y, f1.x, f1.y);
                    reinterpret_cast<float4*>(gs + i * 8)[1] = make_float4(f2.x, f2.y, f3.x, f3.y);
                } else {
                    reinterpret_cast<uint4*>(gs + i * 4)[0] = w[u];
                }
            }
        }
    }
    const int64_t done = nv * EV;
    copy_core(g, n - done, [=](int64_t e) { return done + e; }, [=](int64_t e) { return done + e; }, gs);
    __syncthreads();
    return gs;
}

// Rows [p0, pend) of Z = G_1...G_c (binary32, buffer rows of pitch ldb);
// returns the buffer that holds them.  Level l keeps only the rows of
// Z_{l+1} the tile's prefixes pass through: a contiguous range.
template <typename TC>
__device__ float* left_rows(const SideArgs& a, int64_t p0, int64_t pend, float* buf0, float* buf1, float* gs) {
    float* cur = buf0;
    int64_t lo = p0 / a.D[0];
    {
        const int r1 = a.ranks[1], ldb = a.ldb;
        const int cnt = (int)((pend - 1) / a.D[0] - lo + 1);
        copy_core(static_cast<const TC*>(a.cores[0]), (int64_t)cnt * r1, [=](int64_t e) { return lo * r1 + e; },
                  [=](int64_t e) { return (e / r1) * ldb + e % r1; }, cur);
    }
    __syncthreads();
    for (int l = 1; l < a.c; ++l) {
        const int r0 = a.ranks[l], r1 = a.ranks[l + 1];
        const int64_t nl = a.dims[l];
        const int64_t nlo = p0 / a.D[l];
        const int cnt = (int)((pend - 1) / a.D[l] - nlo + 1);
        float* nxt = (cur == buf0) ? buf1 : buf0;
        const float* G = stage_core<TC>(a, l, gs);
        for (int e = threadIdx.x; e < cnt * r1; e += blockDim.x) {
            const int q = e / r1, b = e - q * r1;
            const int64_t gq = nlo + q, parent = gq / nl;
            const int i = (int)(gq - parent * nl);
            const float* zrow = cur + (parent - lo) * a.ldb;
            const float* gcol = G + (int64_t)i * r1 + b;
            const int kstride = (int)nl * r1;
            float acc = 0.0f;
            for (int k = 0; k < r0; ++k) acc = fmaf(zrow[k], gcol[k * kstride], acc);
            nxt[q * a.ldb + b] = acc;
        }
        __syncthreads();
        cur = nxt;
        lo = nlo;
    }
    return cur;
}

// Columns of S = G_{c+1}...G_d for t in [q0, qend) (binary32, one buffer row
// of pitch ldb per column); returns the buffer, *direct = whether column t
// sits in row t (the whole of S fits one unit) or in row t - q0.  A level
// whose suffix count Qs[l] is at most kUnit computes every suffix (row =
// suffix); otherwise it computes the suffixes t mod Qs[l] of the unit's
// columns (row = t - q0).
template <typename TC>
__device__ float* right_cols(const SideArgs& a, int64_t q0, int64_t qend, float* buf0, float* buf1, float* gs,
                            bool* direct) {
    float* cur = buf0;
    const int last = a.d - 1;
    {
        const int rl = a.ranks[last];
        const int64_t nl = a.dims[last];
        const bool all = a.Qs[last] <= kUnit;
        const int cnt = all ? (int)nl : (int)(qend - q0);
        const int ldb = a.ldb;
        copy_core(static_cast<const TC*>(a.cores[last]), (int64_t)cnt * rl,
                  [=](int64_t e) {
                      const int64_t k = e / cnt, col = e - k * cnt;
                      return k * nl + (all ? col : (q0 + col) % nl);
                  },
                  [=](int64_t e) { return (e % cnt) * ldb + e / cnt; }, cur);
    }
    __syncthreads();
    for (int l = last - 1; l >= a.c; --l) {
        const int r0 = a.ranks[l], r1 = a.ranks[l + 1];
        const int64_t nl = a.dims[l], qn = a.Qs[l + 1];
        const bool all = a.Qs[l] <= kUnit, all_next = qn <= kUnit;
        const int cnt = all ? (int)a.Qs[l] : (int)(qend - q0);
        float* nxt = (cur == buf0) ? buf1 : buf0;
        const float* G = stage_core<TC>(a, l, gs);
        // columns fastest across threads: a warp reads one core row (broadcast)
        // and rows of the column buffer an odd pitch apart (no bank conflicts)
        for (int e = threadIdx.x; e < cnt * r0; e += blockDim.x) {
            const int k = e / cnt, col = e - k * cnt;
            const int64_t sfx = all ? col : (q0 + col) % a.Qs[l];
            const int64_t i = sfx / qn, sn = sfx - i * qn;
            const float* scol = cur + (all_next ? sn : col) * a.ldb;
            const float* grow = G + ((int64_t)k * nl + i) * r1;
            float acc = 0.0f;
            for (int b = 0; b < r1; ++b) acc = fmaf(grow[b], scol[b], acc);
            nxt[col * a.ldb + k] = acc;
        }
        __syncthreads();
        cur = nxt;
    }
    *direct = a.Qs[a.c] <= kUnit;
    return cur;
}

// One CTA per kUnit rows of Z (blockIdx < wunits) or kUnit columns of S:
// forms them and, in image mode (IMG), scales them by one power of two
// (computed operands) and writes their binary16 parts into the operand
// images; otherwise writes them as binary32 Z and S.
template <typename TC, bool IMG>
__global__ void __launch_bounds__(256)
tt_side_kernel(const SideArgs a) {
    constexpr bool BF = std::is_same_v<TC, __nv_bfloat16>;
    extern __shared__ float sbuf[];
    __shared__ float red[8];
    tc::pdl_wait();
    const bool wside = blockIdx.x < a.wunits;
    float* buf0 = sbuf;
    float* buf1 = sbuf + (size_t)a.buf_rows * a.ldb;
    float* gs = sbuf + ((size_t)2 * a.buf_rows * a.ldb + 3) / 4 * 4;     // staged core, 16-byte aligned
    const int kp = (wside ? a.pw.n : a.pu.n) * a.rp;
    if (wside) {
        const int64_t t = blockIdx.x;
        const int64_t p0 = t * kUnit, pend = (p0 + kUnit < a.P) ? p0 + kUnit : a.P;
        const int nrow = (int)(pend - p0);
        const float* z = left_rows<TC>(a, p0, pend, buf0, buf1, gs);
        if constexpr (!IMG) {
            tc::pdl_trigger();
            for (int e = threadIdx.x; e < nrow * a.r; e += blockDim.x)
                a.Zout[p0 * a.r + e] = z[(e / a.r) * a.ldb + e % a.r];
            return;
        }
        float mx = 0.0f;
        for (int e = threadIdx.x; e < nrow * a.r; e += blockDim.x)
            mx = fmaxf(mx, fabsf(z[(e / a.r) * a.ldb + e % a.r]));
        const float tmax = block_max(mx, red);
        const int ex = a.scale_w ? scale_exp(tmax) : 0;
        const float f = pow2(ex);
        tc::pdl_trigger();
        if (threadIdx.x == 0) a.esc_w[t] = ex;
        unsigned char* tile = a.Wimg + (size_t)(p0 / BM) * BM * kp * 2;
        const int ro = (int)(p0 % BM);
        // one thread per (row, 8-column group), rows fastest: a warp writes 512 contiguous bytes
        for (int i = threadIdx.x; i < kUnit * (kp / 8); i += blockDim.x) {
            const int row = i % kUnit, c0 = (i / kUnit) * 8;
            const int p = c0 / a.rp, a0 = c0 - p * a.rp;
            const bool lo = (a.pw.lomask >> p) & 1;
            __align__(16) uint16_t h[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int k = a0 + j;
                h[j] = (k < a.r && row < nrow) ? image_bits<BF>(z[row * a.ldb + k] * f, lo) : (uint16_t)0;
            }
            *reinterpret_cast<uint4*>(tile + tc::w_image_off((uint32_t)(ro + row), (uint32_t)c0)) =
                *reinterpret_cast<const uint4*>(h);
        }
    } else {
        const int64_t t = blockIdx.x - a.wunits;
        const int64_t q0 = t * kUnit, qend = (q0 + kUnit < a.Q) ? q0 + kUnit : a.Q;
        const int nq = (int)(qend - q0);
        bool direct = false;
        const float* sc = right_cols<TC>(a, q0, qend, buf0, buf1, gs, &direct);
        const int64_t base = direct ? q0 : 0;      // buffer row of column q0
        if constexpr (!IMG) {
            tc::pdl_trigger();
            // S[k][q0 + q], columns fastest: 128-byte runs per row of S
            for (int e = threadIdx.x; e < nq * a.r; e += blockDim.x) {
                const int k = e / nq, q = e - k * nq;
                a.Sout[(int64_t)k * a.Q + q0 + q] = sc[(base + q) * a.ldb + k];
            }
            return;
        }
        float mx = 0.0f;
        for (int e = threadIdx.x; e < nq * a.r; e += blockDim.x)
            mx = fmaxf(mx, fabsf(sc[(base + e / a.r) * a.ldb + e % a.r]));
        const float tmax = block_max(mx, red);
        const int ex = a.scale_u ? scale_exp(tmax) : 0;
        const float f = pow2(ex);
        tc::pdl_trigger();
        if (threadIdx.x == 0) a.esc_u[t] = ex;
        const int groups = kp / 8;
        // one thread per (row of U, 8-column group), groups fastest: a warp writes contiguous rows
        for (int i = threadIdx.x; i < nq * groups; i += blockDim.x) {
            const int q = i / groups, c0 = (i - q * groups) * 8;
            const int p = c0 / a.rp, a0 = c0 - p * a.rp;
            const bool lo = (a.pu.lomask >> p) & 1;
            const float* col = sc + (base + q) * a.ldb;
            __align__(16) uint16_t h[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int k = a0 + j;
                h[j] = (k < a.r) ? image_bits<BF>(col[k] * f, lo) : (uint16_t)0;
            }
            *reinterpret_cast<uint4*>(a.Uimg + (q0 + q) * kp + c0) = *reinterpret_cast<const uint4*>(h);
        }
    }
}

size_t r256(size_t v) { return (v + 255) / 256 * 256; }

// SideArgs fields common to both modes; returns the largest rank.
int fill_side(const TTShape& sh, int c, SideArgs& a) {
    const int d = sh.d;
    a.d = d;
    a.c = c;
    a.r = (int)sh.ranks[c];
    a.rp = (a.r + 15) / 16 * 16;
    int rmax = 1;
    for (int l = 0; l < d; ++l) {
        a.dims[l] = sh.dims[l];
        a.ranks[l] = (int)sh.ranks[l];
        a.cores[l] = sh.cores[l];
        if (sh.ranks[l] > rmax) rmax = (int)sh.ranks[l];
    }
    a.ranks[d] = 1;
    a.P = 1;
    for (int l = 0; l < c; ++l) a.P *= sh.dims[l];
    a.Q = 1;
    for (int l = c; l < d; ++l) a.Q *= sh.dims[l];
    for (int l = 0; l < c; ++l) {
        int64_t v = 1;
        for (int j = l + 1; j < c; ++j) v *= sh.dims[j];
        a.D[l] = v;
    }
    a.Qs[d] = 1;
    for (int l = d - 1; l >= 0; --l) a.Qs[l] = a.Qs[l + 1] * sh.dims[l];
    a.ldb = rmax | 1;
    a.buf_rows = kUnit + 1;
    a.wunits = (a.P + kUnit - 1) / kUnit;
    return rmax;
}

// Shared memory of the side kernel: two level buffers and the largest
// interior core (staged in binary32).
size_t side_smem(const TTShape& sh, const SideArgs& a) {
    int64_t core_max = 0;
    for (int l = 1; l <= sh.d - 2; ++l) {
        const int64_t n = sh.ranks[l] * sh.dims[l] * sh.ranks[l + 1];
        if (n > core_max) core_max = n;
    }
    return (((size_t)2 * a.buf_rows * a.ldb + 3) / 4 * 4 + (size_t)core_max) * sizeof(float);
}

}  // namespace

namespace {

// The split product chain for binary16 cores (TC = __half, stored cores exact
// in binary16) or binary32 cores (TC = float: every operand split and scaled).
template <typename TC>
lrc_status launch_split_t(const TTShape& sh, bool out16, void* out, cudaStream_t s, bool* handled) {
    constexpr bool kExactCores = sizeof(TC) == 2;
    constexpr bool kBF = std::is_same_v<TC, __nv_bfloat16>;
    *handled = false;
    const int d = sh.d;
    if (d > 16) return LRC_OK;
    const int c = tt_chain_bond(sh);
    const int r = (int)sh.ranks[c];
    const int rp = (r + 15) / 16 * 16;
    const bool z_core = kExactCores && (c == 1), s_core = kExactCores && (c == d - 1);   // operands exact in binary16
    // parts along the reduction (see the file comment)
    Parts pw{1, 0}, pu{1, 0};
    if (!out16) {
        if (!z_core && !s_core) {
            pw = Parts{3, 0b010};   // [Z_hi | Z_lo | Z_hi]
            pu = Parts{3, 0b100};   // [S_hi | S_hi | S_lo]
        } else if (!z_core) {
            pw = Parts{2, 0b10};    // [Z_hi | Z_lo]
            pu = Parts{2, 0b00};    // [S | S]
        } else if (!s_core) {
            pw = Parts{2, 0b00};    // [Z | Z]
            pu = Parts{2, 0b10};    // [S_hi | S_lo]
        }
    }
    const int kp = pw.n * rp;
    SideArgs a{};
    const int rmax = fill_side(sh, c, a);
    int n2 = 0;
    if (kp > kMaxParts * 64 || rmax > 64 || y_product_plan(a.Q, a.P, kp, out16, &n2) != LRC_OK) return LRC_OK;
    const size_t smem = side_smem(sh, a);
    if (smem > 200 * 1024) return LRC_OK;
    *handled = true;
    a.pw = pw;
    a.pu = pu;
    a.scale_w = z_core ? 0 : 1;
    a.scale_u = s_core ? 0 : 1;
    const int64_t uunits = (a.Q + kUnit - 1) / kUnit;
    const int64_t btiles = (a.P + BM - 1) / BM;
    const size_t w_bytes = r256((size_t)btiles * BM * kp * 2), u_bytes = r256((size_t)a.Q * kp * 2);
    const size_t e_bytes = r256((size_t)(a.wunits + uunits) * sizeof(int));
    void* wsp = nullptr;
    lrc_status st = stream_workspace(s, w_bytes + u_bytes + e_bytes, &wsp);
    if (st != LRC_OK) return st;
    unsigned char* ws = static_cast<unsigned char*>(wsp);
    a.Wimg = ws;
    a.Uimg = reinterpret_cast<uint16_t*>(ws + w_bytes);
    a.esc_w = reinterpret_cast<int*>(ws + w_bytes + u_bytes);
    a.esc_u = a.esc_w + a.wunits;
    cudaError_t e = cudaFuncSetAttribute(tt_side_kernel<TC, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "tt_side_kernel smem attribute");
    e = launch_pdl(tt_side_kernel<TC, true>, dim3((unsigned)(a.wunits + uunits)), dim3(256), smem, s, a);
    if (e != cudaSuccess) return cuda_fail(e, "tt_side_kernel launch");
    if ((st = after_launch("tt_side_kernel")) != LRC_OK) return st;
    return launch_y_product(a.Wimg, kp, a.Uimg, kp, a.Q, a.P, out16, out, a.esc_w, a.esc_u, s, false, kBF);
}

}  // namespace

lrc_status launch_tt_split_f16(const TTShape& sh, bool out16, void* out, cudaStream_t s, bool* handled) {
    return launch_split_t<__half>(sh, out16, out, s, handled);
}

lrc_status launch_tt_split_f32tc(const TTShape& sh, float* out, cudaStream_t s, bool* handled) {
    return launch_split_t<float>(sh, false, out, s, handled);
}

lrc_status launch_tt_bf16(const TTShape& sh, void* out, cudaStream_t s) {
    bool handled = false;
    lrc_status st = launch_split_t<__nv_bfloat16>(sh, true, out, s, &handled);
    if (handled) return st;
    return launch_tt_cc(sh, LRC_BF16, out, s);
}

lrc_status launch_tt_side_f32(const TTShape& sh, float* out, cudaStream_t s, bool* handled) {
    *handled = false;
    const int d = sh.d;
    if (d > 16) return LRC_OK;
    const int c = tt_chain_bond(sh);
    if ((c - 1) + (d - 1 - c) < 2) return LRC_OK;    // at most one chain product per side: nothing to fuse
    SideArgs a{};
    const int rmax = fill_side(sh, c, a);
    int64_t zq;
    if (rmax > 64 || !mul_ok(a.P, a.r, &zq) || zq > ((int64_t)1 << 22) || !mul_ok(a.Q, a.r, &zq) ||
        zq > ((int64_t)1 << 22))
        return LRC_OK;                                 // sides too large for one pass of per-unit chains
    const size_t smem = side_smem(sh, a);
    if (smem > 200 * 1024) return LRC_OK;
    *handled = true;
    const int64_t uunits = (a.Q + kUnit - 1) / kUnit;
    const size_t z_bytes = r256((size_t)a.P * a.r * sizeof(float)), s_bytes = r256((size_t)a.r * a.Q * sizeof(float));
    void* wsp = nullptr;
    lrc_status st = stream_workspace(s, z_bytes + s_bytes, &wsp);
    if (st != LRC_OK) return st;
    a.Zout = static_cast<float*>(wsp);
    a.Sout = reinterpret_cast<float*>(static_cast<unsigned char*>(wsp) + z_bytes);
    cudaError_t e = cudaFuncSetAttribute(tt_side_kernel<float, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "tt_side_kernel smem attribute");
    e = launch_pdl(tt_side_kernel<float, false>, dim3((unsigned)(a.wunits + uunits)), dim3(256), smem, s, a);
    if (e != cudaSuccess) return cuda_fail(e, "tt_side_kernel launch");
    if ((st = after_launch("tt_side_kernel")) != LRC_OK) return st;
    return gemm_cc_f32(a.Zout, a.r, a.Sout, a.Q, false, out, a.Q, a.P, a.Q, a.r, 1, 0, s);
}

}  // namespace lrc
