// tt_cc.cu -- dense TT reconstruction on the CUDA cores, binary64 and binary16 cores
// (Sec. 5.1: T(i_1..i_d) = G_1(i_1)...G_d(i_d); Sec. 7.5,
// Eq. gpu_tt_reconstruction: B_l = Z_{l-1} K_l, Z_l = reshape(B_l)).
//
// The output is T viewed as (prod_{l<d} n_l) prefix rows x n_d columns, C
// order.  A CTA owns a tile of P consecutive prefix rows.  For each level
// l = 1..d-1 it computes only the rows of Z_l that the tile's prefixes pass
// through (a contiguous index range per level, since prefixes are C-order
// consecutive), ping-ponging two shared-memory buffers; the chain's partial
// products therefore never touch global memory.  The last level and the
// final product Z_{d-1} G_d -> out are the only steps whose size scales with
// the tile.  The final product uses a TM x TN register tile per thread and
// writes contiguous output rows.
//
// Element types: binary64 cores with binary64 arithmetic, and binary16 cores
// with binary32 arithmetic and a binary32 or binary16 output (the latter
// rounded once per entry) for the shapes the tensor-core kernels do not take.
// binary32 cores take the product chain of tt_chain.cu.  bfloat16 cores
// (LRC_BF16) take the binary16 form with a bfloat16 output.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "common.cuh"

namespace lrc {
namespace {

constexpr int kThreads = 256;
constexpr int kTM = 4, kTN = 4;

__device__ __forceinline__ float to_acc(__half x) { return __half2float(x); }
__device__ __forceinline__ float to_acc(__nv_bfloat16 x) { return __bfloat162float(x); }
__device__ __forceinline__ float to_acc(float x) { return x; }
__device__ __forceinline__ double to_acc(double x) { return x; }
__device__ __forceinline__ void store_out(float* p, float v) { *p = v; }
__device__ __forceinline__ void store_out(double* p, double v) { *p = v; }
__device__ __forceinline__ void store_out(__half* p, float v) { *p = __float2half_rn(v); }
__device__ __forceinline__ void store_out(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

template <typename TIn>
struct TTParams {
    int d;
    int tile;          // prefix rows per CTA
    int ldz;           // shared row pitch of Z (odd)
    int tx;            // threads along output columns in the final product
    int64_t nprefix;   // prod_{l<d} n_l
    int64_t dims[16];
    int64_t ranks[17];
    int64_t div[16];   // div[l] = prod_{j=l+1}^{d-2} n_j: level-l row of prefix p is p / div[l]
    const TIn* cores[16];
};

// T: arithmetic type; TIn: core element type; TOut: output element type.
template <typename T, typename TIn, typename TOut>
__global__ void __launch_bounds__(kThreads)
tt_cc_kernel(const TTParams<TIn> p, TOut* __restrict__ out) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    T* zbuf[2];
    zbuf[0] = reinterpret_cast<T*>(smem_raw);
    zbuf[1] = zbuf[0] + (size_t)(p.tile + 1) * p.ldz;
    const int tid = threadIdx.x;
    const int d = p.d;

    const int64_t p0 = (int64_t)blockIdx.x * p.tile;
    const int64_t pend = (p0 + p.tile < p.nprefix) ? p0 + p.tile : p.nprefix;
    const int pcount = (int)(pend - p0);

    // level 0 (Z_1 = G_1 rows)
    int cur = 0;
    int64_t lo = p0 / p.div[0];
    int64_t hi = (pend - 1) / p.div[0];
    {
        const int r1 = (int)p.ranks[1];
        const int cnt = (int)(hi - lo + 1);
        const TIn* G = p.cores[0];
        for (int e = tid; e < cnt * r1; e += kThreads) {
            const int q = e / r1, bcol = e % r1;
            zbuf[0][q * p.ldz + bcol] = to_acc(G[(lo + q) * r1 + bcol]);
        }
    }
    __syncthreads();
    // levels 1 .. d-2: Z_{l+1}[q] = Z_l[q / n] G_{l+1}(q % n)
    for (int l = 1; l <= d - 2; ++l) {
        const int r0 = (int)p.ranks[l], r1 = (int)p.ranks[l + 1];
        const int64_t nl = p.dims[l];
        const int64_t nlo = p0 / p.div[l];
        const int64_t nhi = (pend - 1) / p.div[l];
        const int cnt = (int)(nhi - nlo + 1);
        const TIn* G = p.cores[l];
        const T* zin = zbuf[cur];
        T* zout = zbuf[cur ^ 1];
        for (int e = tid; e < cnt * r1; e += kThreads) {
            const int q = e / r1, bcol = e % r1;
            const int64_t gq = nlo + q;
            const int64_t parent = gq / nl;
            const int64_t i = gq - parent * nl;
            const T* zrow = zin + (parent - lo) * p.ldz;
            const TIn* gcol = G + i * r1 + bcol;
            T acc = T(0);
            for (int a = 0; a < r0; ++a) acc = fma(zrow[a], to_acc(gcol[(int64_t)a * nl * r1]), acc);
            zout[q * p.ldz + bcol] = acc;
        }
        __syncthreads();
        cur ^= 1;
        lo = nlo;
        hi = nhi;
    }
    // final product: out[p0 + t, :] = Z_{d-1}[t] G_d   (G_d is r x n_d)
    const int r = (int)p.ranks[d - 1];
    const int64_t nd = p.dims[d - 1];
    const TIn* Gd = p.cores[d - 1];
    const T* z = zbuf[cur];
    const int TX = p.tx, TY = kThreads / TX;
    const int tx = tid % TX, ty = tid / TX;
    for (int rb = 0; rb < pcount; rb += TY * kTM) {
        for (int64_t nc = 0; nc < nd; nc += (int64_t)TX * kTN) {
            T acc[kTM][kTN];
#pragma unroll
            for (int i = 0; i < kTM; ++i)
#pragma unroll
                for (int j = 0; j < kTN; ++j) acc[i][j] = T(0);
            int rows[kTM];
#pragma unroll
            for (int i = 0; i < kTM; ++i) {
                const int t = rb + ty + i * TY;
                rows[i] = t < pcount ? t : pcount - 1;   // clamp reads; store is guarded
            }
            int64_t cols[kTN];
            bool colok[kTN];
#pragma unroll
            for (int j = 0; j < kTN; ++j) {
                cols[j] = nc + tx + (int64_t)j * TX;
                colok[j] = cols[j] < nd;
                if (!colok[j]) cols[j] = nd - 1;
            }
            for (int a = 0; a < r; ++a) {
                T av[kTM], bv[kTN];
#pragma unroll
                for (int i = 0; i < kTM; ++i) av[i] = z[rows[i] * p.ldz + a];
#pragma unroll
                for (int j = 0; j < kTN; ++j) bv[j] = to_acc(__ldg(Gd + (int64_t)a * nd + cols[j]));
#pragma unroll
                for (int i = 0; i < kTM; ++i)
#pragma unroll
                    for (int j = 0; j < kTN; ++j) acc[i][j] = fma(av[i], bv[j], acc[i][j]);
            }
#pragma unroll
            for (int i = 0; i < kTM; ++i) {
                const int t = rb + ty + i * TY;
                if (t >= pcount) continue;
                TOut* orow = out + (p0 + t) * nd;
#pragma unroll
                for (int j = 0; j < kTN; ++j)
                    if (colok[j]) store_out(orow + cols[j], acc[i][j]);
            }
        }
    }
}

template <typename T, typename TIn, typename TOut>
lrc_status launch_tt_cc_t(const TTShape& sh, TOut* out, cudaStream_t s, const char* name) {
    TTParams<TIn> p;
    p.d = sh.d;
    int64_t rmax = 1;
    for (int l = 0; l < sh.d; ++l) {
        p.dims[l] = sh.dims[l];
        p.ranks[l] = sh.ranks[l];
        p.cores[l] = static_cast<const TIn*>(sh.cores[l]);
        if (sh.ranks[l] > rmax) rmax = sh.ranks[l];
    }
    p.ranks[sh.d] = 1;
    p.nprefix = 1;
    for (int l = 0; l < sh.d - 1; ++l) p.nprefix *= sh.dims[l];
    // div[l] = product of dims[l+1 .. d-2]
    for (int l = 0; l < sh.d - 1; ++l) {
        int64_t v = 1;
        for (int j = l + 1; j <= sh.d - 2; ++j) v *= sh.dims[j];
        p.div[l] = v;
    }
    const int64_t nd = sh.dims[sh.d - 1];
    p.tx = nd >= 64 ? 16 : (nd >= 32 ? 8 : (nd >= 16 ? 4 : (nd >= 8 ? 2 : 1)));
    p.ldz = (int)(rmax | 1);
    const int rows_per_pass = (kThreads / p.tx) * kTM;
    int64_t tile = rows_per_pass > 64 ? rows_per_pass : 64;
    const size_t budget = 200 * 1024;
    while (tile > 1 && (size_t)2 * (tile + 1) * p.ldz * sizeof(T) > budget) tile /= 2;
    const size_t smem = (size_t)2 * (tile + 1) * p.ldz * sizeof(T);
    if (smem > budget) {
        set_error("%s: TT rank %lld too large for the on-chip chain", name, (long long)rmax);
        return LRC_ERR_UNSUPPORTED;
    }
    p.tile = (int)tile;
    const int64_t tiles = (p.nprefix + tile - 1) / tile;
    if (tiles > 0x7fffffff) {
        set_error("%s: tensor too large", name);
        return LRC_ERR_UNSUPPORTED;
    }
    cudaError_t e = cudaFuncSetAttribute(tt_cc_kernel<T, TIn, TOut>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, name);
    tt_cc_kernel<T, TIn, TOut><<<(unsigned)tiles, kThreads, smem, s>>>(p, out);
    return after_launch(name);
}

}  // namespace

lrc_status launch_tt_cc(const TTShape& sh, lrc_fmt fmt, void* out, cudaStream_t s) {
    switch (fmt) {
        case LRC_F64:
            return launch_tt_cc_t<double, double, double>(sh, static_cast<double*>(out), s, "tt_cc_kernel<f64>");
        case LRC_F16:
            return launch_tt_cc_t<float, __half, float>(sh, static_cast<float*>(out), s, "tt_cc_kernel<f16,o32>");
        case LRC_BF16:
            return launch_tt_cc_t<float, __nv_bfloat16, __nv_bfloat16>(sh, static_cast<__nv_bfloat16*>(out), s,
                                                                      "tt_cc_kernel<bf16>");
        default:
            return launch_tt_cc_t<float, __half, __half>(sh, static_cast<__half*>(out), s, "tt_cc_kernel<f16,o16>");
    }
}

}  // namespace lrc
