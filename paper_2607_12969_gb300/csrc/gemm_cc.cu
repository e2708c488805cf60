// gemm_cc.cu -- register-tiled products on the CUDA cores with binary32
// arithmetic: C = A B for the binary32 apply (Sec. 4.4, Eq. gpu_matrix_apply,
// both of its products) and for the TT chain (Sec. 7.5,
// Eq. gpu_tt_reconstruction: B_l = Z_{l-1} K_l).
//
// A is M x K row-major.  B is K x N row-major ("NN"), or N x K row-major
// ("NT", B's transpose is what is stored: the factor layouts U and V^T of the
// apply).  A CTA of 256 threads owns a 128 x BN tile of C, BN = 128 or 144;
// each thread owns 8 rows (two groups of 4, 64 apart) x 8 columns (two
// groups of 4, 64 apart) plus, for BN = 144, one column of the last 16, so a
// warp's operand reads are broadcasts (A) or consecutive 16-byte words (B)
// and its stores are 256-byte row segments.
// K advances in slabs of 16: the next slab is fetched into registers while
// the current one is multiplied (two shared-memory buffers, one barrier per
// slab).  Products and sums are binary32 FMAs (no TF32: Sec. 3.4).
//
// A split over K (blockIdx.y) writes one partial product per split at
// C + split * c_split; the caller adds them in a fixed order.
#include "common.cuh"
#include "tc.cuh"

namespace lrc {
namespace {

constexpr int BM = 128, BK = 16, NT = 256;
constexpr int LDA = BM + 4;          // A slab pitch in floats (rows stay 16-byte aligned)

__device__ __forceinline__ float4 ld4(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }
__device__ __forceinline__ float ld1(const float* p) { return __ldg(p); }

// Four consecutive elements (r, c..c+3) of a row-major [R x C] array; zero
// outside.  `vec`: rows are aligned for a vector load.
template <typename TIn>
__device__ __forceinline__ float4 load_quad(const TIn* __restrict__ g, int64_t ld, int64_t R, int64_t C, int64_t r,
                                            int64_t c, bool vec) {
    if (r < R && vec && c + 4 <= C) return ld4(g + r * ld + c);
    float e[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) e[j] = (r < R && c + j < C) ? ld1(g + r * ld + c + j) : 0.0f;
    return make_float4(e[0], e[1], e[2], e[3]);
}

__device__ __forceinline__ void st1(float* p, float v) { __stcs(p, v); }
__device__ __forceinline__ void st4(float* p, const float* v) {
    __stcs(reinterpret_cast<float4*>(p), make_float4(v[0], v[1], v[2], v[3]));
}

template <typename TA, typename TB, typename TOut>
struct GemmArgs {
    const TA* A;
    const TB* B;
    TOut* C;
    int64_t lda, ldb, ldc;
    int64_t M, N, K;
    int64_t ntn;           // column tiles
    int64_t kchunk;        // K per split (multiple of BK)
    int64_t c_split;       // element offset between the splits' outputs
    int vec_a, vec_b, vec_c;
};

// Rows x 16 slabs of a row-major [R x K] operand, transposed into shared
// memory S[k][row] (pitch lds).  Quad f of a slab is row f / 4, elements
// 4 (f % 4) .. + 3; thread t owns quads t, t + 256, ...  Full slabs of an
// aligned operand take one vector load per quad and no bounds test but the
// row's (decided once).
template <typename TIn, int ROWS>
struct RowSlab {
    static constexpr int kQuads = ROWS * BK / 4;
    static constexpr int kPer = (kQuads + NT - 1) / NT;
    float4 v[kPer];
    const TIn* p[kPer];      // row start + first slab's quad; null: row outside
    __device__ __forceinline__ void init(const TIn* __restrict__ g, int64_t ld, int64_t R, int64_t r0, int64_t kbeg) {
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const int f = threadIdx.x + q * NT;
            const int64_t r = r0 + (f >> 2);
            p[q] = (f < kQuads && r < R) ? g + r * ld + kbeg + (f & 3) * 4 : nullptr;
        }
    }
    // slab starting at k0 = kbeg + off; kend bounds the columns of a partial slab
    __device__ __forceinline__ void load(int64_t off, bool fast, int64_t kleft) {
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const int f = threadIdx.x + q * NT;
            if (kQuads % NT != 0 && f >= kQuads) continue;
            if (!p[q]) {
                v[q] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            } else if (fast) {
                v[q] = ld4(p[q] + off);
            } else {
                const int kq = (f & 3) * 4;
                float e[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) e[j] = (kq + j < kleft) ? ld1(p[q] + off + j) : 0.0f;
                v[q] = make_float4(e[0], e[1], e[2], e[3]);
            }
        }
    }
    __device__ __forceinline__ void store(float* S, int lds) const {
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const int f = threadIdx.x + q * NT;
            if (kQuads % NT == 0 || f < kQuads) {
                const int row = f >> 2, k = (f & 3) * 4;
                S[(k + 0) * lds + row] = v[q].x;
                S[(k + 1) * lds + row] = v[q].y;
                S[(k + 2) * lds + row] = v[q].z;
                S[(k + 3) * lds + row] = v[q].w;
            }
        }
    }
};

// 16 x COLS slabs of a row-major [K x C] operand, copied as is: S[k][c].
// Quad f is slab row f / (COLS/4), columns 4 (f % (COLS/4)) .. + 3.
template <typename TIn, int COLS>
struct ColSlab {
    static constexpr int kQuadsRow = COLS / 4;
    static constexpr int kQuads = BK * kQuadsRow;
    static constexpr int kPer = (kQuads + NT - 1) / NT;
    float4 v[kPer];
    const TIn* p[kPer];      // first slab's quad; null: columns outside
    int ncol[kPer];          // columns of the quad inside the operand (0..4)
    __device__ __forceinline__ void init(const TIn* __restrict__ g, int64_t ld, int64_t C, int64_t kbeg, int64_t c0) {
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const int f = threadIdx.x + q * NT;
            const int64_t c = c0 + (f % kQuadsRow) * 4;
            const int64_t in = C - c;
            ncol[q] = in <= 0 ? 0 : (in >= 4 ? 4 : (int)in);
            p[q] = (f < kQuads && ncol[q] > 0) ? g + (kbeg + f / kQuadsRow) * ld + c : nullptr;
        }
    }
    __device__ __forceinline__ void load(int64_t off, bool fast, int64_t kleft) {
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const int f = threadIdx.x + q * NT;
            if (kQuads % NT != 0 && f >= kQuads) continue;
            if (!p[q] || (!fast && f / kQuadsRow >= kleft)) {
                v[q] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            } else if (fast && ncol[q] == 4) {
                v[q] = ld4(p[q] + off);
            } else {
                float e[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) e[j] = (j < ncol[q]) ? ld1(p[q] + off + j) : 0.0f;
                v[q] = make_float4(e[0], e[1], e[2], e[3]);
            }
        }
    }
    __device__ __forceinline__ void store(float* S, int lds) const {
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const int f = threadIdx.x + q * NT;
            if (kQuads % NT == 0 || f < kQuads)
                *reinterpret_cast<float4*>(S + (f / kQuadsRow) * lds + (f % kQuadsRow) * 4) = v[q];
        }
    }
};

// Columns of a thread in a 128 + 16 EX wide tile: tx*4 + j and 64 + tx*4 + j
// (j < 4), then 128 + 16 e + tx (e < EX).
template <int EX>
__device__ __forceinline__ void rank1_update(const float* __restrict__ Ab, const float* __restrict__ Bb, int kk,
                                             int tx, int ty, float (&acc)[8][8 + EX]) {
    constexpr int LDB = 128 + 16 * EX + 4;
    float av[8], bv[8 + EX];
    const float4 a0 = *reinterpret_cast<const float4*>(Ab + kk * LDA + ty * 4);
    const float4 a1 = *reinterpret_cast<const float4*>(Ab + kk * LDA + 64 + ty * 4);
    av[0] = a0.x; av[1] = a0.y; av[2] = a0.z; av[3] = a0.w;
    av[4] = a1.x; av[5] = a1.y; av[6] = a1.z; av[7] = a1.w;
    const float4 b0 = *reinterpret_cast<const float4*>(Bb + kk * LDB + tx * 4);
    const float4 b1 = *reinterpret_cast<const float4*>(Bb + kk * LDB + 64 + tx * 4);
    bv[0] = b0.x; bv[1] = b0.y; bv[2] = b0.z; bv[3] = b0.w;
    bv[4] = b1.x; bv[5] = b1.y; bv[6] = b1.z; bv[7] = b1.w;
#pragma unroll
    for (int e = 0; e < EX; ++e) bv[8 + e] = Bb[kk * LDB + 128 + 16 * e + tx];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8 + EX; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
}

// Two CTAs per SM for 128-wide tiles (128 registers a thread); the 144-wide
// tile needs more and runs one CTA per SM.
template <typename TA, typename TB, typename TOut, bool BT, int EX>
__global__ void __launch_bounds__(NT, EX == 0 ? 2 : 1)
gemm_cc_kernel(const GemmArgs<TA, TB, TOut> a) {
    constexpr int BN = 128 + 16 * EX;
    constexpr int LDB = BN + 4;
    __shared__ __align__(16) float As[2][BK * LDA];
    __shared__ __align__(16) float Bs[2][BK * LDB];

    const int tid = threadIdx.x;
    const int tx = tid & 15, ty = tid >> 4;
    const int64_t tile = blockIdx.x;
    const int64_t mt = tile / a.ntn, nt = tile - mt * a.ntn;
    const int64_t m0 = mt * BM, n0 = nt * BN;
    const int64_t kbeg = (int64_t)blockIdx.y * a.kchunk;
    const int64_t kend = (kbeg + a.kchunk < a.K) ? kbeg + a.kchunk : a.K;
    TOut* C = a.C + (int64_t)blockIdx.y * a.c_split;

    RowSlab<TA, BM> sa;
    ColSlab<TB, BN> sbn;     // NN: 16 x BN slabs of the K x N array
    RowSlab<TB, BN> sbt;     // NT: BN rows of the N x K array
    tc::pdl_wait();          // operands written by the previous kernel of the stream
    sa.init(a.A, a.lda, a.M, m0, kbeg);
    if (BT) sbt.init(a.B, a.ldb, a.N, n0, kbeg);
    else sbn.init(a.B, a.ldb, a.N, kbeg, n0);
    const int64_t klen = kend - kbeg;
    const int64_t nslabs = (klen + BK - 1) / BK;
    const int64_t nfull = klen / BK;
    const bool vec = a.vec_a && a.vec_b;
    auto load = [&](int64_t s) {
        const bool fast = vec && s < nfull;
        const int64_t kleft = klen - s * BK;
        sa.load(s * BK, fast, kleft);
        if (BT) sbt.load(s * BK, fast, kleft);
        else sbn.load(s * BK * a.ldb, fast, kleft);
    };
    auto store = [&](int buf) {
        sa.store(As[buf], LDA);
        if (BT) sbt.store(Bs[buf], LDB);
        else sbn.store(Bs[buf], LDB);
    };

    float acc[8][8 + EX];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8 + EX; ++j) acc[i][j] = 0.0f;

    if (nslabs > 0) {
        load(0);
        store(0);
        __syncthreads();
    }
    for (int64_t s = 0; s < nslabs; ++s) {
        const int buf = (int)(s & 1);
        const bool more = s + 1 < nslabs;
        if (more) load(s + 1);
        const float* Ab = As[buf];
        const float* Bb = Bs[buf];
        if (s < nfull) {
#pragma unroll
            for (int kk = 0; kk < BK; ++kk) rank1_update<EX>(Ab, Bb, kk, tx, ty, acc);
        } else {
            // last, partial slab: only its real columns (the rest are zero-filled)
            const int kn = (int)(klen - s * BK);
#pragma unroll 2
            for (int kk = 0; kk < kn; ++kk) rank1_update<EX>(Ab, Bb, kk, tx, ty, acc);
        }
        if (more) store(buf ^ 1);
        __syncthreads();
    }
    tc::pdl_trigger();

    // epilogue: rows m0 + {ty*4 + i, 64 + ty*4 + i}
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int64_t r = m0 + (i < 4 ? ty * 4 + i : 64 + ty * 4 + (i - 4));
        if (r >= a.M) continue;
        TOut* crow = C + r * a.ldc;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int64_t c = n0 + h * 64 + tx * 4;
            const float* v = &acc[i][h * 4];
            if (a.vec_c && c + 4 <= a.N) {
                st4(crow + c, v);
            } else {
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    if (c + j < a.N) st1(crow + c + j, v[j]);
            }
        }
#pragma unroll
        for (int e = 0; e < EX; ++e) {
            const int64_t c = n0 + 128 + 16 * e + tx;
            if (c < a.N) st1(crow + c, acc[i][8 + e]);
        }
    }
}

template <typename T>
bool vec_ok(const T* p, int64_t ld) {
    constexpr size_t quad = 4 * sizeof(T);
    return (reinterpret_cast<uintptr_t>(p) % quad) == 0 && (ld % 4) == 0;
}

template <typename TA, typename TB, typename TOut, bool BT, int EX>
lrc_status launch_t(const TA* A, int64_t lda, const TB* B, int64_t ldb, TOut* C, int64_t ldc, int64_t M,
                    int64_t N, int64_t K, int splits, int64_t c_split, cudaStream_t s, const char* name) {
    constexpr int BN = 128 + 16 * EX;
    GemmArgs<TA, TB, TOut> a{};
    a.A = A;
    a.B = B;
    a.C = C;
    a.lda = lda;
    a.ldb = ldb;
    a.ldc = ldc;
    a.M = M;
    a.N = N;
    a.K = K;
    a.ntn = (N + BN - 1) / BN;
    const int64_t tiles = ((M + BM - 1) / BM) * a.ntn;
    if (splits < 1) splits = 1;
    a.kchunk = ((K + splits - 1) / splits + BK - 1) / BK * BK;
    splits = (int)((K + a.kchunk - 1) / a.kchunk);
    a.c_split = c_split;
    a.vec_a = vec_ok(A, lda);
    a.vec_b = vec_ok(B, ldb);
    a.vec_c = vec_ok(C, ldc);
    if (tiles > 0x7fffffff || splits > 65535) {
        set_error("%s: product too large (%lld tiles)", name, (long long)tiles);
        return LRC_ERR_UNSUPPORTED;
    }
    if (tiles == 0) return LRC_OK;
    cudaError_t e = launch_pdl(gemm_cc_kernel<TA, TB, TOut, BT, EX>, dim3((unsigned)tiles, (unsigned)splits), dim3(NT), 0,
                               s, a);
    if (e != cudaSuccess) return cuda_fail(e, name);
    return after_launch(name);
}

// ---------------------------------------------------------------------------
// binary64: C = A B (both row-major, B stored K x N), bound by the DFMA rate
// (about 2 per clock per SM on this GPU), so a plain tile is enough: 64 x 64
// tiles, 256 threads, each thread 4 rows x 4 columns strided by 16 (a warp's
// shared reads are two broadcast rows of A and 16 consecutive doubles of B),
// K in 16-wide slabs through two shared-memory buffers with the next slab
// prefetched in registers.
// ---------------------------------------------------------------------------
constexpr int BM64 = 64, BN64 = 64, BK64 = 16;

__global__ void __launch_bounds__(NT)
gemm_f64_kernel(const double* __restrict__ A, int64_t lda, const double* __restrict__ B, int64_t ldb,
                double* __restrict__ C, int64_t ldc, int64_t M, int64_t N, int64_t K, int64_t ntn) {
    __shared__ double As[2][BK64][BM64 + 1];
    __shared__ double Bs[2][BK64][BN64 + 1];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int64_t mt = blockIdx.x / ntn, nt = blockIdx.x - mt * ntn;
    const int64_t m0 = mt * BM64, n0 = nt * BN64;
    tc::pdl_wait();
    double ra[4], rb[4];
    // A slab: element e = tid + 256 q -> row e / 16, k e % 16; B slab: row e / 64, column e % 64
#define LRC_F64_LOAD(k0)                                                                   \
    _Pragma("unroll") for (int q = 0; q < 4; ++q) {                                         \
        const int e = tid + NT * q;                                                        \
        const int64_t ar = m0 + (e >> 4), ak = (k0) + (e & 15);                            \
        ra[q] = (ar < M && ak < K) ? __ldg(A + ar * lda + ak) : 0.0;                       \
        const int64_t bk = (k0) + (e >> 6), bc = n0 + (e & 63);                            \
        rb[q] = (bk < K && bc < N) ? __ldg(B + bk * ldb + bc) : 0.0;                       \
    }
#define LRC_F64_STORE(buf)                                                                 \
    _Pragma("unroll") for (int q = 0; q < 4; ++q) {                                         \
        const int e = tid + NT * q;                                                        \
        As[buf][e & 15][e >> 4] = ra[q];                                                   \
        Bs[buf][e >> 6][e & 63] = rb[q];                                                   \
    }
    double acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.0;
    const int64_t nslabs = (K + BK64 - 1) / BK64;
    if (nslabs > 0) {
        LRC_F64_LOAD(0)
        LRC_F64_STORE(0)
        __syncthreads();
    }
    for (int64_t s = 0; s < nslabs; ++s) {
        const int buf = (int)(s & 1);
        const bool more = s + 1 < nslabs;
        if (more) { LRC_F64_LOAD((s + 1) * BK64) }
        // the last slab multiplies only its real columns
        const int kn = (K - s * BK64) < BK64 ? (int)(K - s * BK64) : BK64;
#pragma unroll 4
        for (int kk = 0; kk < kn; ++kk) {
            double a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[buf][kk][ty + 16 * i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[buf][kk][tx + 16 * j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fma(a[i], b[j], acc[i][j]);
        }
        if (more) { LRC_F64_STORE(buf ^ 1) }
        __syncthreads();
    }
#undef LRC_F64_LOAD
#undef LRC_F64_STORE
    tc::pdl_trigger();
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t r = m0 + ty + 16 * i;
        if (r >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t c = n0 + tx + 16 * j;
            if (c < N) C[r * ldc + c] = acc[i][j];
        }
    }
}

}  // namespace

// Extra 16-column groups per tile for N columns: 128 + 16 ex wide tiles,
// ex = 1 when it removes most of a partial tile (N = 136, 144, 272 ...).
int gemm_cc_ex(int64_t N) {
    const int64_t w0 = (N + 127) / 128 * 128, w1 = (N + 143) / 144 * 144;
    return (w1 < w0) ? 1 : 0;
}

lrc_status gemm_cc_f32(const float* A, int64_t lda, const float* B, int64_t ldb, bool b_trans, float* C,
                       int64_t ldc, int64_t M, int64_t N, int64_t K, int splits, int64_t c_split, cudaStream_t s) {
    const int ex = gemm_cc_ex(N);
    if (b_trans) {
        if (ex)
            return launch_t<float, float, float, true, 1>(A, lda, B, ldb, C, ldc, M, N, K, splits, c_split, s,
                                                          "gemm_cc_kernel<f32,NT,144>");
        return launch_t<float, float, float, true, 0>(A, lda, B, ldb, C, ldc, M, N, K, splits, c_split, s,
                                                      "gemm_cc_kernel<f32,NT,128>");
    }
    if (ex)
        return launch_t<float, float, float, false, 1>(A, lda, B, ldb, C, ldc, M, N, K, splits, c_split, s,
                                                       "gemm_cc_kernel<f32,NN,144>");
    return launch_t<float, float, float, false, 0>(A, lda, B, ldb, C, ldc, M, N, K, splits, c_split, s,
                                                   "gemm_cc_kernel<f32,NN,128>");
}

lrc_status gemm_cc_f64(const double* A, int64_t lda, const double* B, int64_t ldb, double* C, int64_t ldc,
                       int64_t M, int64_t N, int64_t K, cudaStream_t s) {
    const int64_t ntn = (N + BN64 - 1) / BN64;
    const int64_t tiles = ((M + BM64 - 1) / BM64) * ntn;
    if (tiles > 0x7fffffff) {
        set_error("gemm_f64_kernel: product too large (%lld tiles)", (long long)tiles);
        return LRC_ERR_UNSUPPORTED;
    }
    if (tiles == 0) return LRC_OK;
    cudaError_t e = launch_pdl(gemm_f64_kernel, dim3((unsigned)tiles), dim3(NT), 0, s, A, lda, B, ldb, C, ldc, M, N,
                               K, ntn);
    if (e != cudaSuccess) return cuda_fail(e, "gemm_f64_kernel launch");
    return after_launch("gemm_f64_kernel");
}

}  // namespace lrc
