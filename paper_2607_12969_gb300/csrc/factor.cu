// factor.cu -- the factorization side on the GPU (binary64): TT-SVD (Sec. 5,
// the sequential truncated SVDs of Oseledets' algorithm; Alg.
// alg:tt_compensation steps 1-2) and the left-orthogonal gauge (Sec. 6.1).
//
// Both rest on one primitive, a one-sided (Hestenes) Jacobi SVD of a tall
// L x p matrix A held column-major in device memory: column pairs (i, j) are
// rotated until every pair is orthogonal to working precision, accumulating
// the rotations in V (p x p).  Then A V = W with orthogonal columns, the
// singular values are the column norms of W and A = U diag(s) V^T with
// U = W diag(s)^-1.  Rotating A itself, not its Gram matrix, keeps the small
// singular values (the tails E_R of the certificate) accurate to about u s_1
// instead of sqrt(u) s_1.
//
// A sweep visits every pair once in p - 1 rounds of the round-robin
// tournament (p / 2 disjoint pairs per round, one CTA per pair, one launch per
// round); the host checks after each sweep how many rotations were applied
// and stops when none was (at most kMaxSweeps sweeps).  No kernel waits on
// another CTA: rounds are separated by launches.
#include <algorithm>
#include <numeric>
#include <vector>

#include "common.cuh"

namespace lrc {
namespace {

constexpr int kJThreads = 256;
constexpr int kMaxSweeps = 40;
constexpr int kMaxP = 1024;          // columns of one Jacobi problem

__device__ __forceinline__ double block_sum(double v, double* sh) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) sh[warp] = v;
    __syncthreads();
    double s = 0.0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += sh[w];   // same order in every thread
    return s;
}

// Pair k of round `round` of the tournament on pv (even) players: player
// pv - 1 stays, the others turn.
__device__ __forceinline__ void tournament_pair(int pv, int round, int k, int* a, int* b) {
    if (k == 0) {
        *a = pv - 1;
        *b = round;
    } else {
        *a = (round + k) % (pv - 1);
        *b = (round - k + pv - 1) % (pv - 1);
    }
}

// One round: CTA k rotates its column pair of A (L rows) and of V (p rows)
// if the pair is not yet orthogonal: |a_i . a_j| > tol ||a_i|| ||a_j||.
__global__ void __launch_bounds__(kJThreads) jacobi_round_kernel(double* __restrict__ A, int64_t L,
                                                                   double* __restrict__ V, int p, int pv,
                                                                   int round, double tol,
                                                                   unsigned int* __restrict__ rotations) {
    __shared__ double sh[kJThreads / 32];
    __shared__ double cs[2];
    int i, j;
    tournament_pair(pv, round, blockIdx.x, &i, &j);
    if (i >= p || j >= p) return;                 // the dummy player of an odd p
    double* ai = A + (int64_t)i * L;
    double* aj = A + (int64_t)j * L;
    double al = 0.0, be = 0.0, ga = 0.0;
    for (int64_t r = threadIdx.x; r < L; r += kJThreads) {
        const double x = ai[r], y = aj[r];
        al = fma(x, x, al);
        be = fma(y, y, be);
        ga = fma(x, y, ga);
    }
    al = block_sum(al, sh);
    be = block_sum(be, sh);
    ga = block_sum(ga, sh);
    if (threadIdx.x == 0) {
        double c = 1.0, s = 0.0;
        if (ga != 0.0 && fabs(ga) > tol * sqrt(al) * sqrt(be)) {
            // c, s with (c a_i - s a_j) . (s a_i + c a_j) = 0: t = s / c is the
            // smaller root of t^2 + 2 zeta t - 1 = 0, zeta = (be - al) / (2 ga)
            const double zeta = (be - al) / (2.0 * ga);
            const double t = copysign(1.0, zeta) / (fabs(zeta) + sqrt(fma(zeta, zeta, 1.0)));
            c = 1.0 / sqrt(fma(t, t, 1.0));
            s = c * t;
            atomicAdd(rotations, 1u);
        }
        cs[0] = c;
        cs[1] = s;
    }
    __syncthreads();
    const double c = cs[0], s = cs[1];
    if (s == 0.0) return;
    for (int64_t r = threadIdx.x; r < L; r += kJThreads) {
        const double x = ai[r], y = aj[r];
        ai[r] = c * x - s * y;
        aj[r] = fma(s, x, c * y);
    }
    double* vi = V + (int64_t)i * p;
    double* vj = V + (int64_t)j * p;
    for (int r = threadIdx.x; r < p; r += kJThreads) {
        const double x = vi[r], y = vj[r];
        vi[r] = c * x - s * y;
        vj[r] = fma(s, x, c * y);
    }
}

__global__ void identity_kernel(double* V, int p) {
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < (int64_t)p * p;
         e += (int64_t)gridDim.x * blockDim.x)
        V[e] = (e / p == e % p) ? 1.0 : 0.0;
}

__global__ void __launch_bounds__(kJThreads) col_norms_kernel(const double* __restrict__ A, int64_t L,
                                                                double* __restrict__ norms) {
    __shared__ double sh[kJThreads / 32];
    const double* a = A + (int64_t)blockIdx.x * L;
    double s = 0.0;
    for (int64_t r = threadIdx.x; r < L; r += kJThreads) s = fma(a[r], a[r], s);
    s = block_sum(s, sh);
    if (threadIdx.x == 0) norms[blockIdx.x] = sqrt(s);
}

// dst (cols x rows, i.e. the column-major image of the row-major src) = src^T
__global__ void transpose_kernel(const double* __restrict__ src, int64_t rows, int64_t cols,
                                 double* __restrict__ dst) {
    __shared__ double t[32][33];
    const int64_t r0 = (int64_t)blockIdx.y * 32, c0 = (int64_t)blockIdx.x * 32;
    for (int y = threadIdx.y; y < 32; y += blockDim.y) {
        const int64_t r = r0 + y, c = c0 + threadIdx.x;
        if (r < rows && c < cols) t[y][threadIdx.x] = src[r * cols + c];
    }
    __syncthreads();
    for (int y = threadIdx.y; y < 32; y += blockDim.y) {
        const int64_t c = c0 + y, r = r0 + threadIdx.x;
        if (r < rows && c < cols) dst[c * rows + r] = t[threadIdx.x][y];
    }
}

// out[i * r + k] = scale(k) * M[order[k] * ld + i]  (i < n, k < r): columns of
// a column-major matrix M gathered into a row-major n x r matrix, column k
// scaled by sigma[order[k]] (mode 1), by its inverse (mode 2) or not (0).
__global__ void gather_cols_kernel(const double* __restrict__ M, int64_t ld, int64_t n, int r,
                                   const int* __restrict__ order, const double* __restrict__ sigma, int mode,
                                   double* __restrict__ out) {
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n * r;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = e / r;
        const int k = (int)(e - i * r);
        const int o = order[k];
        double f = 1.0;
        if (mode == 1) f = sigma[o];
        else if (mode == 2) f = sigma[o] > 0.0 ? 1.0 / sigma[o] : 0.0;
        out[e] = f * M[(int64_t)o * ld + i];
    }
}

// out[k * n + j] = scale(k) * M[order[k] * ld + j]: the same columns laid out
// as rows (an r x n row-major matrix).
__global__ void gather_rows_kernel(const double* __restrict__ M, int64_t ld, int64_t n, int r,
                                   const int* __restrict__ order, const double* __restrict__ sigma, int mode,
                                   double* __restrict__ out) {
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n * r;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int k = (int)(e / n);
        const int64_t j = e - (int64_t)k * n;
        const int o = order[k];
        const double f = mode == 1 ? sigma[o] : 1.0;
        out[e] = f * M[(int64_t)o * ld + j];
    }
}

int grid_for(int64_t n) {
    const int64_t want = (n + 255) / 256;
    const int64_t cap = (int64_t)sm_count() * 8;
    return (int)(want < 1 ? 1 : (want < cap ? want : cap));
}

// Workspace layout of one factorization: [A: amax][C: cmax][V: p^2]
// [norms: p][order: p ints][rotation counter].
struct FactorWs {
    double* A;
    double* C;
    double* V;
    double* norms;
    int* order;
    unsigned int* rot;
};

lrc_status factor_ws(cudaStream_t s, int64_t amax, int64_t cmax, int p, FactorWs* w) {
    const size_t a = ((size_t)amax * 8 + 255) / 256 * 256, c = ((size_t)cmax * 8 + 255) / 256 * 256;
    const size_t v = ((size_t)p * p * 8 + 255) / 256 * 256, nb = ((size_t)p * 8 + 255) / 256 * 256;
    const size_t ob = ((size_t)p * 4 + 255) / 256 * 256;
    void* base = nullptr;
    lrc_status st = stream_workspace(s, a + c + v + nb + ob + 256, &base);
    if (st != LRC_OK) return st;
    unsigned char* b = static_cast<unsigned char*>(base);
    w->A = reinterpret_cast<double*>(b);
    w->C = reinterpret_cast<double*>(b + a);
    w->V = reinterpret_cast<double*>(b + a + c);
    w->norms = reinterpret_cast<double*>(b + a + c + v);
    w->order = reinterpret_cast<int*>(b + a + c + v + nb);
    w->rot = reinterpret_cast<unsigned int*>(b + a + c + v + nb + ob);
    return LRC_OK;
}

// One-sided Jacobi on A (L x p, column-major, L >= p): on return A holds
// A V (orthogonal columns), V the accumulated rotations, norms the column
// norms and sigma_host the same on the host; order[k] (device and
// order_host) the column of the k-th largest norm.
lrc_status jacobi_svd(const FactorWs& w, int64_t L, int p, std::vector<double>& sigma_host,
                      std::vector<int>& order_host, cudaStream_t s) {
    const int pv = p + (p & 1);
    identity_kernel<<<grid_for((int64_t)p * p), 256, 0, s>>>(w.V, p);
    lrc_status st = after_launch("identity_kernel");
    if (st != LRC_OK) return st;
    // pairs orthogonal within sqrt(L) units of roundoff count as converged
    const double tol = sqrt((double)L) * 0x1p-53;
    for (int sweep = 0; sweep < kMaxSweeps && p > 1; ++sweep) {
        cudaError_t e = cudaMemsetAsync(w.rot, 0, sizeof(unsigned int), s);
        if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync (Jacobi counter)");
        for (int round = 0; round < pv - 1; ++round) {
            jacobi_round_kernel<<<pv / 2, kJThreads, 0, s>>>(w.A, L, w.V, p, pv, round, tol, w.rot);
            if ((st = after_launch("jacobi_round_kernel")) != LRC_OK) return st;
        }
        unsigned int rot = 0;
        e = cudaMemcpyAsync(&rot, w.rot, sizeof rot, cudaMemcpyDeviceToHost, s);
        if (e == cudaSuccess) e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) return cuda_fail(e, "Jacobi sweep count");
        if (rot == 0) break;
        if (sweep == kMaxSweeps - 1) {
            set_error("Jacobi SVD did not converge in %d sweeps (p = %d, L = %lld)", kMaxSweeps, p, (long long)L);
            return LRC_ERR_UNSUPPORTED;
        }
    }
    col_norms_kernel<<<p, kJThreads, 0, s>>>(w.A, L, w.norms);
    if ((st = after_launch("col_norms_kernel")) != LRC_OK) return st;
    sigma_host.resize(p);
    cudaError_t e = cudaMemcpyAsync(sigma_host.data(), w.norms, sizeof(double) * p, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "singular values to host");
    order_host.resize(p);
    std::iota(order_host.begin(), order_host.end(), 0);
    std::stable_sort(order_host.begin(), order_host.end(),
                     [&](int x, int y) { return sigma_host[x] > sigma_host[y]; });
    e = cudaMemcpyAsync(w.order, order_host.data(), sizeof(int) * p, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);     // order_host is the source
    if (e != cudaSuccess) return cuda_fail(e, "column order to device");
    return LRC_OK;
}

// sum of squares from the smallest up, compensated
double tail_sq(const std::vector<double>& sig, const std::vector<int>& order, int from) {
    double s = 0.0, c = 0.0;
    for (int k = (int)order.size() - 1; k >= from; --k) {
        const double t = sig[order[k]] * sig[order[k]];
        const double u = s + t;
        c += (fabs(s) >= fabs(t)) ? ((s - u) + t) : ((t - u) + s);
        s = u;
    }
    return s + c;
}

}  // namespace

int factor_max_cols() { return kMaxP; }

lrc_status run_tt_svd(const double* T, const TTShape& sh, double* const* cores, double* delta2_out,
                      double* spectra_out, cudaStream_t s) {
    const int d = sh.d;
    int pmax = 1;
    int64_t rest = sh.numel;
    for (int l = 0; l < d - 1; ++l) {
        rest /= sh.dims[l];
        const int64_t rows = sh.ranks[l] * sh.dims[l];
        const int64_t p = rows < rest ? rows : rest;
        if (p > kMaxP) {
            set_error("TT-SVD: unfolding %d has %lld x %lld entries; the Jacobi SVD takes at most %d columns",
                      l + 1, (long long)rows, (long long)rest, kMaxP);
            return LRC_ERR_UNSUPPORTED;
        }
        if (p > pmax) pmax = (int)p;
    }
    FactorWs w;
    lrc_status st = factor_ws(s, sh.numel, sh.numel, pmax, &w);
    if (st != LRC_OK) return st;
    const double* C = T;         // the remainder: rows x cols, row-major
    rest = sh.numel;
    int64_t spec_off = 0;
    std::vector<double> sig;
    std::vector<int> order;
    for (int l = 0; l < d - 1; ++l) {
        const int64_t rows = sh.ranks[l] * sh.dims[l];
        const int64_t cols = rest / sh.dims[l];
        rest = cols;
        const int r = (int)sh.ranks[l + 1];
        const bool wide = rows <= cols;          // A = C^T (cols x rows) or A = C (rows x cols)
        const int64_t L = wide ? cols : rows;
        const int p = (int)(wide ? rows : cols);
        cudaError_t e;
        if (wide) {
            // the row-major C is the column-major C^T
            e = cudaMemcpyAsync(w.A, C, sizeof(double) * (size_t)(rows * cols), cudaMemcpyDeviceToDevice, s);
            if (e != cudaSuccess) return cuda_fail(e, "TT-SVD remainder copy");
        } else {
            transpose_kernel<<<dim3((unsigned)((cols + 31) / 32), (unsigned)((rows + 31) / 32)), dim3(32, 8), 0, s>>>(
                C, rows, cols, w.A);
            if ((st = after_launch("transpose_kernel")) != LRC_OK) return st;
        }
        if ((st = jacobi_svd(w, L, p, sig, order, s)) != LRC_OK) return st;
        if (delta2_out) delta2_out[l] = tail_sq(sig, order, r);
        if (spectra_out)
            for (int k = 0; k < p; ++k) spectra_out[spec_off + k] = sig[order[k]];
        spec_off += p;
        double* core = cores[l];                 // rows x r, row-major
        if (wide) {
            // C = V diag(s) W^T: left vectors are V's columns, the next
            // remainder diag(s) W^T is the rows of A V
            gather_cols_kernel<<<grid_for(rows * (int64_t)r), 256, 0, s>>>(w.V, p, rows, r, w.order, w.norms, 0,
                                                                           core);
            if ((st = after_launch("gather_cols_kernel")) != LRC_OK) return st;
            gather_rows_kernel<<<grid_for(cols * (int64_t)r), 256, 0, s>>>(w.A, L, cols, r, w.order, w.norms, 0,
                                                                           w.C);
        } else {
            // C = U diag(s) V^T with U = (A V) diag(s)^-1; next remainder diag(s) V^T
            gather_cols_kernel<<<grid_for(rows * (int64_t)r), 256, 0, s>>>(w.A, L, rows, r, w.order, w.norms, 2,
                                                                           core);
            if ((st = after_launch("gather_cols_kernel")) != LRC_OK) return st;
            gather_rows_kernel<<<grid_for(cols * (int64_t)r), 256, 0, s>>>(w.V, p, cols, r, w.order, w.norms, 1,
                                                                           w.C);
        }
        if ((st = after_launch("gather_rows_kernel")) != LRC_OK) return st;
        C = w.C;
    }
    // the last core is the remainder (r_{d-1} x n_d)
    const size_t last = (size_t)sh.ranks[d - 1] * (size_t)sh.dims[d - 1];
    cudaError_t e = cudaMemcpyAsync(cores[d - 1], C, sizeof(double) * last, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e, "TT-SVD last core");
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "TT-SVD");
    return LRC_OK;
}

lrc_status run_tt_left_orthogonalize(const TTShape& sh, double* const* cores, cudaStream_t s) {
    const int d = sh.d;
    int64_t amax = 1, cmax = 1;
    int pmax = 1;
    for (int l = 0; l < d - 1; ++l) {
        const int64_t rows = sh.ranks[l] * sh.dims[l], p = sh.ranks[l + 1];
        if (p > rows) {
            set_error("left-orthogonalization: core %d is %lld x %lld (rank above r_{l-1} n_l)", l + 1,
                      (long long)rows, (long long)p);
            return LRC_ERR_UNSUPPORTED;
        }
        if (p > kMaxP) {
            set_error("left-orthogonalization: rank %lld above %d", (long long)p, kMaxP);
            return LRC_ERR_UNSUPPORTED;
        }
        amax = std::max(amax, rows * p);
        cmax = std::max(cmax, sh.ranks[l + 1] * sh.dims[l + 1] * sh.ranks[l + 2] + p * p);
        pmax = std::max(pmax, (int)p);
    }
    FactorWs w;
    lrc_status st = factor_ws(s, amax, cmax, pmax, &w);
    if (st != LRC_OK) return st;
    std::vector<double> sig;
    std::vector<int> order;
    for (int l = 0; l < d - 1; ++l) {
        const int64_t rows = sh.ranks[l] * sh.dims[l];
        const int p = (int)sh.ranks[l + 1];
        transpose_kernel<<<dim3((unsigned)((p + 31) / 32), (unsigned)((rows + 31) / 32)), dim3(32, 8), 0, s>>>(
            cores[l], rows, p, w.A);
        if ((st = after_launch("transpose_kernel")) != LRC_OK) return st;
        if ((st = jacobi_svd(w, rows, p, sig, order, s)) != LRC_OK) return st;
        // G = Q R' with Q = (A V) diag(s)^-1 (orthonormal columns) and
        // R' = diag(s) V^T, in the natural column order
        std::iota(order.begin(), order.end(), 0);
        cudaError_t e = cudaMemcpyAsync(w.order, order.data(), sizeof(int) * p, cudaMemcpyHostToDevice, s);
        if (e == cudaSuccess) e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) return cuda_fail(e, "column order to device");
        gather_cols_kernel<<<grid_for(rows * (int64_t)p), 256, 0, s>>>(w.A, rows, rows, p, w.order, w.norms, 2,
                                                                       cores[l]);
        if ((st = after_launch("gather_cols_kernel")) != LRC_OK) return st;
        double* R = w.C;                                // p x p, row-major
        gather_rows_kernel<<<grid_for((int64_t)p * p), 256, 0, s>>>(w.V, p, p, p, w.order, w.norms, 1, R);
        if ((st = after_launch("gather_rows_kernel")) != LRC_OK) return st;
        // core l + 1 <- R' core l + 1  (p x (n_{l+1} r_{l+2}))
        const int64_t ncols = sh.dims[l + 1] * sh.ranks[l + 2];
        double* tmp = w.C + (int64_t)p * p;
        if ((st = gemm_cc_f64(R, p, cores[l + 1], ncols, tmp, ncols, p, ncols, p, s)) != LRC_OK) return st;
        e = cudaMemcpyAsync(cores[l + 1], tmp, sizeof(double) * (size_t)(p * ncols), cudaMemcpyDeviceToDevice, s);
        if (e != cudaSuccess) return cuda_fail(e, "left-orthogonalization core update");
    }
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "left-orthogonalization");
    return LRC_OK;
}

}  // namespace lrc
