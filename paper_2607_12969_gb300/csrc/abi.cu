// abi.cu -- the extern "C" entry points of liblrc.so: argument validation,
// dispatch to the kernels, and the host-side certificate / storage helpers.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <atomic>
#include <mutex>

#include "common.cuh"

namespace lrc {

static thread_local char g_msg[512] = "";
static std::atomic<uint64_t> g_launches{0};

void set_error(const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof g_msg, fmt, ap);
    va_end(ap);
}

lrc_status cuda_fail(cudaError_t e, const char* what) {
    set_error("%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
    return LRC_ERR_CUDA;
}

lrc_status after_launch(const char* what) {
    g_launches.fetch_add(1, std::memory_order_relaxed);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, what);
    return LRC_OK;
}

int sm_count() {
    static std::mutex mu;
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
    std::lock_guard<std::mutex> lock(mu);
    if (cache[dev] == 0) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        cache[dev] = v > 0 ? v : 1;
    }
    return cache[dev];
}

static lrc_status invalid(const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof g_msg, fmt, ap);
    va_end(ap);
    return LRC_ERR_INVALID_ARG;
}

static lrc_status misaligned(const char* name) {
    set_error("%s is not 16-byte aligned", name);
    return LRC_ERR_ALIGNMENT;
}

// Validates a TT shape (Sec. 5.1: ranks r_0 = r_d = 1, core l of size
// r_{l-1} x n_l x r_l) and fills *sh; `es` is the element size of the cores.
static lrc_status tt_shape(const void* const* cores, const int64_t* dims, const int64_t* ranks, int d,
                           int64_t es, const char* what, TTShape* sh) {
    if (!cores || !dims || !ranks) return invalid("null pointer");
    if (d < 2 || d > 16) return invalid("d must be in [2, 16] (d=%d)", d);
    if (ranks[0] != 1 || ranks[d] != 1) return invalid("ranks[0] and ranks[d] must be 1");
    sh->d = d;
    int64_t numel = 1;
    for (int l = 0; l < d; ++l) {
        if (dims[l] <= 0) return invalid("dims[%d] = %lld must be positive", l, (long long)dims[l]);
        if (ranks[l] <= 0 || ranks[l] > 4096) return invalid("ranks[%d] out of range", l);
        if (!cores[l]) return invalid("%s[%d] is null", what, l);
        if ((reinterpret_cast<uintptr_t>(cores[l]) % (uintptr_t)es) != 0) {
            set_error("%s[%d] is not aligned to its element size", what, l);
            return LRC_ERR_ALIGNMENT;
        }
        int64_t c;
        if (!mul_ok(ranks[l], dims[l], &c) || !mul_ok(c, ranks[l + 1], &c) || !mul_ok(c, 8, &c))
            return invalid("core %d size overflow", l);
        if (!mul_ok(numel, dims[l], &numel)) return invalid("tensor size overflow");
        sh->dims[l] = dims[l];
        sh->ranks[l] = ranks[l];
        sh->cores[l] = cores[l];
    }
    sh->ranks[d] = 1;
    sh->numel = numel;
    return LRC_OK;
}

}  // namespace lrc

using namespace lrc;

extern "C" {

int64_t lrc_packed_ld(int64_t cols) {
    if (cols < 0 || cols > INT64_MAX - 15) return -1;
    return (cols + 15) / 16 * 16;
}

lrc_status lrc_round_factors(const double* src, int64_t rows, int64_t cols, int64_t ld_src,
                             void* dst, int64_t ld_dst, lrc_fmt fmt, lrc_stream_t stream) {
    if (!valid_fmt(fmt)) return invalid("unknown format %d", (int)fmt);
    fmt = plain_fmt(fmt);
    if (rows < 0 || cols < 0) return invalid("negative size (rows=%lld cols=%lld)", (long long)rows, (long long)cols);
    if (ld_src < cols || ld_dst < cols) return invalid("leading dimension below cols");
    if (rows == 0 || cols == 0) return LRC_OK;
    int64_t t;
    if (!mul_ok(rows, ld_src, &t) || !mul_ok(rows, ld_dst, &t) || !mul_ok(t, 8, &t))
        return invalid("size overflow");
    if (!src || !dst) return invalid("null pointer");
    if (!aligned16(src)) return misaligned("src");
    if (!aligned16(dst)) return misaligned("dst");
    return launch_round(src, rows, cols, ld_src, dst, ld_dst, fmt, as_stream(stream));
}

lrc_status lrc_widen_factors(const void* src, lrc_fmt fmt, int64_t rows, int64_t cols,
                             int64_t ld_src, double* dst, int64_t ld_dst, lrc_stream_t stream) {
    if (!valid_fmt(fmt)) return invalid("unknown format %d", (int)fmt);
    fmt = plain_fmt(fmt);
    if (rows < 0 || cols < 0) return invalid("negative size");
    if (ld_src < cols || ld_dst < cols) return invalid("leading dimension below cols");
    if (rows == 0 || cols == 0) return LRC_OK;
    int64_t t;
    if (!mul_ok(rows, ld_src, &t) || !mul_ok(rows, ld_dst, &t) || !mul_ok(t, 8, &t))
        return invalid("size overflow");
    if (!src || !dst) return invalid("null pointer");
    if (!aligned16(src)) return misaligned("src");
    if (!aligned16(dst)) return misaligned("dst");
    return launch_widen(src, fmt, rows, cols, ld_src, dst, ld_dst, as_stream(stream));
}

}  // extern "C"

namespace {

// Checks of one apply (sizes, overflow, pointers, alignment) before anything
// is launched.
lrc_status check_apply(const void* U, const void* S, const void* Vt, const void* X, const void* Y, int64_t m,
                       int64_t n, int64_t k, int64_t b) {
    if (m <= 0 || n <= 0 || k <= 0 || b <= 0)
        return invalid("sizes must be positive (m=%lld n=%lld k=%lld b=%lld)", (long long)m,
                       (long long)n, (long long)k, (long long)b);
    int64_t t;
    const int64_t ldk = lrc_packed_ld(k), ldn = lrc_packed_ld(n);
    if (ldk < 0 || ldn < 0 || !mul_ok(m, ldk, &t) || !mul_ok(t, 8, &t) || !mul_ok(k, ldn, &t) ||
        !mul_ok(t, 8, &t) || !mul_ok(b, ldn, &t) || !mul_ok(t, 8, &t) || !mul_ok(b, m, &t) ||
        !mul_ok(t, 8, &t))
        return invalid("size overflow");
    if (!U || !S || !Vt || !X || !Y) return invalid("null pointer");
    if (!aligned16(U)) return misaligned("U");
    if (!aligned16(S)) return misaligned("S");
    if (!aligned16(Vt)) return misaligned("Vt");
    if (!aligned16(X)) return misaligned("X");
    if (!aligned16(Y)) return misaligned("Y");
    return LRC_OK;
}

lrc_status dispatch_apply(const ApplyProblem& p, lrc_fmt fmt, cudaStream_t s) {
    if (apply_skinny_takes(plain_fmt(fmt), p.m, p.n, p.k, p.b))
        return launch_apply_skinny(p.U, p.S, p.Vt, p.X, p.Y, p.m, p.n, p.k, p.b, plain_fmt(fmt), s);
    switch (fmt) {
        case LRC_F64:
            return launch_apply_f64((const double*)p.U, (const double*)p.S, (const double*)p.Vt, (const double*)p.X,
                                    (double*)p.Y, p.m, p.n, p.k, p.b, s);
        case LRC_F32:
        case LRC_F32_TC:
            return launch_apply_f32((const float*)p.U, (const float*)p.S, (const float*)p.Vt, (const float*)p.X,
                                    (float*)p.Y, p.m, p.n, p.k, p.b, fmt == LRC_F32_TC, s);
        case LRC_F16:
        case LRC_F16_O16:
            return launch_apply_f16(p.U, p.S, p.Vt, p.X, p.Y, p.m, p.n, p.k, p.b, fmt == LRC_F16_O16, s);
        case LRC_BF16:
            return launch_apply_f16(p.U, p.S, p.Vt, p.X, p.Y, p.m, p.n, p.k, p.b, true, s, true);
    }
    return invalid("unknown format");
}

}  // namespace

extern "C" {

lrc_status lrc_apply(const void* U, const void* S, const void* Vt, const void* X, void* Y,
                     int64_t m, int64_t n, int64_t k, int64_t b, lrc_fmt fmt,
                     lrc_stream_t stream) {
    if (!valid_fmt(fmt)) return invalid("unknown format %d", (int)fmt);
    lrc_status st = check_apply(U, S, Vt, X, Y, m, n, k, b);
    if (st != LRC_OK) return st;
    return dispatch_apply(ApplyProblem{U, S, Vt, X, Y, m, n, k, b}, fmt, as_stream(stream));
}

lrc_status lrc_apply_batched(int count, const void* const* U, const void* const* S, const void* const* Vt,
                             const void* const* X, void* const* Y, const int64_t* m, const int64_t* n,
                             const int64_t* k, const int64_t* b, lrc_fmt fmt, lrc_stream_t stream) {
    if (!valid_fmt(fmt)) return invalid("unknown format %d", (int)fmt);
    if (count < 0 || count > 4096) return invalid("count must be in [0, 4096] (got %d)", count);
    if (count == 0) return LRC_OK;
    if (!U || !S || !Vt || !X || !Y || !m || !n || !k || !b) return invalid("null array");
    for (int p = 0; p < count; ++p) {
        lrc_status st = check_apply(U[p], S[p], Vt[p], X[p], Y[p], m[p], n[p], k[p], b[p]);
        if (st != LRC_OK) {
            char msg[256];
            snprintf(msg, sizeof msg, "%s", lrc_last_error());
            set_error("problem %d: %s", p, msg);
            return st;
        }
        if ((fmt == LRC_F16 || fmt == LRC_F16_O16 || fmt == LRC_BF16) && k[p] > 512) {
            set_error("problem %d: binary16 / bfloat16 ranks up to 512 (got %lld)", p, (long long)k[p]);
            return LRC_ERR_UNSUPPORTED;
        }
    }
    cudaStream_t s = as_stream(stream);
    ApplyProblem pr[64];
    if (fmt == LRC_F16 || fmt == LRC_F16_O16 || fmt == LRC_BF16) {
        // tensor-core formats: one launch per phase for every group of problems
        const int gmax = apply_f16_group_max();
        for (int p0 = 0; p0 < count; p0 += gmax) {
            const int c = count - p0 < gmax ? count - p0 : gmax;
            for (int i = 0; i < c; ++i)
                pr[i] = ApplyProblem{U[p0 + i], S[p0 + i], Vt[p0 + i], X[p0 + i], Y[p0 + i],
                                     m[p0 + i], n[p0 + i], k[p0 + i], b[p0 + i]};
            lrc_status st = launch_apply_f16_group(pr, c, fmt != LRC_F16, fmt == LRC_BF16, s);
            if (st != LRC_OK) return st;
        }
        return LRC_OK;
    }
    for (int p = 0; p < count; ++p) {
        lrc_status st = dispatch_apply(ApplyProblem{U[p], S[p], Vt[p], X[p], Y[p], m[p], n[p], k[p], b[p]}, fmt, s);
        if (st != LRC_OK) return st;
    }
    return LRC_OK;
}

lrc_status tt_reconstruct(const void* const* cores, const int64_t* dims, const int64_t* ranks,
                          int d, lrc_fmt fmt, void* out, lrc_stream_t stream) {
    if (!valid_fmt(fmt)) return invalid("unknown format %d", (int)fmt);
    if (!out) return invalid("null pointer");
    TTShape sh;
    lrc_status st = tt_shape(cores, dims, ranks, d, storage_bytes(fmt), "cores", &sh);
    if (st != LRC_OK) return st;
    int64_t t;
    if (!mul_ok(sh.numel, 8, &t)) return invalid("tensor size overflow");
    if (!aligned16(out)) return misaligned("out");
    cudaStream_t s = as_stream(stream);
    if (fmt == LRC_F16 || fmt == LRC_F16_O16) return launch_tt_f16(sh, fmt == LRC_F16_O16, out, s);
    if (fmt == LRC_BF16) return launch_tt_bf16(sh, out, s);
    if (fmt == LRC_F32_TC) {
        bool handled = false;
        st = launch_tt_split_f32tc(sh, static_cast<float*>(out), s, &handled);
        if (st != LRC_OK || handled) return st;
        return launch_tt_chain_f32tc(sh, static_cast<float*>(out), s);
    }
    if (fmt == LRC_F32 || fmt == LRC_F32_TC) return launch_tt_chain_f32(sh, static_cast<float*>(out), s);
    if (tt_chain_saves(sh)) return launch_tt_chain_f64(sh, static_cast<double*>(out), s);
    return launch_tt_cc(sh, fmt, out, s);
}

lrc_status tt_gather(const void* const* cores, const int64_t* dims, const int64_t* ranks, int d, lrc_fmt fmt,
                     const int64_t* idx, int64_t count, void* out, lrc_stream_t stream) {
    if (!valid_fmt(fmt)) return invalid("unknown format %d", (int)fmt);
    fmt = plain_fmt(fmt);
    if (count < 0) return invalid("negative count");
    TTShape sh;
    lrc_status st = tt_shape(cores, dims, ranks, d, storage_bytes(fmt), "cores", &sh);
    if (st != LRC_OK) return st;
    for (int l = 0; l <= d; ++l)
        if (ranks[l] > tt_gather_max_rank()) {
            set_error("tt_gather supports ranks up to %d (ranks[%d] = %lld)", tt_gather_max_rank(), l,
                      (long long)ranks[l]);
            return LRC_ERR_UNSUPPORTED;
        }
    if (count == 0) return LRC_OK;
    if (!idx || !out) return invalid("null pointer");
    int64_t t;
    if (!mul_ok(count, 8, &t)) return invalid("size overflow");
    if ((reinterpret_cast<uintptr_t>(idx) & 7u) != 0) {
        set_error("idx is not 8-byte aligned");
        return LRC_ERR_ALIGNMENT;
    }
    const uintptr_t oa = (fmt == LRC_F16_O16 || fmt == LRC_BF16) ? 2u : (fmt == LRC_F64 ? 8u : 4u);
    if ((reinterpret_cast<uintptr_t>(out) % oa) != 0) {
        set_error("out is not aligned to its element size");
        return LRC_ERR_ALIGNMENT;
    }
    return launch_tt_gather(sh, fmt, idx, count, out, as_stream(stream));
}

lrc_status lrc_lowrank_eta(const double* U, const double* S, const double* Vt, const void* Uh, const void* Sh,
                           const void* Vht, lrc_fmt fmt, int64_t m, int64_t n, int64_t k, double* eta_out,
                           double* norm_out, lrc_stream_t stream) {
    if (!valid_fmt(fmt)) return invalid("unknown format %d", (int)fmt);
    fmt = plain_fmt(fmt);
    if (m <= 0 || n <= 0 || k <= 0)
        return invalid("sizes must be positive (m=%lld n=%lld k=%lld)", (long long)m, (long long)n, (long long)k);
    if (k > 4096) return invalid("k = %lld exceeds 4096", (long long)k);
    int64_t t;
    const int64_t ldk = lrc_packed_ld(k), ldn = lrc_packed_ld(n);
    if (!mul_ok(m, ldk, &t) || !mul_ok(t, 8, &t) || !mul_ok(k, ldn, &t) || !mul_ok(t, 8, &t) ||
        !mul_ok(m + n, 2 * k, &t) || !mul_ok(t, 8, &t))
        return invalid("size overflow");
    if (!U || !S || !Vt || !Uh || !Sh || !Vht || !eta_out) return invalid("null pointer");
    if (!aligned16(U)) return misaligned("U");
    if (!aligned16(S)) return misaligned("S");
    if (!aligned16(Vt)) return misaligned("Vt");
    if (!aligned16(Uh)) return misaligned("Uh");
    if (!aligned16(Sh)) return misaligned("Sh");
    if (!aligned16(Vht)) return misaligned("Vht");
    return run_lowrank_eta(U, S, Vt, Uh, Sh, Vht, fmt, m, n, k, eta_out, norm_out, as_stream(stream));
}

lrc_status lrc_tt_eta(const double* const* cores, const void* const* cores_hat, const int64_t* dims,
                      const int64_t* ranks, int d, lrc_fmt fmt, double* eta_out, double* norm_out,
                      lrc_stream_t stream) {
    if (!valid_fmt(fmt)) return invalid("unknown format %d", (int)fmt);
    fmt = plain_fmt(fmt);
    if (!eta_out) return invalid("null eta_out");
    TTShape sh, shh;
    lrc_status st = tt_shape((const void* const*)cores, dims, ranks, d, 8, "cores", &sh);
    if (st != LRC_OK) return st;
    st = tt_shape(cores_hat, dims, ranks, d, storage_bytes(fmt), "cores_hat", &shh);
    if (st != LRC_OK) return st;
    for (int l = 0; l < d; ++l) {
        int64_t c;
        // block cores of an interior level: 2 r_l x n_l x 2 r_{l+1} binary64, twice
        if (!mul_ok(4 * ranks[l] * dims[l], ranks[l + 1], &c) || !mul_ok(c, 16, &c))
            return invalid("core %d too large for eta_TT", l);
    }
    return run_tt_eta(sh, shh.cores, fmt, eta_out, norm_out, as_stream(stream));
}

lrc_status lrc_fro_diff(const void* A, lrc_fmt fa, const void* B, lrc_fmt fb, int64_t count,
                        double* diff_out, double* normA_out, lrc_stream_t stream) {
    if (!valid_fmt(fa) || !valid_fmt(fb)) return invalid("unknown format");
    fa = plain_fmt(fa);
    fb = plain_fmt(fb);
    if (count < 0) return invalid("negative count");
    if (!diff_out) return invalid("null diff_out");
    int64_t t;
    if (!mul_ok(count, 8, &t)) return invalid("size overflow");
    if (count > 0 && !A) return invalid("null A");
    if (count > 0 && !aligned16(A)) return misaligned("A");
    if (B && !aligned16(B)) return misaligned("B");
    if (count == 0) {
        *diff_out = 0.0;
        if (normA_out) *normA_out = 0.0;
        return LRC_OK;
    }
    return run_fro_diff(A, fa, B, fb, count, diff_out, normA_out, as_stream(stream));
}

lrc_status lrc_fro_diff_noalloc(const void* A, lrc_fmt fa, const void* B, lrc_fmt fb, int64_t count,
                                double* diff_out, double* normA_out, lrc_stream_t stream) {
    if (!valid_fmt(fa) || !valid_fmt(fb)) return invalid("unknown format");
    fa = plain_fmt(fa);
    fb = plain_fmt(fb);
    if (count < 0) return invalid("negative count");
    if (!diff_out) return invalid("null diff_out");
    if (count > fro_diff_noalloc_max_count())
        return invalid("lrc_fro_diff_noalloc handles at most %lld elements (got %lld)",
                       (long long)fro_diff_noalloc_max_count(), (long long)count);
    if (count > 0 && !A) return invalid("null A");
    if (count > 0 && !aligned16(A)) return misaligned("A");
    if (B && !aligned16(B)) return misaligned("B");
    if (count == 0) {
        *diff_out = 0.0;
        if (normA_out) *normA_out = 0.0;
        return LRC_OK;
    }
    return run_fro_diff_noalloc(A, fa, B, fb, count, diff_out, normA_out, as_stream(stream));
}

int lrc_certified(double e_base, double e_aug, double eta) { return (e_aug + eta <= e_base) ? 1 : 0; }

double lrc_tail_error(const double* sigma, int64_t len, int64_t k) {
    if (!sigma || len < 0 || k < 0) return -1.0;
    // ascending order (smallest singular values first), compensated
    double s = 0.0, c = 0.0;
    for (int64_t j = len - 1; j >= k; --j) {
        const double term = sigma[j] * sigma[j];
        const double u = s + term;
        c += (fabs(s) >= fabs(term)) ? ((s - u) + term) : ((term - u) + s);
        s = u;
    }
    return sqrt(s + c);
}

double lrc_matrix_storage_ratio(int64_t m, int64_t n, int64_t k_base, int64_t k_aug, lrc_fmt fmt) {
    if (m <= 0 || n <= 0 || k_base <= 0 || k_aug <= 0 || !valid_fmt(fmt)) return -1.0;
    const double per = (double)(m + n + 1);
    return ((double)storage_bytes(fmt) * (double)k_aug * per) / (8.0 * (double)k_base * per);
}

double lrc_tt_storage_bytes(const int64_t* dims, const int64_t* ranks, int d, lrc_fmt fmt) {
    if (!dims || !ranks || d < 1 || !valid_fmt(fmt)) return -1.0;
    double s = 0.0;
    for (int l = 0; l < d; ++l) s += (double)ranks[l] * (double)dims[l] * (double)ranks[l + 1];
    return s * (double)storage_bytes(fmt);
}

const char* lrc_status_string(lrc_status st) {
    switch (st) {
        case LRC_OK: return "ok";
        case LRC_ERR_INVALID_ARG: return "invalid argument";
        case LRC_ERR_ALIGNMENT: return "misaligned pointer";
        case LRC_ERR_UNSUPPORTED: return "unsupported";
        case LRC_ERR_CUDA: return "CUDA error";
        case LRC_ERR_NOMEM: return "out of memory";
        case LRC_ERR_TIMEOUT: return "device wait timed out";
    }
    return "unknown status";
}

const char* lrc_last_error(void) { return g_msg; }

uint64_t lrc_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

lrc_status lrc_device_status(lrc_stream_t stream) {
    cudaError_t e = cudaStreamSynchronize(as_stream(stream));
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    const uint32_t a = take_apply_tc_error();
    const uint32_t t1 = take_tt_tc_error();
    const uint32_t t3 = take_tt3_tc_error();
    const uint32_t tn = take_ttn_tc_error();
    const uint32_t sk = take_skinny_error();
    const uint32_t t = t1 | t3 | tn;
    if (a == 0xffffffffu || t1 == 0xffffffffu || t3 == 0xffffffffu || tn == 0xffffffffu || sk == 0xffffffffu) {
        set_error("could not read the device error words");
        return LRC_ERR_CUDA;
    }
    if (a | t | sk) {
        set_error("a bounded device wait gave up (apply code 0x%x, TT code 0x%x, small-batch apply code 0x%x)", a,
                  t, sk);
        return LRC_ERR_TIMEOUT;
    }
    return LRC_OK;
}

lrc_status lrc_selftest_wait_timeout(int64_t limit_ns, lrc_stream_t stream) {
    if (limit_ns <= 0 || limit_ns > 1000000000LL) return invalid("limit_ns must be in (0, 1e9]");
    return launch_wait_timeout_probe(limit_ns, as_stream(stream));
}

lrc_status lrc_tt_svd(const double* T, const int64_t* dims, const int64_t* ranks, int d, double* const* cores,
                      double* delta2_out, double* spectra_out, lrc_stream_t stream) {
    TTShape sh;
    lrc_status st = tt_shape((const void* const*)cores, dims, ranks, d, 8, "cores", &sh);
    if (st != LRC_OK) return st;
    if (!T) return invalid("null T");
    if ((reinterpret_cast<uintptr_t>(T) & 7u) != 0) return misaligned("T");
    int64_t rest = sh.numel;
    for (int l = 0; l < d - 1; ++l) {
        rest /= dims[l];
        const int64_t rows = ranks[l] * dims[l], p = rows < rest ? rows : rest;
        if (ranks[l + 1] > p)
            return invalid("ranks[%d] = %lld exceeds the smaller side (%lld) of unfolding %d", l + 1,
                           (long long)ranks[l + 1], (long long)p, l + 1);
        if (p > factor_max_cols()) {
            set_error("TT-SVD: unfolding %d's smaller side is %lld; at most %d", l + 1, (long long)p,
                      factor_max_cols());
            return LRC_ERR_UNSUPPORTED;
        }
    }
    int64_t t;
    if (!mul_ok(sh.numel, 16, &t)) return invalid("tensor too large");
    return run_tt_svd(T, sh, cores, delta2_out, spectra_out, as_stream(stream));
}

lrc_status lrc_tt_left_orthogonalize(double* const* cores, const int64_t* dims, const int64_t* ranks, int d,
                                     lrc_stream_t stream) {
    TTShape sh;
    lrc_status st = tt_shape((const void* const*)cores, dims, ranks, d, 8, "cores", &sh);
    if (st != LRC_OK) return st;
    for (int l = 0; l < d - 1; ++l) {
        if (ranks[l + 1] > ranks[l] * dims[l])
            return invalid("ranks[%d] = %lld exceeds ranks[%d] * dims[%d] = %lld", l + 1, (long long)ranks[l + 1], l,
                           l, (long long)(ranks[l] * dims[l]));
        if (ranks[l + 1] > factor_max_cols()) {
            set_error("left-orthogonalization: rank %lld above %d", (long long)ranks[l + 1], factor_max_cols());
            return LRC_ERR_UNSUPPORTED;
        }
    }
    return run_tt_left_orthogonalize(sh, cores, as_stream(stream));
}

lrc_status lrc_probe_peak(int kind, int64_t iters, double* flops_out, lrc_stream_t stream) {
    if (kind < 0 || kind > 3) return invalid("kind must be 0..3");
    if (iters < 1 || iters > (1LL << 30)) return invalid("iters must be in [1, 2^30]");
    if (!flops_out) return invalid("null flops_out");
    return run_probe_peak(kind, iters, flops_out, as_stream(stream));
}

lrc_status lrc_shutdown(void) {
    release_scratch();
    release_workspaces();
    return LRC_OK;
}

}  // extern "C"
