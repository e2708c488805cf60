/*
 * lrc.h -- C ABI of the GB300 (sm_103a) rank-compensation hot path.
 *
 * The library implements the resident downstream kernels of "Low-Precision
 * Rank Compensation for Matrices and Tensor Trains": factor rounding, the
 * batched low-rank apply, dense Tensor-Train reconstruction, and the
 * Frobenius-difference reduction that measures the storage perturbation eta
 * used by the certificates of Thm 4.1 and Thm 6.1.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - All arrays are C order (row-major).  "Device" pointers are CUDA global
 *    memory addresses of the current device; "host" pointers are ordinary
 *    process memory.  The caller owns every buffer; the library keeps no
 *    pointer after a call returns.
 *  - `stream` is a cudaStream_t passed as an opaque pointer (NULL = the
 *    legacy default stream).  Calls are asynchronous on it unless stated.
 *  - Every argument is validated before anything is launched; on a
 *    validation error nothing is written and the call returns a negative
 *    lrc_status.  A failed launch returns LRC_ERR_CUDA.  Faults of a kernel
 *    that already ran surface at the next synchronising call, as in CUDA.
 *    lrc_last_error() gives a message for the last failure of the calling
 *    thread.
 *  - Sizes are int64_t; products of sizes must not overflow int64.
 *  - The library never traps and has no CPU fallback: it needs an sm_103a
 *    GPU.  Device scratch is allocated only where an entry point says so
 *    (library workspaces, allocated on first use and reused).
 *  - Stream order holds as for any kernel: work the caller enqueues after a
 *    call starts after the call's kernels have completed.  Inside a call the
 *    kernels are chained by programmatic dependent launch, and the last
 *    kernel of a call may let the next kernel of the stream begin its
 *    prologue early; that only affects a caller's own kernel launched with
 *    the programmatic-serialization attribute, which (as CUDA requires of
 *    such a kernel) must execute griddepcontrol.wait before it reads the
 *    call's outputs.  A library kernel launched that way reads memory an
 *    earlier kernel of the stream may have written only after its
 *    griddepcontrol.wait, or after a kernel of its own call that has
 *    already waited for everything before the call.
 */
#ifndef LRC_H
#define LRC_H

#include <stdint.h>

#if defined(__GNUC__)
#define LRC_API __attribute__((visibility("default")))
#else
#define LRC_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Storage / arithmetic formats (Sec. 3.2, Table "precision comparison";
 * Sec. 3.4: FP16 products accumulate in FP32, TF32 is never used). */
typedef enum {
    LRC_F64 = 0,      /* binary64 storage, binary64 arithmetic, binary64 output             */
    LRC_F32 = 1,      /* binary32 storage, binary32 FMA arithmetic, binary32 output         */
    LRC_F16 = 2,      /* binary16 storage, binary32 accumulation, binary32 output           */
    LRC_F16_O16 = 3,  /* binary16 storage, binary32 accumulation, binary16 workspaces and
                         output: the method-precision FP16 path of Sec. 3.4                 */
    LRC_F32_TC = 4,   /* binary32 storage and output; the output product of lrc_apply and
                         tt_reconstruct on the tensor cores: each binary32 operand is scaled
                         by a power of two per 32 rows and split into binary16 parts
                         hi + lo, and Z S ~ Z_hi S_hi + Z_lo S_hi + Z_hi S_lo accumulates in
                         binary32 (about 22 significand bits per operand).  A variant of
                         LRC_F32; every other call treats it as LRC_F32                      */
    LRC_BF16 = 5      /* bfloat16 storage (8 significand bits, binary32's exponent range:
                         Sec. 3.2 precision table), binary32 accumulation, bfloat16
                         workspaces and output: the method-precision policy of Sec. 3.4
                         applied to bfloat16                                                  */
} lrc_fmt;

typedef enum {
    LRC_OK = 0,
    LRC_ERR_INVALID_ARG = -1,   /* null pointer, size <= 0, overflow, bad rank vector ... */
    LRC_ERR_ALIGNMENT = -2,     /* a pointer is not 16-byte aligned                       */
    LRC_ERR_UNSUPPORTED = -3,   /* valid request outside what this build implements       */
    LRC_ERR_CUDA = -4,          /* a CUDA call or launch failed                           */
    LRC_ERR_NOMEM = -5,         /* library scratch could not be allocated                 */
    LRC_ERR_TIMEOUT = -6        /* a bounded device-side wait gave up                     */
} lrc_status;

typedef void* lrc_stream_t;     /* cudaStream_t */

/* Row pitch (in elements) of a packed factor with `cols` logical columns:
 * cols rounded up to a multiple of 16, so that every row starts on a
 * 16-byte boundary in every format.  Returns -1 for cols < 0. */
LRC_API int64_t lrc_packed_ld(int64_t cols);

/*
 * lrc_round_factors -- store a factor in a lower precision (Sec. 3.2-3.3;
 * the remark after Thm 4.1: U, Sigma and V^T are rounded individually, and
 * Alg. 1 step 4 rounds TT cores).
 *
 *   src     device, binary64, rows x cols with row pitch ld_src (>= cols)
 *   dst     device, rows x ld_dst elements of the format `fmt`
 *           (LRC_F64: binary64 copy; LRC_F32: binary32; LRC_F16 and
 *           LRC_F16_O16: binary16)
 *   ld_dst  row pitch of dst in elements, >= cols
 *
 * Each element is converted directly from binary64 with IEEE 754
 * round-to-nearest, ties to even (no intermediate format), subnormals kept,
 * overflow to +-infinity, NaN to a quiet NaN of the same sign.  Columns
 * [cols, ld_dst) of every dst row are written with +0.  src and dst must be
 * 16-byte aligned; rows*ld of either may be zero only if rows or cols is 0
 * (then nothing happens).
 */
LRC_API lrc_status lrc_round_factors(const double* src, int64_t rows, int64_t cols, int64_t ld_src,
                             void* dst, int64_t ld_dst, lrc_fmt fmt, lrc_stream_t stream);

/*
 * lrc_widen_factors -- exact binary64 value of a stored factor, so that the
 * rounded factors can be contracted in FP64 as the paper does for eta
 * (remark after Thm 4.1; Sec. 6.1: rounded cores reconstructed in FP64).
 *
 *   src     device, rows x cols, row pitch ld_src, format `fmt`
 *   dst     device, binary64, rows x ld_dst; columns [cols, ld_dst) get +0
 */
LRC_API lrc_status lrc_widen_factors(const void* src, lrc_fmt fmt, int64_t rows, int64_t cols,
                             int64_t ld_src, double* dst, int64_t ld_dst, lrc_stream_t stream);

/*
 * lrc_apply -- batched low-rank apply (Sec. 4.4, Eq. gpu_matrix_apply):
 *
 *     Y = [(X V) diag(s)] U^T,   i.e. Y^T = U (diag(s) (V^T X^T)),
 *
 * with the factors of a rank-k approximation A_k = U diag(s) V^T of an
 * m x n matrix, applied to b queries at once.
 *
 *   U    device, m x k, row pitch lrc_packed_ld(k)
 *   S    device, k singular values s_1..s_k
 *   Vt   device, V^T: k x n, row pitch lrc_packed_ld(n)
 *   X    device, b x n queries (one per row), row pitch lrc_packed_ld(n)
 *   Y    device, b x m results, row pitch m
 *
 * Element types: LRC_F64 -> U, S, Vt, X, Y binary64; LRC_F32 -> all
 * binary32; LRC_F16 -> U, S, Vt, X binary16 and Y binary32; LRC_F16_O16 ->
 * all binary16 (the intermediate is rounded to binary16 as well); LRC_BF16
 * -> all bfloat16 (intermediate too), on the tensor-core path at every b.  Pad
 * columns of U, Vt and X are never read.  All five pointers must be 16-byte
 * aligned.  k may exceed min(m, n).  Asynchronous on `stream`.
 *
 * Intermediate: for LRC_F64 and LRC_F32 the b x k product (X V) diag(s)
 * stays in shared memory.  For LRC_F16 and LRC_F16_O16 the reduction over n
 * is split over all multiprocessors, so its partial sums and the scaled
 * intermediate (binary16, a hi/lo pair for LRC_F16) pass through a device
 * workspace owned by the library: one buffer per (device, stream),
 * allocated on first use and reallocated -- after synchronizing `stream` --
 * when a larger problem arrives, freed by lrc_shutdown().  Calls on
 * different streams use different buffers.  Small batches add their
 * per-chunk partial sums in the same workspace and keep a per-stream buffer
 * of 1024 arrival counters (zeroed once when made, left at zero by every
 * call, freed by lrc_shutdown()): at most 16 queries in binary64 and
 * binary32 on the CUDA cores (binary16 too when the tensor-core products
 * do not take the shape), and up to 64 queries in binary16 and bfloat16 as
 * two tensor-core products when n <= 32768 and k <= 512 (the second
 * product's tiles must fit in shared memory).  Binary16 ranks: up to 512,
 * and up to 320 for LRC_F16 where the small-batch tensor-core products do
 * not take the call (more than 64 queries, n > 32768), else
 * LRC_ERR_UNSUPPORTED.
 */
/* LRC_F32_TC: as LRC_F32, with the second product (W U^T) on the tensor
 * cores when b > 32 and k <= 192; otherwise the LRC_F32 kernels. */
LRC_API lrc_status lrc_apply(const void* U, const void* S, const void* Vt, const void* X, void* Y,
                     int64_t m, int64_t n, int64_t k, int64_t b, lrc_fmt fmt,
                     lrc_stream_t stream);

/*
 * lrc_apply_batched -- `count` independent applies of lrc_apply in one call:
 * problem p applies its own rank-k[p] factors U[p], S[p], Vt[p] of an
 * m[p] x n[p] matrix to its own b[p] queries X[p], writing Y[p].  The paper
 * times its matrix applies aggregated over a set of matrices (Sec. 4.4, ten
 * matrices per measurement); this is that aggregate as one call.
 *
 *   U, S, Vt, X, Y   HOST arrays of `count` DEVICE pointers, each with the
 *                    layout, element type and alignment of lrc_apply
 *   m, n, k, b       HOST arrays of `count` sizes
 *   fmt              one format for every problem
 *
 * LRC_F16, LRC_F16_O16 and LRC_BF16: the problems share the tensor-core
 * kernels' launches -- one launch per phase for up to 16 problems (the
 * multiprocessors are divided among the problems in proportion to their
 * work; larger counts take one set of launches per 16), and every batch size
 * takes the tensor-core path.  Other formats: the problems are launched one
 * after another as lrc_apply would.  Results equal lrc_apply's on each
 * problem up to the summation order of the split reduction (same tolerance).
 * 0 <= count <= 4096.  Every problem is validated before anything is
 * launched; the message of a failure names the problem.  Workspace: the
 * stream's library workspace, the sum of the problems' (see lrc_apply).
 * Asynchronous on `stream`.
 */
LRC_API lrc_status lrc_apply_batched(int count, const void* const* U, const void* const* S, const void* const* Vt,
                                     const void* const* X, void* const* Y, const int64_t* m, const int64_t* n,
                                     const int64_t* k, const int64_t* b, lrc_fmt fmt, lrc_stream_t stream);

/*
 * tt_reconstruct -- dense Tensor-Train reconstruction (Sec. 5.1:
 * T(i_1..i_d) = G_1(i_1) ... G_d(i_d); Sec. 7.5, Eq. gpu_tt_reconstruction:
 * the chain B_l = Z_{l-1} K_l, Z_l = reshape(B_l)).
 *
 *   cores   HOST array of d DEVICE pointers; cores[l] holds G_{l+1}, an
 *           unpadded C-order ranks[l] x dims[l] x ranks[l+1] array
 *   dims    host, d mode sizes n_1..n_d (> 0)
 *   ranks   host, d+1 TT ranks with ranks[0] = ranks[d] = 1 (> 0)
 *   d       number of cores, 2 <= d <= 16
 *   out     device, prod(dims) entries in C order (i_1 slowest): the
 *           vectorised tensor of Eq. gpu_tt_reconstruction
 *
 * Element types: LRC_F64 cores/out binary64; LRC_F32 binary32; LRC_F16
 * binary16 cores, binary32 out; LRC_F16_O16 binary16 cores, workspaces and
 * out.  Cores must be aligned to their element size, out to 16 bytes.
 * Intermediate products Z_l stay on chip.  Asynchronous on `stream`.
 */
/* LRC_F32_TC: binary32 cores and output; the chain's output product on the
 * tensor cores when the chain's sides fit its one-pass side kernel
 * (bond rank <= 64), otherwise the LRC_F32 kernels. */
LRC_API lrc_status tt_reconstruct(const void* const* cores, const int64_t* dims, const int64_t* ranks,
                          int d, lrc_fmt fmt, void* out, lrc_stream_t stream);

/*
 * tt_gather -- sampled entries T(i_1..i_d) = G_1(i_1) G_2(i_2) ... G_d(i_d)
 * of a Tensor Train (Sec. 5.1), each evaluated by its own core chain: the
 * independent check of a dense reconstruction on sampled entries.
 *
 *   cores, dims, ranks, d, fmt  as in tt_reconstruct; ranks up to 256, else
 *           LRC_ERR_UNSUPPORTED
 *   idx     device, `count` int64 flat indices into the C-order vectorised
 *           tensor (i_1 slowest), 8-byte aligned; an index outside
 *           [0, prod(dims)) yields a quiet NaN in its output slot
 *   count   number of entries, >= 0 (0: nothing is launched)
 *   out     device, `count` values: binary64 for LRC_F64, binary32 for
 *           LRC_F32 and LRC_F16, binary16 for LRC_F16_O16; aligned to the
 *           element size
 *
 * Arithmetic: binary64 FMA for LRC_F64; binary32 FMA for LRC_F32 and for
 * binary16 cores (products of binary16 values accumulated in binary32,
 * Sec. 3.4); LRC_F16_O16 rounds the binary32 result to binary16 once.
 * Entries are independent: duplicates and any order are allowed.
 * Asynchronous on `stream`.
 */
LRC_API lrc_status tt_gather(const void* const* cores, const int64_t* dims, const int64_t* ranks, int d,
                             lrc_fmt fmt, const int64_t* idx, int64_t count, void* out,
                             lrc_stream_t stream);

/*
 * lrc_fro_diff -- Frobenius norm of a difference (Sec. 5.1 "Frobenius norm";
 * eta of Thm 4.1 and eta_TT of Thm 6.1 are ||A_k' - Ahat_k'||_F and
 * ||T_R+ - That_R+||_F of the FP64 reconstructions).
 *
 *   A, B        device arrays of `count` elements in formats fa, fb
 *               (LRC_F64, LRC_F32, or LRC_F16 / LRC_F16_O16 = binary16);
 *               B may be NULL, meaning B = 0
 *   diff_out    host: sqrt(sum_i (A_i - B_i)^2), sums in binary64
 *   normA_out   host, may be NULL: sqrt(sum_i A_i^2)
 *
 * Arithmetic: differences are binary64.  When both inputs are binary64, each
 * square d^2 with 2^-48 <= |d| < 2^60 is formed from a binary32 pair split of
 * d (its leading 24 and next 23 significand bits; the last 6 bits are
 * dropped, a relative change of d of at most 2^-47) as an exact binary32
 * two-product plus correction terms, summed in binary32 pairs and flushed to
 * binary64 every 128 elements; other squares, and all squares of binary32 or
 * binary16 inputs, are binary64 FMAs.  The result is within about 2^-46
 * relative of the exactly rounded binary64 sum of squares.
 *
 * Summation is deterministic: fixed per-block partial sums reduced in a
 * fixed order, so repeated calls on the same data give identical bits.
 * Uses library-held device scratch (allocated on first use per device,
 * released by lrc_shutdown), so concurrent calls on different streams of
 * the same device must not overlap.  The two results are written by the
 * final kernel into a per-stream slot of mapped pinned host memory
 * (allocated on first use, released by lrc_shutdown) and read once the
 * stream has synchronised, so they never wait behind other copies on the
 * copy engines.  SYNCHRONISES `stream`.
 */
LRC_API lrc_status lrc_fro_diff(const void* A, lrc_fmt fa, const void* B, lrc_fmt fb, int64_t count,
                        double* diff_out, double* normA_out, lrc_stream_t stream);

/*
 * lrc_fro_diff_noalloc -- the same reduction as lrc_fro_diff for callers that
 * must not allocate device memory.  The paper has no counterpart: this is a
 * deployment variant.  Callers that run under a fixed device-memory budget
 * whose memory is owned by another allocator (a serving framework's caching
 * pool, say), or that cannot afford the implicit device synchronisation a
 * cudaMalloc can cause in the middle of a latency-critical loop, can use it:
 * it calls no cudaMalloc, cudaFree or other allocating routine.
 *
 * Arguments and results are those of lrc_fro_diff; A and B are still the
 * caller's buffers.  The per-block partial sums live in a fixed array of
 * 8194 doubles (about 64 KB) compiled into the library, which every GPU that
 * loads the library keeps until the process exits.  That array bounds the
 * input: count <= 268435456 (4096 blocks x 65536 elements); a larger count
 * returns LRC_ERR_INVALID_ARG without launching.  The first call on each
 * device looks up the array's device address (cudaGetSymbolAddress) with that
 * device current; make that first call before any stream capture.  All calls
 * share the one array and every call overwrites the entries it uses, so no
 * state carries over between calls, but calls whose kernels overlap on the
 * GPU (different streams, other threads) race on it and must be serialised by
 * the caller.  The looked-up address is cached per device; a caller that
 * resets a device (cudaDeviceReset) calls lrc_shutdown first, which forgets
 * it.  Synchronises `stream`.
 */
LRC_API lrc_status lrc_fro_diff_noalloc(const void* A, lrc_fmt fa, const void* B, lrc_fmt fb,
                                        int64_t count, double* diff_out, double* normA_out,
                                        lrc_stream_t stream);

/*
 * lrc_lowrank_eta -- eta = ||U diag(s) V^T - Uh diag(sh) Vh^T||_F, the
 * perturbation of Thm 4.1 (remark after it: the three factors are rounded
 * individually), without forming either m x n matrix.
 *
 *   U, S, Vt     device, the binary64 rank-k factors in the layout of
 *                lrc_apply: U m x k with row pitch lrc_packed_ld(k), S k
 *                values, Vt = V^T k x n with row pitch lrc_packed_ld(n)
 *   Uh, Sh, Vht  device, the stored factors in format `fmt`, same layout
 *                (what lrc_round_factors writes)
 *   eta_out      host: eta
 *   norm_out     host, may be NULL: ||U diag(s) V^T||_F
 *
 * With the rounding errors dU = U - Uh, dV = V - Vh, ds = s - sh (exact in
 * binary64) the difference is exactly [dU, Uh] M [dV, Vh]^T with
 * M = [[S, S], [S, dS]] (diagonal blocks), so eta^2 = tr(M^T Gu M Gv) with
 * the 2k x 2k Gram matrices Gu = [dU, Uh]^T [dU, Uh], Gv = [dV, Vh]^T
 * [dV, Vh].  Every term carries the rounding errors explicitly, so nothing
 * of the size of ||A|| cancels: the result is accurate relative to eta,
 * where the dense route (lrc_apply with X = I, lrc_fro_diff) is accurate
 * relative to ||A||.  Work: about 2 (m + n) k (2k + 1) binary64 flops.
 * All arithmetic binary64; deterministic on a device.  k <= 4096.  Pointers
 * 16-byte aligned.  Scratch: the stream's library workspace (see
 * lrc_apply), 16 (m + n) k bytes plus O(k^2); the results come back through
 * the stream's mapped host slot (see lrc_fro_diff).  SYNCHRONISES `stream`.
 */
LRC_API lrc_status lrc_lowrank_eta(const double* U, const double* S, const double* Vt,
                                   const void* Uh, const void* Sh, const void* Vht, lrc_fmt fmt,
                                   int64_t m, int64_t n, int64_t k, double* eta_out,
                                   double* norm_out, lrc_stream_t stream);

/*
 * lrc_tt_eta -- eta_TT = ||T(G_1..G_d) - T(Gh_1..Gh_d)||_F, the perturbation
 * of Thm 6.1 (Sec. 6.1: rounded cores compared in FP64), without forming
 * either tensor.
 *
 *   cores      HOST array of d DEVICE pointers to the binary64 cores, layout
 *              of tt_reconstruct (core l: ranks[l] x dims[l] x ranks[l+1])
 *   cores_hat  HOST array of d DEVICE pointers to the stored cores in format
 *              `fmt`, same shapes
 *   dims, ranks, d  as in tt_reconstruct
 *   eta_out    host: eta_TT
 *   norm_out   host, may be NULL: ||T(G)||_F
 *
 * With D_l = Z_l - Zh_l the difference of the partial products of Eq.
 * gpu_tt_reconstruction, [D_l, Zh_l] = [D_{l-1}, Zh_{l-1}] C_l(i_l) with the
 * block core C_l(i) = [[G_l(i), 0], [G_l(i) - Gh_l(i), Gh_l(i)]], and
 * T - Th = [D_{d-1}, Zh_{d-1}] [G_d; G_d - Gh_d].  The 2 r_l x 2 r_l Gram
 * matrix of [D_l, Zh_l] over all prefixes is carried from core to core
 * (M_l = sum_i C_l(i)^T M_{l-1} C_l(i)) and contracted with the last core.
 * Work: about sum over interior cores of 8 r_{l-1} n_l r_l (2 r_{l-1} +
 * r_l) binary64 flops.  Deterministic on a device.  Cores aligned to their
 * element size.  Scratch: the stream's workspace, two buffers of
 * 4 r_{l-1} n_l r_l binary64 for the largest interior core plus O(r^2); the
 * results come back through the stream's mapped host slot (see
 * lrc_fro_diff).  SYNCHRONISES `stream`.
 */
LRC_API lrc_status lrc_tt_eta(const double* const* cores, const void* const* cores_hat,
                              const int64_t* dims, const int64_t* ranks, int d, lrc_fmt fmt,
                              double* eta_out, double* norm_out, lrc_stream_t stream);

/* Thm 4.1 Eq. matrix_condition and Thm 6.1 Eq. tt_condition:
 * returns 1 if e_aug + eta <= e_base (certified non-increase), else 0. */
LRC_API int lrc_certified(double e_base, double e_aug, double eta);

/* Sec. 4: E_k = (sum_{j>k} sigma_j^2)^(1/2) for host sigma[0..len) (sigma_1
 * first), summed from the smallest term up.  Returns -1 on bad arguments. */
LRC_API double lrc_tail_error(const double* sigma, int64_t len, int64_t k);

/* Eq. matrix_storage_ratio generalised to k_aug >= k_base: storage of the
 * rank-k_aug factors in `fmt` over the FP64 rank-k_base factors. */
LRC_API double lrc_matrix_storage_ratio(int64_t m, int64_t n, int64_t k_base, int64_t k_aug, lrc_fmt fmt);

/* Sec. 5.1: TT storage in bytes, sum_l R_{l-1} n_l R_l scalars of `fmt`. */
LRC_API double lrc_tt_storage_bytes(const int64_t* dims, const int64_t* ranks, int d, lrc_fmt fmt);

/* Message for a status code, and the last error message of this thread. */
LRC_API const char* lrc_status_string(lrc_status status);
LRC_API const char* lrc_last_error(void);

/* Number of kernels this library has launched in this process. */
LRC_API uint64_t lrc_launch_count(void);

/* Synchronises `stream`, then reports whether a bounded device-side wait in
 * a tensor-core kernel gave up since the last call: LRC_ERR_TIMEOUT if so
 * (the error words are cleared), LRC_ERR_CUDA if the stream reported an
 * error, LRC_OK otherwise.  Kernels never hang: every wait on a barrier is
 * limited in time, after which the CTA records the event and exits. */
LRC_API lrc_status lrc_device_status(lrc_stream_t stream);

/* Test hook for the failure path above: launches one CTA that waits, with a
 * time limit of `limit_ns` (0 < limit_ns <= 1e9), on a barrier that nothing
 * arrives on.  The next lrc_device_status() returns LRC_ERR_TIMEOUT. */
LRC_API lrc_status lrc_selftest_wait_timeout(int64_t limit_ns, lrc_stream_t stream);

/*
 * lrc_tt_svd -- TT-SVD of a dense tensor on the GPU (Sec. 5: Oseledets'
 * sequential truncated SVDs; Alg. alg:tt_compensation steps 1-2, the FP64
 * baseline T_R and the augmented T_{R+delta}), in binary64.
 *
 *   T       device, the dense tensor, prod(dims) binary64 entries, C order
 *           (i_1 slowest), 8-byte aligned; not modified
 *   dims, ranks, d  as in tt_reconstruct: the ranks to truncate to, with
 *           ranks[0] = ranks[d] = 1 and every ranks[l] at most the smaller
 *           side of unfolding l, min(ranks[l-1] dims[l-1], dims[l] ... dims[d-1]),
 *           which must itself be at most 1024
 *   cores   HOST array of d DEVICE pointers, core l receives
 *           ranks[l] x dims[l] x ranks[l+1] binary64 values (C order)
 *   delta2_out   host, may be NULL: d - 1 values, the sum of the discarded
 *           squared singular values at each bond; ||T - T_R||_F^2 is their sum
 *           (the discarded parts of the sequential steps are orthogonal)
 *   spectra_out  host, may be NULL: every singular value of every unfolding
 *           remainder, bond after bond, each bond's in descending order
 *           (min(rows, cols) values per bond) -- the local spectra of the
 *           certificate's diagnostics
 *
 * Each bond's SVD is a one-sided Jacobi SVD of the tall side of the
 * remainder (column pairs rotated until orthogonal to sqrt(L) units of
 * roundoff; at most 40 sweeps, else LRC_ERR_UNSUPPORTED), so small singular
 * values are accurate to about u times the largest.  The cores 1..d-1 are
 * left-orthonormal.  d = 2 is the truncated SVD of a dims[0] x dims[1]
 * matrix: cores[0] = U_k, cores[1] = diag(s_k) V_k^T, spectra_out = all
 * singular values.  Scratch: the stream's library workspace, about
 * 16 prod(dims) bytes.  SYNCHRONISES `stream`.
 */
LRC_API lrc_status lrc_tt_svd(const double* T, const int64_t* dims, const int64_t* ranks, int d,
                              double* const* cores, double* delta2_out, double* spectra_out,
                              lrc_stream_t stream);

/*
 * lrc_tt_left_orthogonalize -- the left-orthogonal gauge (Sec. 6.1), in
 * place, binary64: for l = 1..d-1 the unfolding (r_{l-1} n_l) x r_l of core
 * l is factored Q R' (Q with orthonormal columns, from a one-sided Jacobi
 * SVD: Q = U, R' = diag(s) V^T), core l becomes Q and core l + 1 becomes
 * R' core l + 1.  The tensor is unchanged (to rounding) and ||G_d||_F =
 * ||T||_F.  Requires r_l <= r_{l-1} n_l and r_l <= 1024; a zero singular
 * value leaves a zero column in Q (still exact).  cores: HOST array of d
 * DEVICE pointers (binary64, layout of tt_reconstruct).  SYNCHRONISES `stream`.
 */
LRC_API lrc_status lrc_tt_left_orthogonalize(double* const* cores, const int64_t* dims, const int64_t* ranks, int d,
                                             lrc_stream_t stream);

/*
 * lrc_probe_peak -- measured rate of one arithmetic unit of this GPU, the
 * denominator of the roofline fractions of the binary32 and binary64 paths
 * (their products run on the CUDA cores' FMA units or on the binary64 tensor
 * cores, Sec. 3.4 fixing only the precision).  Runs a kernel of independent
 * multiply-add chains (no memory traffic in the loop) on every SM:
 *
 *   kind  0 = binary32 FMA, 1 = binary32 two-lane packed FMA,
 *         2 = binary64 FMA, 3 = binary64 tensor-core MMA (m8n8k4)
 *   iters loop steps per thread, 1 <= iters <= 2^30 (about 2^20 gives a
 *         launch of a few to a few hundred milliseconds)
 *   flops_out  host: flops per second, CUDA-event time of one launch after
 *         a shorter warm-up launch
 *
 * Uses the stream's library workspace for one value per thread.
 * SYNCHRONISES `stream`.
 */
LRC_API lrc_status lrc_probe_peak(int kind, int64_t iters, double* flops_out, lrc_stream_t stream);

/* Release library-held scratch on every device; the library stays usable. */
LRC_API lrc_status lrc_shutdown(void);

#ifdef __cplusplus
}
#endif

#endif /* LRC_H */
