// common.cuh -- internal helpers shared by the translation units of liblrc.so.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "lrc.h"

namespace lrc {

// Records a message for lrc_last_error() on the calling thread.
void set_error(const char* fmt, ...);

// Maps a CUDA error to LRC_ERR_CUDA with a message naming `what`.
lrc_status cuda_fail(cudaError_t e, const char* what);

// Checks cudaGetLastError() after a launch; counts the launch.
lrc_status after_launch(const char* what);

// Multiprocessor count of the current device (cached per device).
int sm_count();

// Launch with programmatic stream serialization: the kernel may begin before
// the previous kernel of the stream has finished and synchronizes with it
// through pdl_wait().
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, Args&&... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline cudaStream_t as_stream(lrc_stream_t s) { return reinterpret_cast<cudaStream_t>(s); }

// Bytes of one stored element of a format (binary16 for both F16 variants).
inline int64_t storage_bytes(lrc_fmt f) {
    switch (f) {
        case LRC_F64: return 8;
        case LRC_F32:
        case LRC_F32_TC: return 4;
        case LRC_F16:
        case LRC_F16_O16:
        case LRC_BF16: return 2;
    }
    return 0;
}

inline bool valid_fmt(int f) { return f >= LRC_F64 && f <= LRC_BF16; }
// LRC_F32_TC is LRC_F32 everywhere but in the output products of lrc_apply
// and tt_reconstruct
inline lrc_fmt plain_fmt(lrc_fmt f) { return f == LRC_F32_TC ? LRC_F32 : f; }

// a * b with overflow detection (both >= 0).
inline bool mul_ok(int64_t a, int64_t b, int64_t* out) {
    if (a < 0 || b < 0) return false;
    if (a != 0 && b > INT64_MAX / a) return false;
    *out = a * b;
    return true;
}

// ---- launchers (implemented in the .cu files) ----------------------------
lrc_status launch_round(const double* src, int64_t rows, int64_t cols, int64_t ld_src, void* dst,
                        int64_t ld_dst, lrc_fmt fmt, cudaStream_t s);
lrc_status launch_widen(const void* src, lrc_fmt fmt, int64_t rows, int64_t cols, int64_t ld_src,
                        double* dst, int64_t ld_dst, cudaStream_t s);
lrc_status launch_apply_f64(const double* U, const double* S, const double* Vt, const double* X,
                            double* Y, int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s);
// LRC_F32_TC output product C (P x Q, row pitch Q) = A B^T on the tensor
// cores through the scaled binary16 split (apply_cc.cu): A(i, j) =
// A[i a_rs + j a_cs] is P x k (a scale per row), B(i, j) = B[i b_rs + j b_cs]
// is Q x k (a scale per 32 rows); ws holds split_product_bytes(P, Q, k)
// bytes (256-byte aligned); split_product_fits says whether the product
// kernel takes the shape.
size_t split_product_bytes(int64_t P, int64_t Q, int64_t k);
bool split_product_fits(int64_t P, int64_t Q, int64_t k);
lrc_status launch_split_product(const float* A, int64_t a_rs, int64_t a_cs, const float* B, int64_t b_rs,
                                int64_t b_cs, int64_t P, int64_t Q, int64_t k, unsigned char* ws, float* C,
                                cudaStream_t s);
// tc: the second product on the tensor cores (LRC_F32_TC) where it applies
lrc_status launch_apply_f32(const float* U, const float* S, const float* Vt, const float* X,
                            float* Y, int64_t m, int64_t n, int64_t k, int64_t b, bool tc, cudaStream_t s);
// small-batch split path of the CUDA-core apply (apply_split.cu)
lrc_status launch_apply_split_f64(const double* U, const double* S, const double* Vt, const double* X, double* Y,
                                  int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s);
lrc_status launch_apply_split_f32(const float* U, const float* S, const float* Vt, const float* X, float* Y,
                                  int64_t m, int64_t n, int64_t k, int64_t b, cudaStream_t s);
// One apply of a batch (lrc_apply_batched); layouts of lrc_apply.
struct ApplyProblem {
    const void* U;
    const void* S;
    const void* Vt;
    const void* X;
    void* Y;
    int64_t m, n, k, b;
};
// Up to apply_f16_group_max() binary16 / bfloat16 problems in one launch per
// phase (apply_tc.cu); every problem is validated by the caller.
int apply_f16_group_max();
lrc_status launch_apply_f16_group(const ApplyProblem* pr, int count, bool out16, bool bf16, cudaStream_t s);
// bf16: bfloat16 operands and output (out16 must be set)
lrc_status launch_apply_f16(const void* U, const void* S, const void* Vt, const void* X, void* Y,
                            int64_t m, int64_t n, int64_t k, int64_t b, bool out16, cudaStream_t s,
                            bool bf16 = false);
// small batches (apply_skinny.cu): on the tensor cores at most 64 queries in
// binary16 and bfloat16, rank at most 512, n at most 32768; otherwise on the
// CUDA cores at most 16 queries in binary32 and binary64 and 4 in binary16,
// ranks up to 1024 whose tiles fit in shared memory
bool apply_skinny_takes(lrc_fmt fmt, int64_t m, int64_t n, int64_t k, int64_t b);
lrc_status launch_apply_skinny(const void* U, const void* S, const void* Vt, const void* X, void* Y, int64_t m,
                               int64_t n, int64_t k, int64_t b, lrc_fmt fmt, cudaStream_t s);

// Register-tiled binary32 products on the CUDA cores (gemm_cc.cu):
// C[M x N] = A[M x K] B with B stored K x N (b_trans = false) or N x K
// (b_trans = true), all row-major; `splits` > 1 splits K and writes split z's
// partial product at C + z * c_split.  gemm_cc_ex(N): the tile width the
// launcher uses for N columns is 128 + 16 * gemm_cc_ex(N).  The kernels wait
// for the previous kernel of the stream (programmatic dependent launch).
int gemm_cc_ex(int64_t N);
// binary64 C[M x N] = A[M x K] B[K x N], all row-major (DFMA-bound tiles)
lrc_status gemm_cc_f64(const double* A, int64_t lda, const double* B, int64_t ldb, double* C, int64_t ldc,
                       int64_t M, int64_t N, int64_t K, cudaStream_t s);
lrc_status gemm_cc_f32(const float* A, int64_t lda, const float* B, int64_t ldb, bool b_trans, float* C,
                       int64_t ldc, int64_t M, int64_t N, int64_t K, int splits, int64_t c_split, cudaStream_t s);

// The second product of the binary16 apply for other callers (apply_tc.cu):
// Y[b x m] = W U^T on the tensor cores, binary32 accumulation, binary32 or
// binary16 output.  W is given as 128-row tile images (canonical K-major
// layout, tc::w_image_off, 128 x kp binary16 each), U as m rows of kp
// binary16 with row pitch ldu elements.  esc_w / esc_u (nullable together)
// scale entry (i, j) by 2^-(esc_w[i / 32] + esc_u[j / 32]) -- esc_w[i] when
// w_per_row -- each in [-60, 60]; y_product_plan checks that the product
// fits the kernel.
lrc_status y_product_plan(int64_t m, int64_t b, int kp, bool out16, int* n2);
lrc_status launch_y_product(const unsigned char* Wimg, int kp, const void* U, int64_t ldu, int64_t m, int64_t b,
                            bool out16, void* Y, const int* esc_w, const int* esc_u, cudaStream_t s,
                            bool w_per_row = false, bool bf16 = false);

struct TTShape {
    int d;
    int64_t dims[16];
    int64_t ranks[17];
    const void* cores[16];
    int64_t numel;
};
lrc_status launch_tt_cc(const TTShape& sh, lrc_fmt fmt, void* out, cudaStream_t s);
// binary32 / binary64 TT as a chain of products meeting at one bond
// (tt_chain.cu); binary64 takes it where it saves at least a fifth of the
// left-to-right chain's multiplies (tt_chain_saves)
lrc_status launch_tt_chain_f32(const TTShape& sh, float* out, cudaStream_t s);
lrc_status launch_tt_chain_f64(const TTShape& sh, double* out, cudaStream_t s);
bool tt_chain_saves(const TTShape& sh);
// multiply count (x2) of that chain at its cheapest bond
double tt_chain_flops(const TTShape& sh);
lrc_status launch_tt_f16(const TTShape& sh, bool out16, void* out, cudaStream_t s);
// binary16 TT as a product chain with the output product on the tensor cores
// (tt_split.cu); *handled = false when the shape is outside it (nothing launched)
lrc_status launch_tt_split_f16(const TTShape& sh, bool out16, void* out, cudaStream_t s, bool* handled);
// the same product chain for binary32 cores (LRC_F32_TC): both operands split
// into scaled hi/lo binary16 parts; *handled = false when the shape is outside it
lrc_status launch_tt_split_f32tc(const TTShape& sh, float* out, cudaStream_t s, bool* handled);
// bfloat16 cores, bfloat16 workspaces and output: the same product chain with
// bfloat16 tensor-core operands where the shape fits it, else the CUDA-core
// chain of tt_cc.cu
lrc_status launch_tt_bf16(const TTShape& sh, void* out, cudaStream_t s);
// the FP32 product chain with its output product on the tensor cores
// (LRC_F32_TC) when split_product_fits, else on the CUDA cores (tt_chain.cu)
lrc_status launch_tt_chain_f32tc(const TTShape& sh, float* out, cudaStream_t s);
// binary32 TT whose chain has several small products at its ends: one side
// launch forms Z and S, one product forms the tensor (tt_split.cu);
// *handled = false when the shape is outside it
lrc_status launch_tt_side_f32(const TTShape& sh, float* out, cudaStream_t s, bool* handled);
// bond at which the product chain of tt_chain.cu meets
int tt_chain_bond(const TTShape& sh);

// 2-D TMA map over a row-major [rows x cols] array with a row pitch of
// `pitch_bytes`: boxes of box_cols x box_rows elements, 128-byte swizzle or
// none, elements outside the array read as zero.
lrc_status encode_map_2d(CUtensorMap* map, CUtensorMapDataType dt, const void* base, int64_t cols, int64_t rows,
                         int64_t pitch_bytes, uint32_t box_cols, uint32_t box_rows, bool swizzle128,
                         const char* what);

// Device error words of the tensor-core kernels (bounded waits that gave up);
// read and cleared by lrc_device_status().  0xffffffff = could not be read.
uint32_t take_apply_tc_error();
uint32_t take_tt_tc_error();
uint32_t take_tt3_tc_error();
// 3-way binary16 TT on the tensor cores; *handled = false when the shape is
// outside the kernel (nothing launched).
lrc_status launch_tt3_f16_tc(const TTShape& sh, bool out16, void* out, cudaStream_t s, bool* handled);
// binary16 TT with narrow last two modes on the tensor cores (tt_narrow_tc.cu);
// *handled = false when the shape is outside the kernel (nothing launched).
lrc_status launch_ttn_f16_tc(const TTShape& sh, bool out16, void* out, cudaStream_t s, bool* handled);
uint32_t take_ttn_tc_error();
uint32_t take_skinny_error();
lrc_status launch_wait_timeout_probe(int64_t limit_ns, cudaStream_t s);

lrc_status run_fro_diff(const void* A, lrc_fmt fa, const void* B, lrc_fmt fb, int64_t count,
                        double* diff_out, double* normA_out, cudaStream_t s);
void release_scratch();
// Per-(device, stream) workspace, grown on demand; freed by release_workspaces().
lrc_status stream_workspace(cudaStream_t s, size_t bytes, void** out);
// Per-(device, stream) arrival counters, zero between kernels: kStreamCounters
// of them, made (and zeroed in stream order) on first use.
constexpr int kStreamCounters = 1024;
lrc_status stream_counters(cudaStream_t s, unsigned int** out);
// Per-(device, stream) slot of kResultSlots doubles in mapped pinned host
// memory: `dev` is the address kernels write, `host` the one the host reads
// once the stream has synchronised.
constexpr int kResultSlots = 8;
lrc_status stream_result_slot(cudaStream_t s, double** host, double** dev);
void release_workspaces();
lrc_status run_fro_diff_noalloc(const void* A, lrc_fmt fa, const void* B, lrc_fmt fb, int64_t count,
                                double* diff_out, double* normA_out, cudaStream_t s);
int64_t fro_diff_noalloc_max_count();

// Sampled TT entries (tt_gather.cu); ranks up to tt_gather_max_rank().
int tt_gather_max_rank();
lrc_status launch_tt_gather(const TTShape& sh, lrc_fmt fmt, const int64_t* idx, int64_t count, void* out,
                            cudaStream_t s);

// eta of Thm 4.1 / eta_TT of Thm 6.1 from Gram blocks (eta.cu); synchronise s.
lrc_status run_lowrank_eta(const double* U, const double* S, const double* Vt, const void* Uh, const void* Sh,
                           const void* Vht, lrc_fmt fmt, int64_t m, int64_t n, int64_t k, double* eta_out,
                           double* norm_out, cudaStream_t s);
lrc_status run_tt_eta(const TTShape& sh, const void* const* hats, lrc_fmt fmt, double* eta_out, double* norm_out,
                      cudaStream_t s);

// Factorization side (factor.cu), binary64; synchronise s.  The caller has
// checked the shapes (every rank at most the smaller side of its unfolding).
int factor_max_cols();
lrc_status run_tt_svd(const double* T, const TTShape& sh, double* const* cores, double* delta2_out,
                      double* spectra_out, cudaStream_t s);
lrc_status run_tt_left_orthogonalize(const TTShape& sh, double* const* cores, cudaStream_t s);

// Measured rate of one arithmetic unit (peak_probe.cu); synchronises s.
lrc_status run_probe_peak(int kind, int64_t iters, double* flops_out, cudaStream_t s);

}  // namespace lrc
