// tc_pending.cu -- binary16 TT reconstruction runs on the CUDA-core chain
// kernel (binary32 arithmetic) until the tensor-core version replaces it.
#include "common.cuh"

namespace lrc {

lrc_status launch_tt_f16(const TTShape& sh, bool out16, void* out, cudaStream_t s) {
    return launch_tt_cc(sh, out16 ? LRC_F16_O16 : LRC_F16, out, s);
}

uint32_t take_tt_tc_error() { return 0; }

}  // namespace lrc
