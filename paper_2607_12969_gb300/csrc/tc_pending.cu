// tc_pending.cu -- the binary16 paths are not built yet: they report
// LRC_ERR_UNSUPPORTED instead of falling back to anything else.
#include "common.cuh"

namespace lrc {

lrc_status launch_apply_f16(const void*, const void*, const void*, const void*, void*, int64_t,
                            int64_t, int64_t, int64_t, bool, cudaStream_t) {
    set_error("binary16 apply is not built in this version");
    return LRC_ERR_UNSUPPORTED;
}

lrc_status launch_tt_f16(const TTShape&, bool, void*, cudaStream_t) {
    set_error("binary16 TT reconstruction is not built in this version");
    return LRC_ERR_UNSUPPORTED;
}

}  // namespace lrc
