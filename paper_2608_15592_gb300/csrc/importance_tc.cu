// tcgen05 path of the attention kernels (bf16).
#include "importance_tc.cuh"

namespace estp {

bool tc_supported(estp_dtype, int) { return false; }
int tc_tile() { return 128; }
int tc_qc() { return 4; }

estp_status launch_lse_tc(estp_ctx*, const void*, const void*, int, int, int, float,
                          const ImpHeads&, const int32_t*, int, int64_t, int, float*,
                          cudaStream_t, size_t) {
    return fail(ESTP_ERR_UNSUPPORTED, "tensor-core LSE path not built");
}

estp_status launch_imp_tc(estp_ctx*, const void*, const void*, const float*, int, int, int,
                          float, const ImpHeads&, const int32_t*, int, int64_t, bool,
                          const int32_t*, const PlanInfo*, float*, cudaStream_t) {
    return fail(ESTP_ERR_UNSUPPORTED, "tensor-core importance path not built");
}

}  // namespace estp
