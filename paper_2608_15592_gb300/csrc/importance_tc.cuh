// tcgen05 (tensor-core) path of the attention kernels for bf16 inputs.
#pragma once
#include "importance_plan.cuh"

namespace estp {

bool tc_supported(estp_dtype dtype, int d);
int tc_tile();  // keys (and queries) per tile
// pairs of query tiles per column-sum item for a call over B prompts, sumT tokens and
// n_groups KV groups on num_sms SMs
int tc_qc(int B, int64_t sumT, int n_groups, int num_sms);

estp_status launch_lse_tc(estp_ctx* ctx, const void* Q, const void* K, int Hq, int Hkv, int d,
                          float scale, const ImpHeads& hs, const int32_t* cu, int B, int64_t sumT,
                          int max_seqlen, float* lse, cudaStream_t st, size_t ws_off = 0);

estp_status launch_imp_tc(estp_ctx* ctx, const void* Q, const void* K, const float* lse, int Hq,
                          int Hkv, int d, float scale, const ImpHeads& hs, const int32_t* cu,
                          int B, int64_t sumT, bool exclude_self, const int32_t* base,
                          const PlanInfo* info, float* part, int c_max, int qc, cudaStream_t st);

}  // namespace estp
