// Internal declarations shared by the ESTP CUDA translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <nvtx3/nvToolsExt.h>

#include "estp.h"

// Bounded device waits: about 2 s of SM clock.
constexpr long long kWaitCycles = 4000000000ll;

struct estp_ctx {
    int device = 0;
    int num_sms = 0;
    int* status = nullptr;      // device status word (estp_status codes)
    void* ws = nullptr;         // growable scratch for one call's intermediates
    size_t ws_bytes = 0;
    float* imp_acc = nullptr;   // importance accumulator C_j, fp32 [imp_cap]
    int64_t imp_cap = 0;
    // state of the open importance accumulation
    bool imp_open = false;
    int64_t imp_sumT = 0;
    int32_t imp_B = 0;
    const int32_t* imp_cu = nullptr;
    int32_t imp_n_heads = 0;
    uint32_t imp_flags = 0;     // flags of the opening call (divisor variant, self term)
    uint32_t* pool_done = nullptr;      // per-prompt arrival counters of the pooling kernel
    int32_t pool_done_cap = 0;
    // limit of the attention kernels' abortable waits (estp_set_wait_limit)
    long long wait_cycles = kWaitCycles;
};

namespace estp {

// An NVTX range named after the entry point for the length of the host call (a no-op
// unless a profiler is attached), so that a timeline groups each call's launches.
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange&) = delete;
    NvtxRange& operator=(const NvtxRange&) = delete;
};
#define ESTP_NVTX_RANGE(name) ::estp::NvtxRange estp_nvtx_range_(name)

// ---------------------------------------------------------------- host helpers
estp_status fail(estp_status st, const char* fmt, ...);
estp_status cuda_fail(cudaError_t e, const char* what);
estp_status ws_reserve(estp_ctx* ctx, size_t bytes);
estp_status set_device(estp_ctx* ctx);

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline int esize(estp_dtype t) { return t == ESTP_BF16 ? 2 : 4; }

// --------------------------------------------------------------- device helpers
__device__ __forceinline__ void report(int* status, int code) { atomicCAS(status, 0, code); }

// Debug builds (-DESTP_CHECKS): bounds checks on the kernels' global accesses.  A failed
// check records ESTP_ERR_BOUNDS in the status word (when the launch has one) and the
// caller skips the access; nothing traps.  Release builds compile the checks away.
__device__ __forceinline__ bool in_bounds(bool ok, int* status) {
#ifdef ESTP_CHECKS
    if (!ok && status != nullptr) report(status, ESTP_ERR_BOUNDS);
    return ok;
#else
    (void)ok;
    (void)status;
    return true;
#endif
}

// 16-byte streaming load that bypasses L1 (data read exactly once).
__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float lg2(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Binary search: largest b in [0, n) with base[b] <= x (base non-decreasing, base[0] <= x).
__device__ __forceinline__ int upper_slot(const int32_t* base, int n, int64_t x) {
    int lo = 0, hi = n - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (base[mid] <= x) lo = mid; else hi = mid - 1;
    }
    return lo;
}

// ------------------------------------------------------------------ launchers
estp_status launch_entropy(estp_ctx* ctx, const void* logits, estp_dtype dtype, int64_t n_rows,
                           int64_t V, int64_t ld, const int32_t* cu, int32_t B, float* H,
                           cudaStream_t st);

struct ImpHeads {
    int n_heads;          // selected query heads
    int n_groups;         // KV groups that hold at least one selected head
    int16_t group[256];   // KV head index of group slot g
    int16_t begin[257];   // heads of group slot g: head_list[begin[g] .. begin[g+1])
    int16_t head_list[256];
};

estp_status build_heads(const int32_t* heads, int n_heads, int Hq, int Hkv, ImpHeads* out);

estp_status launch_lse(estp_ctx* ctx, const void* Q, const void* K, estp_dtype dtype, int Hq,
                       int Hkv, int d, float scale, const ImpHeads& hs, const int32_t* cu,
                       int B, int64_t sumT, int max_seqlen, float* lse, cudaStream_t st);

estp_status launch_importance(estp_ctx* ctx, const void* Q, const void* K, estp_dtype dtype,
                              const float* lse, int Hq, int Hkv, int d, float scale,
                              const ImpHeads& hs, const int32_t* cu, int B, int64_t sumT,
                              int max_seqlen, bool accumulate, uint32_t flags, float* acc,
                              cudaStream_t st);

estp_status launch_head_loss(estp_ctx* ctx, const float* pooled, int B, int64_t D,
                             const estp_head& head, const float* targets, float lambda3,
                             float* loss, float* grad_W, float* grad_bias, float* grad_pooled,
                             cudaStream_t st);
estp_status launch_lm_head_entropy(estp_ctx* ctx, const void* hidden, int64_t ldh, const void* W,
                                   int64_t ldw, int64_t n_rows, int64_t D, int64_t V, float* H,
                                   cudaStream_t st);
estp_status launch_mlp_head_predict(estp_ctx* ctx, const float* pooled, int B, int64_t D,
                                    const estp_mlp_head& head, float* pred, float* probs,
                                    cudaStream_t st);
estp_status launch_mlp_head_loss(estp_ctx* ctx, const float* pooled, int B, int64_t D,
                                 const estp_mlp_head& head, const float* targets, float lambda3,
                                 float* loss, const estp_mlp_grads& g, cudaStream_t st);
estp_status launch_misalignment(estp_ctx* ctx, const float* H, const float* S, const int32_t* cu,
                                int B, int64_t sumT, int pct, int32_t* counts, cudaStream_t st);
estp_status launch_attn_forward(estp_ctx* ctx, const void* Q, const void* K, const void* V,
                                const float* lse, int Hq, int Hkv, float scale, const int32_t* cu,
                                int B, int64_t sumT, int max_seqlen, bool exclude_self,
                                bool accumulate, float* acc, void* O, cudaStream_t st);
estp_status launch_importance_finalize(estp_ctx* ctx, const float* acc, const int32_t* cu, int B,
                                       int64_t sumT, int n_layers, int n_heads, uint32_t flags,
                                       float* out, cudaStream_t st);

estp_status launch_pool(estp_ctx* ctx, const void* hidden, estp_dtype dtype, int64_t D,
                        int64_t ldh, const float* H, const float* S, const int32_t* cu, int B,
                        int64_t sumT, estp_mix_params mix, const estp_head* head, float* pooled,
                        float* pred, cudaStream_t st);

}  // namespace estp
