// Inline-PTX helpers shared by the TMA / mbarrier / tcgen05 kernels (sm_100+).
#pragma once
#include <stdint.h>

#include "estp_internal.cuh"

namespace estp {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: false (and the CTA's abort flag set) when the barrier does not
// complete within `limit` SM cycles or another role of the CTA has already aborted.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                         int* status, long long limit = kWaitCycles) {
    if (mbar_try_wait(bar, parity)) return true;  // fast path: no flag read
    if (*abort_flag) return false;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (*abort_flag) return false;
        if (clock64() - t0 > limit) {
            *abort_flag = 1;
            report(status, ESTP_ERR_TIMEOUT);
            return false;
        }
    }
    return true;
}

// Bounded wait that ignores the abort flag (used to drain outstanding async work); its
// limit is always the full kWaitCycles, so that every copy and MMA a CTA issued has
// completed before it frees its tensor memory and exits.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity, int* status) {
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > kWaitCycles) {
            report(status, ESTP_ERR_TIMEOUT);
            return;
        }
    }
}

// Warp-uniform bounded wait: every lane polls the barrier (one broadcast shared-memory
// access), so the warp takes no divergent branch, and a vote gives every lane the same
// answer.  (Polling by lane 0 with a shuffle of the result was 6 % slower in the column-sum
// kernel.)
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          int* status, long long limit = kWaitCycles) {
    const bool r = wait_bar(bar, parity, abort_flag, status, limit);
    return __all_sync(0xffffffffu, r ? 1 : 0) != 0;
}

// max of three floats in one instruction (sm_100+)
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

}  // namespace estp

