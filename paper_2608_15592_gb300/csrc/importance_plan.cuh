// Work plans for the attention kernels (shared by the CUDA-core and tcgen05 paths).
//
// Importance items.  A prompt of T tokens has nt = ceil(T / tile) key tiles.  Key
// tile kt receives mass only from query tiles kt .. nt-1 (causal), which are cut
// into chunks of qc query tiles:  item (group slot g, key tile kt, chunk c) covers
// query tiles kt + c*qc .. min(nt, kt + (c+1)*qc) - 1.  Items of one prompt are
// numbered g-major, then kt, then c.  The number of items of one group is
//   f(nt) = sum_{m=1..nt} ceil(m / qc) = qc*a*(a+1)/2 + r*(a+1),  nt = a*qc + r,
// and key tile kt starts at item F(kt) = f(nt) - f(nt - kt).
//
// LSE items: (query tile, head slot), numbered from the last query tile (longest
// rows, most key tiles) to the first, so that a dynamic scheduler hands out the
// largest items of a prompt first.
#pragma once
#include "estp_internal.cuh"

namespace estp {

__host__ __device__ __forceinline__ int64_t items_f(int64_t n, int qc) {
    const int64_t a = n / qc, r = n % qc;
    return (int64_t)qc * a * (a + 1) / 2 + r * (a + 1);
}

struct PlanInfo {
    int32_t ok;      // 1 when cu_seqlens passed the device checks
    int32_t total;   // total items
    int32_t next;    // dynamic work counter of the persistent kernels (zeroed by the plan)
    int32_t pad;
};

// Per-prompt count of a plan of kind 0: importance items f(nt); kind 1: one per tile, nt;
// kind 2: one per pair of tiles (query tile, key tile <= query tile), nt (nt + 1) / 2.
__host__ __device__ __forceinline__ int64_t plan_count(int64_t nt, int qc, int kind) {
    return kind == 0 ? items_f(nt, qc) : kind == 1 ? nt : nt * (nt + 1) / 2;
}

// Prefix of per-prompt counts (base[B+1]) and validation.  One CTA of 1024.
// Each prompt counts mult * plan_count(nt, qc, kind).
__global__ void __launch_bounds__(1024) attn_plan_kernel(const int32_t* cu, int B, int64_t sumT,
                                                         int max_seqlen, int tile, int qc,
                                                         int mult, int kind, int32_t* base,
                                                         PlanInfo* info, int* status);

// Two plans of the same prompts in one launch of 2 blocks: block 0 writes (kind0, base0,
// info0), block 1 (kind1, base1, info1).
__global__ void __launch_bounds__(1024) attn_plan2_kernel(const int32_t* cu, int B, int64_t sumT,
                                                          int max_seqlen, int tile, int qc,
                                                          int mult, int kind0, int32_t* base0,
                                                          PlanInfo* info0, int kind1,
                                                          int32_t* base1, PlanInfo* info1,
                                                          int* status);

struct ImpItem {
    int b, g, kt, qt0, qt1;
    int64_t t0;
    int T;
};

// Item `item` of prompt b (the prompt whose items contain it: upper_slot(base, B, item)).
__device__ __forceinline__ ImpItem decode_imp_item_at(int item, int b, const int32_t* base,
                                                      const int32_t* cu, int tile, int qc) {
    ImpItem it;
    it.b = b;
    it.t0 = cu[it.b];
    it.T = cu[it.b + 1] - cu[it.b];
    const int nt = (it.T + tile - 1) / tile;
    const int64_t per_group = items_f(nt, qc);
    const int64_t local = item - base[it.b];
    it.g = (int)(local / per_group);
    const int64_t rem = local - (int64_t)it.g * per_group;
    const int64_t fnt = per_group;
    int lo = 0, hi = nt - 1;  // largest kt with F(kt) <= rem
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (fnt - items_f(nt - mid, qc) <= rem) lo = mid; else hi = mid - 1;
    }
    it.kt = lo;
    const int c = (int)(rem - (fnt - items_f(nt - lo, qc)));
    it.qt0 = lo + c * qc;
    it.qt1 = min(nt, it.qt0 + qc);
    return it;
}

__device__ __forceinline__ ImpItem decode_imp_item(int item, const int32_t* base, int B,
                                                   const int32_t* cu, int tile, int qc) {
    return decode_imp_item_at(item, upper_slot(base, B, item), base, cu, tile, qc);
}

struct LseItem {
    int b, hslot, qt;
    int64_t t0;
    int T;
};

__device__ __forceinline__ LseItem decode_lse_item_at(int item, int b, const int32_t* base,
                                                      const int32_t* cu, int tile, int n_heads) {
    LseItem it;
    it.b = b;
    it.t0 = cu[it.b];
    it.T = cu[it.b + 1] - cu[it.b];
    const int nt = (it.T + tile - 1) / tile;
    const int local = item - base[it.b];
    const int rank = local / n_heads;
    it.hslot = local - rank * n_heads;
    it.qt = nt - 1 - rank;
    return it;
}

__device__ __forceinline__ LseItem decode_lse_item(int item, const int32_t* base, int B,
                                                   const int32_t* cu, int tile, int n_heads) {
    return decode_lse_item_at(item, upper_slot(base, B, item), base, cu, tile, n_heads);
}

// Number of chunks of key tile kt of a prompt with nt tiles.
__host__ __device__ __forceinline__ int chunks_of(int nt, int kt, int qc) {
    return (nt - kt + qc - 1) / qc;
}

}  // namespace estp
