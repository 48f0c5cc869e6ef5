// The prefill's causal attention output with the importance column sums taken from the
// same probability tiles (Sec. 3.1, Eq. 2-0): O = A V for every query head, and
// C_j += sum_h sum_{i >= j} A^h_ij for the importance accumulator.
//
// Two passes.  The row normalisers lse come first (the caller's, or the row-normaliser
// kernel's).  Then attn_fwd_kernel forms, per (query tile of 128 rows, head), the exact
// probabilities P = exp(scale q.k - lse) of each causal key tile, with no running
// rescale, on the tensor cores:
//   S   = Q K^T       tcgen05.mma, M = N = 128, K = 16 x 8 steps over d = 128, into TMEM
//   P   = 2^(S scale log2e - lse log2e)   epilogue, written back to TMEM as bf16
//   O  += P V         tcgen05.mma with A = P from TMEM, B = the key tile of V
// and the column sums of P over the tile's 128 query rows (a warp reduce-scatter, then the
// four TMEM lane quarters in order) go to a partial buffer, one slot per (prompt, head,
// query tile, key tile).  imp_fwd_reduce_kernel adds a key's slots in a fixed order into
// the accumulator: no floating-point atomics, repeated calls give identical bits.
//
// V enters the second MMA as it is stored, [sumT, Hkv, 128]: a 128-key tile lands in shared
// memory as rows of keys with d contiguous, which is B in the MN-major form (N = d
// contiguous, 128-byte swizzle; the two 64-wide d blocks 16 KB apart, the 8-key groups
// 1 KB apart).  Keys past the prompt meet P = 0.
//
// attn_fwd_kernel: one persistent CTA per SM, 320 threads.
//   warp 0      TMA producer: claims items, stages Q (1 buffer: the next item's Q loads
//               once the item's last S is done), K (a ring of 3: a load takes ~1500 cycles,
//               a slot frees when its S is done) and V (a ring of 2, a slot frees when
//               its P V is done)
//   warp 1      issues S = Q K^T (as soon as a K tile and an S buffer are free)
//   warp 2      issues O += P V (as soon as the epilogue has written P).  S and P V have
//               one issuing thread each (lane 0 of warps 1 and 2), because one thread
//               that issues 16 MMAs, makes 4 barrier checks and 5 commits per tile takes
//               longer than the tensor pipe needs for them
//   warps 3-18  epilogue, two groups of 8 that take the even and the odd key-tile steps
//               (each S / P buffer belongs to one group); warp w reads TMEM lanes
//               32 (w % 4) .. (one query row each) and one 64-column half: P, the column
//               sums of its 32 rows, and O at the end of an item (by the group of its
//               last step)
//   warp 19     adds the four lane quarters' column sums of every tile, in order, and
//               writes the tile's partial slot
// TMEM: S double-buffered (2 x 128 columns), O (128), P double-buffered (2 x 64 columns of
// bf16 pairs): all 512.  Every mbarrier wait is bounded (a test may lower the limit of the
// abortable waits through estp_set_wait_limit); on expiry the CTA records ESTP_ERR_TIMEOUT
// and drains: the producer waits for the last copy into each Q, K and V slot, each issuer
// for all its MMAs, before the TMEM is freed.
#include <cstddef>

#include "importance_tc.cuh"
#include "tcgen05.cuh"

namespace estp {
namespace {

constexpr int kT = 128;                     // rows of a query or key tile
constexpr int kD = 128;                     // head dim of this path
constexpr int kAtomBytes = kT * 128;        // 128 rows x 64 bf16
constexpr int kTileBytes = 2 * kAtomBytes;  // 128 rows x 128 bf16
constexpr int kEpiWarp0 = 3, kEpiWarps = 16;
constexpr int kGroupWarps = kEpiWarps / 2;        // warps of one epilogue group
constexpr int kRedWarp = kEpiWarp0 + kEpiWarps;  // the column-sum reducer
constexpr int kThreads = 32 * (kRedWarp + 1);
constexpr int kSched = 4;
// dynamic shared memory (offsets from a 1024-aligned base)
constexpr int kQBufs = 1;                         // Q tiles (the next item's Q loads
                                                  // once the last S of the item is done)
constexpr int kKStages = 3;                       // K ring: a K load takes ~1500 cycles
constexpr int kQOff = 0;
constexpr int kKOff = kQBufs * kTileBytes;
constexpr int kVOff = kKOff + kKStages * kTileBytes;  // [2 stages] V tiles
constexpr int kCsOff = kVOff + 2 * kTileBytes;        // [2][4 quarters][128] column sums
constexpr int kBarOff = kCsOff + 2 * 4 * kT * 4;
constexpr int kNumBars = 2 * kQBufs + 2 * kKStages + 2 + 8 + 3 + 2 + 4 + 2 * kSched;
constexpr int kMiscOff = kBarOff + kNumBars * 8;  // tmem address, abort flag
constexpr int kItemOff = kMiscOff + 16;           // [kSched] decoded items of the sched ring
// TMEM columns
constexpr uint32_t kColS = 0, kColO = 256, kColP = 384;
constexpr uint32_t kIdesc = idesc_bf16(kT, kT);   // M = N = 128 for both products
constexpr uint32_t kIdescPV = kIdesc | (1u << 16);  // P V: B (the V tile) MN-major

// Shared-memory descriptor of an MN-major B tile with 128-byte swizzle: 64 d values per
// 128-byte row of one key, 8-key groups 1 KB apart (stride byte offset), the second
// 64-wide d block 16 KB on (leading byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t sw128_mn_desc(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)(16384 >> 4) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

struct FwdArgs {
    const int32_t* cu;
    const int32_t* base;    // items plan: prompt b's items start at base[b] (Hq per tile)
    const int32_t* base2;   // partial slots: prompt b's start at base2[b] (Hq per tile pair)
    PlanInfo* info;
    const PlanInfo* info2;  // validity of the partial-slot plan
    int B, Hq, Hkv;
    int64_t sumT;
    float scale_log2;
    int exclude_self;
    const float* lse;       // [Hq, sumT] natural log
    __nv_bfloat16* O;       // [sumT, Hq, 128]
    float* part;            // [slots][128]
    int64_t n_slots;        // slots of part (bounds checks of debug builds)
    int* status;
    long long wait_cycles;  // limit of the abortable waits (kWaitCycles unless a test lowers it)
};

// O += P V: A from TMEM, B an MN-major shared-memory tile (+ D when acc != 0).
__device__ __forceinline__ void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(kIdescPV), "r"(acc));
}


// tcgen05.st .16x128b.x8: 16 lanes from the lane of taddr, 32 columns.  Thread t writes,
// for k = 0..7, w[2k] to lane t/4, column 4k + t%4, and w[2k + 1] to lane t/4 + 8.
__device__ __forceinline__ void tmem_st16x128_x8(uint32_t taddr, const uint32_t* w) {
    asm volatile(
        "tcgen05.st.sync.aligned.16x128b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
        "%11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7]),
        "r"(w[8]), "r"(w[9]), "r"(w[10]), "r"(w[11]), "r"(w[12]), "r"(w[13]), "r"(w[14]), "r"(w[15])
        : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);  // .x = lo (low half)
    return *reinterpret_cast<const uint32_t*>(&v);
}

__device__ __forceinline__ int64_t tri(int64_t n) { return n * (n + 1) / 2; }

struct FwdItem {
    int valid;              // 0: no more items
    int h, qt, T;
    int64_t t0;
    int64_t slot0;          // partial slot of (this head, query tile, key tile 0)
};
constexpr int kSmemBytes = kItemOff + kSched * (int)sizeof(FwdItem) + 1024;
// the decoded items are copied with 8-byte accesses at most: every slot and every int64
// field must sit on an 8-byte boundary of the 1024-aligned shared-memory base
static_assert(alignof(FwdItem) == 8 && sizeof(FwdItem) % 8 == 0, "FwdItem layout");
static_assert(kItemOff % 8 == 0 && offsetof(FwdItem, t0) % 8 == 0 && offsetof(FwdItem, slot0) % 8 == 0,
              "FwdItem alignment in shared memory");
static_assert(kSmemBytes <= 227 * 1024, "shared memory per CTA");

__device__ __forceinline__ FwdItem fwd_item(const FwdArgs& a, int item) {
    const LseItem li = decode_lse_item(item, a.base, a.B, a.cu, kT, a.Hq);
    FwdItem t;
    t.valid = 1;
    t.h = li.hslot;
    t.qt = li.qt;
    t.t0 = li.t0;
    t.T = li.T;
    const int nt = (li.T + kT - 1) / kT;
    t.slot0 = a.base2[li.b] + (int64_t)li.hslot * tri(nt) + tri(li.qt);
    return t;
}

__global__ void __launch_bounds__(kThreads, 1)
    attn_fwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                    const __grid_constant__ CUtensorMap tm_v, const FwdArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    float* cs = reinterpret_cast<float*>(sm + kCsOff);
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + kBarOff);
    uint64_t* q_full = bars;                         // [kQBufs]
    uint64_t* q_empty = q_full + kQBufs;             // [kQBufs]
    uint64_t* k_full = q_empty + kQBufs;             // [kKStages]
    uint64_t* k_empty = k_full + kKStages;           // [kKStages]
    uint64_t* v_full = k_empty + kKStages;           // [2] (a V slot is free when p_empty completes)
    uint64_t* s_full = v_full + 2;                   // [2]
    uint64_t* s_empty = s_full + 2;                  // [2]
    uint64_t* p_full = s_empty + 2;                  // [2]
    uint64_t* p_empty = p_full + 2;                  // [2]
    // [2] O complete, for the group that takes the parity of the item's last step: each
    // group waits on every phase of its own barrier
    uint64_t* o_full = p_empty + 2;
    uint64_t* o_empty = o_full + 2;
    uint64_t* drain = o_empty + 1;     // [2] each issuer's MMAs done
    uint64_t* cs_full = drain + 2;     // [2] column sums of every quarter written
    uint64_t* cs_empty = cs_full + 2;  // [2] column sums added up by the reducer warp
    uint64_t* sched_full = cs_empty + 2;  // [kSched]
    uint64_t* sched_empty = sched_full + kSched;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + kMiscOff);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + kMiscOff + 4);
    FwdItem* sched_item = reinterpret_cast<FwdItem*>(sm + kItemOff);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kQBufs; ++i) {
            mbar_init(&q_full[i], 1);
            mbar_init(&q_empty[i], 1);
        }
        for (int i = 0; i < kKStages; ++i) {
            mbar_init(&k_full[i], 1);
            mbar_init(&k_empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&v_full[i], 1);
            mbar_init(&s_full[i], 1);
            mbar_init(&s_empty[i], kGroupWarps);
            mbar_init(&p_full[i], kGroupWarps);
            mbar_init(&p_empty[i], 1);
        }
        mbar_init(&o_full[0], 1);
        mbar_init(&o_full[1], 1);
        mbar_init(o_empty, kGroupWarps);
        mbar_init(&drain[0], 1);
        mbar_init(&drain[1], 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&cs_full[i], kGroupWarps);
            mbar_init(&cs_empty[i], 1);  // the reducer warp
        }
        for (int i = 0; i < kSched; ++i) {
            mbar_init(&sched_full[i], 1);
            mbar_init(&sched_empty[i], 3 + kEpiWarps);  // issuers, epilogue and reducer warps
        }
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(512));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // the plans (and the lse values) are complete past this point
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int total = a.info->ok && a.info2->ok ? a.info->total : 0;

    // the k-th item of this CTA, decoded by the producer (valid = 0: no more items)
    auto consume_item = [&](int k, bool warp_uniform) -> FwdItem {
        const int slot = k % kSched;
        const uint32_t par = (uint32_t)((k / kSched) & 1);
        bool got;
        if (warp_uniform) got = warp_wait(&sched_full[slot], par, abort_flag, a.status, a.wait_cycles);
        else got = wait_bar(&sched_full[slot], par, abort_flag, a.status, a.wait_cycles);
        FwdItem t{};
        if (!got) return t;
        t = sched_item[slot];
        if (warp_uniform) __syncwarp();
        if (!warp_uniform || lane == 0) mbar_arrive(&sched_empty[slot]);
        return t;
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_q)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_k)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_v)) : "memory");
            // V of step s is issued after K of step s + 1: it is needed one MMA pair
            // later, and its ring slot frees later
            struct VLoad {
                int pos, g;
                uint32_t step;
            };
            VLoad vp{0, 0, 0};
            bool have_v = false, ok = true;
            auto load_v = [&](const VLoad& v) -> bool {
                const int stage = (int)(v.step & 1);
                const uint32_t u = v.step >> 1;
                // P V of step - 2 is complete (p_empty completes with it): its V slot is free
                if (u >= 1 && !wait_bar(&p_empty[stage], (u - 1) & 1, abort_flag, a.status, a.wait_cycles)) return false;
                mbar_expect_tx(&v_full[stage], kTileBytes);
                for (int at = 0; at < 2; ++at)
                    tma_load_3d(sm + kVOff + stage * kTileBytes + at * kAtomBytes, &tm_v,
                                at * 64, v.g, v.pos, &v_full[stage]);
                return true;
            };
            // K copies issued (copy n into ring slot n % kKStages): counted apart from the
            // steps, because a step whose V load gives up leaves the loop after its K copy
            uint32_t step = 0, v_issued = 0, k_issued = 0;
            int n_items = 0;
            int item = blockIdx.x;
            for (int it = 0; ok; ++it) {
                if (item >= total) item = -1;
                const int slot = it % kSched;
                if (it >= kSched &&
                    !wait_bar(&sched_empty[slot], (uint32_t)(((it / kSched) - 1) & 1), abort_flag, a.status, a.wait_cycles))
                    break;
                FwdItem t{};
                if (item >= 0) t = fwd_item(a, item);
                sched_item[slot] = t;
                mbar_arrive(&sched_full[slot]);
                if (item < 0) break;
                const int g = t.h / (a.Hq / a.Hkv);
                const int fb = it % kQBufs;
                if (it >= kQBufs && !wait_bar(&q_empty[fb], ((it / kQBufs) - 1) & 1, abort_flag, a.status, a.wait_cycles)) break;
                mbar_expect_tx(&q_full[fb], kTileBytes);
                for (int at = 0; at < 2; ++at)
                    tma_load_3d(sm + kQOff + fb * kTileBytes + at * kAtomBytes, &tm_q, at * 64, t.h,
                                (int)(t.t0 + t.qt * kT), &q_full[fb]);
                ++n_items;
                for (int kt = 0; kt <= t.qt; ++kt, ++step) {
                    const int stage = (int)(step % kKStages);
                    const uint32_t u = step / kKStages;
                    if (u >= 1 && !wait_bar(&k_empty[stage], (u - 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(&k_full[stage], kTileBytes);
                    for (int at = 0; at < 2; ++at)
                        tma_load_3d(sm + kKOff + stage * kTileBytes + at * kAtomBytes, &tm_k, at * 64, g,
                                    (int)(t.t0 + kt * kT), &k_full[stage]);
                    ++k_issued;
                    if (have_v) {
                        if (!load_v(vp)) {
                            ok = false;
                            break;
                        }
                        ++v_issued;
                    }
                    vp = VLoad{(int)(t.t0 + kt * kT), g, step};
                    have_v = true;
                }
                if (!ok) break;
                item = (int)gridDim.x + atomicAdd(&a.info->next, 1);
            }
            if (ok && have_v && load_v(vp)) ++v_issued;
            // every copy in flight lands before the CTA exits
            for (uint32_t i = 0; i < (uint32_t)kKStages && i < k_issued; ++i)
                drain_wait(&k_full[(k_issued - 1 - i) % kKStages], ((k_issued - 1 - i) / kKStages) & 1,
                           a.status);
            for (uint32_t i = 0; i < 2 && i < v_issued; ++i)
                drain_wait(&v_full[(v_issued - 1 - i) & 1], ((v_issued - 1 - i) >> 1) & 1, a.status);
            for (int i = 0; i < kQBufs && i < n_items; ++i) {  // the last load of each Q buffer
                const int last = n_items - 1 - i;
                drain_wait(&q_full[last % kQBufs], (uint32_t)((last / kQBufs) & 1), a.status);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ S issuer
        if (lane == 0) {
            uint32_t step = 0;
            bool issued = false, ok = true;
            for (int it = 0; ok; ++it) {
                const FwdItem t = consume_item(it, false);
                if (!t.valid) break;
                const int fb = it % kQBufs;
                if (!wait_bar(&q_full[fb], (it / kQBufs) & 1, abort_flag, a.status, a.wait_cycles)) break;
                const uint32_t qa = smem_u32(sm + kQOff + fb * kTileBytes);
                for (int kt = 0; kt <= t.qt; ++kt, ++step) {
                    const int kst = (int)(step % kKStages);
                    const int stage = (int)(step & 1);  // S buffer
                    const uint32_t u = step >> 1;
                    if (!wait_bar(&k_full[kst], (step / kKStages) & 1, abort_flag, a.status, a.wait_cycles) ||
                        (u >= 1 && !wait_bar(&s_empty[stage], (u - 1) & 1, abort_flag, a.status, a.wait_cycles))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    issued = true;
                    const uint32_t ka = smem_u32(sm + kKOff + kst * kTileBytes);
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const uint32_t off = (uint32_t)((kk >> 2) * kAtomBytes + (kk & 3) * 32);
                        mma_bf16<kIdesc>(tmem + kColS + stage * 128, sw128_desc(qa + off),
                                         sw128_desc(ka + off), kk > 0 ? 1u : 0u);
                    }
                    mma_commit(&k_empty[kst]);
                    mma_commit(&s_full[stage]);
                    if (kt == t.qt) mma_commit(&q_empty[fb]);  // the item's last use of Q
                }
            }
            if (issued) {
                mma_commit(&drain[0]);
                drain_wait(&drain[0], 0, a.status);
            }
        }
    } else if (warp == 2) {
        // ----------------------------------------------------------- PV issuer
        // O += P(s) V(s): P from TMEM, the key tile of V from its ring; the first tile of an
        // item overwrites O (once the epilogue has read the previous item's O), the last
        // one hands O to the epilogue group that takes its parity
        if (lane == 0) {
            uint32_t step = 0;
            bool issued = false, ok = true;
            for (int it = 0; ok; ++it) {
                const FwdItem t = consume_item(it, false);
                if (!t.valid) break;
                for (int kt = 0; kt <= t.qt; ++kt, ++step) {
                    const int pb = (int)(step & 1);
                    if (!wait_bar(&v_full[pb], (step >> 1) & 1, abort_flag, a.status, a.wait_cycles) ||
                        !wait_bar(&p_full[pb], (step >> 1) & 1, abort_flag, a.status, a.wait_cycles) ||
                        (kt == 0 && it >= 1 && !wait_bar(o_empty, (it - 1) & 1, abort_flag, a.status, a.wait_cycles))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    issued = true;
                    const uint32_t va = smem_u32(sm + kVOff + pb * kTileBytes);
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk)
                        mma_ts(tmem + kColO, tmem + kColP + pb * 64 + kk * 8,
                               sw128_mn_desc(va + kk * 16 * 128),  // keys 16 kk ..
                               (kt == 0 && kk == 0) ? 0u : 1u);
                    mma_commit(&p_empty[pb]);  // also frees the V slot for the producer
                    if (kt == t.qt) mma_commit(&o_full[pb]);
                }
            }
            if (issued) {
                mma_commit(&drain[1]);
                drain_wait(&drain[1], 0, a.status);
            }
        }
    } else if (warp == kRedWarp) {
        // ------------------------------------------------------ column-sum reducer
        // every tile of every item, in order: the sums of the four lane quarters, added
        // in quarter order, 4 columns per lane, written as the tile's partial slot
        uint32_t step = 0;
        bool ok = true;
        for (int it = 0; ok; ++it) {
            const FwdItem t = consume_item(it, true);
            if (!t.valid) break;
            for (int kt = 0; kt <= t.qt; ++kt, ++step) {
                const int sb = (int)(step & 1);
                if (!warp_wait(&cs_full[sb], (step >> 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                    ok = false;
                    break;
                }
                const float4* c4 = reinterpret_cast<const float4*>(cs + sb * 4 * kT) + lane;
                const float4 x0 = c4[0], x1 = c4[kT / 4], x2 = c4[2 * kT / 4], x3 = c4[3 * kT / 4];
                __syncwarp();
                if (lane == 0) mbar_arrive(&cs_empty[sb]);
                const float4 sum = make_float4((x0.x + x1.x) + (x2.x + x3.x), (x0.y + x1.y) + (x2.y + x3.y),
                                               (x0.z + x1.z) + (x2.z + x3.z), (x0.w + x1.w) + (x2.w + x3.w));
                if (in_bounds(t.slot0 + kt >= 0 && t.slot0 + kt < a.n_slots, a.status))
                    reinterpret_cast<float4*>(a.part + (t.slot0 + kt) * kT)[lane] = sum;
            }
        }
    } else {
        // ------------------------------------------------------------- epilogue
        const int e = warp - kEpiWarp0;
        const int q = warp & 3;                // TMEM lane quarter
        const int grp = (e >> 2) & 1;          // takes the steps of this parity
        const int half = e >> 3;               // 64-column half of S / P and of O's columns
        const int row = q * 32 + lane;         // query row of the tile owned by this thread
        const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16);
        // S / P layout (16x256b / 16x128b): thread (g, c) = (lane / 4, lane % 4) holds rows
        // 32q + g + 8r, r = 0..3, and key columns 8k + 2c + 0..1, k = 0..7, of its half
        const int g8 = lane >> 2, c4 = lane & 3;
        uint32_t step = 0, n_out = 0;  // n_out: items whose O this group has read
        bool ok = true;
        for (int it = 0; ok; ++it) {
            const FwdItem t = consume_item(it, true);
            if (!t.valid) break;
            const int i_loc = t.qt * kT + row;                 // query index in the prompt
            const bool valid = i_loc < t.T;
            // the row normalisers (log2 units) of the 4 rows of the S / P layout; a row past
            // the prompt gets +inf, so its probabilities are exactly 0
            float lr[4];
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int ir = t.qt * kT + q * 32 + g8 + 8 * r;
                lr[r] = ir < t.T ? a.lse[(int64_t)t.h * a.sumT + t.t0 + ir] * kLog2e : INFINITY;
            }
            for (int kt = 0; kt <= t.qt; ++kt, ++step) {
                if ((int)(step & 1) != grp) continue;
                const int sb = grp;
                if (!warp_wait(&s_full[sb], (step >> 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                float* csb = cs + sb * 4 * kT;
                const bool diag = kt == t.qt;
                float csum[16];  // column sums of this thread's rows: [2k + e] for column 8k + 2c4 + e
                uint32_t w[2][16];  // packed P of both 16-lane halves, stored once all is computed
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {  // lanes 32q + 16 hh .., rows r = 2 hh, 2 hh + 1
                    uint32_t raw[32];
                    tmem_ld16x256_x8(lane_base + ((uint32_t)(16 * hh) << 16) + kColS + sb * 128 + half * 64, raw);
                    tmem_wait_ld();
                    if (hh == 1) {  // S of this warp read: the buffer may take the next tile
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&s_empty[sb]);
                    }
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
#pragma unroll
                        for (int rr = 0; rr < 2; ++rr) {
                            const int r = 2 * hh + rr;
                            float p0 = ex2(fmaf(__uint_as_float(raw[4 * k + 2 * rr]), a.scale_log2, -lr[r]));
                            float p1 = ex2(fmaf(__uint_as_float(raw[4 * k + 2 * rr + 1]), a.scale_log2, -lr[r]));
                            float c0 = p0, c1 = p1;
                            if (diag) {  // causal mask, and the self term of the column sums
                                const int dd = half * 64 + 8 * k + 2 * c4 - (q * 32 + g8 + 8 * r);
                                p0 = dd <= 0 ? p0 : 0.f;
                                p1 = dd + 1 <= 0 ? p1 : 0.f;
                                c0 = a.exclude_self && dd == 0 ? 0.f : p0;
                                c1 = a.exclude_self && dd + 1 == 0 ? 0.f : p1;
                            }
                            w[hh][2 * k + rr] = pack_bf16(p0, p1);
                            if (hh == 0 && rr == 0) {
                                csum[2 * k] = c0;
                                csum[2 * k + 1] = c1;
                            } else {
                                csum[2 * k] += c0;
                                csum[2 * k + 1] += c1;
                            }
                        }
                    }
                }
                // reduce-scatter over g8 (lane bits 2..4): lane (g8, c4) ends with columns
                // 8 g8 + 2 c4 + 0..1 = 2 lane + 0..1 of the warp's 32 rows
#pragma unroll
                for (int lvl = 0; lvl < 3; ++lvl) {
                    const int wdt = 8 >> lvl;            // values kept after this level
                    const int bit = 16 >> lvl;           // lane bit exchanged
                    const bool upper = (lane & bit) != 0;
#pragma unroll
                    for (int i = 0; i < wdt; ++i) {
                        const float send = upper ? csum[i] : csum[i + wdt];
                        const float keep = upper ? csum[i + wdt] : csum[i];
                        csum[i] = keep + __shfl_xor_sync(0xffffffffu, send, bit);
                    }
                }
                // the reducer warp is done with this buffer's sums of step - 2
                if (step >= 2 && !warp_wait(&cs_empty[sb], ((step >> 1) - 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                    ok = false;
                    break;
                }
                *reinterpret_cast<float2*>(csb + q * kT + half * 64 + 2 * lane) = make_float2(csum[0], csum[1]);
                // P V of step - 2 has read this P buffer
                if (step >= 2 && !warp_wait(&p_empty[sb], ((step >> 1) - 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                    ok = false;
                    break;
                }
                tmem_st16x128_x8(lane_base + kColP + sb * 64 + half * 32, w[0]);
                tmem_st16x128_x8(lane_base + (16u << 16) + kColP + sb * 64 + half * 32, w[1]);
                asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&p_full[sb]);
                    mbar_arrive(&cs_full[sb]);
                }
            }
            if (!ok) break;
            if ((int)((step - 1) & 1) != grp) continue;  // the other group ends this item
            // O of the item: this warp's 32 rows x 64 columns
            if (!warp_wait(&o_full[grp], n_out & 1, abort_flag, a.status, a.wait_cycles)) break;
            ++n_out;
            tc_fence_after();
#pragma unroll
            for (int ch = 0; ch < 2; ++ch) {
                float v[32];
                tmem_ld32(lane_base + kColO + half * 64 + ch * 32, v);
                tmem_wait_ld();
                if (valid && in_bounds(t.t0 + i_loc < a.sumT && t.h >= 0 && t.h < a.Hq, a.status)) {
                    uint4* out = reinterpret_cast<uint4*>(
                        a.O + ((t.t0 + i_loc) * a.Hq + t.h) * (int64_t)kD + half * 64 + ch * 32);
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        out[k] = make_uint4(pack_bf16(v[8 * k], v[8 * k + 1]), pack_bf16(v[8 * k + 2], v[8 * k + 3]),
                                            pack_bf16(v[8 * k + 4], v[8 * k + 5]), pack_bf16(v[8 * k + 6], v[8 * k + 7]));
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(o_empty);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        __syncwarp();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512));
    }
}

// C_j (+)= sum over heads h and query tiles qt >= kt(j) of the partial slots of key j.  A block
// takes 32 keys; its warp w sums heads w, w + 8, .. (each over qt in order), and the 8 warp
// sums are added in order: a fixed order, whatever the launch.
constexpr int kRedHeadLanes = 8;
__global__ void __launch_bounds__(32 * kRedHeadLanes)
    imp_fwd_reduce_kernel(const float* __restrict__ part, const int32_t* cu, const int32_t* base2,
                          const PlanInfo* info, const PlanInfo* info2, int B, int Hq, int64_t sumT,
                          int accumulate, float* acc, int64_t n_slots, int* status) {
    __shared__ float red[kRedHeadLanes][32];
    asm volatile("griddepcontrol.wait;" ::: "memory");  // the forward's partial slots are complete
    const int jj = threadIdx.x & 31, hl = threadIdx.x >> 5;
    const int64_t j = (int64_t)blockIdx.x * 32 + jj;
    float v = 0.f;
    if (j < sumT && info->ok && info2->ok) {
        const int b = upper_slot(cu, B, j);
        const int T = cu[b + 1] - cu[b];
        const int nt = (T + kT - 1) / kT;
        const int jl = (int)(j - cu[b]), kt = jl / kT, col = jl - kt * kT;
        const bool ok = in_bounds(b >= 0 && b < B && base2[b] + (int64_t)Hq * tri(nt) <= n_slots, status);
        for (int h = hl; ok && h < Hq; h += kRedHeadLanes) {
            const int64_t s0 = base2[b] + (int64_t)h * tri(nt);
            float vh = 0.f;
            constexpr int kBatch = 8;  // loads in flight before they are added, in order
            for (int q0 = kt; q0 < nt; q0 += kBatch) {
                float pv[kBatch];
#pragma unroll
                for (int i = 0; i < kBatch; ++i)
                    pv[i] = q0 + i < nt ? part[(s0 + tri(q0 + i) + kt) * kT + col] : 0.f;
#pragma unroll
                for (int i = 0; i < kBatch; ++i)
                    if (q0 + i < nt) vh += pv[i];
            }
            v += vh;
        }
    }
    red[hl][jj] = v;
    __syncthreads();
    if (hl == 0 && j < sumT) {
        float sum = 0.f;
#pragma unroll
        for (int k = 0; k < kRedHeadLanes; ++k) sum += red[k][jj];
        acc[j] = accumulate ? acc[j] + sum : sum;
    }
}

// bf16 tensor map of 3 dimensions (d0 innermost), box b0 x b1 x b2, 128-byte swizzle.
estp_status make_map3(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                      uint64_t s1, uint64_t s2, uint32_t b0, uint32_t b1, uint32_t b2) {
    auto fn = tensor_map_encoder();
    if (!fn) return fail(ESTP_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    cuuint64_t dims[3] = {d0, d1, d2};
    cuuint64_t strides[2] = {s1, s2};
    cuuint32_t box[3] = {b0, b1, b2};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                    box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(ESTP_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    return ESTP_OK;
}

}  // namespace

estp_status launch_attn_forward(estp_ctx* ctx, const void* Q, const void* K, const void* V,
                                const float* lse_in, int Hq, int Hkv, float scale,
                                const int32_t* cu, int B, int64_t sumT, int max_seqlen,
                                bool exclude_self, bool accumulate, float* acc, void* O,
                                cudaStream_t st) {
    // workspace: partial slots | lse (when not given) | plans | row-normaliser plan
    const int64_t max_nt = (max_seqlen + kT - 1) / kT;
    const int64_t tiles_bound = (sumT + kT - 1) / kT + B;          // sum of nt_b
    const int64_t slots_bound = (int64_t)Hq * tiles_bound * (max_nt + 1) / 2 + Hq;
    const size_t off_part = 0;
    const size_t off_lse = off_part + align_up(sizeof(float) * (size_t)slots_bound * kT, 256);
    const size_t off_plan = off_lse + (lse_in ? 0 : align_up(sizeof(float) * (size_t)Hq * sumT, 256));
    const size_t off_base2 = off_plan + align_up(sizeof(int32_t) * (size_t)(B + 1), 256);
    const size_t off_info = off_base2 + align_up(sizeof(int32_t) * (size_t)(B + 1), 256);
    const size_t off_info2 = off_info + 256;
    const size_t off_lse_plan = off_info2 + 256;
    // the row-normaliser kernel's own plan comes after ours: reserve for it too
    estp_status s = ws_reserve(ctx, off_lse_plan + align_up(sizeof(int32_t) * (size_t)(B + 1), 256) +
                                        sizeof(PlanInfo) + 256);
    if (s != ESTP_OK) return s;
    char* ws = static_cast<char*>(ctx->ws);
    float* part = reinterpret_cast<float*>(ws + off_part);
    int32_t* base = reinterpret_cast<int32_t*>(ws + off_plan);
    int32_t* base2 = reinterpret_cast<int32_t*>(ws + off_base2);
    PlanInfo* info = reinterpret_cast<PlanInfo*>(ws + off_info);
    PlanInfo* info2 = reinterpret_cast<PlanInfo*>(ws + off_info2);
    const float* lse = lse_in;
    if (!lse_in) {  // pass 1: the row normalisers of every head
        float* l = reinterpret_cast<float*>(ws + off_lse);
        ImpHeads all;
        if ((s = build_heads(nullptr, Hq, Hq, Hkv, &all)) != ESTP_OK) return s;
        if ((s = launch_lse_tc(ctx, Q, K, Hq, Hkv, kD, scale, all, cu, B, sumT, max_seqlen, l, st,
                               off_lse_plan)) != ESTP_OK)
            return s;
        lse = l;
    }
    // plans: items (prompt, query tile, head), and the partial slots (tile pairs x heads)
    attn_plan2_kernel<<<2, 1024, 0, st>>>(cu, B, sumT, max_seqlen, kT, 1, Hq, 1, base, info, 2, base2,
                                          info2, ctx->status);
    // the forward and the reduce are programmatic dependents of the launch before them:
    // each starts its prologue early and waits on the device for its inputs
    cudaLaunchAttribute pdl[1];
    pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    pdl[0].val.programmaticStreamSerializationAllowed = 1;
    auto config = [&](dim3 grid, dim3 block, size_t smem) {
        cudaLaunchConfig_t c = {};
        c.gridDim = grid;
        c.blockDim = block;
        c.dynamicSmemBytes = smem;
        c.stream = st;
        c.attrs = pdl;
        c.numAttrs = 1;
        return c;
    };
    cudaError_t e;
    CUtensorMap mq, mk, mv;
    // Q, K, V: (d, head, token), one head's 64 d x 128 tokens per box
    if ((s = make_map3(&mq, Q, kD, Hq, sumT, (uint64_t)kD * 2, (uint64_t)Hq * kD * 2, 64, 1, kT)) != ESTP_OK) return s;
    if ((s = make_map3(&mk, K, kD, Hkv, sumT, (uint64_t)kD * 2, (uint64_t)Hkv * kD * 2, 64, 1, kT)) != ESTP_OK) return s;
    if ((s = make_map3(&mv, V, kD, Hkv, sumT, (uint64_t)kD * 2, (uint64_t)Hkv * kD * 2, 64, 1, kT)) != ESTP_OK) return s;
    FwdArgs a{};
    a.cu = cu; a.base = base; a.base2 = base2; a.info = info; a.info2 = info2;
    a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.sumT = sumT;
    a.scale_log2 = scale * kLog2e;
    a.exclude_self = exclude_self ? 1 : 0;
    a.lse = lse; a.O = static_cast<__nv_bfloat16*>(O); a.part = part; a.status = ctx->status;
    a.n_slots = slots_bound;
    a.wait_cycles = ctx->wait_cycles;
    e = cudaFuncSetAttribute(attn_fwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (e != cudaSuccess) return cuda_fail(e, "attention forward smem attribute");
    cudaLaunchConfig_t cf = config(dim3((unsigned)ctx->num_sms), dim3(kThreads), kSmemBytes);
    e = cudaLaunchKernelEx(&cf, attn_fwd_kernel, mq, mk, mv, a);
    if (e != cudaSuccess) return cuda_fail(e, "attention forward launch");
    cudaLaunchConfig_t cr = config(dim3((unsigned)((sumT + 31) / 32)), dim3(32 * kRedHeadLanes), 0);
    e = cudaLaunchKernelEx(&cr, imp_fwd_reduce_kernel, (const float*)part, cu, (const int32_t*)base2,
                           (const PlanInfo*)info, (const PlanInfo*)info2, B, Hq, sumT, accumulate ? 1 : 0, acc,
                           slots_bound, ctx->status);
    if (e != cudaSuccess) return cuda_fail(e, "attention forward reduce launch");
    e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "attention forward reduce launch");
}

}  // namespace estp
