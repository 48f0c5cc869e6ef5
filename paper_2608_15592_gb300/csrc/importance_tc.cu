// tcgen05 path of the attention kernels (bf16 Q/K, head_dim 64 or 128).
//
// Both kernels recompute S = Q K^T tile by tile on the 5th-generation tensor cores
// and never materialise the attention matrix A (Sec. 3.1).  One persistent CTA per
// SM runs a warp-specialised pipeline:
//   warp 0      TMA producer: the item's fixed 128-row tile, then a ring of streamed
//               128-row tiles (128B-swizzled, one 64-column atom per TMA box)
//   warp 1      MMA issuer: D[128 x 128] (fp32, TMEM) = fixed (M side) x streamed^T,
//               double-buffered accumulators (2 x 128 TMEM columns)
//   warps 2-9   epilogue: tcgen05.ld of the accumulator, exp2 and row reductions;
//               warp w reads TMEM lanes 32*(w%4).. (its quarter), and the two warps
//               of a quarter split the 128 columns (halves)
//
// LSE mode (rows = queries): lse_i = ln sum_{j<=i} exp(scale q_i.k_j), streaming the
//   key tiles 0..qt with a running max (flash-style online normaliser).
// Column-sum mode (rows = keys): C_j += sum_{i>=j} 2^(scale*log2e q_i.k_j - log2e*lse_i),
//   streaming the query tiles of the item for every selected head of the KV group, so
//   the sum over queries stays in the thread that owns key j.
//
// Every mbarrier wait is bounded (about 2 s of SM clock); on expiry the CTA records
// ESTP_ERR_TIMEOUT in the status word and drains without further waits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "importance_tc.cuh"
#include "ptx.cuh"

namespace estp {
namespace {

constexpr int kTile = 128;
constexpr int kQcTc = 4;
constexpr int kThreads = 320;          // 10 warps
constexpr int kEpiWarp0 = 2;           // warps 2..9
constexpr int kAccCols = 128;
constexpr int kSched = 4;              // depth of the item-index ring (producer -> consumers)

enum Mode { kModeLse = 0, kModeImp = 1 };

template <int D>
struct Cfg {
    static constexpr int kAtoms = D / 64;
    static constexpr int kTileBytes = kTile * 128 * kAtoms;  // 128 rows x D bf16
    static constexpr int kStages = D == 64 ? 8 : 4;
    static constexpr int kKSteps = D / 16;
    // dynamic smem layout (offsets from a 1024-aligned base)
    static constexpr int kFixOff = 0;
    static constexpr int kRingOff = 2 * kTileBytes;
    static constexpr int kNlOff = kRingOff + kStages * kTileBytes;  // [8 warps][64] f32
    static constexpr int kMergeOff = kNlOff + 8 * 64 * 4;             // [2][4][32] float2
    static constexpr int kBarOff = kMergeOff + 2 * 4 * 32 * 8;
    // fix_full/empty[2], ring_full/empty[kStages], acc_full/empty[2], drain,
    // sched_full/empty[kSched], xfull/xempty[2][4]
    static constexpr int kNumBars = 2 + 2 + 2 * kStages + 2 + 2 + 1 + 2 * kSched + 16;
    static constexpr int kMiscOff = kBarOff + kNumBars * 8;  // tmem addr, abort flag, sched items
    static constexpr int kSmemBytes = kMiscOff + 16 + 4 * kSched + 1024;  // + alignment slack
};

struct TcArgs {
    const int32_t* cu;
    const int32_t* base;
    const PlanInfo* info;
    int B, Hq, Hkv;
    int64_t sumT;
    float scale_log2;
    int exclude_self;
    const float* lse;   // column-sum mode input [Hq, sumT]
    float* part;        // column-sum mode output [c][G][sumT]
    float* lse_out;     // LSE mode output [Hq, sumT]
    int* status;
    ImpHeads hs;
};

// ------------------------------------------------------------------ PTX helpers
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int x, int y, int z,
                                            uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row groups
// 1024 bytes apart (stride byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr) {
    return (uint64_t)((addr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both K-major,
// N = 128, M = 128.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kTile >> 3) << 17) |
                            ((uint32_t)(kTile >> 4) << 24);

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(kIdesc), "r"(acc));
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_u32(bar))
        : "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
        "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
        "%28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr));
#pragma unroll
    for (int k = 0; k < 32; ++k) v[k] = __uint_as_float(r[k]);
}

__device__ __forceinline__ void tmem_wait_ld() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}


// --------------------------------------------------------------- item description
struct TcItem {
    int b, T;
    int64_t t0;
    int fix_y, fix_row0;       // fixed tile: head (LSE: query head, IMP: KV head), first row
    int n_steps;
    // LSE: the query head; IMP: group slot, key tile, query-tile range, chunk slot
    int h, g, kt, qt0, qt1, chunk;
};

template <int MODE>
__device__ __forceinline__ TcItem make_item(const TcArgs& a, int item) {
    TcItem t;
    if (MODE == kModeLse) {
        const LseItem li = decode_lse_item(item, a.base, a.B, a.cu, kTile, a.hs.n_heads);
        t.b = li.b; t.T = li.T; t.t0 = li.t0;
        t.h = a.hs.head_list[li.hslot];
        t.fix_y = t.h;
        t.fix_row0 = li.qt * kTile;
        t.qt0 = li.qt;
        t.n_steps = li.qt + 1;  // key tiles 0..qt
        t.g = 0; t.kt = 0; t.qt1 = li.qt + 1; t.chunk = 0;
    } else {
        const ImpItem ii = decode_imp_item(item, a.base, a.B, a.cu, kTile, kQcTc);
        t.b = ii.b; t.T = ii.T; t.t0 = ii.t0;
        t.g = ii.g; t.kt = ii.kt; t.qt0 = ii.qt0; t.qt1 = ii.qt1;
        t.chunk = (ii.qt0 - ii.kt) / kQcTc;
        t.fix_y = a.hs.group[ii.g];
        t.fix_row0 = ii.kt * kTile;
        const int nh = a.hs.begin[ii.g + 1] - a.hs.begin[ii.g];
        t.n_steps = nh * (ii.qt1 - ii.qt0);
        t.h = 0;
    }
    return t;
}

// Streamed tile of step s of an item: (head for TMA y, first row).
template <int MODE>
__device__ __forceinline__ void step_tile(const TcArgs& a, const TcItem& t, int s, int& y, int& row0,
                                          int& head, int& qt) {
    if (MODE == kModeLse) {
        y = t.h / (a.Hq / a.Hkv);
        row0 = s * kTile;  // key tile s
        head = t.h;
        qt = t.qt0;
    } else {
        const int nq = t.qt1 - t.qt0;
        const int hi = s / nq;
        qt = t.qt0 + (s - hi * nq);
        head = a.hs.head_list[a.hs.begin[t.g] + hi];
        y = head;
        row0 = qt * kTile;
    }
}

template <int D, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_fix, const __grid_constant__ CUtensorMap tm_str,
                   const TcArgs a) {
    using C = Cfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    uint8_t* fix = sm + C::kFixOff;
    uint8_t* ring = sm + C::kRingOff;
    float* nl_all = reinterpret_cast<float*>(sm + C::kNlOff);
    float2* merge = reinterpret_cast<float2*>(sm + C::kMergeOff);
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + C::kBarOff);
    uint64_t* fix_full = bars;                    // [2]
    uint64_t* fix_empty = bars + 2;               // [2]
    uint64_t* ring_full = bars + 4;               // [kStages]
    uint64_t* ring_empty = bars + 4 + C::kStages; // [kStages]
    uint64_t* acc_full = bars + 4 + 2 * C::kStages;
    uint64_t* acc_empty = acc_full + 2;
    uint64_t* drain = acc_empty + 2;
    uint64_t* sched_full = drain + 1;             // [kSched]
    uint64_t* sched_empty = sched_full + kSched;  // [kSched]
    uint64_t* xfull = sched_empty + kSched;       // [2][4]: half-1 partials ready
    uint64_t* xempty = xfull + 8;                 // [2][4]: half-0 has read them
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + C::kMiscOff);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + C::kMiscOff + 4);
    volatile int* sched_item = reinterpret_cast<volatile int*>(sm + C::kMiscOff + 16);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&fix_full[i], 1);
            mbar_init(&fix_empty[i], 1);
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 8);  // one arrival per epilogue warp
        }
        for (int i = 0; i < C::kStages; ++i) {
            mbar_init(&ring_full[i], 1);
            mbar_init(&ring_empty[i], 1);
        }
        mbar_init(drain, 1);
        for (int i = 0; i < kSched; ++i) {
            mbar_init(&sched_full[i], 1);
            mbar_init(&sched_empty[i], 1 + 8);  // MMA thread + 8 epilogue warps
        }
        for (int i = 0; i < 8; ++i) {
            mbar_init(&xfull[i], 1);
            mbar_init(&xempty[i], 1);
        }
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 1) {  // TMEM: 2 accumulators x 128 columns
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(2 * kAccCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    PlanInfo* info = const_cast<PlanInfo*>(a.info);
    const int total = info->total;

    // Item k of this CTA, published by the producer in slot k % kSched (-1 = no more).
    auto consume_item = [&](int k, bool warp_uniform) -> int {
        const int slot = k % kSched;
        const uint32_t par = (uint32_t)((k / kSched) & 1);
        bool got;
        if (warp_uniform) got = warp_wait(&sched_full[slot], par, abort_flag, a.status);
        else got = wait_bar(&sched_full[slot], par, abort_flag, a.status);
        if (!got) return -1;
        const int item = sched_item[slot];
        if (warp_uniform) __syncwarp();
        if (!warp_uniform || lane == 0) mbar_arrive(&sched_empty[slot]);
        return item;
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_fix)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_str)) : "memory");
            long long step = 0;
            int item = blockIdx.x;
            for (int it = 0;; ++it) {
                if (item >= total) item = -1;
                const int slot = it % kSched;
                if (it >= kSched &&
                    !wait_bar(&sched_empty[slot], (uint32_t)(((it / kSched) - 1) & 1), abort_flag, a.status))
                    break;
                sched_item[slot] = item;
                mbar_arrive(&sched_full[slot]);  // release: the item index is visible to waiters
                if (item < 0) break;
                const TcItem t = make_item<MODE>(a, item);
                const int fb = it & 1;
                if (it >= 2 && !wait_bar(&fix_empty[fb], ((it >> 1) - 1) & 1, abort_flag, a.status)) break;
                mbar_expect_tx(&fix_full[fb], C::kTileBytes);
#pragma unroll
                for (int at = 0; at < C::kAtoms; ++at)
                    tma_load_3d(fix + fb * C::kTileBytes + at * kTile * 128, &tm_fix, at * 64, t.fix_y,
                                (int)(t.t0 + t.fix_row0), &fix_full[fb]);
                bool ok = true;
                for (int s = 0; s < t.n_steps; ++s, ++step) {
                    const int stage = (int)(step % C::kStages);
                    const long long u = step / C::kStages;
                    if (u >= 1 && !wait_bar(&ring_empty[stage], (uint32_t)((u - 1) & 1), abort_flag, a.status)) {
                        ok = false;
                        break;
                    }
                    int y, row0, head, qt;
                    step_tile<MODE>(a, t, s, y, row0, head, qt);
                    mbar_expect_tx(&ring_full[stage], C::kTileBytes);
#pragma unroll
                    for (int at = 0; at < C::kAtoms; ++at)
                        tma_load_3d(ring + stage * C::kTileBytes + at * kTile * 128, &tm_str, at * 64, y,
                                    (int)(t.t0 + row0), &ring_full[stage]);
                }
                if (!ok) break;
                item = (int)gridDim.x + atomicAdd(&info->next, 1);
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0) {
            long long step = 0;
            bool issued = false;
            for (int it = 0;; ++it) {
                const int item = consume_item(it, false);
                if (item < 0) break;
                const TcItem t = make_item<MODE>(a, item);
                const int fb = it & 1;
                if (!wait_bar(&fix_full[fb], (it >> 1) & 1, abort_flag, a.status)) break;
                const uint32_t fix_addr = smem_u32(fix + fb * C::kTileBytes);
                bool ok = true;
                for (int s = 0; s < t.n_steps; ++s, ++step) {
                    const int stage = (int)(step % C::kStages);
                    const long long u = step / C::kStages;
                    const int ab = (int)(step & 1);
                    const long long ua = step >> 1;
                    if (!wait_bar(&ring_full[stage], (uint32_t)(u & 1), abort_flag, a.status) ||
                        (ua >= 1 && !wait_bar(&acc_empty[ab], (uint32_t)((ua - 1) & 1), abort_flag, a.status))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t str_addr = smem_u32(ring + stage * C::kTileBytes);
#pragma unroll
                    for (int kk = 0; kk < C::kKSteps; ++kk) {
                        const uint32_t off = (uint32_t)((kk >> 2) * kTile * 128 + (kk & 3) * 32);
                        mma_bf16(tmem + (uint32_t)(ab * kAccCols), sw128_desc(fix_addr + off),
                                 sw128_desc(str_addr + off), kk > 0 ? 1u : 0u);
                    }
                    mma_commit(&ring_empty[stage]);
                    mma_commit(&acc_full[ab]);
                    issued = true;
                }
                if (!ok) break;
                mma_commit(&fix_empty[fb]);
            }
            if (issued) {  // every MMA done before the TMEM is released
                mma_commit(drain);
                drain_wait(drain, 0, a.status);
            }
        }
    } else {
        // ------------------------------------------------------------- epilogue
        const int q = warp & 3;                    // TMEM lane quarter
        const int half = (warp - kEpiWarp0) >> 2;  // column half
        const int row = q * 32 + lane;             // accumulator row owned by this thread
        float* nl = nl_all + (warp - kEpiWarp0) * 64;
        long long step = 0;
        bool ok = true;
        for (int it = 0; ok; ++it) {
            const int item = consume_item(it, true);
            if (item < 0) break;
            const TcItem t = make_item<MODE>(a, item);
            float2 acc2 = make_float2(0.f, 0.f);   // column-sum mode
            float m = -1e30f, ssum = 0.f;          // LSE mode
            float pre0 = 0.f, pre1 = 0.f;
            auto load_nl = [&](int s, float& r0, float& r1) {
                int y, row0, head, qt;
                step_tile<MODE>(a, t, s, y, row0, head, qt);
                const int i0 = row0 + half * 64 + lane, i1 = i0 + 32;
                const float* l = a.lse + (int64_t)head * a.sumT + t.t0;
                r0 = i0 < t.T ? -l[i0] * kLog2e : -INFINITY;
                r1 = i1 < t.T ? -l[i1] * kLog2e : -INFINITY;
            };
            if (MODE == kModeImp) load_nl(0, pre0, pre1);
            for (int s = 0; s < t.n_steps && ok; ++s, ++step) {
                int y, row0, head, qt;
                step_tile<MODE>(a, t, s, y, row0, head, qt);
                if (MODE == kModeImp) {
                    __syncwarp();
                    nl[lane] = pre0;
                    nl[lane + 32] = pre1;
                    __syncwarp();
                    if (s + 1 < t.n_steps) load_nl(s + 1, pre0, pre1);
                }
                const int ab = (int)(step & 1);
                ok = warp_wait(&acc_full[ab], (uint32_t)((step >> 1) & 1), abort_flag, a.status);
                if (!ok) break;
                tc_fence_after();
                float v[64];
                const uint32_t taddr = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * kAccCols + half * 64);
                tmem_ld32(taddr, v);
                tmem_ld32(taddr + 32, v + 32);
                tmem_wait_ld();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&acc_empty[ab]);
                const int col0 = half * 64;
                if (MODE == kModeImp) {
                    const float2 sc = make_float2(a.scale_log2, a.scale_log2);
                    if (qt != t.kt) {
#pragma unroll
                        for (int c = 0; c < 64; c += 4) {
                            const float4 n4 = *reinterpret_cast<const float4*>(nl + c);
                            float2 x0 = __ffma2_rn(make_float2(v[c], v[c + 1]), sc, make_float2(n4.x, n4.y));
                            float2 x1 = __ffma2_rn(make_float2(v[c + 2], v[c + 3]), sc, make_float2(n4.z, n4.w));
                            acc2 = __fadd2_rn(acc2, make_float2(ex2(x0.x), ex2(x0.y)));
                            acc2 = __fadd2_rn(acc2, make_float2(ex2(x1.x), ex2(x1.y)));
                        }
                    } else {  // diagonal tile: query i = col, key j = row (local); keep i >= j
#pragma unroll
                        for (int c = 0; c < 64; c += 2) {
                            const float2 n2 = *reinterpret_cast<const float2*>(nl + c);
                            float2 x = __ffma2_rn(make_float2(v[c], v[c + 1]), sc, n2);
                            const int i0 = col0 + c, i1 = i0 + 1;
                            const bool k0 = a.exclude_self ? i0 > row : i0 >= row;
                            const bool k1 = a.exclude_self ? i1 > row : i1 >= row;
                            acc2 = __fadd2_rn(acc2, make_float2(k0 ? ex2(x.x) : 0.f, k1 ? ex2(x.y) : 0.f));
                        }
                    }
                } else {
                    const bool diag = (s == t.qt0);  // key tile == query tile
                    float mx = -1e30f;
#pragma unroll
                    for (int c = 0; c < 64; ++c) {
                        if (diag && col0 + c > row) v[c] = -INFINITY;
                        mx = fmaxf(mx, v[c]);
                    }
                    const float nm = fmaxf(m, mx * a.scale_log2);
                    ssum *= ex2(m - nm);
                    m = nm;
                    const float2 sc = make_float2(a.scale_log2, a.scale_log2);
                    const float2 nm2 = make_float2(-nm, -nm);
                    float2 s2 = make_float2(0.f, 0.f);
#pragma unroll
                    for (int c = 0; c < 64; c += 2) {
                        float2 x = __ffma2_rn(make_float2(v[c], v[c + 1]), sc, nm2);
                        s2 = __fadd2_rn(s2, make_float2(ex2(x.x), ex2(x.y)));
                    }
                    ssum += s2.x + s2.y;
                }
            }
            if (!ok) break;
            // merge the two column halves of each row (bounded mbarrier hand-off), then write
            const int pb = it & 1;
            const uint32_t use = (uint32_t)(it >> 1);
            float2* mb = merge + pb * 128;
            uint64_t* xf = &xfull[pb * 4 + q];
            uint64_t* xe = &xempty[pb * 4 + q];
            if (half == 1) {
                if (use >= 1) ok = warp_wait(xe, (use - 1) & 1, abort_flag, a.status);
                if (!ok) break;
                mb[q * 32 + lane] = MODE == kModeImp ? make_float2(acc2.x + acc2.y, 0.f)
                                                     : make_float2(m, ssum);
                __syncwarp();
                if (lane == 0) mbar_arrive(xf);
            } else {
                ok = warp_wait(xf, use & 1, abort_flag, a.status);
                if (!ok) break;
                const float2 o = mb[q * 32 + lane];
                __syncwarp();
                if (lane == 0) mbar_arrive(xe);
                if (MODE == kModeImp) {
                    const int j = t.fix_row0 + row;
                    if (j < t.T)
                        a.part[((int64_t)t.chunk * a.hs.n_groups + t.g) * a.sumT + t.t0 + j] =
                            acc2.x + acc2.y + o.x;
                } else {
                    const float mm = fmaxf(m, o.x);
                    const float ss = ssum * ex2(m - mm) + o.y * ex2(o.x - mm);
                    const int i = t.fix_row0 + row;
                    if (i < t.T) a.lse_out[(int64_t)t.h * a.sumT + t.t0 + i] = (mm + lg2(ss)) * kLn2;
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        __syncwarp();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(2 * kAccCols));
    }
}

// ------------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

// [sumT, heads, d] bf16 viewed as a 3-D tensor (d, heads, sumT); box 64 x 1 x 128.
estp_status make_map(CUtensorMap* m, const void* base, int heads, int d, int64_t sumT) {
    auto fn = encode_fn();
    if (!fn) return fail(ESTP_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)heads, (cuuint64_t)sumT};
    cuuint64_t strides[2] = {(cuuint64_t)d * 2, (cuuint64_t)heads * d * 2};
    cuuint32_t box[3] = {64, 1, (cuuint32_t)kTile};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                    box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(ESTP_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    return ESTP_OK;
}

template <int D, int MODE>
estp_status launch_tc(estp_ctx* ctx, const CUtensorMap& fixm, const CUtensorMap& strm,
                      const TcArgs& a, cudaStream_t st) {
    auto kern = attn_tc_kernel<D, MODE>;
    const int smem = Cfg<D>::kSmemBytes;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "tc kernel smem attribute");
    kern<<<ctx->num_sms, kThreads, smem, st>>>(fixm, strm, a);
    e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "tc kernel launch");
}

}  // namespace

bool tc_supported(estp_dtype dtype, int d) { return dtype == ESTP_BF16 && (d == 64 || d == 128); }
int tc_tile() { return kTile; }
int tc_qc() { return kQcTc; }

estp_status launch_lse_tc(estp_ctx* ctx, const void* Q, const void* K, int Hq, int Hkv, int d,
                          float scale, const ImpHeads& hs, const int32_t* cu, int B, int64_t sumT,
                          int max_seqlen, float* lse, cudaStream_t st, size_t ws_off) {
    const size_t off_info = ws_off + align_up(sizeof(int32_t) * (size_t)(B + 1), 256);
    estp_status s = ws_reserve(ctx, off_info + sizeof(PlanInfo));
    if (s != ESTP_OK) return s;
    char* ws = static_cast<char*>(ctx->ws);
    TcArgs a{};
    a.cu = cu; a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.sumT = sumT;
    a.base = reinterpret_cast<int32_t*>(ws + ws_off);
    a.info = reinterpret_cast<PlanInfo*>(ws + off_info);
    a.scale_log2 = scale * kLog2e;
    a.lse_out = lse;
    a.status = ctx->status;
    a.hs = hs;
    CUtensorMap mq, mk;
    if ((s = make_map(&mq, Q, Hq, d, sumT)) != ESTP_OK) return s;
    if ((s = make_map(&mk, K, Hkv, d, sumT)) != ESTP_OK) return s;
    attn_plan_kernel<<<1, 1024, 0, st>>>(cu, B, sumT, max_seqlen, kTile, 1, hs.n_heads, 1,
                                         const_cast<int32_t*>(a.base), const_cast<PlanInfo*>(a.info),
                                         ctx->status);
    return d == 64 ? launch_tc<64, kModeLse>(ctx, mq, mk, a, st)
                   : launch_tc<128, kModeLse>(ctx, mq, mk, a, st);
}

estp_status launch_imp_tc(estp_ctx* ctx, const void* Q, const void* K, const float* lse, int Hq,
                          int Hkv, int d, float scale, const ImpHeads& hs, const int32_t* cu,
                          int B, int64_t sumT, bool exclude_self, const int32_t* base,
                          const PlanInfo* info, float* part, cudaStream_t st) {
    TcArgs a{};
    a.cu = cu; a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.sumT = sumT;
    a.base = base; a.info = info;
    a.scale_log2 = scale * kLog2e;
    a.exclude_self = exclude_self ? 1 : 0;
    a.lse = lse;
    a.part = part;
    a.status = ctx->status;
    a.hs = hs;
    CUtensorMap mq, mk;
    estp_status s;
    if ((s = make_map(&mq, Q, Hq, d, sumT)) != ESTP_OK) return s;
    if ((s = make_map(&mk, K, Hkv, d, sumT)) != ESTP_OK) return s;
    return d == 64 ? launch_tc<64, kModeImp>(ctx, mk, mq, a, st)
                   : launch_tc<128, kModeImp>(ctx, mk, mq, a, st);
}

}  // namespace estp
