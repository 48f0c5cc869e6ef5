// tcgen05 path of the attention kernels (bf16 Q/K, head_dim 64 or 128).
//
// Both kernels recompute S = Q K^T tile by tile on the 5th-generation tensor cores
// and never materialise the attention matrix A (Sec. 3.1).  One persistent CTA per
// SM works on "pair items": two fixed 128-row tiles (2p and 2p+1) multiplied by the
// same sequence of streamed 128-row tiles, so that every streamed tile feeds two MMAs.
// The CTA runs a warp-specialised pipeline:
//   warp 0       TMA producer: the item's two fixed tiles, then a ring of streamed tiles
//                (128B-swizzled, one 64-column atom per TMA box) and, for column sums,
//                the lse values of each streamed query tile
//   warps 1, 18  MMA issuers, one per fixed tile: D_A = A x S^T (warp 1) and
//                D_B = B x S^T (warp 18), M = 128, N = 128, fp32 in TMEM, each
//                double-buffered: 2 x 2 x 128 = all 512 TMEM columns
//   warps 2-17   epilogue: tcgen05.ld, exp2 and row reductions; warp w reads TMEM lanes
//                32*(w%4).. (its quarter).  LSE mode: 8 warps per fixed tile, two per
//                quarter splitting the 128 columns, at every step.  Column-sum mode: a
//                group of 4 warps per fixed tile and accumulator buffer reads all 128
//                columns at every other step, so the two buffers' groups work a step
//                apart and each step's lse values pass through 8 warps instead of 16
//                (12 % faster there; in LSE mode the longer hold on the accumulator
//                before it is released costs more than it gains)
// Two issuers because the tensor core's instruction queue is shallow: a check of an
// mbarrier costs an issuing thread ~150-180 cycles even when the phase has completed,
// and with a single issuer the pipe idles through its two waits and commits per step;
// with one issuer per tile those waits overlap the other tile's MMAs.
//
// LSE mode (rows = queries): a pair = query tiles q, q+1 of one head (q odd when the
//   prompt's tile count is odd, so that the unpaired tile is tile 0), streaming the key
//   tiles 0..q+1 with a running max (flash-style normaliser); a tile skips the key tiles
//   after its own query tile.
// Column-sum mode (rows = keys): pair p = key tiles 2p, 2p+1 of one KV group,
//   C_j += sum_{i>=j} 2^(scale*log2e q_i.k_j - log2e*lse_i), streaming the query tiles
//   of the item's chunk for every selected head of the group, so the sum over queries
//   stays in the thread that owns key j; a tile skips query tiles before its own key
//   tile.
//
// Every mbarrier wait is bounded (about 2 s of SM clock; a test may lower the limit of
// the abortable waits through estp_set_wait_limit); on expiry the CTA records
// ESTP_ERR_TIMEOUT in the status word, skips every further abortable wait, and drains:
// the producer waits (full limit) for its last copies into each ring slot, fixed-tile
// buffer and lse slot, the issuers for all their MMAs, before the TMEM is freed.
#include "importance_tc.cuh"
#include "tcgen05.cuh"

namespace estp {
namespace {

constexpr int kTile = 128;             // rows of a fixed or streamed tile
constexpr int kPair = 2 * kTile;       // rows of the fixed pair (the plan's tile)
// Pairs of query tiles per column-sum item: the largest of kQcChoices that still gives the
// persistent grid about kItemsPerSm items per SM (tc_qc).  Longer items cost fewer item
// hand-offs; too few items leave SMs idle at the end of a launch.
constexpr int kQcChoices[4] = {16, 8, 4, 2};
constexpr int kItemsPerSm = 16;
constexpr int kEpiWarp0 = 2;           // warps 2..17
constexpr int kEpiWarps = 16;          // 8 per fixed tile (LSE) or 4 per tile and buffer (column sums)
// MMA issuers: warp 1 for fixed tile A, warp 18 for tile B, so that one issuer's barrier
// waits and commits overlap the other's MMAs in the tensor pipe
constexpr int kMmaWarpB = kEpiWarp0 + kEpiWarps;
constexpr int kThreads = 32 * (kMmaWarpB + 1);
constexpr int kAccCols = 128;
constexpr int kAccBufs = 2;            // accumulator pairs in TMEM (kAccBufs x 2 x 128 columns)
constexpr int kSched = 4;              // depth of the item-index ring (producer -> consumers)
// Column-sum mode: the lse values of each streamed query tile reach shared memory by
// TMA, in a ring of their own that the epilogue releases (plain loads from the epilogue
// queue behind the tile stream and stall it for several steps).
constexpr int kLseSlots = 8;
constexpr int kLseBox = kTile + 4;     // floats per copy: the tile's 128, from a 16-byte boundary
constexpr int kLseSlotBytes = 640;     // >= kLseBox * 4, multiple of 128

enum Mode { kModeLse = 0, kModeImp = 1 };

template <int D>
struct Cfg {
    static constexpr int kAtoms = D / 64;
    static constexpr int kTileBytes = kTile * 128 * kAtoms;  // 128 rows x D bf16
    static constexpr int kStages = D == 64 ? 6 : 2;
    // dynamic smem layout (offsets from a 1024-aligned base)
    static constexpr int kFixOff = 0;                               // [2 buffers][A, B]
    static constexpr int kRingOff = 4 * kTileBytes;
    static constexpr int kNlOff = kRingOff + kStages * kTileBytes;  // [16 warps][128] f32
    static constexpr int kMergeOff = kNlOff + kEpiWarps * 128 * 4;   // [2][A, B][4][32] float2
    static constexpr int kBarOff = kMergeOff + 2 * 2 * 4 * 32 * 8;
    // fix_full/empty[2], ring_full/empty[kStages], acc_full/empty[A, B][kAccBufs],
    // drain[A, B], sched_full/empty[kSched], xfull/xempty[2][A, B][4], lse_full/empty[kLseSlots]
    static constexpr int kNumBars =
        2 + 2 + 2 * kStages + 4 * kAccBufs + 2 + 2 * kSched + 32 + 2 * kLseSlots;
    // tmem addr, abort flag, then the sched ring's item indices and their prompts (int32)
    static constexpr int kMiscOff = kBarOff + kNumBars * 8;
    static constexpr int kLseOff = (kMiscOff + 16 + 8 * kSched + 127) / 128 * 128;  // lse ring
    static constexpr int kSmemBytes = kLseOff + kLseSlots * kLseSlotBytes + 1024;  // + alignment slack
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
    long long wait_cycles;  // limit of the abortable waits (kWaitCycles unless a test lowers it)
    int c_max;              // column-sum mode: chunk slots of the partial buffer (bounds checks)
    int qc;                 // column-sum mode: pairs of query tiles per item
    int head_pairs;         // LSE mode: an item is one query tile of two heads of a group
    ImpHeads hs;
};

// Instruction descriptor: M = N = 128.
constexpr uint32_t kIdesc = idesc_bf16(kTile, kTile);

// --------------------------------------------------------------- item description
struct TcItem {
    int b, T;
    int64_t t0;
    int fix_y, fix_row0;       // fixed tile A: head (LSE: query head, IMP: KV head), first row
    int fix_y2, dq;            // fixed tile B: head, and its tile offset from A (1 or 0)
    int n_steps;
    // LSE: the query heads of tiles A and B and tile A's query tile (qt0);
    // IMP: group slot, the pair's first key tile (kt), query-tile range, chunk slot
    int h, h2, g, kt, qt0, qt1, chunk;
};

// Item `item`, which belongs to prompt b (looked up once by the producer).
template <int MODE>
__device__ __forceinline__ TcItem make_item(const TcArgs& a, int item, int b) {
    TcItem t;
    if (MODE == kModeLse) {
        t.g = 0; t.kt = 0; t.chunk = 0;
        if (a.head_pairs) {
            // Query tile qt0 of heads head_list[2u] (A) and head_list[2u + 1] (B), two heads of
            // one KV group: both need the key tiles 0 .. qt0, so no step leaves a tile idle.
            const LseItem li = decode_lse_item_at(item, b, a.base, a.cu, kTile, a.hs.n_heads >> 1);
            t.b = li.b; t.T = li.T; t.t0 = li.t0;
            t.h = a.hs.head_list[2 * li.hslot];
            t.h2 = a.hs.head_list[2 * li.hslot + 1];
            t.qt0 = li.qt;
            t.dq = 0;
            t.n_steps = t.qt0 + 1;
        } else {
            const LseItem li = decode_lse_item_at(item, b, a.base, a.cu, kPair, a.hs.n_heads);
            t.b = li.b; t.T = li.T; t.t0 = li.t0;
            t.h = t.h2 = a.hs.head_list[li.hslot];
            const int nt = (t.T + kTile - 1) / kTile;
            // Query tiles qt0 (A) and qt0 + 1 (B).  Pairs end at the prompt's last tile, so
            // with an odd tile count the unpaired tile is tile 0: the pair (-1, 0) streams one
            // key tile, where a lone last tile would stream all of them for nothing.
            t.qt0 = 2 * li.qt - (nt & 1);
            t.dq = 1;
            t.n_steps = t.qt0 + 2;         // key tiles 0 .. the pair's last tile
        }
        t.fix_y = t.h;
        t.fix_y2 = t.h2;
        t.fix_row0 = t.qt0 * kTile;        // -128 for the pair (-1, 0): rows outside the prompt
        t.qt1 = t.qt0 + 1 + t.dq;
    } else {
        const ImpItem ii = decode_imp_item_at(item, b, a.base, a.cu, kPair, a.qc);
        t.b = ii.b; t.T = ii.T; t.t0 = ii.t0;
        const int nt = (t.T + kTile - 1) / kTile;
        t.g = ii.g;
        t.kt = 2 * ii.kt;                  // key tiles kt (A) and kt + 1 (B, may be >= nt)
        t.qt0 = 2 * ii.qt0;
        t.qt1 = min(nt, 2 * ii.qt1);
        t.chunk = (ii.qt0 - ii.kt) / a.qc;
        t.fix_y = t.fix_y2 = a.hs.group[ii.g];
        t.fix_row0 = t.kt * kTile;
        t.dq = 1;
        const int nh = a.hs.begin[ii.g + 1] - a.hs.begin[ii.g];
        t.n_steps = nh * (t.qt1 - t.qt0);
        t.h = t.h2 = 0;
    }
    return t;
}

// Streamed tiles of an item, step by step: TMA head coordinate y, first row, the query
// head of the tile and (column sums) its query tile.  Column-sum steps run over the
// item's query tiles for each selected head of the group in turn; the counters advance
// without divisions or per-step table lookups.
template <int MODE>
struct StepIter {
    int y, row0, head, qt;
    int hi;  // column sums: index of the head within the group

    __device__ __forceinline__ StepIter(const TcArgs& a, const TcItem& t) {
        if (MODE == kModeLse) {
            head = t.h;
            y = t.h / (a.Hq / a.Hkv);
            qt = t.qt0;
            row0 = 0;  // key tile 0
        } else {
            hi = 0;
            head = a.hs.head_list[a.hs.begin[t.g]];
            y = head;
            qt = t.qt0;
            row0 = qt * kTile;
        }
    }
    __device__ __forceinline__ void next(const TcArgs& a, const TcItem& t) {
        if (MODE == kModeLse) {
            row0 += kTile;
        } else if (++qt < t.qt1) {
            row0 += kTile;
        } else {
            qt = t.qt0;
            row0 = qt * kTile;
            ++hi;
            if (hi < a.hs.begin[t.g + 1] - a.hs.begin[t.g]) head = a.hs.head_list[a.hs.begin[t.g] + hi];
            y = head;
        }
    }
};

template <int D, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_fix, const __grid_constant__ CUtensorMap tm_str,
                   const __grid_constant__ CUtensorMap tm_lse, const TcArgs a) {
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
    uint64_t* ring_empty = ring_full + C::kStages;  // [kStages]
    uint64_t* acc_full = ring_empty + C::kStages;
    uint64_t* acc_empty = acc_full + 2 * kAccBufs;   // [A, B][kAccBufs], like acc_full
    uint64_t* drain = acc_empty + 2 * kAccBufs;   // [A, B]
    uint64_t* sched_full = drain + 2;             // [kSched]
    uint64_t* sched_empty = sched_full + kSched;  // [kSched]
    uint64_t* xfull = sched_empty + kSched;       // [2][A, B][4]: partial 1 of the rows written
    uint64_t* xempty = xfull + 16;                // [2][A, B][4]: partial 0's warp has read it
    uint64_t* lse_full = xempty + 16;             // [kLseSlots]
    uint64_t* lse_empty = lse_full + kLseSlots;   // [kLseSlots]
    float* lse_ring = reinterpret_cast<float*>(sm + C::kLseOff);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + C::kMiscOff);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + C::kMiscOff + 4);
    volatile int* sched_item = reinterpret_cast<volatile int*>(sm + C::kMiscOff + 16);
    volatile int* sched_b = sched_item + kSched;  // prompt of each published item

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&fix_full[i], 1);
            mbar_init(&fix_empty[i], 2);  // both issuers
        }
        for (int i = 0; i < 2 * kAccBufs; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], MODE == kModeLse ? kEpiWarps / 2 : kEpiWarps / 4);  // its readers
        }
        for (int i = 0; i < C::kStages; ++i) {
            mbar_init(&ring_full[i], 1);
            mbar_init(&ring_empty[i], 2);  // both issuers
        }
        mbar_init(&drain[0], 1);
        mbar_init(&drain[1], 1);
        for (int i = 0; i < kSched; ++i) {
            mbar_init(&sched_full[i], 1);
            mbar_init(&sched_empty[i], 2 + kEpiWarps);  // MMA issuers + epilogue warps
        }
        for (int i = 0; i < 16; ++i) {
            mbar_init(&xfull[i], 1);
            mbar_init(&xempty[i], 1);
        }
        for (int i = 0; i < kLseSlots; ++i) {
            mbar_init(&lse_full[i], 1);
            mbar_init(&lse_empty[i], kEpiWarps / 2);  // one arrival per warp that reads the step
        }
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 1) {  // TMEM: kAccBufs x (A, B) x 128 columns
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(kAccBufs * 2 * kAccCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    // the column-sum reduce (a programmatic dependent) may launch now; it waits for
    // this grid before reading the partials
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // the plan (and, in column-sum mode, the lse values) are complete past this point
    asm volatile("griddepcontrol.wait;" ::: "memory");
    PlanInfo* info = const_cast<PlanInfo*>(a.info);
    const int total = info->total;

    // Item k of this CTA and its prompt, published by the producer in slot k % kSched
    // (item -1 = no more).
    auto consume_item = [&](int k, bool warp_uniform, int& b) -> int {
        const int slot = k % kSched;
        const uint32_t par = (uint32_t)((k / kSched) & 1);
        bool got;
        if (warp_uniform) got = warp_wait(&sched_full[slot], par, abort_flag, a.status, a.wait_cycles);
        else got = wait_bar(&sched_full[slot], par, abort_flag, a.status, a.wait_cycles);
        if (!got) return -1;
        const int item = sched_item[slot];
        b = sched_b[slot];
        if (warp_uniform) __syncwarp();
        if (!warp_uniform || lane == 0) mbar_arrive(&sched_empty[slot]);
        return item;
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_fix)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_str)) : "memory");
            if (MODE == kModeImp)
                asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_lse)) : "memory");
            uint32_t step = 0;
            // lse copies issued: one per step, issued before the step's ring wait, so an
            // abort at that wait leaves one more lse copy than ring copies in flight
            uint32_t lse_issued = 0;
            int n_items = 0;
            int item = blockIdx.x;
            for (int it = 0;; ++it) {
                if (item >= total) item = -1;
                const int slot = it % kSched;
                if (it >= kSched &&
                    !wait_bar(&sched_empty[slot], (uint32_t)(((it / kSched) - 1) & 1), abort_flag, a.status, a.wait_cycles))
                    break;
                // the item's prompt: one lookup here instead of one in every consumer role
                const int b = item >= 0 ? upper_slot(a.base, a.B, item) : 0;
                sched_item[slot] = item;
                sched_b[slot] = b;
                mbar_arrive(&sched_full[slot]);  // release: item and prompt visible to waiters
                if (item < 0) break;
                const TcItem t = make_item<MODE>(a, item, b);
                const int fb = it & 1;
                if (it >= 2 && !wait_bar(&fix_empty[fb], ((it >> 1) - 1) & 1, abort_flag, a.status, a.wait_cycles)) break;
                mbar_expect_tx(&fix_full[fb], 2 * C::kTileBytes);
#pragma unroll
                for (int tau = 0; tau < 2; ++tau)
#pragma unroll
                    for (int at = 0; at < C::kAtoms; ++at)
                        tma_load_3d(fix + (fb * 2 + tau) * C::kTileBytes + at * kTile * 128, &tm_fix,
                                    at * 64, tau ? t.fix_y2 : t.fix_y,
                                    (int)(t.t0 + t.fix_row0) + tau * t.dq * kTile,
                                    &fix_full[fb]);
                ++n_items;
                bool ok = true;
                StepIter<MODE> si(a, t);
                for (int s = 0; s < t.n_steps; ++s, ++step, si.next(a, t)) {
                    const int stage = (int)(step % C::kStages);
                    const uint32_t u = step / C::kStages;
                    const int y = si.y, row0 = si.row0, head = si.head;
                    if (MODE == kModeImp) {  // the tile's lse values, from a 16-byte boundary
                        const int ls = (int)(step % kLseSlots);
                        const uint32_t lu = step / kLseSlots;
                        if (lu >= 1 && !wait_bar(&lse_empty[ls], (lu - 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                            ok = false;
                            break;
                        }
                        const int64_t x = (int64_t)head * a.sumT + t.t0 + row0;
                        if (!in_bounds(x >= 0 && x < (int64_t)a.Hq * a.sumT, a.status)) {
                            *abort_flag = 1;  // the consumers leave at their next wait
                            ok = false;
                            break;
                        }
                        mbar_expect_tx(&lse_full[ls], kLseBox * 4);
                        tma_load_1d(lse_ring + ls * (kLseSlotBytes / 4), &tm_lse, (int)(x & ~int64_t(3)),
                                    &lse_full[ls]);
                        ++lse_issued;
                    }
                    if (u >= 1 && !wait_bar(&ring_empty[stage], (u - 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(&ring_full[stage], C::kTileBytes);
#pragma unroll
                    for (int at = 0; at < C::kAtoms; ++at)
                        tma_load_3d(ring + stage * C::kTileBytes + at * kTile * 128, &tm_str, at * 64, y,
                                    (int)(t.t0 + row0), &ring_full[stage]);
                    if (!ok) break;
                }
                if (!ok) break;
                item = (int)gridDim.x + atomicAdd(&info->next, 1);
            }
            // Every copy this thread issued has landed before the CTA can exit (on the
            // normal path the consumers already waited for all of them).
            for (uint32_t st = 0; st < (uint32_t)C::kStages && st < step; ++st)
                drain_wait(&ring_full[(step - 1 - st) % C::kStages], ((step - 1 - st) / C::kStages) & 1,
                           a.status);
            if (MODE == kModeImp)
                for (uint32_t k = 0; k < (uint32_t)kLseSlots && k < lse_issued; ++k) {
                    const uint32_t s2 = lse_issued - 1 - k;  // the last copy into each slot
                    drain_wait(&lse_full[s2 % kLseSlots], (s2 / kLseSlots) & 1, a.status);
                }
            for (int fb = 0; fb < 2 && fb < n_items; ++fb)
                drain_wait(&fix_full[fb], (uint32_t)(((n_items - 1 - fb) / 2) & 1), a.status);
        }
    } else if (warp == 1 || warp == kMmaWarpB) {
        // --------------------------------------------- MMA issuers (tile A, tile B)
        const int tau = warp == 1 ? 0 : 1;
        if (lane == 0) {
            uint32_t step = 0;
            bool issued = false;
            for (int it = 0;; ++it) {
                int b = 0;
                const int item = consume_item(it, false, b);
                if (item < 0) break;
                const TcItem t = make_item<MODE>(a, item, b);
                const int fb = it & 1;
                if (!wait_bar(&fix_full[fb], (it >> 1) & 1, abort_flag, a.status, a.wait_cycles)) break;
                const uint32_t fix_addr = smem_u32(fix + (fb * 2 + tau) * C::kTileBytes);
                bool ok = true;
                int q_it = t.qt0;  // column sums: the step's query tile
                for (int s = 0; s < t.n_steps; ++s, ++step) {
                    const int stage = (int)(step % C::kStages);
                    const uint32_t u = step / C::kStages;
                    const int ab = (int)(step % kAccBufs);
                    const uint32_t ua = step / kAccBufs;
                    const uint32_t str_addr = smem_u32(ring + stage * C::kTileBytes);
                    if (!wait_bar(&ring_full[stage], u & 1, abort_flag, a.status, a.wait_cycles)) {
                        ok = false;
                        break;
                    }
                    if (ua >= 1 && !wait_bar(&acc_empty[tau * kAccBufs + ab], (ua - 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    issued = true;
                    // a tile wholly above the diagonal (queries all before keys) is not
                    // computed: the epilogue skips it, and its commit still hands it over
                    const bool skip = MODE == kModeImp ? q_it < t.kt + tau : s > t.qt0 + tau * t.dq;
                    if (!skip) {
#pragma unroll
                        for (int kk = 0; kk < 4 * C::kAtoms; ++kk) {  // K steps of 16
                            const uint32_t off = (uint32_t)((kk >> 2) * kTile * 128 + (kk & 3) * 32);
                            mma_bf16<kIdesc>(tmem + (uint32_t)((ab * 2 + tau) * kAccCols), sw128_desc(fix_addr + off),
                                     sw128_desc(str_addr + off), kk > 0 ? 1u : 0u);
                        }
                    }
                    mma_commit(&acc_full[tau * kAccBufs + ab]);
                    mma_commit(&ring_empty[stage]);
                    if (MODE == kModeImp && ++q_it == t.qt1) q_it = t.qt0;
                }
                if (!ok) break;
                mma_commit(&fix_empty[fb]);
            }
            if (issued) {  // every MMA done before the TMEM is released
                mma_commit(&drain[tau]);
                drain_wait(&drain[tau], 0, a.status);
            }
        }
    } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + kEpiWarps) {
        // ------------------------------------------------------------- epilogue
        const int e = warp - kEpiWarp0;
        // LSE mode: warps 8 tau .. 8 tau + 7 read fixed tile tau at every step, two warps per
        //   quarter, one per column half (sub).
        // Column-sum mode: warps 4 g .. 4 g + 3 read fixed tile g & 1 at the steps of parity
        //   sub = g >> 1 (all 128 columns), so that the groups of the two accumulator buffers
        //   work a step apart and each step's lse values are read by 8 warps.
        constexpr int kChunks = MODE == kModeLse ? 2 : 4;  // 32-column chunks per step
        const int tau = MODE == kModeLse ? e >> 3 : (e >> 2) & 1;  // fixed tile: 0 = A, 1 = B
        const int sub = MODE == kModeLse ? (e >> 2) & 1 : e >> 3;  // which of a row's two partials
        const int col0 = MODE == kModeLse ? sub * 64 : 0;
        const int q = warp & 3;                    // TMEM lane quarter
        const int row = q * 32 + lane;             // accumulator row owned by this thread
        float* nl = nl_all + e * 128;
        uint32_t step = 0;
        bool ok = true;
        for (int it = 0; ok; ++it) {
            int b = 0;
            const int item = consume_item(it, true, b);
            if (item < 0) break;
            const TcItem t = make_item<MODE>(a, item, b);
            // column-sum mode: partial sums of this thread's four key rows 8 s + g8 (s = 0..3)
            // of the quarter, over its columns (16x256b layout, see below)
            float2 acc4[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                              make_float2(0.f, 0.f)};
            float m = -1e30f, ssum = 0.f;          // LSE mode
            StepIter<MODE> si(a, t);
            auto do_step = [&](int s) -> bool {
                const int row0 = si.row0, head = si.head, qt = si.qt;
                if (MODE == kModeImp) {  // -log2e * lse of the step's 128 query columns
                    const int ls = (int)(step % kLseSlots);
                    if (!warp_wait(&lse_full[ls], (step / kLseSlots) & 1, abort_flag, a.status, a.wait_cycles))
                        return false;
                    const int64_t x = (int64_t)head * a.sumT + t.t0 + row0;
                    const float* lr = lse_ring + ls * (kLseSlotBytes / 4) + (int)(x & 3);
                    float r[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int i = row0 + 32 * k + lane;
                        r[k] = i < t.T ? -lr[32 * k + lane] * kLog2e : -INFINITY;
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&lse_empty[ls]);
#pragma unroll
                    for (int k = 0; k < 4; ++k) nl[32 * k + lane] = r[k];
                    __syncwarp();
                }
                const int ab = (int)(step % kAccBufs);
                const int abar = tau * kAccBufs + ab;  // accumulator barrier
                if (!warp_wait(&acc_full[abar], (step / kAccBufs) & 1, abort_flag, a.status, a.wait_cycles))
                    return false;
                tc_fence_after();
                // column-sum mode: this warp's key tile against the streamed query tile
                const int kt = t.kt + tau;
                const bool imp_skip = MODE == kModeImp && qt < kt;   // queries all before keys
                const bool imp_diag = MODE == kModeImp && qt == kt;
                // LSE mode: this warp's query tile against streamed key tile s
                const int my_qt = t.qt0 + tau * t.dq;
                const bool lse_skip = MODE == kModeLse && s > my_qt;  // keys all after queries
                const bool lse_diag = MODE == kModeLse && s == my_qt;
                if (imp_skip || lse_skip) {  // nothing to read: hand the accumulator back
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&acc_empty[abar]);
                    return true;
                }
                const uint32_t taddr =
                    tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)((ab * 2 + tau) * kAccCols + col0);
                const float2 sc = make_float2(a.scale_log2, a.scale_log2);
                if constexpr (MODE == kModeImp) {
                    // 16x256b loads: thread (g8, c4) = (lane / 4, lane % 4) holds key rows
                    // q*32 + 16 lh + 8 jj + g8 and query columns 64 h + 8 k + 2 c4 + {0, 1}.
                    // Each query column's -lse log2e is then needed by 8 lanes only: 8
                    // two-float shared loads per 64 columns, each one wavefront, instead of
                    // every lane reading all 128 values (the shared-memory pipe was the bound).
                    const int g8 = lane >> 2, c4 = lane & 3;
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        float2 n2[8];
#pragma unroll
                        for (int k = 0; k < 8; ++k)
                            n2[k] = *reinterpret_cast<const float2*>(nl + h * 64 + 8 * k + 2 * c4);
#pragma unroll
                        for (int lh = 0; lh < 2; ++lh) {
                            uint32_t raw[32];
                            tmem_ld16x256_x8(taddr + ((uint32_t)(16 * lh) << 16) + (uint32_t)(h * 64), raw);
                            tmem_wait_ld();
                            if (h == 1 && lh == 1) {  // all 128 columns read: release the accumulator
                                tc_fence_before();
                                __syncwarp();
                                if (lane == 0) mbar_arrive(&acc_empty[abar]);
                            }
                            if (!imp_diag) {
#pragma unroll
                                for (int k = 0; k < 8; ++k) {
                                    const float2 x0 = __ffma2_rn(
                                        make_float2(__uint_as_float(raw[4 * k]), __uint_as_float(raw[4 * k + 1])),
                                        sc, n2[k]);
                                    const float2 x1 = __ffma2_rn(
                                        make_float2(__uint_as_float(raw[4 * k + 2]), __uint_as_float(raw[4 * k + 3])),
                                        sc, n2[k]);
                                    acc4[2 * lh] = __fadd2_rn(acc4[2 * lh], make_float2(ex2(x0.x), ex2(x0.y)));
                                    acc4[2 * lh + 1] = __fadd2_rn(acc4[2 * lh + 1], make_float2(ex2(x1.x), ex2(x1.y)));
                                }
                            } else {  // diagonal tile: query i = column, key j = row; keep i >= j
#pragma unroll
                                for (int k = 0; k < 8; ++k) {
#pragma unroll
                                    for (int jj = 0; jj < 2; ++jj) {
                                        const float2 x = __ffma2_rn(
                                            make_float2(__uint_as_float(raw[4 * k + 2 * jj]),
                                                        __uint_as_float(raw[4 * k + 2 * jj + 1])),
                                            sc, n2[k]);
                                        const int i0 = h * 64 + 8 * k + 2 * c4;
                                        const int j = q * 32 + 16 * lh + 8 * jj + g8;
                                        const bool k0 = a.exclude_self ? i0 > j : i0 >= j;
                                        const bool k1 = a.exclude_self ? i0 + 1 > j : i0 + 1 >= j;
                                        acc4[2 * lh + jj] = __fadd2_rn(
                                            acc4[2 * lh + jj], make_float2(k0 ? ex2(x.x) : 0.f, k1 ? ex2(x.y) : 0.f));
                                    }
                                }
                            }
                        }
                    }
                    return true;
                } else {
                // LSE mode: chunks of 32 columns of this thread's query row: load, (release the
                // accumulator after the last), reduce
#pragma unroll
                for (int ch = 0; ch < kChunks; ++ch) {
                    float v[32];
                    tmem_ld32(taddr + ch * 32, v);
                    tmem_wait_ld();
                    if (ch == kChunks - 1) {
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&acc_empty[abar]);
                    }
                    const int cb = col0 + ch * 32;  // tile column of v[0]
                    {
                        if (lse_diag) {  // diagonal tile: keys j = col after the query i = row
#pragma unroll
                            for (int c = 0; c < 32; ++c)
                                if (cb + c > row) v[c] = -INFINITY;
                        }
                        // chunk max: four independent 3-input max chains, then a short tree
                        float mk[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const float* w8 = v + 8 * k;
                            mk[k] = fmaxf(fmax3(fmax3(w8[0], w8[1], w8[2]), w8[3], w8[4]),
                                          fmax3(w8[5], w8[6], w8[7]));
                        }
                        const float mx = fmaxf(fmax3(mk[0], mk[1], mk[2]), mk[3]);
                        const float nm = fmaxf(m, mx * a.scale_log2);
                        ssum *= ex2(m - nm);
                        m = nm;
                        const float2 nm2 = make_float2(-nm, -nm);
                        float2 s2[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                                        make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
                        for (int c = 0; c < 32; c += 2) {
                            float2 x = __ffma2_rn(make_float2(v[c], v[c + 1]), sc, nm2);
                            s2[(c >> 1) & 3] = __fadd2_rn(s2[(c >> 1) & 3], make_float2(ex2(x.x), ex2(x.y)));
                        }
                        const float2 s01 = __fadd2_rn(s2[0], s2[1]), s23 = __fadd2_rn(s2[2], s2[3]);
                        const float2 st = __fadd2_rn(s01, s23);
                        ssum += st.x + st.y;
                    }
                }
                return true;
                }
            };
            for (int s = 0; s < t.n_steps; ++s, ++step, si.next(a, t))
                if ((MODE == kModeLse || (int)(step & 1) == sub) && !(ok = do_step(s))) break;
            if (!ok) break;
            // column-sum mode: the four lanes c4 of a g8 hold columns of the same four rows;
            // a butterfly over them gives each the rows' sums (the same bits in all four,
            // as the additions pair the same operands), and lane (g8, c4) keeps row
            // 8 c4 + g8 of the quarter
            int my_row = lane;  // row of the quarter this thread merges and writes
            float my_sum = 0.f;
            if constexpr (MODE == kModeImp) {
                float rs[4];
#pragma unroll
                for (int r4 = 0; r4 < 4; ++r4) rs[r4] = acc4[r4].x + acc4[r4].y;
#pragma unroll
                for (int r4 = 0; r4 < 4; ++r4) {
                    rs[r4] += __shfl_xor_sync(0xffffffffu, rs[r4], 1);
                    rs[r4] += __shfl_xor_sync(0xffffffffu, rs[r4], 2);
                }
                const int c4 = lane & 3;
                my_row = 8 * c4 + (lane >> 2);
                my_sum = c4 == 0 ? rs[0] : c4 == 1 ? rs[1] : c4 == 2 ? rs[2] : rs[3];
            }
            // merge the two partials of each row (bounded mbarrier hand-off), then write
            const int pb = it & 1;
            const uint32_t use = (uint32_t)(it >> 1);
            float2* mb = merge + (pb * 2 + tau) * 128;
            uint64_t* xf = &xfull[(pb * 2 + tau) * 4 + q];
            uint64_t* xe = &xempty[(pb * 2 + tau) * 4 + q];
            if (sub == 1) {
                if (use >= 1) ok = warp_wait(xe, (use - 1) & 1, abort_flag, a.status, a.wait_cycles);
                if (!ok) break;
                mb[q * 32 + my_row] = MODE == kModeImp ? make_float2(my_sum, 0.f) : make_float2(m, ssum);
                __syncwarp();
                if (lane == 0) mbar_arrive(xf);
            } else {
                ok = warp_wait(xf, use & 1, abort_flag, a.status, a.wait_cycles);
                if (!ok) break;
                const float2 o = mb[q * 32 + my_row];
                __syncwarp();
                if (lane == 0) mbar_arrive(xe);
                if (MODE == kModeImp) {
                    const int j = t.fix_row0 + tau * kTile + q * 32 + my_row;
                    if (j < t.T && in_bounds(t.chunk >= 0 && t.chunk < a.c_max && t.g >= 0 &&
                                                 t.g < a.hs.n_groups && t.t0 + j < a.sumT,
                                             a.status))
                        a.part[((int64_t)t.chunk * a.hs.n_groups + t.g) * a.sumT + t.t0 + j] =
                            my_sum + o.x;
                } else {
                    const float mm = fmaxf(m, o.x);
                    const float ss = ssum * ex2(m - mm) + o.y * ex2(o.x - mm);
                    const int i = t.fix_row0 + tau * t.dq * kTile + row;
                    const int h = tau ? t.h2 : t.h;
                    if (i >= 0 && i < t.T && in_bounds(h >= 0 && h < a.Hq && t.t0 + i < a.sumT, a.status))
                        a.lse_out[(int64_t)h * a.sumT + t.t0 + i] = (mm + lg2(ss)) * kLn2;
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
                     "r"(kAccBufs * 2 * kAccCols));
    }
}

// ------------------------------------------------------------------- host side

// [sumT, heads, d] bf16 viewed as a 3-D tensor (d, heads, sumT); box 64 x 1 x 128.
estp_status make_map(CUtensorMap* m, const void* base, int heads, int d, int64_t sumT) {
    auto fn = tensor_map_encoder();
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

// lse [Hq * sumT] fp32 as a 1-D tensor; box kLseBox (outside the array reads zero).
estp_status make_lse_map(CUtensorMap* m, const float* lse, int64_t n) {
    auto fn = tensor_map_encoder();
    if (!fn) return fail(ESTP_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    cuuint64_t dims[1] = {(cuuint64_t)n};
    cuuint64_t strides[1] = {0};
    cuuint32_t box[1] = {(cuuint32_t)kLseBox};
    cuuint32_t es[1] = {1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 1, const_cast<float*>(lse), dims, strides,
                    box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                    CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(ESTP_ERR_CUDA, "cuTensorMapEncodeTiled (lse) failed (%d)", (int)r);
    return ESTP_OK;
}

template <int D, int MODE>
estp_status launch_tc(estp_ctx* ctx, const CUtensorMap& fixm, const CUtensorMap& strm,
                      const CUtensorMap& lsem, const TcArgs& a, cudaStream_t st) {
    auto kern = attn_tc_kernel<D, MODE>;
    const int smem = Cfg<D>::kSmemBytes;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "tc kernel smem attribute");
    // a programmatic dependent of the plan kernel: the launch and the prologue (barriers,
    // TMEM, tensor-map prefetch) overlap the plan, which the kernel waits for on the device
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)ctx->num_sms);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = (size_t)smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kern, fixm, strm, lsem, a);
    if (e != cudaSuccess) return cuda_fail(e, "tc kernel launch");
    e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "tc kernel launch");
}

}  // namespace

bool tc_supported(estp_dtype dtype, int d) { return dtype == ESTP_BF16 && (d == 64 || d == 128); }
int tc_tile() { return kPair; }
int tc_qc(int B, int64_t sumT, int n_groups, int num_sms) {
    // the prompts' lengths stay on the device: estimate the item count from the mean length
    const int64_t t_mean = B > 0 ? (sumT + B - 1) / B : 0;
    const int64_t nt = (t_mean + kPair - 1) / kPair;
    for (int qc : kQcChoices)
        if ((int64_t)B * n_groups * items_f(nt, qc) >= (int64_t)kItemsPerSm * num_sms) return qc;
    return kQcChoices[3];
}

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
    a.wait_cycles = ctx->wait_cycles;
    a.hs = hs;
    CUtensorMap mq, mk;
    if ((s = make_map(&mq, Q, Hq, d, sumT)) != ESTP_OK) return s;
    if ((s = make_map(&mk, K, Hkv, d, sumT)) != ESTP_OK) return s;
    // LSE items: (prompt, query tile, pair of heads of one KV group) when every group holds
    // an even number of the selected heads, else (prompt, pair of query tiles, head)
    a.head_pairs = 1;
    for (int g = 0; g < hs.n_groups; ++g)
        if ((hs.begin[g + 1] - hs.begin[g]) & 1) a.head_pairs = 0;
    attn_plan_kernel<<<1, 1024, 0, st>>>(cu, B, sumT, max_seqlen, a.head_pairs ? kTile : kPair, 1,
                                         a.head_pairs ? hs.n_heads / 2 : hs.n_heads, 1,
                                         const_cast<int32_t*>(a.base), const_cast<PlanInfo*>(a.info),
                                         ctx->status);
    // (the lse map argument is unused in this mode)
    return d == 64 ? launch_tc<64, kModeLse>(ctx, mq, mk, mq, a, st)
                   : launch_tc<128, kModeLse>(ctx, mq, mk, mq, a, st);
}

estp_status launch_imp_tc(estp_ctx* ctx, const void* Q, const void* K, const float* lse, int Hq,
                          int Hkv, int d, float scale, const ImpHeads& hs, const int32_t* cu,
                          int B, int64_t sumT, bool exclude_self, const int32_t* base,
                          const PlanInfo* info, float* part, int c_max, int qc, cudaStream_t st) {
    TcArgs a{};
    a.c_max = c_max;
    a.qc = qc;
    a.cu = cu; a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.sumT = sumT;
    a.base = base; a.info = info;
    a.scale_log2 = scale * kLog2e;
    a.exclude_self = exclude_self ? 1 : 0;
    a.lse = lse;
    a.part = part;
    a.status = ctx->status;
    a.wait_cycles = ctx->wait_cycles;
    a.hs = hs;
    // the lse coordinate of a TMA copy is a 32-bit element index
    if ((int64_t)Hq * sumT + kLseBox >= ((int64_t)1 << 31))
        return fail(ESTP_ERR_UNSUPPORTED, "Hq * sumT = %lld lse values exceed 2^31 - %d",
                    (long long)Hq * sumT, kLseBox);
    CUtensorMap mq, mk, ml;
    estp_status s;
    if ((s = make_map(&mq, Q, Hq, d, sumT)) != ESTP_OK) return s;
    if ((s = make_map(&mk, K, Hkv, d, sumT)) != ESTP_OK) return s;
    if ((s = make_lse_map(&ml, lse, (int64_t)Hq * sumT)) != ESTP_OK) return s;
    return d == 64 ? launch_tc<64, kModeImp>(ctx, mk, mq, ml, a, st)
                   : launch_tc<128, kModeImp>(ctx, mk, mq, ml, a, st);
}

}  // namespace estp
