// Entropy of the next-token distribution with the logits formed on the tensor cores
// (Eq. 2-1 of z = h W^T, where W is the model's output projection): the [rows, V] logits
// are never written to memory.
//
// lm_head_kernel: one persistent CTA per SM.  A work item is (row block rb of 128 tokens,
// vocabulary split sp); items run split-fastest, so the CTAs working at one time share a
// few row blocks (kept in L2) and stream W.  For every 256-entry vocabulary tile of its
// split the CTA forms the 128 x 256 logit tile in TMEM,
//   D = sum over 64-wide chunks c of the hidden size of A_c B_c^T,
// with A_c = hidden[rows of rb, c] and B_c = W[entries of the tile, c] staged by TMA in a
// 4-stage ring (128B-swizzled, 48 KB per stage), 4 tcgen05.mma (M = 128, N = 256, K = 16)
// per stage, and two accumulators of 256 fp32 columns (all 512 TMEM columns), so that the
// epilogue of one tile overlaps the MMAs of the next.
//   warp 0      TMA producer
//   warp 1      MMA issuer (one thread)
//   warps 2-5   epilogue: warp w reads TMEM lanes 32 (w % 4) .. (one token each) in
//               32-column chunks and folds them into the token's running
//               m = max y, s = sum 2^(y - m), t = sum 2^(y - m) (y - m), y = z log2(e)
// At the end of an item each token's (m, s, t) for the split goes to a partial buffer;
// lm_head_merge_kernel combines the splits in split order,
//   M = max m_k, S = sum 2^(m_k - M) s_k, T = sum 2^(m_k - M) (t_k + s_k (m_k - M)),
// and writes H = ln 2 (log2 S - T / S) (nats).
//
// Every mbarrier wait is bounded (a test may lower the limit of the abortable waits
// through estp_set_wait_limit); on expiry the CTA records ESTP_ERR_TIMEOUT in the status
// word, drains its own copies and MMAs and frees its TMEM.
#include "tcgen05.cuh"

namespace estp {
namespace {

constexpr int kM = 128;                       // tokens per tile (TMEM lanes)
constexpr int kN = 256;                       // vocabulary entries per tile (MMA N)
constexpr int kKc = 64;                       // hidden-size chunk per stage (one swizzle atom)
constexpr int kStages = 4;
constexpr int kABytes = kM * kKc * 2;         // 16 KB
constexpr int kBBytes = kN * kKc * 2;         // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kAccBufs = 2;                   // 2 x 256 TMEM columns
constexpr int kEpiWarp0 = 2;
constexpr int kEpiWarps = 4;
constexpr int kThreads = 32 * (kEpiWarp0 + kEpiWarps);
// dynamic shared memory (offsets from a 1024-aligned base)
constexpr int kBarOff = kStages * kStageBytes;
constexpr int kNumBars = 2 * kStages + 2 * kAccBufs + 1;  // full, empty, acc_full, acc_empty, drain
constexpr int kMiscOff = kBarOff + kNumBars * 8;           // tmem address, abort flag
constexpr int kSmemBytes = kMiscOff + 16 + 1024;           // + alignment slack
static_assert(kSmemBytes <= 227 * 1024, "shared memory per CTA");

// Instruction descriptor: M = 128, N = 256.
constexpr uint32_t kIdesc = idesc_bf16(kM, kN);

struct LmArgs {
    int64_t n_rows;
    int64_t V;
    int nk;            // hidden-size chunks (D / 64)
    int n_vt;          // vocabulary tiles
    int S;             // vocabulary splits
    int64_t n_items;   // row blocks x splits
    float* part;       // [3][S][n_rows]: m, s, t (log2 units)
    int* status;
    long long wait_cycles;  // limit of the abortable waits (kWaitCycles unless a test lowers it)
};

// Vocabulary tiles [vt0, vt1) of split sp.
__device__ __forceinline__ void split_range(const LmArgs& a, int sp, int& vt0, int& vt1) {
    vt0 = (int)((int64_t)sp * a.n_vt / a.S);
    vt1 = (int)((int64_t)(sp + 1) * a.n_vt / a.S);
}

// Fold 32 logits z (one chunk of this token's row) into (m, s, t), log2 units.  Columns
// at or past `valid` are outside the vocabulary.
__device__ __forceinline__ void fold_chunk(float* v, int valid, float& m, float& s, float& t) {
    if (valid < 32) {
#pragma unroll
        for (int c = 0; c < 32; ++c)
            if (c >= valid) v[c] = -1e30f;  // 2^(y - m) = 0 and 0 * (y - m) = 0 (finite)
    }
    float mk[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float* w8 = v + 8 * k;
        mk[k] = fmaxf(fmax3(fmax3(w8[0], w8[1], w8[2]), w8[3], w8[4]), fmax3(w8[5], w8[6], w8[7]));
    }
    const float my = fmaxf(fmax3(mk[0], mk[1], mk[2]), mk[3]) * kLog2e;
    if (my > m) {  // rescale (s, t) to the new max: t' = f (t + s (m - m')), s' = f s
        if (m == -INFINITY) {
            s = 0.f;
            t = 0.f;
        } else {
            const float dm = m - my, f = ex2(dm);
            t = f * fmaf(s, dm, t);
            s *= f;
        }
        m = my;
    }
    const float2 l2 = make_float2(kLog2e, kLog2e), nm = make_float2(-m, -m);
    float2 s2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
    float2 t2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
    for (int c = 0; c < 32; c += 2) {
        const float2 d = __ffma2_rn(make_float2(v[c], v[c + 1]), l2, nm);  // y - m
        const float2 e = make_float2(ex2(d.x), ex2(d.y));
        const int j = (c >> 1) & 1;
        s2[j] = __fadd2_rn(s2[j], e);
        t2[j] = __ffma2_rn(e, d, t2[j]);
    }
    const float2 ss = __fadd2_rn(s2[0], s2[1]), tt = __fadd2_rn(t2[0], t2[1]);
    s += ss.x + ss.y;
    t += tt.x + tt.y;
}

__global__ void __launch_bounds__(kThreads, 1)
    lm_head_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                   const LmArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + kBarOff);
    uint64_t* full = bars;                       // [kStages]
    uint64_t* empty = full + kStages;            // [kStages]
    uint64_t* acc_full = empty + kStages;        // [kAccBufs]
    uint64_t* acc_empty = acc_full + kAccBufs;   // [kAccBufs]
    uint64_t* drain = acc_empty + kAccBufs;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + kMiscOff);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(sm + kMiscOff + 4);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < kAccBufs; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], kEpiWarps);  // one arrival per epilogue warp
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 1) {  // TMEM: kAccBufs x 256 columns
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(kAccBufs * kN));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_a)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_b)) : "memory");
            uint32_t step = 0;
            bool ok = true;
            for (int64_t item = blockIdx.x; ok && item < a.n_items; item += gridDim.x) {
                const int sp = (int)(item % a.S), rb = (int)(item / a.S);
                int vt0, vt1;
                split_range(a, sp, vt0, vt1);
                for (int vt = vt0; ok && vt < vt1; ++vt) {
                    for (int kc = 0; kc < a.nk; ++kc, ++step) {
                        const int stage = (int)(step % kStages);
                        const uint32_t u = step / kStages;
                        if (u >= 1 && !wait_bar(&empty[stage], (u - 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                            ok = false;
                            break;
                        }
                        uint8_t* st = sm + stage * kStageBytes;
                        mbar_expect_tx(&full[stage], kStageBytes);
                        tma_load_2d(st, &tm_a, kc * kKc, rb * kM, &full[stage]);
                        tma_load_2d(st + kABytes, &tm_b, kc * kKc, vt * kN, &full[stage]);
                    }
                }
            }
            // every copy this thread issued has landed before the CTA can exit
            for (uint32_t i = 0; i < (uint32_t)kStages && i < step; ++i)
                drain_wait(&full[(step - 1 - i) % kStages], ((step - 1 - i) / kStages) & 1, a.status);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0) {
            uint32_t step = 0, tile = 0;
            bool ok = true, issued = false;
            for (int64_t item = blockIdx.x; ok && item < a.n_items; item += gridDim.x) {
                const int sp = (int)(item % a.S);
                int vt0, vt1;
                split_range(a, sp, vt0, vt1);
                for (int vt = vt0; ok && vt < vt1; ++vt, ++tile) {
                    const int ab = (int)(tile % kAccBufs);
                    const uint32_t ua = tile / kAccBufs;
                    if (ua >= 1 && !wait_bar(&acc_empty[ab], (ua - 1) & 1, abort_flag, a.status, a.wait_cycles)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t d = tmem + (uint32_t)(ab * kN);
                    for (int kc = 0; kc < a.nk; ++kc, ++step) {
                        const int stage = (int)(step % kStages);
                        if (!wait_bar(&full[stage], (step / kStages) & 1, abort_flag, a.status, a.wait_cycles)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        issued = true;
                        const uint32_t sa = smem_u32(sm + stage * kStageBytes);
#pragma unroll
                        for (int kk = 0; kk < kKc / 16; ++kk)
                            mma_bf16<kIdesc>(d, sw128_desc(sa + kk * 32), sw128_desc(sa + kABytes + kk * 32),
                                     (kc > 0 || kk > 0) ? 1u : 0u);
                        mma_commit(&empty[stage]);
                    }
                    if (ok) mma_commit(&acc_full[ab]);
                }
            }
            if (issued) {  // every MMA done before the TMEM is released
                mma_commit(drain);
                drain_wait(drain, 0, a.status);
            }
        }
    } else {
        // ------------------------------------------------------------- epilogue
        const int q = warp & 3;               // TMEM lane quarter
        const int row_l = q * 32 + lane;      // token of the tile owned by this thread
        uint32_t tile = 0;
        bool ok = true;
        for (int64_t item = blockIdx.x; ok && item < a.n_items; item += gridDim.x) {
            const int sp = (int)(item % a.S), rb = (int)(item / a.S);
            int vt0, vt1;
            split_range(a, sp, vt0, vt1);
            float m = -INFINITY, s = 0.f, t = 0.f;
            for (int vt = vt0; vt < vt1; ++vt, ++tile) {
                const int ab = (int)(tile % kAccBufs);
                if (!warp_wait(&acc_full[ab], (tile / kAccBufs) & 1, abort_flag, a.status, a.wait_cycles)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t taddr = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(ab * kN);
                const int64_t v0 = (int64_t)vt * kN;
#pragma unroll 1
                for (int ch = 0; ch < kN / 32; ++ch) {
                    float v[32];
                    tmem_ld32(taddr + ch * 32, v);
                    tmem_wait_ld();
                    if (ch == kN / 32 - 1) {  // the whole tile is in registers: release it
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&acc_empty[ab]);
                    }
                    const int64_t left = a.V - (v0 + ch * 32);
                    if (left <= 0) continue;
                    fold_chunk(v, left < 32 ? (int)left : 32, m, s, t);
                }
            }
            if (!ok) break;
            const int64_t row = (int64_t)rb * kM + row_l;
            if (row < a.n_rows) {
                const int64_t plane = (int64_t)a.S * a.n_rows;
                float* p = a.part + (int64_t)sp * a.n_rows + row;
                p[0] = m;
                p[plane] = s;
                p[2 * plane] = t;
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        __syncwarp();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(kAccBufs * kN));
    }
}

// Per token: the splits' (m, s, t) combined in split order, H in nats.
__global__ void lm_head_merge_kernel(const float* __restrict__ part, int64_t n_rows, int S,
                                     float* __restrict__ H) {
    const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= n_rows) return;
    const int64_t plane = (int64_t)S * n_rows;
    float M = -INFINITY;
    for (int k = 0; k < S; ++k) M = fmaxf(M, part[(int64_t)k * n_rows + r]);
    float Sx = 0.f, Tx = 0.f;
    for (int k = 0; k < S; ++k) {
        const float mk = part[(int64_t)k * n_rows + r];
        const float sk = part[plane + (int64_t)k * n_rows + r];
        const float tk = part[2 * plane + (int64_t)k * n_rows + r];
        if (mk == -INFINITY) continue;  // a split without vocabulary entries
        const float dm = mk - M, f = ex2(dm);
        Sx = fmaf(f, sk, Sx);
        Tx = fmaf(f, fmaf(sk, dm, tk), Tx);
    }
    H[r] = kLn2 * (lg2(Sx) - Tx / Sx);
}


// [rows, ld] bf16 row-major viewed as a 2-D tensor (D, rows); box 64 x box_rows, 128B
// swizzle; rows past the end read as zero.
estp_status make_map_2d(CUtensorMap* m, const void* base, int64_t D, int64_t rows, int64_t ld,
                        int box_rows) {
    auto fn = tensor_map_encoder();
    if (!fn) return fail(ESTP_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)kKc, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                    box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(ESTP_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    return ESTP_OK;
}

}  // namespace

estp_status launch_lm_head_entropy(estp_ctx* ctx, const void* hidden, int64_t ldh, const void* W,
                                   int64_t ldw, int64_t n_rows, int64_t D, int64_t V, float* H,
                                   cudaStream_t st) {
    CUtensorMap tma, tmb;
    estp_status s = make_map_2d(&tma, hidden, D, n_rows, ldh, kM);
    if (s != ESTP_OK) return s;
    s = make_map_2d(&tmb, W, D, V, ldw, kN);
    if (s != ESTP_OK) return s;
    LmArgs a{};
    a.n_rows = n_rows;
    a.V = V;
    a.nk = (int)(D / kKc);
    a.n_vt = (int)((V + kN - 1) / kN);
    const int64_t n_rb = (n_rows + kM - 1) / kM;
    // splits: at least four items per SM; the fewest splits whose items fill the last
    // wave of the persistent grid to 97 % (else the best fill up to four times as many).
    // Fewer splits keep more row blocks in flight at once, so that each W tile read from
    // DRAM serves more of them.
    // At least as many splits that the row blocks in flight at once (G / S of them, 256 D
    // bytes each) fit in ~48 MB of L2 beside the W tiles streaming through.
    const int64_t G = ctx->num_sms;
    const int64_t l2_budget = 48ll << 20, rb_bytes = (int64_t)kM * D * 2;
    const int64_t s_l2 = (G * rb_bytes + l2_budget - 1) / l2_budget;
    int64_t s_lo = (4 * G + n_rb - 1) / n_rb;
    if (s_lo < s_l2) s_lo = s_l2;
    int64_t S = s_lo < a.n_vt ? s_lo : a.n_vt;  // small problems: one tile per split
    double best = -1.0;
    for (int64_t c = s_lo; c <= a.n_vt && c <= 4 * s_lo; ++c) {
        const int64_t items = n_rb * c, waves = (items + G - 1) / G;
        const double fill = (double)items / (double)(waves * G);
        if (fill > best + 1e-9) {
            best = fill;
            S = c;
        }
        if (fill >= 0.97) break;
    }
    a.S = (int)S;
    a.n_items = n_rb * S;
    s = ws_reserve(ctx, sizeof(float) * 3 * (size_t)S * (size_t)n_rows);
    if (s != ESTP_OK) return s;
    a.part = static_cast<float*>(ctx->ws);
    a.status = ctx->status;
    a.wait_cycles = ctx->wait_cycles;
    cudaError_t e = cudaFuncSetAttribute(lm_head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemBytes);
    if (e != cudaSuccess) return cuda_fail(e, "lm-head kernel smem attribute");
    const int64_t grid = a.n_items < ctx->num_sms ? a.n_items : ctx->num_sms;
    lm_head_kernel<<<(unsigned)grid, kThreads, kSmemBytes, st>>>(tma, tmb, a);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "lm-head kernel launch");
    lm_head_merge_kernel<<<(unsigned)((n_rows + 255) / 256), 256, 0, st>>>(a.part, n_rows, a.S, H);
    e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "lm-head merge launch");
}

}  // namespace estp
