// Attention importance (Eq. 2-0, Sec. 3.1): row log-normalisers, causal column sums
// of the softmax attention, the deterministic partial reduce and the final scaling.
//
// This file holds the device plan, the CUDA-core kernels (fp32 inputs, and any
// shape the tensor-core path does not take) and the launchers that pick a path.
//
// Column sums are formed in the transposed orientation: a CTA owns a tile of KEYS
// and streams the query tiles that may attend to it, so the sum over queries of
// A_ij = 2^(s_ij log2e - lse_i log2e) stays in the thread that owns key j.  Each
// item writes its keys' partial sums to its own slot of a partial buffer; the reduce
// kernel adds the slots of every key in a fixed order (no float atomics).
#include "importance_plan.cuh"
#include "importance_tc.cuh"

namespace estp {

// One plan, computed by all 1024 threads of the calling block.
static __device__ void plan_body(const int32_t* cu, int B, int64_t sumT, int max_seqlen, int tile,
                                 int qc, int mult, int kind, int32_t* base, PlanInfo* info,
                                 int* status) {
    // thread t owns prompts [t*per, (t+1)*per); one read of cu, warp-shuffle scans
    __shared__ int64_t warp_sum[32];
    __shared__ int bad;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    if (tid == 0) bad = 0;
    __syncthreads();
    if (tid == 0 && (cu[0] != 0 || (int64_t)cu[B] != sumT)) bad = 1;
    const int per = (B + 1023) / 1024;
    const int b0 = min(B, tid * per), b1 = min(B, b0 + per);
    int64_t local = 0;
    for (int b = b0; b < b1; ++b) {
        const int32_t len = cu[b + 1] - cu[b];
        if (len < 0 || len > max_seqlen) { bad = 1; continue; }
        const int nt = (len + tile - 1) / tile;
        local += (int64_t)mult * plan_count(nt, qc, kind);
    }
    int64_t inc = local;  // inclusive scan within the warp
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int64_t v = __shfl_up_sync(0xffffffffu, inc, off);
        if (lane >= off) inc += v;
    }
    if (lane == 31) warp_sum[wid] = inc;
    __syncthreads();
    if (wid == 0) {
        int64_t w = warp_sum[lane];
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int64_t v = __shfl_up_sync(0xffffffffu, w, off);
            if (lane >= off) w += v;
        }
        warp_sum[lane] = w;  // inclusive over warps
    }
    __syncthreads();
    const int64_t total = warp_sum[31];
    const bool ok = !bad && total < INT32_MAX / 2;  // item indices stay 32-bit
    int64_t run = inc - local + (wid > 0 ? warp_sum[wid - 1] : 0);
    for (int b = b0; b < b1; ++b) {
        base[b] = ok ? (int32_t)run : 0;
        const int32_t len = cu[b + 1] - cu[b];
        const int nt = (len + tile - 1) / tile;
        if (len >= 0) run += (int64_t)mult * plan_count(nt, qc, kind);
    }
    if (tid == 1023) {
        base[B] = ok ? (int32_t)total : 0;
        info->ok = ok ? 1 : 0;
        info->total = ok ? (int32_t)total : 0;
        info->next = 0;
    }
    if (tid == 0 && !ok) report(status, ESTP_ERR_INVALID_ARG);
}

__global__ void __launch_bounds__(1024) attn_plan_kernel(const int32_t* cu, int B, int64_t sumT,
                                                         int max_seqlen, int tile, int qc,
                                                         int mult, int kind, int32_t* base,
                                                         PlanInfo* info, int* status) {
    // the tensor-core kernel that consumes the plan may launch now and run its prologue;
    // it waits for this grid before its first read of the plan
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    plan_body(cu, B, sumT, max_seqlen, tile, qc, mult, kind, base, info, status);
}

__global__ void __launch_bounds__(1024) attn_plan2_kernel(const int32_t* cu, int B, int64_t sumT,
                                                          int max_seqlen, int tile, int qc,
                                                          int mult, int kind0, int32_t* base0,
                                                          PlanInfo* info0, int kind1,
                                                          int32_t* base1, PlanInfo* info1,
                                                          int* status) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (blockIdx.x == 0) plan_body(cu, B, sumT, max_seqlen, tile, qc, mult, kind0, base0, info0, status);
    else plan_body(cu, B, sumT, max_seqlen, tile, qc, mult, kind1, base1, info1, status);
}

namespace {

// ----------------------------------------------------------- CUDA-core kernels
constexpr int kSTile = 64;      // rows per tile (keys or queries)
constexpr int kSQc = 8;         // query tiles per importance item
constexpr int kSThreads = 256;  // 16 x 16 threads, 4 x 4 scores each

struct SimtArgs {
    const void* Q;
    const void* K;
    const float* lse;          // [Hq, sumT] natural log
    const int32_t* cu;
    const int32_t* base;
    const PlanInfo* info;
    int B, Hq, Hkv, d;
    int64_t sumT;
    float scale_log2;          // softmax_scale * log2(e)
    ImpHeads hs;
    int exclude_self;
    float* part;               // [c_max][n_groups][sumT]
    float* lse_out;            // LSE kernel output [Hq, sumT]
    int c_max;                 // chunk slots of part (bounds checks of debug builds)
    int* status;
};

// Rows [row0, row0 + n) of a [rows, heads, d] tensor, head h, into smem as fp32
// row-major with stride d + 4; rows past n are zero.
template <bool kBf16>
__device__ __forceinline__ void load_tile(float* sm, const void* src, int64_t row0, int n,
                                          int heads, int h, int d) {
    const int stride = d + 4;
    const int vec = kBf16 ? 8 : 4;
    const int per_row = d / vec;
    for (int idx = threadIdx.x; idx < kSTile * per_row; idx += kSThreads) {
        const int r = idx / per_row, x = (idx - r * per_row) * vec;
        float4 lo = make_float4(0.f, 0.f, 0.f, 0.f), hi = lo;
        if (r < n) {
            const int64_t off = ((row0 + r) * heads + h) * (int64_t)d + x;
            if (kBf16) {
                uint4 v = *reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(src) + off);
                lo = make_float4(bf16lo(v.x), bf16hi(v.x), bf16lo(v.y), bf16hi(v.y));
                hi = make_float4(bf16lo(v.z), bf16hi(v.z), bf16lo(v.w), bf16hi(v.w));
            } else {
                lo = *reinterpret_cast<const float4*>(static_cast<const float*>(src) + off);
            }
        }
        *reinterpret_cast<float4*>(sm + r * stride + x) = lo;
        if (kBf16) *reinterpret_cast<float4*>(sm + r * stride + x + 4) = hi;
    }
}

// acc[a][b] = A-row (ty*4+a) . B-row (tx*4+b)
__device__ __forceinline__ void tile_dot(const float* As, const float* Bs, int d, int ty, int tx,
                                         float acc[4][4]) {
    const int stride = d + 4;
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
    for (int x = 0; x < d; x += 4) {
        float4 av[4], bv[4];
#pragma unroll
        for (int a = 0; a < 4; ++a) av[a] = *reinterpret_cast<const float4*>(As + (ty * 4 + a) * stride + x);
#pragma unroll
        for (int b = 0; b < 4; ++b) bv[b] = *reinterpret_cast<const float4*>(Bs + (tx * 4 + b) * stride + x);
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                acc[a][b] = fmaf(av[a].x, bv[b].x, acc[a][b]);
                acc[a][b] = fmaf(av[a].y, bv[b].y, acc[a][b]);
                acc[a][b] = fmaf(av[a].z, bv[b].z, acc[a][b]);
                acc[a][b] = fmaf(av[a].w, bv[b].w, acc[a][b]);
            }
    }
}

// Row log-normalisers: rows = queries of one tile, streamed over key tiles 0..qt.
template <bool kBf16>
__global__ void __launch_bounds__(kSThreads) lse_simt_kernel(SimtArgs a) {
    extern __shared__ float smem[];
    float* Qs = smem;
    float* Ks = smem + kSTile * (a.d + 4);
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int total = a.info->total;
    const int rep = a.Hq / a.Hkv;
    for (int item = blockIdx.x; item < total; item += gridDim.x) {
        const LseItem it = decode_lse_item(item, a.base, a.B, a.cu, kSTile, a.hs.n_heads);
        const int h = a.hs.head_list[it.hslot];
        const int q0 = it.qt * kSTile;
        __syncthreads();
        load_tile<kBf16>(Qs, a.Q, it.t0 + q0, min(kSTile, it.T - q0), a.Hq, h, a.d);
        float m[4], s[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) { m[r] = -1e30f; s[r] = 0.f; }
        for (int kt = 0; kt <= it.qt; ++kt) {
            const int k0 = kt * kSTile;
            __syncthreads();
            load_tile<kBf16>(Ks, a.K, it.t0 + k0, min(kSTile, it.T - k0), a.Hkv, h / rep, a.d);
            __syncthreads();
            float acc[4][4];
            tile_dot(Qs, Ks, a.d, ty, tx, acc);
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int i = q0 + ty * 4 + r;
                float v[4];
                float mx = -1e30f;
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const int j = k0 + tx * 4 + c;
                    const bool ok = j <= i && j < it.T;
                    v[c] = ok ? acc[r][c] * a.scale_log2 : -1e30f;
                    mx = fmaxf(mx, v[c]);
                }
                const float nm = fmaxf(m[r], mx);
                s[r] *= ex2(m[r] - nm);
                m[r] = nm;
#pragma unroll
                for (int c = 0; c < 4; ++c) s[r] += ex2(v[c] - nm);
            }
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) {
#pragma unroll
            for (int off = 8; off > 0; off >>= 1) {
                const float m2 = __shfl_xor_sync(0xffffffffu, m[r], off);
                const float s2 = __shfl_xor_sync(0xffffffffu, s[r], off);
                const float nm = fmaxf(m[r], m2);
                s[r] = s[r] * ex2(m[r] - nm) + s2 * ex2(m2 - nm);
                m[r] = nm;
            }
            const int i = q0 + ty * 4 + r;
            if (tx == 0 && i < it.T) a.lse_out[(int64_t)h * a.sumT + it.t0 + i] = (m[r] + lg2(s[r])) * kLn2;
        }
    }
}

// Column sums: rows = keys of one tile, streamed over the item's query tiles and
// the selected heads of one KV group.
template <bool kBf16>
__global__ void __launch_bounds__(kSThreads) imp_simt_kernel(SimtArgs a) {
    extern __shared__ float smem[];
    float* Ks = smem;
    float* Qs = smem + kSTile * (a.d + 4);
    float* lse_s = Qs + kSTile * (a.d + 4);
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int total = a.info->total;
    for (int item = blockIdx.x; item < total; item += gridDim.x) {
        const ImpItem it = decode_imp_item(item, a.base, a.B, a.cu, kSTile, kSQc);
        const int grp = a.hs.group[it.g];
        const int k0 = it.kt * kSTile;
        __syncthreads();
        load_tile<kBf16>(Ks, a.K, it.t0 + k0, min(kSTile, it.T - k0), a.Hkv, grp, a.d);
        float col[4] = {0.f, 0.f, 0.f, 0.f};
        for (int hi = a.hs.begin[it.g]; hi < a.hs.begin[it.g + 1]; ++hi) {
            const int h = a.hs.head_list[hi];
            for (int qt = it.qt0; qt < it.qt1; ++qt) {
                const int q0 = qt * kSTile;
                __syncthreads();
                load_tile<kBf16>(Qs, a.Q, it.t0 + q0, min(kSTile, it.T - q0), a.Hq, h, a.d);
                if (threadIdx.x < kSTile) {
                    const int i = q0 + threadIdx.x;
                    lse_s[threadIdx.x] = i < it.T ? a.lse[(int64_t)h * a.sumT + it.t0 + i] * kLog2e : INFINITY;
                }
                __syncthreads();
                float acc[4][4];
                tile_dot(Ks, Qs, a.d, ty, tx, acc);
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    const int j = k0 + ty * 4 + r;
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const int i = q0 + tx * 4 + c;
                        const bool ok = i >= j && i < it.T && !(a.exclude_self && i == j);
                        col[r] += ok ? ex2(acc[r][c] * a.scale_log2 - lse_s[tx * 4 + c]) : 0.f;
                    }
                }
            }
        }
        const int c_slot = (it.qt0 - it.kt) / kSQc;
        if (!in_bounds(c_slot >= 0 && c_slot < a.c_max, a.status)) continue;
        float* out = a.part + ((int64_t)c_slot * a.hs.n_groups + it.g) * a.sumT + it.t0;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
#pragma unroll
            for (int off = 8; off > 0; off >>= 1) col[r] += __shfl_xor_sync(0xffffffffu, col[r], off);
            const int j = k0 + ty * 4 + r;
            if (tx == 0 && j < it.T) out[j] = col[r];
        }
    }
}

// acc[j] (+)= sum over chunk slots c (in order) and group slots g (in order) of part.
// Largest b with cu[b] <= j: cu staged in shared memory when it fits (kCuStage entries).
constexpr int kCuStage = 2048;

__device__ __forceinline__ const int32_t* stage_cu(const int32_t* cu, int B, int32_t* cu_s) {
    if (B + 1 > kCuStage) return cu;
    for (int i = threadIdx.x; i <= B; i += blockDim.x) cu_s[i] = cu[i];
    __syncthreads();
    return cu_s;
}

__global__ void imp_reduce_kernel(const float* part, const PlanInfo* info, const int32_t* cu,
                                  int B, int64_t sumT, int n_groups, int tile, int qc,
                                  int accumulate, float* acc, int c_max, int* status) {
    __shared__ int32_t cu_s[kCuStage];
    const int32_t* cuv = stage_cu(cu, B, cu_s);
    // the partials are complete past this point (launched as a programmatic dependent
    // of the column-sum kernel; a no-op after an ordinary launch)
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= sumT) return;
    float v = 0.f;
    if (info->ok) {
        const int b = upper_slot(cuv, B, j);
        const int T = cuv[b + 1] - cuv[b];
        const int nt = (T + tile - 1) / tile;
        const int kt = (int)((j - cuv[b]) / tile);
        int n = chunks_of(nt, kt, qc) * n_groups;  // partials (c, g), c-major
        if (!in_bounds(n <= c_max * n_groups && b >= 0 && b < B, status)) n = 0;
        // up to 16 partials are loaded before any is added (independent loads in flight),
        // then added in the same (c, g) order
        constexpr int kBatch = 16;
        for (int i0 = 0; i0 < n; i0 += kBatch) {
            float p[kBatch];
#pragma unroll
            for (int i = 0; i < kBatch; ++i) p[i] = i0 + i < n ? part[(int64_t)(i0 + i) * sumT + j] : 0.f;
#pragma unroll
            for (int i = 0; i < kBatch; ++i)
                if (i0 + i < n) v += p[i];
        }
    }
    acc[j] = accumulate ? acc[j] + v : v;
}

// S_j = C_j / (n_j * layers * heads): n_j = N_b (Eq. 2-0), the causal count of the
// queries whose terms enter C_j (div 1: N_b - j, one fewer without the diagonal;
// S_j = 0 where it is 0), or 1 (div 2).
__global__ void imp_finalize_kernel(const float* acc, const int32_t* cu, int B, int64_t sumT,
                                    float inv_lh, int div, int exclude_self, float* out) {
    __shared__ int32_t cu_s[kCuStage];
    const int32_t* cuv = stage_cu(cu, B, cu_s);
    const int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= sumT) return;
    const int b = upper_slot(cuv, B, j);
    if (!in_bounds(b >= 0 && b < B, nullptr)) return;
    int64_t n = cuv[b + 1] - cuv[b];
    if (div == 1) n = (int64_t)cuv[b + 1] - j - (exclude_self ? 1 : 0);
    else if (div == 2) n = 1;
    out[j] = n > 0 ? acc[j] * inv_lh / (float)n : 0.f;
}

size_t simt_smem(int d, bool with_lse) {
    return sizeof(float) * (2 * kSTile * (d + 4) + (with_lse ? kSTile : 0));
}

}  // namespace

// Launch geometry shared by both paths.
static int persistent_grid(estp_ctx* ctx, const void* kernel, int threads, size_t smem) {
    int occ = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kernel, threads, smem);
    return ctx->num_sms * (occ > 0 ? occ : 1);
}

estp_status launch_lse(estp_ctx* ctx, const void* Q, const void* K, estp_dtype dtype, int Hq,
                       int Hkv, int d, float scale, const ImpHeads& hs, const int32_t* cu,
                       int B, int64_t sumT, int max_seqlen, float* lse, cudaStream_t st) {
    if (tc_supported(dtype, d))
        return launch_lse_tc(ctx, Q, K, Hq, Hkv, d, scale, hs, cu, B, sumT, max_seqlen, lse, st);
    const size_t off_info = align_up(sizeof(int32_t) * (size_t)(B + 1), 256);
    estp_status s = ws_reserve(ctx, off_info + sizeof(PlanInfo));
    if (s != ESTP_OK) return s;
    char* ws = static_cast<char*>(ctx->ws);
    SimtArgs a{};
    a.Q = Q; a.K = K; a.cu = cu; a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.d = d; a.sumT = sumT;
    a.base = reinterpret_cast<int32_t*>(ws);
    a.info = reinterpret_cast<PlanInfo*>(ws + off_info);
    a.scale_log2 = scale * kLog2e;
    a.hs = hs;
    a.lse_out = lse;
    attn_plan_kernel<<<1, 1024, 0, st>>>(cu, B, sumT, max_seqlen, kSTile, 1, hs.n_heads, 1,
                                         reinterpret_cast<int32_t*>(ws),
                                         reinterpret_cast<PlanInfo*>(ws + off_info), ctx->status);
    const size_t smem = simt_smem(d, false);
    const void* kfn = dtype == ESTP_BF16 ? (const void*)lse_simt_kernel<true> : (const void*)lse_simt_kernel<false>;
    cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    const int grid = persistent_grid(ctx, kfn, kSThreads, smem);
    if (dtype == ESTP_BF16) lse_simt_kernel<true><<<grid, kSThreads, smem, st>>>(a);
    else lse_simt_kernel<false><<<grid, kSThreads, smem, st>>>(a);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "lse launch");
}

estp_status launch_importance(estp_ctx* ctx, const void* Q, const void* K, estp_dtype dtype,
                              const float* lse, int Hq, int Hkv, int d, float scale,
                              const ImpHeads& hs, const int32_t* cu, int B, int64_t sumT,
                              int max_seqlen, bool accumulate, uint32_t flags, float* acc,
                              cudaStream_t st) {
    const bool tc = tc_supported(dtype, d);
    const int tile = tc ? tc_tile() : kSTile;
    const int qc = tc ? tc_qc(B, sumT, hs.n_groups, ctx->num_sms) : kSQc;
    const int nt_max = (max_seqlen + tile - 1) / tile;
    const int c_max = nt_max > 0 ? chunks_of(nt_max, 0, qc) : 0;
    // workspace: [own lse][plan base][info][partials]
    const size_t lse_bytes = lse ? 0 : align_up(sizeof(float) * (size_t)Hq * (size_t)sumT, 256);
    const size_t off_base = lse_bytes;
    const size_t off_info = off_base + align_up(sizeof(int32_t) * (size_t)(B + 1), 256);
    const size_t off_part = off_info + 256;
    const size_t part_bytes = sizeof(float) * (size_t)c_max * (size_t)hs.n_groups * (size_t)sumT;
    estp_status s = ws_reserve(ctx, off_part + part_bytes);
    if (s != ESTP_OK) return s;
    char* ws = static_cast<char*>(ctx->ws);
    // The LSE launch keeps its own plan at the start of the workspace, so an internal
    // LSE goes first and sits below the importance plan.
    float* lse_use = const_cast<float*>(lse);
    if (!lse) {
        lse_use = reinterpret_cast<float*>(ws);
        // LSE kernels only need rows of the selected heads.
        if (tc) s = launch_lse_tc(ctx, Q, K, Hq, Hkv, d, scale, hs, cu, B, sumT, max_seqlen,
                                  lse_use, st, off_base);
        else {
            SimtArgs a{};
            a.Q = Q; a.K = K; a.cu = cu; a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.d = d; a.sumT = sumT;
            a.base = reinterpret_cast<int32_t*>(ws + off_base);
            a.info = reinterpret_cast<PlanInfo*>(ws + off_info);
            a.scale_log2 = scale * kLog2e;
            a.hs = hs;
            a.lse_out = lse_use;
            attn_plan_kernel<<<1, 1024, 0, st>>>(cu, B, sumT, max_seqlen, kSTile, 1, hs.n_heads, 1,
                                                 reinterpret_cast<int32_t*>(ws + off_base),
                                                 reinterpret_cast<PlanInfo*>(ws + off_info),
                                                 ctx->status);
            const size_t smem = simt_smem(d, false);
            const void* kfn = dtype == ESTP_BF16 ? (const void*)lse_simt_kernel<true> : (const void*)lse_simt_kernel<false>;
            cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            const int grid = persistent_grid(ctx, kfn, kSThreads, smem);
            if (dtype == ESTP_BF16) lse_simt_kernel<true><<<grid, kSThreads, smem, st>>>(a);
            else lse_simt_kernel<false><<<grid, kSThreads, smem, st>>>(a);
        }
        if (s != ESTP_OK) return s;
    }
    int32_t* base = reinterpret_cast<int32_t*>(ws + off_base);
    PlanInfo* info = reinterpret_cast<PlanInfo*>(ws + off_info);
    float* part = reinterpret_cast<float*>(ws + off_part);
    attn_plan_kernel<<<1, 1024, 0, st>>>(cu, B, sumT, max_seqlen, tile, qc, hs.n_groups, 0, base,
                                         info, ctx->status);
    if (tc) {
        s = launch_imp_tc(ctx, Q, K, lse_use, Hq, Hkv, d, scale, hs, cu, B, sumT,
                          (flags & ESTP_IMP_EXCLUDE_SELF) != 0, base, info, part, c_max, qc, st);
        if (s != ESTP_OK) return s;
    } else {
        SimtArgs a{};
        a.Q = Q; a.K = K; a.lse = lse_use; a.cu = cu; a.base = base; a.info = info; a.B = B;
        a.Hq = Hq; a.Hkv = Hkv; a.d = d; a.sumT = sumT; a.scale_log2 = scale * kLog2e;
        a.hs = hs; a.exclude_self = (flags & ESTP_IMP_EXCLUDE_SELF) != 0; a.part = part;
        a.c_max = c_max; a.status = ctx->status;
        const size_t smem = simt_smem(d, true);
        const void* kfn = dtype == ESTP_BF16 ? (const void*)imp_simt_kernel<true> : (const void*)imp_simt_kernel<false>;
        cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        const int grid = persistent_grid(ctx, kfn, kSThreads, smem);
        if (dtype == ESTP_BF16) imp_simt_kernel<true><<<grid, kSThreads, smem, st>>>(a);
        else imp_simt_kernel<false><<<grid, kSThreads, smem, st>>>(a);
    }
    {  // a programmatic dependent of the column-sum kernel: it waits on it on the device
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)((sumT + 255) / 256));
        cfg.blockDim = dim3(256);
        cfg.stream = st;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        cudaError_t e = cudaLaunchKernelEx(&cfg, imp_reduce_kernel, (const float*)part,
                                           (const PlanInfo*)info, cu, B, sumT, hs.n_groups, tile,
                                           qc, accumulate ? 1 : 0, acc, c_max, ctx->status);
        if (e != cudaSuccess) return cuda_fail(e, "importance reduce launch");
    }
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "importance launch");
}

estp_status launch_importance_finalize(estp_ctx* ctx, const float* acc, const int32_t* cu, int B,
                                       int64_t sumT, int n_layers, int n_heads, uint32_t flags,
                                       float* out, cudaStream_t st) {
    (void)ctx;
    const float inv_lh = 1.f / ((float)n_layers * (float)n_heads);
    const int div = (flags & ESTP_IMP_DIV_CAUSAL) ? 1 : (flags & ESTP_IMP_DIV_NONE) ? 2 : 0;
    imp_finalize_kernel<<<(unsigned)((sumT + 255) / 256), 256, 0, st>>>(
        acc, cu, B, sumT, inv_lh, div, (flags & ESTP_IMP_EXCLUDE_SELF) ? 1 : 0, out);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "finalize launch");
}

}  // namespace estp
