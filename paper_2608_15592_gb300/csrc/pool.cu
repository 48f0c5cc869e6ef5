// K-POOL: mixing, tempered softmax and weighted pooling (Eqs. 2-2..2-4, Sec. 3.2),
// then the linear length head (Eq. 3-2, Sec. 3.3).  Two launches, one pass over the
// hidden states.
//
// pool_stream_kernel: the packed token axis is cut evenly over a persistent grid (one
// wave): CTA c owns tokens [t_c, t_{c+1}) with t_c = floor(c * sumT / G).  Its range
// splits at prompt boundaries into segments; for the segment of prompt b it writes,
// over the segment's tokens i,
//   M = max w_i,  Z = sum 2^(w_i - M),  P = sum 2^(w_i - M) h_i,
//   w_i = (lambda1 S_i + lambda2 H_i) log2(e) / alpha
// (online over windows of up to 4096 tokens, rescaling when the running max grows) to
// slot c + b.  Slots are ordered like the tokens, so the segments of a prompt occupy
// consecutive slots.
//
// pool_finish_kernel: CTA (b, column block) merges the slots of prompt b in order,
//   M* = max M_s,  Z* = sum 2^(M_s - M*) Z_s,  pooled = sum 2^(M_s - M*) P_s / Z*
// (= sum_i e_i h_i of Eq. 2-4; zero for a prompt without tokens), and forms the partial
// logits of the length head over its columns; the last CTA of the prompt (an arrival
// counter) adds the partials in column-block order and reduces the head.  The merge
// and the head run after the stream, when their short dependent reads meet an idle
// memory system.  No floating-point atomics: every sum runs in a fixed order.
#include "estp_internal.cuh"

namespace estp {
namespace {

constexpr int kWin = 4096;        // tokens whose weights are staged at once (one window)
constexpr int kMaxThreads = 512;  // stream CTA: 16-byte column units of one slice
constexpr int kBatch = 4;         // rows per load batch; two batches in flight per thread
constexpr int kFinThreads = 512;  // finish CTA: 2 columns per thread
constexpr int kFinCols = 2 * kFinThreads;
constexpr int kMaxSlots = 1024;   // slot factors staged per pass of the finish kernel

struct StreamArgs {
    const char* hidden;
    int64_t ld_bytes;
    int64_t D;
    int64_t units;           // 16-byte units per row covering D
    int64_t slice_units;     // units per column slice (grid.y)
    const float* H;
    const float* S;
    const int32_t* cu;
    int B;
    int64_t sumT;
    int G;                   // CTAs along the token axis (grid.x)
    float w_l1, w_l2;        // lambda * log2(e) / alpha
    float* P;                // [G + B slots, D]
    float2* MZ;              // [G + B slots] (M, Z)
    int* status;
};

struct FinishArgs {
    const float* P;
    const float2* MZ;
    const int32_t* cu;
    int B;
    int64_t sumT;
    int G;
    int64_t D;
    int n_cb;                // column blocks (grid.y)
    int vec2;                // D even and P, pooled, W 8-byte aligned: float2 access
    float* pooled;           // [B, D]
    uint32_t* done;          // [B] arrival counters (back to zero after the last arrival)
    float* zpart;            // [B, n_cb, K] partial logits
    const float* W;          // length head (NULL: pooling only)
    const float* bias;
    const float* centers;
    int K;
    float* pred;
    int* status;             // bounds checks of debug builds
};

// Eight bf16 (or four fp32) values of one 16-byte unit, weighted by e, added to acc.
template <bool kBf16>
__device__ __forceinline__ void acc_unit(float* acc, const uint4& v, float e) {
    if (kBf16) {
        acc[0] = fmaf(e, bf16lo(v.x), acc[0]);
        acc[1] = fmaf(e, bf16hi(v.x), acc[1]);
        acc[2] = fmaf(e, bf16lo(v.y), acc[2]);
        acc[3] = fmaf(e, bf16hi(v.y), acc[3]);
        acc[4] = fmaf(e, bf16lo(v.z), acc[4]);
        acc[5] = fmaf(e, bf16hi(v.z), acc[5]);
        acc[6] = fmaf(e, bf16lo(v.w), acc[6]);
        acc[7] = fmaf(e, bf16hi(v.w), acc[7]);
    } else {
        acc[0] = fmaf(e, __uint_as_float(v.x), acc[0]);
        acc[1] = fmaf(e, __uint_as_float(v.y), acc[1]);
        acc[2] = fmaf(e, __uint_as_float(v.z), acc[2]);
        acc[3] = fmaf(e, __uint_as_float(v.w), acc[3]);
    }
}

__device__ float block_reduce(float v, bool is_max, float* sh) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        float o = __shfl_xor_sync(0xffffffffu, v, off);
        v = is_max ? fmaxf(v, o) : v + o;
    }
    __syncthreads();
    if (lane == 0) sh[wid] = v;
    __syncthreads();
    float r = sh[0];
    for (int k = 1; k < nw; ++k) r = is_max ? fmaxf(r, sh[k]) : r + sh[k];
    __syncthreads();  // sh may be reused right away
    return r;
}

// First token of CTA c's range, and the CTA that owns token i (0 <= i < sumT).
__device__ __forceinline__ int64_t range_start(int64_t c, int64_t sumT, int G) {
    return c * sumT / G;
}
__device__ __forceinline__ int owner_cta(int64_t i, int64_t sumT, int G) {
    const int64_t c = ((i + 1) * G - 1) / sumT;
    return (int)(c < G - 1 ? c : G - 1);
}

template <bool kBf16>
__global__ void __launch_bounds__(kMaxThreads, 2) pool_stream_kernel(const StreamArgs a) {
    __shared__ float e_s[kWin];
    __shared__ float sh[32];
    const int c = blockIdx.x, tid = threadIdx.x;
    const int64_t t_lo = range_start(c, a.sumT, a.G), t_hi = range_start(c + 1, a.sumT, a.G);
    const int64_t u = (int64_t)blockIdx.y * a.slice_units + tid;
    const bool active = tid < a.slice_units && u < a.units;
    constexpr int kPer = kBf16 ? 8 : 4;

    // Every CTA checks all of cu_seqlens the same way (bad metadata: nothing is written
    // but the status word).
    int bad = 0;
    if (tid == 0) bad = a.cu[0] != 0 || (int64_t)a.cu[a.B] != a.sumT;
    for (int b = tid; b < a.B; b += blockDim.x) bad |= a.cu[b + 1] < a.cu[b];
    bad = __syncthreads_or(bad);
    // the finish kernel may be scheduled now: it waits for this grid before reading its output
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (bad && c == 0 && blockIdx.y == 0 && tid == 0) report(a.status, ESTP_ERR_INVALID_ARG);
    if (bad || t_lo >= t_hi) return;

    const char* p = a.hidden + (active ? u : 0) * 16;
    int b = upper_slot(a.cu, a.B, t_lo);  // the prompt of token t_lo (never an empty one)
    for (int64_t s0 = t_lo; s0 < t_hi;) {
        const int64_t s1 = min((int64_t)a.cu[b + 1], t_hi);  // segment [s0, s1) of prompt b
        float acc[kPer];
#pragma unroll
        for (int k = 0; k < kPer; ++k) acc[k] = 0.f;
        float m = -INFINITY, z = 0.f;  // running max and sum (uniform over the CTA)
        for (int64_t i0 = s0; i0 < s1; i0 += kWin) {
            const int n = (int)min((int64_t)kWin, s1 - i0);
            uint4 va[kBatch], vb[kBatch];  // the first rows are requested before the weights
#pragma unroll
            for (int k = 0; k < kBatch; ++k)
                if (active && k < n) va[k] = ld_stream(p + (i0 + k) * a.ld_bytes);
            // the window's weights, its max, and 2^(w - max) staged in shared memory
            float wmax = -INFINITY;
            for (int i = tid; i < n; i += blockDim.x) {
                const float w = fmaf(a.w_l1, a.S[i0 + i], a.w_l2 * a.H[i0 + i]);
                e_s[i] = w;
                wmax = fmaxf(wmax, w);
            }
            const float nm = fmaxf(m, block_reduce(wmax, true, sh));
            float zw = 0.f;
            for (int i = tid; i < n; i += blockDim.x) {
                const float e = ex2(e_s[i] - nm);
                e_s[i] = e;
                zw += e;
            }
            zw = block_reduce(zw, false, sh);  // fixed-order sum (also a barrier for e_s)
            const float f = m == -INFINITY ? 0.f : ex2(m - nm);  // rescale to the new max
#pragma unroll
            for (int k = 0; k < kPer; ++k) acc[k] *= f;
            z = z * f + zw;
            m = nm;
            if (active) {  // rows in two alternating batches: one reduced while one loads
                for (int i = 0; i < n; i += 2 * kBatch) {
#pragma unroll
                    for (int k = 0; k < kBatch; ++k)
                        if (i + kBatch + k < n) vb[k] = ld_stream(p + (i0 + i + kBatch + k) * a.ld_bytes);
#pragma unroll
                    for (int k = 0; k < kBatch; ++k)
                        if (i + k < n) acc_unit<kBf16>(acc, va[k], e_s[i + k]);
#pragma unroll
                    for (int k = 0; k < kBatch; ++k)
                        if (i + 2 * kBatch + k < n) va[k] = ld_stream(p + (i0 + i + 2 * kBatch + k) * a.ld_bytes);
#pragma unroll
                    for (int k = 0; k < kBatch; ++k)
                        if (i + kBatch + k < n) acc_unit<kBf16>(acc, vb[k], e_s[i + kBatch + k]);
                }
            }
            __syncthreads();  // e_s is rewritten by the next window
        }
        const int slot = c + b;
        if (!in_bounds(slot >= 0 && slot < a.G + a.B && b < a.B, a.status)) return;
        if (active) {
            float* out = a.P + (int64_t)slot * a.D + u * kPer;
            const int64_t left = a.D - u * kPer;
#pragma unroll
            for (int k = 0; k < kPer; ++k)
                if (k < left) out[k] = acc[k];
        }
        if (blockIdx.y == 0 && tid == 0) a.MZ[slot] = make_float2(m, z);
        s0 = s1;
        ++b;
        while (b < a.B && a.cu[b + 1] == a.cu[b]) ++b;  // empty prompts own no tokens
    }
}

// Online merge of (max, sum) pairs: (m, z) <- (m, z) + (m2, z2) rescaled to the larger max.
__device__ __forceinline__ void merge_mz(float& m, float& z, float m2, float z2) {
    const float nm = fmaxf(m, m2);
    if (nm == -INFINITY) return;
    z = z * ex2(m - nm) + z2 * ex2(m2 - nm);
    m = nm;
}

// 2 columns at `col` of a float row (float2 when aligned, else bounds-checked scalars).
__device__ __forceinline__ float2 load2(const float* row, int64_t col, int64_t D, bool v2) {
    if (v2) return *reinterpret_cast<const float2*>(row + col);
    return make_float2(row[col], col + 1 < D ? row[col + 1] : 0.f);
}

// Reduce-scatter over a warp: on entry lane l holds v[0..31] (32 bins), on exit it holds
// in v[0] the warp sum of bin l.  Five butterfly rounds of halving width; every lane
// adds in the same order, so the result is deterministic.
__device__ __forceinline__ float warp_reduce_scatter32(float* v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int w = 16; w >= 1; w >>= 1) {
        const bool upper = (lane & w) != 0;  // keep bins [w, 2w) of the current block, else [0, w)
#pragma unroll
        for (int j = 0; j < w; ++j) {
            const float send = upper ? v[j] : v[j + w];
            const float keep = upper ? v[j + w] : v[j];
            v[j] = keep + __shfl_xor_sync(0xffffffffu, send, w);
        }
    }
    return v[0];
}

// CTA (b, column block): merge of prompt b's slots over kFinCols columns, partial logits.
__global__ void __launch_bounds__(kFinThreads) pool_finish_kernel(const FinishArgs a) {
    __shared__ float f_s[kMaxSlots];
    __shared__ float2 mz_s[kFinThreads / 32];
    __shared__ float red[kFinThreads / 32][32];
    __shared__ float z_s[1024];
    __shared__ float sh[32];
    __shared__ int last;
    const int b = blockIdx.x, cb = blockIdx.y, tid = threadIdx.x;
    const int lane = tid & 31, wid = tid >> 5, nw = blockDim.x >> 5;
    const int64_t col = (int64_t)cb * kFinCols + 2 * tid;  // this thread's 2 columns
    const bool in = col < a.D;
    const bool v2 = a.vec2 != 0;
    // head rows of the first 32 bins: requested before the stream kernel has finished
    float2 wv[32];
#pragma unroll
    for (int j = 0; j < 32; ++j)
        wv[j] = a.W && j < a.K && in ? load2(a.W + (int64_t)j * a.D, col, a.D, v2) : make_float2(0.f, 0.f);
    // cu_seqlens is an input: checked here as the stream kernel checks it (which reports)
    const int32_t t0 = a.cu[b], t1 = a.cu[b + 1];
    int bad = 0;
    if (tid == 0) bad = a.cu[0] != 0 || (int64_t)a.cu[a.B] != a.sumT;
    for (int k = tid; k < a.B; k += blockDim.x) bad |= a.cu[k + 1] < a.cu[k];
    if (__syncthreads_or(bad)) return;
    // the stream kernel's slots are complete past this point
    asm volatile("griddepcontrol.wait;" ::: "memory");
    float2 h = make_float2(0.f, 0.f);
    if (t1 > t0 && in_bounds(owner_cta(t1 - 1, a.sumT, a.G) + b < a.G + a.B, a.status)) {
        const int c0 = owner_cta(t0, a.sumT, a.G), c1 = owner_cta(t1 - 1, a.sumT, a.G);
        const int n = c1 - c0 + 1;
        // (M*, Z*) in one pass: online per thread, then warps and the CTA in fixed order
        float m = -INFINITY, z = 0.f;
        for (int k = tid; k < n; k += blockDim.x) {
            const float2 mz = a.MZ[c0 + k + b];
            if (k < kMaxSlots) f_s[k] = mz.x;
            merge_mz(m, z, mz.x, mz.y);
        }
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float m2 = __shfl_xor_sync(0xffffffffu, m, off), z2 = __shfl_xor_sync(0xffffffffu, z, off);
            merge_mz(m, z, m2, z2);
        }
        if (lane == 0) mz_s[wid] = make_float2(m, z);
        __syncthreads();
        m = -INFINITY;
        z = 0.f;
        for (int w = 0; w < nw; ++w) merge_mz(m, z, mz_s[w].x, mz_s[w].y);
        const float mx = m, inv = 1.f / z;
        for (int cc = 0; cc < n; cc += kMaxSlots) {  // slots in passes of kMaxSlots factors
            const int nn = min(kMaxSlots, n - cc);
            if (cc > 0) {
                __syncthreads();
                for (int k = tid; k < nn; k += blockDim.x) f_s[k] = a.MZ[c0 + cc + k + b].x;
            }
            __syncthreads();
            for (int k = tid; k < nn; k += blockDim.x) f_s[k] = ex2(f_s[k] - mx);
            __syncthreads();
            if (in) {
                int k = 0;
                for (; k + 16 <= nn; k += 16) {  // sixteen slots in flight
                    float2 p[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) p[j] = load2(a.P + (int64_t)(c0 + cc + k + j + b) * a.D, col, a.D, v2);
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        h.x = fmaf(f_s[k + j], p[j].x, h.x);
                        h.y = fmaf(f_s[k + j], p[j].y, h.y);
                    }
                }
                for (; k < nn; ++k) {
                    const float2 p = load2(a.P + (int64_t)(c0 + cc + k + b) * a.D, col, a.D, v2);
                    h.x = fmaf(f_s[k], p.x, h.x);
                    h.y = fmaf(f_s[k], p.y, h.y);
                }
            }
        }
        h.x *= inv;
        h.y *= inv;
    }
    if (in) {
        float* out = a.pooled + (int64_t)b * a.D;
        if (v2) *reinterpret_cast<float2*>(out + col) = h;
        else {
            out[col] = h.x;
            if (col + 1 < a.D) out[col + 1] = h.y;
        }
    }
    if (!a.W) return;
    // partial logits of these columns, 32 bins per pass: products, reduce-scatter over the
    // warp (lane l ends with bin l), warp partials added in warp order
    for (int k0 = 0; k0 < a.K; k0 += 32) {
        float part[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            if (k0 > 0)
                wv[j] = k0 + j < a.K && in ? load2(a.W + (int64_t)(k0 + j) * a.D, col, a.D, v2)
                                           : make_float2(0.f, 0.f);
            part[j] = fmaf(wv[j].x, h.x, wv[j].y * h.y);
        }
        red[wid][lane] = warp_reduce_scatter32(part);
        __syncthreads();
        if (tid < 32 && k0 + tid < a.K) {
            float zk = 0.f;
            for (int w = 0; w < nw; ++w) zk += red[w][tid];
            a.zpart[((int64_t)b * a.n_cb + cb) * a.K + k0 + tid] = zk;
        }
        __syncthreads();
    }
    // arrival; the last CTA of prompt b adds the column blocks in order and reduces the head
    __threadfence();
    __syncthreads();
    if (tid == 0) last = atomicInc(&a.done[b], (uint32_t)a.n_cb - 1) == (uint32_t)a.n_cb - 1;
    __syncthreads();
    if (!last) return;
    __threadfence();
    for (int k = tid; k < a.K; k += blockDim.x) {
        float zk = a.bias ? a.bias[k] : 0.f;
        for (int j = 0; j < a.n_cb; ++j) zk += __ldcg(a.zpart + ((int64_t)b * a.n_cb + j) * a.K + k);
        z_s[k] = zk;
    }
    __syncthreads();
    float mx = -INFINITY;
    for (int k = tid; k < a.K; k += blockDim.x) mx = fmaxf(mx, z_s[k]);
    mx = block_reduce(mx, true, sh);
    float zs = 0.f, ys = 0.f;
    for (int k = tid; k < a.K; k += blockDim.x) {
        const float e = ex2((z_s[k] - mx) * kLog2e);
        zs += e;
        ys = fmaf(e, a.centers[k], ys);
    }
    zs = block_reduce(zs, false, sh);
    ys = block_reduce(ys, false, sh);
    if (tid == 0) a.pred[b] = ys / zs;
}

}  // namespace

estp_status launch_pool(estp_ctx* ctx, const void* hidden, estp_dtype dtype, int64_t D,
                        int64_t ldh, const float* H, const float* S, const int32_t* cu, int B,
                        int64_t sumT, estp_mix_params mix, const estp_head* head, float* pooled,
                        float* pred, cudaStream_t st) {
    StreamArgs a{};
    a.hidden = static_cast<const char*>(hidden);
    a.ld_bytes = ldh * esize(dtype);
    a.D = D;
    const int per = dtype == ESTP_BF16 ? 8 : 4;
    a.units = (D + per - 1) / per;
    const int n_slices = (int)((a.units + kMaxThreads - 1) / kMaxThreads);
    a.slice_units = (a.units + n_slices - 1) / n_slices;
    const int threads = (int)((a.slice_units + 31) / 32 * 32);
    const void* kfn = dtype == ESTP_BF16 ? (const void*)pool_stream_kernel<true>
                                         : (const void*)pool_stream_kernel<false>;
    int occ = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kfn, threads, 0);
    if (e != cudaSuccess) return cuda_fail(e, "pool occupancy");
    // one wave: G token ranges x n_slices column slices; every range holds >= 1 token
    int64_t G = (int64_t)ctx->num_sms * (occ > 0 ? occ : 1) / n_slices;
    if (G < 1) G = 1;
    if (sumT > 0 && G > sumT) G = sumT;
    a.G = (int)G;
    a.H = H;
    a.S = S;
    a.cu = cu;
    a.B = B;
    a.sumT = sumT;
    a.w_l1 = mix.lambda1 * kLog2e / mix.alpha;
    a.w_l2 = mix.lambda2 * kLog2e / mix.alpha;
    a.status = ctx->status;
    const bool with_head = head && pred;
    const int K = with_head ? head->K : 0;
    const int n_cb = (int)((D + kFinCols - 1) / kFinCols);
    // arrival counters persist in the context (zero, and back to zero after each prompt)
    if (with_head && ctx->pool_done_cap < B) {
        cudaFree(ctx->pool_done);
        ctx->pool_done = nullptr;
        ctx->pool_done_cap = 0;
        e = cudaMalloc(&ctx->pool_done, sizeof(uint32_t) * (size_t)B);
        if (e == cudaSuccess) e = cudaMemset(ctx->pool_done, 0, sizeof(uint32_t) * (size_t)B);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(ESTP_ERR_WORKSPACE, "pool counters: %s", cudaGetErrorString(e));
        }
        ctx->pool_done_cap = B;
    }
    // workspace: [MZ slots][zpart B x n_cb x K][P slots x D], G + B slots
    const int64_t slots = G + B;
    const size_t off_mz = 0;
    const size_t off_z = align_up(off_mz + sizeof(float2) * (size_t)slots, 256);
    const size_t off_p = align_up(off_z + sizeof(float) * (size_t)B * n_cb * K, 256);
    estp_status s = ws_reserve(ctx, off_p + sizeof(float) * (size_t)slots * (size_t)D);
    if (s != ESTP_OK) return s;
    char* ws = static_cast<char*>(ctx->ws);
    a.MZ = reinterpret_cast<float2*>(ws + off_mz);
    a.P = reinterpret_cast<float*>(ws + off_p);
    dim3 grid((unsigned)G, (unsigned)n_slices);
    if (dtype == ESTP_BF16) pool_stream_kernel<true><<<grid, threads, 0, st>>>(a);
    else pool_stream_kernel<false><<<grid, threads, 0, st>>>(a);
    FinishArgs f{};
    f.status = ctx->status;
    f.P = a.P;
    f.MZ = a.MZ;
    f.cu = cu;
    f.B = B;
    f.sumT = sumT;
    f.G = a.G;
    f.D = D;
    f.n_cb = n_cb;
    f.vec2 = D % 2 == 0 && aligned16(pooled) && (!with_head || aligned16(head->W));
    f.pooled = pooled;
    if (with_head) {
        f.done = ctx->pool_done;
        f.zpart = reinterpret_cast<float*>(ws + off_z);
        f.W = head->W;
        f.bias = head->bias;
        f.centers = head->centers;
        f.K = K;
        f.pred = pred;
    }
    // launched as a programmatic dependent of the stream kernel (it waits on it on the device)
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)B, (unsigned)n_cb);
    cfg.blockDim = dim3(kFinThreads);
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, pool_finish_kernel, f);
    if (e != cudaSuccess) return cuda_fail(e, "pool finish launch");
    e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "pool launch");
}

}  // namespace estp
