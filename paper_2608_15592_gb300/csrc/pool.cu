// K-POOL: mixing, tempered softmax and weighted pooling (Eqs. 2-2..2-4, Sec. 3.2),
// then the linear length head (Eq. 3-2, Sec. 3.3).
//
// One pass over the hidden states.  Each prompt is cut into chunks of kChunk
// tokens; a CTA owns (chunk c, slice of D) and produces
//   M_c = max_{i in c} w_i,  Z_c = sum_{i in c} 2^(w_i - M_c),
//   P_c = sum_{i in c} 2^(w_i - M_c) h_i,     w_i = (lambda1 S_i + lambda2 H_i) log2(e) / alpha
// so the prompt-wide softmax of Eq. 2-3 never needs a separate pre-pass.  The merge
// kernel combines chunks in index order:  M = max M_c,  Z = sum 2^(M_c - M) Z_c,
// pooled = sum 2^(M_c - M) P_c / Z  (= sum_i e_i h_i, Eq. 2-4).
#include "estp_internal.cuh"

namespace estp {
namespace {

constexpr int kChunk = 64;        // tokens per chunk
constexpr int kPoolThreads = 256;
constexpr int kMergeThreads = 256;

// Exclusive prefix of ceil(len_b / kChunk) over prompts, validated.  One CTA.
__global__ void __launch_bounds__(1024) chunk_plan_kernel(const int32_t* cu, int B, int64_t sumT,
                                                          int32_t* base, int* status) {
    __shared__ int32_t sums[1024];
    __shared__ int bad;
    const int tid = threadIdx.x;
    if (tid == 0) bad = (cu[0] != 0 || (int64_t)cu[B] != sumT);
    __syncthreads();
    const int per = (B + 1023) / 1024;
    const int b0 = min(B, tid * per), b1 = min(B, b0 + per);
    int32_t local = 0;
    for (int b = b0; b < b1; ++b) {
        int32_t len = cu[b + 1] - cu[b];
        if (len < 0) bad = 1;
        else local += (len + kChunk - 1) / kChunk;
    }
    sums[tid] = local;
    __syncthreads();
    for (int off = 1; off < 1024; off <<= 1) {  // inclusive Hillis-Steele scan
        int32_t v = tid >= off ? sums[tid - off] : 0;
        __syncthreads();
        sums[tid] += v;
        __syncthreads();
    }
    int32_t run = sums[tid] - local;
    const bool ok = !bad;
    for (int b = b0; b < b1; ++b) {
        base[b] = ok ? run : 0;
        int32_t len = cu[b + 1] - cu[b];
        run += len > 0 ? (len + kChunk - 1) / kChunk : 0;
    }
    if (tid == 1023) base[B] = ok ? sums[1023] : 0;
    if (tid == 0 && !ok) report(status, ESTP_ERR_INVALID_ARG);
}

struct PoolArgs {
    const char* hidden;
    int64_t ld_bytes;
    int64_t D;
    int64_t units;           // 16-byte units per row covering D
    const float* H;
    const float* S;
    const int32_t* cu;
    const int32_t* base;     // chunk plan [B+1]
    int B;
    float w_l1, w_l2;        // lambda * log2(e) / alpha
    float* P;                // [n_chunks, D]
    float2* MZ;              // [n_chunks] (M_c, Z_c)
};

template <bool kBf16>
__global__ void __launch_bounds__(kPoolThreads) pool_chunk_kernel(PoolArgs a) {
    __shared__ float e_s[kChunk];
    __shared__ float red[2];
    const int c = blockIdx.x;
    if (c >= a.base[a.B]) return;
    const int b = upper_slot(a.base, a.B, c);
    const int64_t i0 = a.cu[b] + (int64_t)(c - a.base[b]) * kChunk;
    const int64_t left_tokens = a.cu[b + 1] - i0;
    const int n = left_tokens < kChunk ? (int)left_tokens : kChunk;
    const int tid = threadIdx.x;
    if (tid < 32) {  // chunk weights: one warp, two tokens per lane
        float w0 = -INFINITY, w1 = -INFINITY;
        if (tid < n) w0 = fmaf(a.w_l1, a.S[i0 + tid], a.w_l2 * a.H[i0 + tid]);
        if (tid + 32 < n) w1 = fmaf(a.w_l1, a.S[i0 + tid + 32], a.w_l2 * a.H[i0 + tid + 32]);
        float mx = fmaxf(w0, w1);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
        float e0 = tid < n ? ex2(w0 - mx) : 0.f;
        float e1 = tid + 32 < n ? ex2(w1 - mx) : 0.f;
        e_s[tid] = e0;
        e_s[tid + 32] = e1;
        float z = e0 + e1;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(0xffffffffu, z, off);
        if (tid == 0) { red[0] = mx; red[1] = z; }
    }
    __syncthreads();
    const int64_t u = (int64_t)blockIdx.y * kPoolThreads + tid;
    if (blockIdx.y == 0 && tid == 0) a.MZ[c] = make_float2(red[0], red[1]);
    if (u >= a.units) return;
    constexpr int kPer = kBf16 ? 8 : 4;
    float acc[kPer];
#pragma unroll
    for (int k = 0; k < kPer; ++k) acc[k] = 0.f;
    const char* p = a.hidden + i0 * a.ld_bytes + u * 16;
    int i = 0;
    for (; i + 8 <= n; i += 8) {
        uint4 v[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) v[k] = ld_stream(p + (int64_t)(i + k) * a.ld_bytes);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const float e = e_s[i + k];
            if (kBf16) {
                acc[0] = fmaf(e, bf16lo(v[k].x), acc[0]);
                acc[1] = fmaf(e, bf16hi(v[k].x), acc[1]);
                acc[2] = fmaf(e, bf16lo(v[k].y), acc[2]);
                acc[3] = fmaf(e, bf16hi(v[k].y), acc[3]);
                acc[4] = fmaf(e, bf16lo(v[k].z), acc[4]);
                acc[5] = fmaf(e, bf16hi(v[k].z), acc[5]);
                acc[6] = fmaf(e, bf16lo(v[k].w), acc[6]);
                acc[7] = fmaf(e, bf16hi(v[k].w), acc[7]);
            } else {
                acc[0] = fmaf(e, __uint_as_float(v[k].x), acc[0]);
                acc[1] = fmaf(e, __uint_as_float(v[k].y), acc[1]);
                acc[2] = fmaf(e, __uint_as_float(v[k].z), acc[2]);
                acc[3] = fmaf(e, __uint_as_float(v[k].w), acc[3]);
            }
        }
    }
    for (; i < n; ++i) {
        uint4 v = ld_stream(p + (int64_t)i * a.ld_bytes);
        const float e = e_s[i];
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
    float* out = a.P + (int64_t)c * a.D + u * kPer;
    const int64_t left = a.D - u * kPer;
#pragma unroll
    for (int k = 0; k < kPer; ++k)
        if (k < left) out[k] = acc[k];
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
    return r;
}

// pooled[b, cols of this CTA] from the prompt's chunks, in chunk order.
__global__ void __launch_bounds__(kMergeThreads) pool_merge_kernel(const float* P, const float2* MZ,
                                                                   const int32_t* base, int64_t D,
                                                                   float* pooled) {
    __shared__ float f_s[kMergeThreads];
    __shared__ float sh[32];
    const int b = blockIdx.x;
    const int c0 = base[b], c1 = base[b + 1];
    const int64_t col = ((int64_t)blockIdx.y * kMergeThreads + threadIdx.x) * 4;
    float mx = -INFINITY;
    for (int c = c0 + threadIdx.x; c < c1; c += kMergeThreads) mx = fmaxf(mx, MZ[c].x);
    mx = block_reduce(mx, true, sh);
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    float zpart = 0.f;
    for (int cb = c0; cb < c1; cb += kMergeThreads) {
        __syncthreads();
        const int c = cb + threadIdx.x;
        float f = 0.f;
        if (c < c1) {
            float2 mz = MZ[c];
            f = ex2(mz.x - mx);
            zpart += f * mz.y;
        }
        f_s[threadIdx.x] = f;
        __syncthreads();
        const int nb = min(kMergeThreads, c1 - cb);
        if (col < D) {
            for (int k = 0; k < nb; ++k) {
                const float* row = P + (int64_t)(cb + k) * D + col;
                const float f2 = f_s[k];
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (col + q < D) acc[q] = fmaf(f2, row[q], acc[q]);
            }
        }
    }
    const float Z = block_reduce(zpart, false, sh);
    if (col < D) {
        const float inv = c1 > c0 ? 1.f / Z : 0.f;
#pragma unroll
        for (int q = 0; q < 4; ++q)
            if (col + q < D) pooled[(int64_t)b * D + col + q] = acc[q] * inv;
    }
}

// Linear head + softmax over K bins + expectation (Eq. 3-2).  One CTA of 32 warps per
// prompt; warp w forms the logits z_k = W_k . h + bias_k of bins k = w, w + 32, ...
// (float4 loads when rows are 16-byte aligned), then the CTA reduces the softmax and
// the expectation in a fixed order.
__global__ void __launch_bounds__(1024) head_kernel(const float* pooled, int64_t D, const float* W,
                                                    const float* bias, const float* centers, int K,
                                                    int vec4, float* pred) {
    __shared__ float z_s[1024];
    __shared__ float sh[32];
    const int b = blockIdx.x;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const float* h = pooled + (int64_t)b * D;
    for (int k = wid; k < K; k += 32) {
        const float* w = W + (int64_t)k * D;
        float acc0 = 0.f, acc1 = 0.f;
        if (vec4) {
            const float4* w4 = reinterpret_cast<const float4*>(w);
            const float4* h4 = reinterpret_cast<const float4*>(h);
            const int64_t n4 = D / 4;
            int64_t x = lane;
            for (; x + 32 < n4; x += 64) {
                const float4 a0 = w4[x], b0 = h4[x], a1 = w4[x + 32], b1 = h4[x + 32];
                acc0 = fmaf(a0.x, b0.x, fmaf(a0.y, b0.y, fmaf(a0.z, b0.z, fmaf(a0.w, b0.w, acc0))));
                acc1 = fmaf(a1.x, b1.x, fmaf(a1.y, b1.y, fmaf(a1.z, b1.z, fmaf(a1.w, b1.w, acc1))));
            }
            for (; x < n4; x += 32) {
                const float4 a0 = w4[x], b0 = h4[x];
                acc0 = fmaf(a0.x, b0.x, fmaf(a0.y, b0.y, fmaf(a0.z, b0.z, fmaf(a0.w, b0.w, acc0))));
            }
        } else {
            for (int64_t x = lane; x < D; x += 32) acc0 = fmaf(w[x], h[x], acc0);
        }
        float acc = acc0 + acc1;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
        if (lane == 0) z_s[k] = acc + (bias ? bias[k] : 0.f);
    }
    __syncthreads();
    float mx = -INFINITY;
    for (int k = threadIdx.x; k < K; k += 1024) mx = fmaxf(mx, z_s[k]);
    mx = block_reduce(mx, true, sh);
    float zs = 0.f, ys = 0.f;
    for (int k = threadIdx.x; k < K; k += 1024) {
        const float e = ex2((z_s[k] - mx) * kLog2e);
        zs += e;
        ys = fmaf(e, centers[k], ys);
    }
    zs = block_reduce(zs, false, sh);
    ys = block_reduce(ys, false, sh);
    if (threadIdx.x == 0) pred[b] = ys / zs;
}

}  // namespace

estp_status launch_pool(estp_ctx* ctx, const void* hidden, estp_dtype dtype, int64_t D,
                        int64_t ldh, const float* H, const float* S, const int32_t* cu, int B,
                        int64_t sumT, estp_mix_params mix, const estp_head* head, float* pooled,
                        float* pred, cudaStream_t st) {
    const int64_t n_chunks = (sumT + kChunk - 1) / kChunk + B;  // upper bound
    const size_t off_base = 0;
    const size_t off_mz = align_up(sizeof(int32_t) * (size_t)(B + 1), 256);
    const size_t off_p = align_up(off_mz + sizeof(float2) * (size_t)n_chunks, 256);
    const size_t bytes = off_p + sizeof(float) * (size_t)n_chunks * (size_t)D;
    estp_status s = ws_reserve(ctx, bytes);
    if (s != ESTP_OK) return s;
    char* ws = static_cast<char*>(ctx->ws);
    PoolArgs a;
    a.hidden = static_cast<const char*>(hidden);
    a.ld_bytes = ldh * esize(dtype);
    a.D = D;
    const int per = dtype == ESTP_BF16 ? 8 : 4;
    a.units = (D + per - 1) / per;
    a.H = H;
    a.S = S;
    a.cu = cu;
    a.base = reinterpret_cast<int32_t*>(ws + off_base);
    a.B = B;
    a.w_l1 = mix.lambda1 * kLog2e / mix.alpha;
    a.w_l2 = mix.lambda2 * kLog2e / mix.alpha;
    a.P = reinterpret_cast<float*>(ws + off_p);
    a.MZ = reinterpret_cast<float2*>(ws + off_mz);
    chunk_plan_kernel<<<1, 1024, 0, st>>>(cu, B, sumT, reinterpret_cast<int32_t*>(ws + off_base), ctx->status);
    if (n_chunks > 0 && sumT > 0) {
        dim3 grid((unsigned)n_chunks, (unsigned)((a.units + kPoolThreads - 1) / kPoolThreads));
        if (dtype == ESTP_BF16) pool_chunk_kernel<true><<<grid, kPoolThreads, 0, st>>>(a);
        else pool_chunk_kernel<false><<<grid, kPoolThreads, 0, st>>>(a);
    }
    dim3 mgrid((unsigned)B, (unsigned)((D + 4 * kMergeThreads - 1) / (4 * kMergeThreads)));
    pool_merge_kernel<<<mgrid, kMergeThreads, 0, st>>>(a.P, a.MZ, a.base, D, pooled);
    if (head && pred) {
        const int vec4 = (D % 4 == 0) && aligned16(head->W) && aligned16(pooled);
        head_kernel<<<B, 1024, 0, st>>>(pooled, D, head->W, head->bias, head->centers, head->K,
                                        vec4, pred);
    }
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "pool launch");
}

}  // namespace estp
