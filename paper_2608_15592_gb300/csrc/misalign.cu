// Entropy/importance misalignment counts (the diagnostic behind Fig. 1b): per prompt,
// the k = floor(pct * T / 100) tokens with the largest and the smallest entropy H and
// importance S, and how many of the high-entropy tokens are among the low-importance
// ones (and the reverse).
//
// CTA b handles prompt b.  Each token gets a 64-bit key: the order-preserving unsigned
// image of its value in the high half and its index in the low half (the index reversed
// for "largest first"), so all keys are distinct and ties go to the lower index.  Four
// radix selections (8 passes of 8-bit digits, shared-memory histograms) find the k-th
// key of each order; a last pass counts the two intersections.  Integer counts: the
// result is exact.
#include "estp_internal.cuh"

namespace estp {
namespace {

constexpr int kThreads = 1024;

// monotone map float -> uint32 (larger float, larger image); inputs are finite, and
// -0 maps with +0 (they are equal values, so their order falls to the index)
__device__ __forceinline__ uint32_t ordered(float f) {
    const uint32_t u = f == 0.f ? 0u : __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// "k largest, lower index first": the earlier token has the larger key
__device__ __forceinline__ uint64_t key_top(float x, int i) {
    return ((uint64_t)ordered(x) << 32) | (uint32_t)(0xFFFFFFFFu - (uint32_t)i);
}
// "k smallest, lower index first": the earlier token has the smaller key
__device__ __forceinline__ uint64_t key_bot(float x, int i) {
    return ((uint64_t)ordered(x) << 32) | (uint32_t)i;
}

// The r-th smallest (1-based) of the n keys key(v[i], i): eight passes, most significant
// digit first, each keeping the keys that share the digits found so far.
template <bool kTop>
__device__ uint64_t select_rank(const float* v, int n, int r, uint32_t* hist, uint64_t* sh) {
    uint64_t prefix = 0, mask = 0;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int d = threadIdx.x; d < 256; d += blockDim.x) hist[d] = 0;
        __syncthreads();
        for (int i = threadIdx.x; i < n; i += blockDim.x) {
            const uint64_t key = kTop ? key_top(v[i], i) : key_bot(v[i], i);
            if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255], 1u);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            int cum = 0, d = 0;
            for (; d < 255; ++d) {
                if (cum + (int)hist[d] >= r) break;
                cum += (int)hist[d];
            }
            sh[0] = prefix | ((uint64_t)d << shift);
            sh[1] = (uint64_t)(r - cum);
        }
        __syncthreads();
        prefix = sh[0];
        r = (int)sh[1];
        mask |= (uint64_t)255 << shift;
        __syncthreads();  // sh is rewritten by the next pass
    }
    return prefix;
}

__global__ void __launch_bounds__(kThreads) misalign_kernel(const float* __restrict__ H,
                                                            const float* __restrict__ S,
                                                            const int32_t* __restrict__ cu, int B,
                                                            int64_t sumT, int pct,
                                                            int32_t* __restrict__ counts,
                                                            int* status) {
    __shared__ uint32_t hist[256];
    __shared__ uint64_t sh[2];
    __shared__ int n_hl, n_lh;
    const int b = blockIdx.x;
    // cu_seqlens is checked by every CTA the same way; CTA 0 reports
    int bad = 0;
    if (threadIdx.x == 0) bad = cu[0] != 0 || (int64_t)cu[B] != sumT;
    for (int q = threadIdx.x; q < B; q += blockDim.x) bad |= cu[q + 1] < cu[q];
    if (__syncthreads_or(bad)) {
        if (b == 0 && threadIdx.x == 0) report(status, ESTP_ERR_INVALID_ARG);
        return;
    }
    const int64_t t0 = cu[b];
    const int T = cu[b + 1] - cu[b];
    const int k = (int)((int64_t)pct * T / 100);
    if (k == 0) {
        if (threadIdx.x == 0) {
            counts[3 * b] = 0;
            counts[3 * b + 1] = 0;
            counts[3 * b + 2] = 0;
        }
        return;
    }
    const float* h = H + t0;
    const float* s = S + t0;
    // TopX: the keys at or above the (T - k + 1)-th smallest key_top; BotX: at or below
    // the k-th smallest key_bot
    const uint64_t top_h = select_rank<true>(h, T, T - k + 1, hist, sh);
    const uint64_t bot_h = select_rank<false>(h, T, k, hist, sh);
    const uint64_t top_s = select_rank<true>(s, T, T - k + 1, hist, sh);
    const uint64_t bot_s = select_rank<false>(s, T, k, hist, sh);
    if (threadIdx.x == 0) n_hl = n_lh = 0;
    __syncthreads();
    int hl = 0, lh = 0;
    for (int i = threadIdx.x; i < T; i += blockDim.x) {
        const bool th = key_top(h[i], i) >= top_h, bh = key_bot(h[i], i) <= bot_h;
        const bool ts = key_top(s[i], i) >= top_s, bs = key_bot(s[i], i) <= bot_s;
        hl += th && bs;
        lh += bh && ts;
    }
    atomicAdd(&n_hl, hl);
    atomicAdd(&n_lh, lh);
    __syncthreads();
    if (threadIdx.x == 0) {
        counts[3 * b] = k;
        counts[3 * b + 1] = n_hl;
        counts[3 * b + 2] = n_lh;
    }
}

}  // namespace

estp_status launch_misalignment(estp_ctx* ctx, const float* H, const float* S, const int32_t* cu,
                                int B, int64_t sumT, int pct, int32_t* counts, cudaStream_t st) {
    misalign_kernel<<<B, kThreads, 0, st>>>(H, S, cu, B, sumT, pct, counts, ctx->status);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "misalignment launch");
}

}  // namespace estp
