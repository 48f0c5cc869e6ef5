// Training loss of the length head (Sec. 3.3): the soft label of Eq. 3-1, the linear
// head of Eq. 3-2 and the loss of Eq. 3-3 averaged over the prompts, with its gradients.
//
// head_fwd_kernel: CTA b forms z = W h_b + bias (warp w takes logits k = w, w + 8, ...:
//   lanes stride the D columns, then a fixed butterfly), p_hat = softmax(z),
//   y_hat = sum p_hat_k c_k (relative to the centre of the largest logit), the soft
//   label around the bin nearest to y_b, the prompt's CE and squared error, and dL/dz_b
//   (with the batch mean's 1/B).
// head_grad_kernel: one thread per output element of dL/dW = sum_b dz_b h_b^T,
//   dL/dbias = sum_b dz_b and dL/dpooled_b = W^T dz_b, each summed in a fixed order,
//   and the loss itself.  Everything is fp32.
#include "estp_internal.cuh"

namespace estp {
namespace {

constexpr int kFwdThreads = 256;
constexpr int kMaxK = 1024;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    return v;
}

__global__ void __launch_bounds__(kFwdThreads) head_fwd_kernel(
    const float* __restrict__ pooled, int64_t D, const float* __restrict__ W,
    const float* __restrict__ bias, const float* __restrict__ centers, int K,
    const float* __restrict__ targets, int B, float lambda3, float* __restrict__ dz,
    float2* __restrict__ part) {
    __shared__ float z_s[kMaxK];
    const int b = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    const float* h = pooled + (int64_t)b * D;
    for (int k = warp; k < K; k += nw) {
        const float* wk = W + (int64_t)k * D;
        float acc = 0.f;
        for (int64_t x = lane; x < D; x += 32) acc = fmaf(wk[x], h[x], acc);
        acc = warp_sum(acc);
        if (lane == 0) z_s[k] = acc + (bias ? bias[k] : 0.f);
    }
    __syncthreads();
    if (warp != 0) return;
    // softmax over the K bins, the expectation of Eq. 3-2, and the nearest bin of y_b.
    // y_hat is formed relative to the centre of the largest logit r: y_hat = c_r + dy with
    // dy = sum_k p_hat_k (c_k - c_r), so that c_k - y_hat = (c_k - c_r) - dy does not
    // cancel when p_hat is concentrated on r.
    const float y = targets[b];
    float m = -INFINITY;
    int r = 0;
    for (int k = lane; k < K; k += 32)
        if (z_s[k] > m) { m = z_s[k]; r = k; }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {  // (max, first index)
        const float om = __shfl_xor_sync(0xffffffffu, m, off);
        const int orr = __shfl_xor_sync(0xffffffffu, r, off);
        if (om > m || (om == m && orr < r)) { m = om; r = orr; }
    }
    const float cr = centers[r];
    float Z = 0.f, dy = 0.f;
    float best_d = INFINITY;
    int best_k = 0;
    for (int k = lane; k < K; k += 32) {
        const float e = __expf(z_s[k] - m);
        Z += e;
        dy = fmaf(e, centers[k] - cr, dy);
        const float d = fabsf(y - centers[k]);
        if (d < best_d) { best_d = d; best_k = k; }  // lowest k of this lane on a tie
    }
    Z = warp_sum(Z);
    dy = warp_sum(dy) / Z;
    const float yh = cr + dy;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {  // (distance, index): the lowest index wins ties
        const float od = __shfl_xor_sync(0xffffffffu, best_d, off);
        const int ok = __shfl_xor_sync(0xffffffffu, best_k, off);
        if (od < best_d || (od == best_d && ok < best_k)) { best_d = od; best_k = ok; }
    }
    const int i = best_k;
    float norm = 0.f;
    for (int k = lane; k < K; k += 32) norm += __expf(-fabsf((float)(k - i)));
    norm = warp_sum(norm);
    const float lnZ = __logf(Z), err = yh - y, inv_b = 1.f / (float)B;
    float ce = 0.f;
    for (int k = lane; k < K; k += 32) {
        const float p = __expf(-fabsf((float)(k - i))) / norm;
        const float lp_hat = z_s[k] - m - lnZ;  // ln p_hat_k
        const float p_hat = __expf(lp_hat);
        ce -= p * lp_hat;
        dz[(int64_t)b * K + k] =
            (lambda3 * (p_hat - p) + (1.f - lambda3) * 2.f * err * p_hat * ((centers[k] - cr) - dy)) * inv_b;
    }
    ce = warp_sum(ce);
    if (lane == 0) part[b] = make_float2(ce, err * err);
}

__global__ void head_grad_kernel(const float* __restrict__ pooled, int B, int64_t D,
                                 const float* __restrict__ W, int K, const float* __restrict__ dz,
                                 const float2* __restrict__ part, float lambda3,
                                 float* __restrict__ loss, float* __restrict__ grad_W,
                                 float* __restrict__ grad_bias, float* __restrict__ grad_pooled) {
    const int64_t n_w = grad_W ? (int64_t)K * D : 0;
    const int64_t n_b = grad_bias ? K : 0;
    const int64_t n_p = grad_pooled ? (int64_t)B * D : 0;
    const int64_t total = n_w + n_b + n_p + 1;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        if (t < n_w) {  // dL/dW[k, x] = sum_b dz[b, k] h[b, x]
            const int k = (int)(t / D);
            const int64_t x = t - (int64_t)k * D;
            float g = 0.f;
            for (int b = 0; b < B; ++b) g = fmaf(dz[(int64_t)b * K + k], pooled[(int64_t)b * D + x], g);
            grad_W[t] = g;
        } else if (t < n_w + n_b) {  // dL/dbias[k] = sum_b dz[b, k]
            const int k = (int)(t - n_w);
            float g = 0.f;
            for (int b = 0; b < B; ++b) g += dz[(int64_t)b * K + k];
            grad_bias[k] = g;
        } else if (t < n_w + n_b + n_p) {  // dL/dpooled[b, x] = sum_k W[k, x] dz[b, k]
            const int64_t r = t - n_w - n_b;
            const int b = (int)(r / D);
            const int64_t x = r - (int64_t)b * D;
            float g = 0.f;
            for (int k = 0; k < K; ++k) g = fmaf(W[(int64_t)k * D + x], dz[(int64_t)b * K + k], g);
            grad_pooled[r] = g;
        } else {  // the loss: batch means of the CE and squared-error terms
            float ce = 0.f, se = 0.f;
            for (int b = 0; b < B; ++b) {
                ce += part[b].x;
                se += part[b].y;
            }
            loss[0] = (lambda3 * ce + (1.f - lambda3) * se) / (float)B;
        }
    }
}

}  // namespace

estp_status launch_head_loss(estp_ctx* ctx, const float* pooled, int B, int64_t D,
                             const estp_head& head, const float* targets, float lambda3,
                             float* loss, float* grad_W, float* grad_bias, float* grad_pooled,
                             cudaStream_t st) {
    const int K = head.K;
    const size_t off_part = align_up(sizeof(float) * (size_t)B * K, 256);
    estp_status s = ws_reserve(ctx, off_part + sizeof(float2) * (size_t)B);
    if (s != ESTP_OK) return s;
    char* ws = static_cast<char*>(ctx->ws);
    float* dz = reinterpret_cast<float*>(ws);
    float2* part = reinterpret_cast<float2*>(ws + off_part);
    head_fwd_kernel<<<B, kFwdThreads, 0, st>>>(pooled, D, head.W, head.bias, head.centers, K,
                                               targets, B, lambda3, dz, part);
    const int64_t total = (grad_W ? (int64_t)K * D : 0) + (grad_bias ? K : 0) +
                          (grad_pooled ? (int64_t)B * D : 0) + 1;
    const int blocks = (int)((total + 255) / 256 < 4 * (int64_t)ctx->num_sms ? (total + 255) / 256
                                                                           : 4 * (int64_t)ctx->num_sms);
    head_grad_kernel<<<blocks, 256, 0, st>>>(pooled, B, D, head.W, K, dz, part, lambda3, loss,
                                             grad_W, grad_bias, grad_pooled);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "head loss launch");
}

}  // namespace estp
