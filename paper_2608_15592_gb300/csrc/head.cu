// Training loss of the length head (Sec. 3.3): the soft label of Eq. 3-1, the linear
// head of Eq. 3-2 and the loss of Eq. 3-3 averaged over the prompts, with its gradients;
// and the MLP predictor of Sec. 3.3 / Fig. 2 (one hidden layer of F ReLU units in front
// of the K-bin softmax projection), its prediction and its loss.
//
// head_fwd_kernel: CTA b forms z = W h_b + bias (warp w takes logits k = w, w + 8, ...:
//   lanes stride the D columns, then a fixed butterfly), p_hat = softmax(z),
//   y_hat = sum p_hat_k c_k (relative to the centre of the largest logit), the soft
//   label around the bin nearest to y_b, the prompt's CE and squared error, and dL/dz_b
//   (with the batch mean's 1/B).
// head_grad_kernel: one thread per output element of dL/dW = sum_b dz_b h_b^T,
//   dL/dbias = sum_b dz_b and dL/dpooled_b = W^T dz_b, each summed in a fixed order,
//   and the loss itself.  Everything is fp32.
// mlp_hidden_kernel: u = max(W1 h + b1, 0), one warp per hidden unit and 8 prompts at a
//   time (lanes stride D, then a fixed butterfly).  The MLP reuses the two kernels above
//   layer by layer: head_fwd_kernel and head_grad_kernel on u with W2 (dL/dW2, dL/db2,
//   dL/du and the loss), then head_grad_kernel on h with W1, gated by u > 0 (the ReLU's
//   derivative), for dL/dW1, dL/db1 and dL/dh.
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
    float2* __restrict__ part, float* __restrict__ pred, float* __restrict__ probs) {
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
    for (int k = lane; k < K; k += 32) {
        const float e = __expf(z_s[k] - m);
        Z += e;
        dy = fmaf(e, centers[k] - cr, dy);
    }
    Z = warp_sum(Z);
    dy = warp_sum(dy) / Z;
    const float yh = cr + dy;
    if (pred && lane == 0) pred[b] = yh;
    if (probs)
        for (int k = lane; k < K; k += 32) probs[(int64_t)b * K + k] = __expf(z_s[k] - m) / Z;
    if (!targets) return;  // prediction only
    const float y = targets[b];
    float best_d = INFINITY;
    int best_k = 0;
    for (int k = lane; k < K; k += 32) {
        const float d = fabsf(y - centers[k]);
        if (d < best_d) { best_d = d; best_k = k; }  // lowest k of this lane on a tie
    }
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

// gate (NULL: none): dz[b, k] counts only where gate[b, k] > 0 (a ReLU's derivative);
// loss NULL: no loss element.
__global__ void head_grad_kernel(const float* __restrict__ pooled, int B, int64_t D,
                                 const float* __restrict__ W, int K, const float* __restrict__ dz,
                                 const float* __restrict__ gate, const float2* __restrict__ part,
                                 float lambda3, float* __restrict__ loss, float* __restrict__ grad_W,
                                 float* __restrict__ grad_bias, float* __restrict__ grad_pooled) {
    const int64_t n_w = grad_W ? (int64_t)K * D : 0;
    const int64_t n_b = grad_bias ? K : 0;
    const int64_t n_p = grad_pooled ? (int64_t)B * D : 0;
    const int64_t total = n_w + n_b + n_p + (loss ? 1 : 0);
    auto dzg = [&](int b, int k) -> float {
        const float v = dz[(int64_t)b * K + k];
        return gate && !(gate[(int64_t)b * K + k] > 0.f) ? 0.f : v;
    };
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        if (t < n_w) {  // dL/dW[k, x] = sum_b dz[b, k] h[b, x]
            const int k = (int)(t / D);
            const int64_t x = t - (int64_t)k * D;
            float acc = 0.f;
            for (int b = 0; b < B; ++b) acc = fmaf(dzg(b, k), pooled[(int64_t)b * D + x], acc);
            grad_W[t] = acc;
        } else if (t < n_w + n_b) {  // dL/dbias[k] = sum_b dz[b, k]
            const int k = (int)(t - n_w);
            float acc = 0.f;
            for (int b = 0; b < B; ++b) acc += dzg(b, k);
            grad_bias[k] = acc;
        } else if (t < n_w + n_b + n_p) {  // dL/dpooled[b, x] = sum_k W[k, x] dz[b, k]
            const int64_t r = t - n_w - n_b;
            const int b = (int)(r / D);
            const int64_t x = r - (int64_t)b * D;
            float acc = 0.f;
            for (int k = 0; k < K; ++k) acc = fmaf(W[(int64_t)k * D + x], dzg(b, k), acc);
            grad_pooled[r] = acc;
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

constexpr int kHidB = 16;  // prompts per warp pass of the hidden layer
constexpr int kDhB = 4;    // prompts per block of the input gradient

// Four consecutive floats of a row at column x (a 16-byte load when vec, else scalar
// loads, zero past D).
__device__ __forceinline__ float4 ld4(const float* __restrict__ row, int64_t x, int64_t D, bool vec) {
    if (vec) return __ldg(reinterpret_cast<const float4*>(row + x));
    return make_float4(x < D ? __ldg(row + x) : 0.f, x + 1 < D ? __ldg(row + x + 1) : 0.f,
                       x + 2 < D ? __ldg(row + x + 2) : 0.f, x + 3 < D ? __ldg(row + x + 3) : 0.f);
}

// u[b, f] = max(sum_x W1[f, x] h[b, x] + b1[f], 0): one warp per hidden unit f, lanes
// stride D four columns at a time, kHidB prompts per pass, then a fixed butterfly.
__global__ void __launch_bounds__(128) mlp_hidden_kernel(const float* __restrict__ pooled, int B,
                                                         int64_t D, const float* __restrict__ W1,
                                                         const float* __restrict__ b1, int F,
                                                         float* __restrict__ u, int vec) {
    const int lane = threadIdx.x & 31;
    const int64_t f = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (f >= F) return;
    const float* w = W1 + f * D;
    const float bias = b1 ? b1[f] : 0.f;
    for (int b0 = 0; b0 < B; b0 += kHidB) {
        const int nb = B - b0 < kHidB ? B - b0 : kHidB;
        float acc[kHidB];
#pragma unroll
        for (int j = 0; j < kHidB; ++j) acc[j] = 0.f;
        for (int64_t x = 4 * lane; x < D; x += 128) {
            // every load of the pass first (rows past B repeat the last row, unused), then the FMAs
            const float4 wv = ld4(w, x, D, vec);
            float4 hv[kHidB];
#pragma unroll
            for (int j = 0; j < kHidB; ++j)
                hv[j] = ld4(pooled + (int64_t)(b0 + (j < nb ? j : nb - 1)) * D, x, D, vec);
#pragma unroll
            for (int j = 0; j < kHidB; ++j)
                acc[j] = fmaf(wv.x, hv[j].x, fmaf(wv.y, hv[j].y, fmaf(wv.z, hv[j].z, fmaf(wv.w, hv[j].w, acc[j]))));
        }
#pragma unroll
        for (int j = 0; j < kHidB; ++j) {
            const float a = warp_sum(acc[j]) + bias;
            if (lane == 0 && j < nb) u[(int64_t)(b0 + j) * F + f] = a > 0.f ? a : 0.f;
        }
    }
}

// dL/dh[b, x] = sum_f W1[f, x] g[b, f], g = dL/du where u > 0 (the ReLU's derivative), else 0.
// Block (128 columns, kDhB prompts): g of the block's prompts is staged in shared memory
// (dynamic, kDhB x F floats); warp w takes f = w, w + 8, ... (four W1 rows in flight);
// the 8 warp partials are added in warp order.
__global__ void __launch_bounds__(256) mlp_dh_kernel(const float* __restrict__ W1, int64_t D, int F,
                                                     const float* __restrict__ du,
                                                     const float* __restrict__ u, int B,
                                                     float* __restrict__ dh, int vec) {
    extern __shared__ float g_s[];  // [kDhB][F]
    __shared__ float4 red[8][kDhB][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t x = (int64_t)blockIdx.x * 128 + 4 * lane;
    const int b0 = blockIdx.y * kDhB;
    const int nb = B - b0 < kDhB ? B - b0 : kDhB;
    for (int q = threadIdx.x; q < kDhB * F; q += blockDim.x) {
        const int j = q / F, f = q - j * F;
        float gv = 0.f;
        if (j < nb) {
            const int64_t i = (int64_t)(b0 + j) * F + f;
            gv = u[i] > 0.f ? du[i] : 0.f;
        }
        g_s[q] = gv;
    }
    __syncthreads();
    float4 acc[kDhB];
#pragma unroll
    for (int j = 0; j < kDhB; ++j) acc[j] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (x < D) {
        int f = warp;
        for (; f + 24 < F; f += 32) {  // four rows f, f + 8, f + 16, f + 24 in flight
            float4 wv[4];
#pragma unroll
            for (int r = 0; r < 4; ++r) wv[r] = ld4(W1 + (int64_t)(f + 8 * r) * D, x, D, vec);
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int j = 0; j < kDhB; ++j) {
                    const float gv = g_s[j * F + f + 8 * r];
                    acc[j].x = fmaf(gv, wv[r].x, acc[j].x);
                    acc[j].y = fmaf(gv, wv[r].y, acc[j].y);
                    acc[j].z = fmaf(gv, wv[r].z, acc[j].z);
                    acc[j].w = fmaf(gv, wv[r].w, acc[j].w);
                }
        }
        for (; f < F; f += 8) {
            const float4 wv = ld4(W1 + (int64_t)f * D, x, D, vec);
#pragma unroll
            for (int j = 0; j < kDhB; ++j) {
                const float gv = g_s[j * F + f];
                acc[j].x = fmaf(gv, wv.x, acc[j].x);
                acc[j].y = fmaf(gv, wv.y, acc[j].y);
                acc[j].z = fmaf(gv, wv.z, acc[j].z);
                acc[j].w = fmaf(gv, wv.w, acc[j].w);
            }
        }
    }
#pragma unroll
    for (int j = 0; j < kDhB; ++j) red[warp][j][lane] = acc[j];
    __syncthreads();
    if (warp == 0 && x < D) {
        for (int j = 0; j < nb; ++j) {
            float4 t = red[0][j][lane];
            for (int w = 1; w < 8; ++w) {
                const float4 o = red[w][j][lane];
                t.x += o.x;
                t.y += o.y;
                t.z += o.z;
                t.w += o.w;
            }
            float* out = dh + (int64_t)(b0 + j) * D + x;
            out[0] = t.x;
            if (x + 1 < D) out[1] = t.y;
            if (x + 2 < D) out[2] = t.z;
            if (x + 3 < D) out[3] = t.w;
        }
    }
}

// dL/dW1[f, x] = sum_b g[b, f] h[b, x] and dL/db1[f] = sum_b g[b, f], g = dL/du where u > 0:
// thread (f, four columns x) sums the prompts in order; the threads with x = 0 also write
// dL/db1[f].  Either output may be NULL.
__global__ void __launch_bounds__(256) mlp_dw1_kernel(const float* __restrict__ pooled, int B,
                                                      int64_t D, int F, const float* __restrict__ du,
                                                      const float* __restrict__ u,
                                                      float* __restrict__ gW1,
                                                      float* __restrict__ gb1, int vec) {
    const int64_t per_row = (D + 3) / 4;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= (int64_t)F * per_row) return;
    const int f = (int)(t / per_row);
    const int64_t x = 4 * (t - (int64_t)f * per_row);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    float gs = 0.f;
    for (int b = 0; b < B; ++b) {
        const int64_t i = (int64_t)b * F + f;
        const float gv = u[i] > 0.f ? du[i] : 0.f;
        gs += gv;
        if (gW1) {
            const float4 hv = ld4(pooled + (int64_t)b * D, x, D, vec);
            acc.x = fmaf(gv, hv.x, acc.x);
            acc.y = fmaf(gv, hv.y, acc.y);
            acc.z = fmaf(gv, hv.z, acc.z);
            acc.w = fmaf(gv, hv.w, acc.w);
        }
    }
    if (gb1 && x == 0) gb1[f] = gs;
    if (!gW1) return;
    float* out = gW1 + (int64_t)f * D + x;
    if (vec) {
        *reinterpret_cast<float4*>(out) = acc;
    } else {
        out[0] = acc.x;
        if (x + 1 < D) out[1] = acc.y;
        if (x + 2 < D) out[2] = acc.z;
        if (x + 3 < D) out[3] = acc.w;
    }
}

int grad_blocks(estp_ctx* ctx, int64_t total) {
    const int64_t b = (total + 255) / 256, cap = 4 * (int64_t)ctx->num_sms;
    return (int)(b < cap ? (b > 0 ? b : 1) : cap);
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
                                               targets, B, lambda3, dz, part, nullptr, nullptr);
    const int64_t total = (grad_W ? (int64_t)K * D : 0) + (grad_bias ? K : 0) +
                          (grad_pooled ? (int64_t)B * D : 0) + 1;
    head_grad_kernel<<<grad_blocks(ctx, total), 256, 0, st>>>(pooled, B, D, head.W, K, dz, nullptr,
                                                              part, lambda3, loss, grad_W, grad_bias,
                                                              grad_pooled);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "head loss launch");
}

// The MLP's hidden units u [B, F] into the workspace at `u`.
static bool vec4(const float* a, const float* b, int64_t D) {
    return D % 4 == 0 && aligned16(a) && aligned16(b);
}

static cudaError_t mlp_hidden(estp_ctx* ctx, const float* pooled, int B, int64_t D,
                              const estp_mlp_head& head, float* u, cudaStream_t st) {
    const int64_t threads = 32 * (int64_t)head.F;
    mlp_hidden_kernel<<<(unsigned)((threads + 127) / 128), 128, 0, st>>>(
        pooled, B, D, head.W1, head.b1, head.F, u, vec4(pooled, head.W1, D) ? 1 : 0);
    return cudaGetLastError();
}

estp_status launch_mlp_head_predict(estp_ctx* ctx, const float* pooled, int B, int64_t D,
                                    const estp_mlp_head& head, float* pred, float* probs,
                                    cudaStream_t st) {
    estp_status s = ws_reserve(ctx, sizeof(float) * (size_t)B * head.F);
    if (s != ESTP_OK) return s;
    float* u = static_cast<float*>(ctx->ws);
    cudaError_t e = mlp_hidden(ctx, pooled, B, D, head, u, st);
    if (e != cudaSuccess) return cuda_fail(e, "mlp hidden launch");
    head_fwd_kernel<<<B, kFwdThreads, 0, st>>>(u, head.F, head.W2, head.b2, head.centers, head.K,
                                               nullptr, B, 0.f, nullptr, nullptr, pred, probs);
    e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "mlp head launch");
}

estp_status launch_mlp_head_loss(estp_ctx* ctx, const float* pooled, int B, int64_t D,
                                 const estp_mlp_head& head, const float* targets, float lambda3,
                                 float* loss, const estp_mlp_grads& g, cudaStream_t st) {
    const int F = head.F, K = head.K;
    // workspace: u [B, F] | du [B, F] | dz [B, K] | part [B]
    const size_t off_du = align_up(sizeof(float) * (size_t)B * F, 256);
    const size_t off_dz = off_du + align_up(sizeof(float) * (size_t)B * F, 256);
    const size_t off_part = off_dz + align_up(sizeof(float) * (size_t)B * K, 256);
    estp_status s = ws_reserve(ctx, off_part + sizeof(float2) * (size_t)B);
    if (s != ESTP_OK) return s;
    char* ws = static_cast<char*>(ctx->ws);
    float* u = reinterpret_cast<float*>(ws);
    float* du = reinterpret_cast<float*>(ws + off_du);
    float* dz = reinterpret_cast<float*>(ws + off_dz);
    float2* part = reinterpret_cast<float2*>(ws + off_part);
    const bool lower = g.W1 || g.b1 || g.pooled;  // gradients below the hidden layer
    cudaError_t e = mlp_hidden(ctx, pooled, B, D, head, u, st);
    if (e != cudaSuccess) return cuda_fail(e, "mlp hidden launch");
    head_fwd_kernel<<<B, kFwdThreads, 0, st>>>(u, F, head.W2, head.b2, head.centers, K, targets, B,
                                               lambda3, dz, part, nullptr, nullptr);
    // second layer: dL/dW2, dL/db2, dL/du and the loss
    int64_t total = (g.W2 ? (int64_t)K * F : 0) + (g.b2 ? K : 0) + (lower ? (int64_t)B * F : 0) + 1;
    head_grad_kernel<<<grad_blocks(ctx, total), 256, 0, st>>>(u, B, F, head.W2, K, dz, nullptr, part,
                                                              lambda3, loss, g.W2, g.b2,
                                                              lower ? du : nullptr);
    if (g.W1 || g.b1) {  // first layer, through the ReLU (u > 0): dL/dW1, dL/db1
        const int64_t threads = (int64_t)F * ((D + 3) / 4);
        mlp_dw1_kernel<<<(unsigned)((threads + 255) / 256), 256, 0, st>>>(
            pooled, B, D, F, du, u, g.W1, g.b1, vec4(pooled, g.W1 ? g.W1 : pooled, D) ? 1 : 0);
    }
    const size_t smem = sizeof(float) * kDhB * (size_t)F;
    if (g.pooled && smem > 200 * 1024) {  // very wide hidden layer: the general kernel
        total = (int64_t)B * D;
        head_grad_kernel<<<grad_blocks(ctx, total), 256, 0, st>>>(pooled, B, D, head.W1, F, du, u,
                                                                  nullptr, 0.f, nullptr, nullptr,
                                                                  nullptr, g.pooled);
    } else if (g.pooled) {  // dL/dpooled = W1^T (dL/du where u > 0)
        const dim3 grid((unsigned)((D + 127) / 128), (unsigned)((B + kDhB - 1) / kDhB));
        if (smem > 48 * 1024) {
            e = cudaFuncSetAttribute(mlp_dh_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return cuda_fail(e, "mlp input-gradient smem attribute");
        }
        mlp_dh_kernel<<<grid, 256, smem, st>>>(head.W1, D, F, du, u, B, g.pooled,
                                               vec4(head.W1, head.W1, D) ? 1 : 0);
    }
    e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "mlp head loss launch");
}

}  // namespace estp
