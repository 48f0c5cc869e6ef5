// C ABI of the ESTP library: contexts, argument validation and dispatch.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>

#include "estp_internal.cuh"
#include "tcgen05.cuh"

namespace estp {

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
        return (PFN_cuTensorMapEncodeTiled_v12000) nullptr;
    }();
    return fn;
}

static thread_local char g_msg[512] = "no error";

estp_status fail(estp_status st, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof g_msg, fmt, ap);
    va_end(ap);
    return st;
}

estp_status cuda_fail(cudaError_t e, const char* what) {
    return fail(ESTP_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

estp_status set_device(estp_ctx* ctx) {
    cudaError_t e = cudaSetDevice(ctx->device);
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "cudaSetDevice");
}

// Grows the workspace to at least `bytes`.  cudaFree waits for the device, so work
// already enqueued on the old buffer finishes before it is released.
estp_status ws_reserve(estp_ctx* ctx, size_t bytes) {
    if (bytes <= ctx->ws_bytes) return ESTP_OK;
    size_t want = align_up(bytes + bytes / 4, size_t(1) << 20);
    if (ctx->ws) cudaFree(ctx->ws);
    ctx->ws = nullptr;
    ctx->ws_bytes = 0;
    cudaError_t e = cudaMalloc(&ctx->ws, want);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(ESTP_ERR_WORKSPACE, "workspace of %zu bytes: %s", want, cudaGetErrorString(e));
    }
    ctx->ws_bytes = want;
    return ESTP_OK;
}

estp_status build_heads(const int32_t* heads, int n_heads, int Hq, int Hkv, ImpHeads* out) {
    int rep = Hq / Hkv;
    int list[256];
    if (!heads) {
        n_heads = Hq;
        for (int h = 0; h < Hq; ++h) list[h] = h;
    } else {
        if (n_heads <= 0 || n_heads > 256)
            return fail(ESTP_ERR_INVALID_ARG, "n_heads=%d must be in 1..256", n_heads);
        for (int s = 0; s < n_heads; ++s) {
            if (heads[s] < 0 || heads[s] >= Hq)
                return fail(ESTP_ERR_INVALID_ARG, "heads[%d]=%d outside [0, %d)", s, heads[s], Hq);
            list[s] = heads[s];
        }
    }
    out->n_heads = n_heads;
    out->n_groups = 0;
    int pos = 0;
    for (int g = 0; g < Hkv; ++g) {
        int start = pos;
        for (int s = 0; s < n_heads; ++s)
            if (list[s] / rep == g) out->head_list[pos++] = (int16_t)list[s];
        if (pos > start) {
            out->group[out->n_groups] = (int16_t)g;
            out->begin[out->n_groups] = (int16_t)start;
            out->n_groups++;
        }
    }
    out->begin[out->n_groups] = (int16_t)pos;
    return ESTP_OK;
}

}  // namespace estp

using namespace estp;

extern "C" {

estp_status estp_create(estp_ctx** out, int device) {
    if (!out) return fail(ESTP_ERR_INVALID_ARG, "ctx out-pointer is NULL");
    *out = nullptr;
    int n = 0;
    cudaError_t e = cudaGetDeviceCount(&n);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDeviceCount");
    if (device < 0 || device >= n)
        return fail(ESTP_ERR_INVALID_ARG, "device %d outside [0, %d)", device, n);
    estp_ctx* ctx = new (std::nothrow) estp_ctx();
    if (!ctx) return fail(ESTP_ERR_WORKSPACE, "out of host memory");
    ctx->device = device;
    estp_status st = set_device(ctx);
    if (st != ESTP_OK) { delete ctx; return st; }
    e = cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) { delete ctx; return cuda_fail(e, "cudaDeviceGetAttribute"); }
    e = cudaMalloc(&ctx->status, sizeof(int));
    if (e == cudaSuccess) e = cudaMemset(ctx->status, 0, sizeof(int));
    if (e != cudaSuccess) { cudaFree(ctx->status); delete ctx; return cuda_fail(e, "status word"); }
    *out = ctx;
    return ESTP_OK;
}

void estp_destroy(estp_ctx* ctx) {
    if (!ctx) return;
    cudaSetDevice(ctx->device);
    cudaDeviceSynchronize();
    cudaFree(ctx->ws);
    cudaFree(ctx->imp_acc);
    cudaFree(ctx->pool_done);
    cudaFree(ctx->status);
    delete ctx;
}

const char* estp_last_error(const estp_ctx*) { return g_msg; }

estp_status estp_set_wait_limit(estp_ctx* ctx, int64_t cycles) {
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    ctx->wait_cycles = cycles > 0 ? (long long)cycles : kWaitCycles;
    return ESTP_OK;
}

estp_status estp_sync_status(estp_ctx* ctx, estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_sync_status");
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    estp_status st = set_device(ctx);
    if (st != ESTP_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    int code = 0;
    e = cudaMemcpyAsync(&code, ctx->status, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(ctx->status, 0, sizeof(int), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "reading the status word");
    switch (code) {
        case ESTP_OK: return ESTP_OK;
        case ESTP_ERR_INVALID_ARG:
            return fail(ESTP_ERR_INVALID_ARG, "device check failed: cu_seqlens or max_seqlen");
        case ESTP_ERR_TIMEOUT: return fail(ESTP_ERR_TIMEOUT, "a device-side wait timed out");
        default: return fail((estp_status)code, "device status %d", code);
    }
}

estp_status estp_token_entropy(estp_ctx* ctx, const void* logits, estp_dtype dtype,
                               int64_t n_rows, int64_t V, int64_t ld,
                               const int32_t* cu_seqlens, int32_t B, float* entropy_out,
                               estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_token_entropy");
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    if (dtype != ESTP_F32 && dtype != ESTP_BF16) return fail(ESTP_ERR_INVALID_ARG, "dtype");
    if (n_rows < 0 || V < 1 || ld < V)
        return fail(ESTP_ERR_INVALID_ARG, "need n_rows >= 0, V >= 1, ld >= V");
    if (cu_seqlens && B < 0) return fail(ESTP_ERR_INVALID_ARG, "B < 0");
    if (n_rows == 0) return ESTP_OK;
    if (!logits || !entropy_out) return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    if (!aligned16(logits) || (ld * esize(dtype)) % 16)
        return fail(ESTP_ERR_INVALID_ARG, "logits base and row stride must be 16-byte aligned");
    estp_status st = set_device(ctx);
    if (st != ESTP_OK) return st;
    return launch_entropy(ctx, logits, dtype, n_rows, V, ld, cu_seqlens, B, entropy_out,
                          reinterpret_cast<cudaStream_t>(stream));
}

static estp_status check_attn(estp_ctx* ctx, const void* Q, const void* K, estp_dtype dtype,
                              int32_t Hq, int32_t Hkv, int32_t head_dim, float scale,
                              const int32_t* cu, int32_t B, int64_t sumT, int32_t max_seqlen) {
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    if (dtype != ESTP_F32 && dtype != ESTP_BF16) return fail(ESTP_ERR_INVALID_ARG, "dtype");
    if (Hq < 1 || Hkv < 1 || Hq > 256 || Hq % Hkv)
        return fail(ESTP_ERR_INVALID_ARG, "need 1 <= Hkv, Hq <= 256, Hq %% Hkv == 0");
    if (head_dim != 64 && head_dim != 128)
        return fail(ESTP_ERR_UNSUPPORTED, "head_dim %d (64 or 128 supported)", head_dim);
    if (!(scale > 0.f) || !std::isfinite(scale))
        return fail(ESTP_ERR_INVALID_ARG, "softmax_scale must be finite and > 0");
    if (B < 0 || sumT < 0 || max_seqlen < 0 || (int64_t)max_seqlen > sumT)
        return fail(ESTP_ERR_INVALID_ARG, "need B, sumT >= 0 and 0 <= max_seqlen <= sumT");
    if (sumT > INT32_MAX) return fail(ESTP_ERR_INVALID_ARG, "sumT exceeds int32");
    if (B > 0 && !cu) return fail(ESTP_ERR_INVALID_ARG, "cu_seqlens is NULL");
    if (sumT > 0 && (!Q || !K)) return fail(ESTP_ERR_INVALID_ARG, "NULL Q or K");
    if (sumT > 0 && (!aligned16(Q) || !aligned16(K)))
        return fail(ESTP_ERR_INVALID_ARG, "Q and K must be 16-byte aligned");
    return ESTP_OK;
}

estp_status estp_attn_lse(estp_ctx* ctx, const void* Q, const void* K, estp_dtype dtype,
                          int32_t Hq, int32_t Hkv, int32_t head_dim, float softmax_scale,
                          const int32_t* cu_seqlens, int32_t B, int64_t sumT,
                          int32_t max_seqlen, float* lse_out, estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_attn_lse");
    estp_status st = check_attn(ctx, Q, K, dtype, Hq, Hkv, head_dim, softmax_scale, cu_seqlens,
                                B, sumT, max_seqlen);
    if (st != ESTP_OK) return st;
    if (sumT == 0 || B == 0) return ESTP_OK;
    if (!lse_out) return fail(ESTP_ERR_INVALID_ARG, "lse_out is NULL");
    ImpHeads hs;
    st = build_heads(nullptr, Hq, Hq, Hkv, &hs);
    if (st == ESTP_OK) st = set_device(ctx);
    if (st != ESTP_OK) return st;
    return launch_lse(ctx, Q, K, dtype, Hq, Hkv, head_dim, softmax_scale, hs, cu_seqlens, B,
                      sumT, max_seqlen, lse_out, reinterpret_cast<cudaStream_t>(stream));
}

// Opens (accumulate = 0) or continues (accumulate = 1) the context's importance
// accumulation over n_heads heads; checks the flags and the lse alignment, sets the device
// and sizes the accumulator.
static estp_status open_importance(estp_ctx* ctx, const float* lse, int n_heads,
                                   const int32_t* cu_seqlens, int32_t B, int64_t sumT,
                                   int accumulate, uint32_t flags) {
    constexpr uint32_t kDiv = ESTP_IMP_DIV_CAUSAL | ESTP_IMP_DIV_NONE;
    if (flags & ~(ESTP_IMP_EXCLUDE_SELF | kDiv)) return fail(ESTP_ERR_INVALID_ARG, "unknown flags");
    if ((flags & kDiv) == kDiv)
        return fail(ESTP_ERR_INVALID_ARG, "ESTP_IMP_DIV_CAUSAL and ESTP_IMP_DIV_NONE together");
    estp_status st;
    if (accumulate) {
        if (!ctx->imp_open)
            return fail(ESTP_ERR_INVALID_ARG, "accumulate=1 without an open accumulation");
        if (ctx->imp_sumT != sumT || ctx->imp_B != B || ctx->imp_cu != cu_seqlens ||
            ctx->imp_n_heads != n_heads)
            return fail(ESTP_ERR_INVALID_ARG,
                        "accumulate=1 with different cu_seqlens/B/sumT/head count");
        // the finalize divisor is fixed when the accumulation opens; the causal count
        // also depends on whether the self term is summed
        const uint32_t fixed = (ctx->imp_flags & ESTP_IMP_DIV_CAUSAL) ? (kDiv | ESTP_IMP_EXCLUDE_SELF) : kDiv;
        if ((flags & fixed) != (ctx->imp_flags & fixed))
            return fail(ESTP_ERR_INVALID_ARG,
                        "accumulate=1 with divisor flags that differ from the opening call");
    }
    if (lse && !aligned16(lse)) return fail(ESTP_ERR_INVALID_ARG, "lse must be 16-byte aligned");
    st = set_device(ctx);
    if (st != ESTP_OK) return st;
    if (ctx->imp_cap < sumT) {
        cudaFree(ctx->imp_acc);
        ctx->imp_acc = nullptr;
        ctx->imp_cap = 0;
        ctx->imp_open = false;
        if (accumulate) return fail(ESTP_ERR_INVALID_ARG, "accumulator lost");
        cudaError_t e = cudaMalloc(&ctx->imp_acc, sizeof(float) * (size_t)(sumT > 0 ? sumT : 1));
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(ESTP_ERR_WORKSPACE, "importance accumulator: %s", cudaGetErrorString(e));
        }
        ctx->imp_cap = sumT > 0 ? sumT : 1;
    }
    ctx->imp_open = true;
    ctx->imp_sumT = sumT;
    ctx->imp_B = B;
    ctx->imp_cu = cu_seqlens;
    ctx->imp_n_heads = n_heads;
    if (!accumulate) ctx->imp_flags = flags;
    return ESTP_OK;
}

estp_status estp_attn_importance(estp_ctx* ctx, const void* Q, const void* K,
                                 estp_dtype dtype, const float* lse, int32_t Hq, int32_t Hkv,
                                 int32_t head_dim, float softmax_scale, const int32_t* heads,
                                 int32_t n_heads, const int32_t* cu_seqlens, int32_t B,
                                 int64_t sumT, int32_t max_seqlen, int accumulate,
                                 uint32_t flags, estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_attn_importance");
    estp_status st = check_attn(ctx, Q, K, dtype, Hq, Hkv, head_dim, softmax_scale, cu_seqlens,
                                B, sumT, max_seqlen);
    if (st != ESTP_OK) return st;
    ImpHeads hs;
    st = build_heads(heads, n_heads, Hq, Hkv, &hs);
    if (st != ESTP_OK) return st;
    st = open_importance(ctx, lse, hs.n_heads, cu_seqlens, B, sumT, accumulate, flags);
    if (st != ESTP_OK) return st;
    if (sumT == 0 || B == 0) return ESTP_OK;
    return launch_importance(ctx, Q, K, dtype, lse, Hq, Hkv, head_dim, softmax_scale, hs,
                             cu_seqlens, B, sumT, max_seqlen, accumulate != 0, flags,
                             ctx->imp_acc, reinterpret_cast<cudaStream_t>(stream));
}

estp_status estp_attn_forward_importance(estp_ctx* ctx, const void* Q, const void* K,
                                         const void* V, estp_dtype dtype, const float* lse,
                                         int32_t Hq, int32_t Hkv, int32_t head_dim,
                                         float softmax_scale, const int32_t* cu_seqlens,
                                         int32_t B, int64_t sumT, int32_t max_seqlen,
                                         int accumulate, uint32_t flags, void* out,
                                         estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_attn_forward_importance");
    estp_status st = check_attn(ctx, Q, K, dtype, Hq, Hkv, head_dim, softmax_scale, cu_seqlens,
                                B, sumT, max_seqlen);
    if (st != ESTP_OK) return st;
    if (dtype != ESTP_BF16) return fail(ESTP_ERR_UNSUPPORTED, "attention forward: bf16 only");
    if (head_dim != 128) return fail(ESTP_ERR_UNSUPPORTED, "attention forward: head_dim 128 only");
    if (sumT > 0 && (!V || !out)) return fail(ESTP_ERR_INVALID_ARG, "NULL V or out");
    if (sumT > 0 && (!aligned16(V) || !aligned16(out)))
        return fail(ESTP_ERR_INVALID_ARG, "V and out must be 16-byte aligned");
    st = open_importance(ctx, lse, Hq, cu_seqlens, B, sumT, accumulate, flags);
    if (st != ESTP_OK) return st;
    if (sumT == 0 || B == 0) return ESTP_OK;
    return launch_attn_forward(ctx, Q, K, V, lse, Hq, Hkv, softmax_scale, cu_seqlens, B, sumT,
                               max_seqlen, (flags & ESTP_IMP_EXCLUDE_SELF) != 0, accumulate != 0,
                               ctx->imp_acc, out, reinterpret_cast<cudaStream_t>(stream));
}

estp_status estp_attn_importance_finalize(estp_ctx* ctx, int32_t n_layers,
                                          float* importance_out, estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_attn_importance_finalize");
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    if (!ctx->imp_open) return fail(ESTP_ERR_INVALID_ARG, "no open importance accumulation");
    if (n_layers < 1) return fail(ESTP_ERR_INVALID_ARG, "n_layers must be >= 1");
    if (ctx->imp_sumT == 0 || ctx->imp_B == 0) return ESTP_OK;
    if (!importance_out) return fail(ESTP_ERR_INVALID_ARG, "importance_out is NULL");
    estp_status st = set_device(ctx);
    if (st != ESTP_OK) return st;
    return launch_importance_finalize(ctx, ctx->imp_acc, ctx->imp_cu, ctx->imp_B, ctx->imp_sumT,
                                      n_layers, ctx->imp_n_heads, ctx->imp_flags, importance_out,
                                      reinterpret_cast<cudaStream_t>(stream));
}

estp_status estp_pool(estp_ctx* ctx, const void* hidden, estp_dtype dtype, int64_t D,
                      int64_t ldh, const float* entropy, const float* importance,
                      const int32_t* cu_seqlens, int32_t B, int64_t sumT,
                      estp_mix_params mix, const estp_head* head, float* pooled_out,
                      float* pred_len_out, estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_pool");
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    if (dtype != ESTP_F32 && dtype != ESTP_BF16) return fail(ESTP_ERR_INVALID_ARG, "dtype");
    if (D < 1 || ldh < D || B < 0 || sumT < 0 || sumT > INT32_MAX)
        return fail(ESTP_ERR_INVALID_ARG, "need D >= 1, ldh >= D, B >= 0, 0 <= sumT < 2^31");
    if (!(mix.alpha > 0.f) || !std::isfinite(mix.alpha) || !std::isfinite(mix.lambda1) ||
        !std::isfinite(mix.lambda2))
        return fail(ESTP_ERR_INVALID_ARG, "mix params must be finite with alpha > 0");
    if (pred_len_out && !head) return fail(ESTP_ERR_INVALID_ARG, "pred_len_out needs a head");
    if (head && (!head->W || !head->centers || head->K < 1 || head->K > 1024))
        return fail(ESTP_ERR_INVALID_ARG, "head needs W, centers and 1 <= K <= 1024");
    if (B == 0) return ESTP_OK;
    if (!cu_seqlens || !pooled_out) return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    if (sumT > 0 && (!hidden || !entropy || !importance))
        return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    if (sumT > 0 && (!aligned16(hidden) || (ldh * esize(dtype)) % 16))
        return fail(ESTP_ERR_INVALID_ARG, "hidden base and row stride must be 16-byte aligned");
    estp_status st = set_device(ctx);
    if (st != ESTP_OK) return st;
    return launch_pool(ctx, hidden, dtype, D, ldh, entropy, importance, cu_seqlens, B, sumT, mix,
                       head, pooled_out, pred_len_out, reinterpret_cast<cudaStream_t>(stream));
}

estp_status estp_head_loss(estp_ctx* ctx, const float* pooled, int32_t B, int64_t D,
                           const estp_head* head, const float* targets, float lambda3,
                           float* loss_out, float* grad_W, float* grad_bias,
                           float* grad_pooled, estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_head_loss");
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    if (B < 1 || D < 1) return fail(ESTP_ERR_INVALID_ARG, "need B >= 1 and D >= 1");
    if (!head || !head->W || !head->centers || head->K < 1 || head->K > 1024)
        return fail(ESTP_ERR_INVALID_ARG, "head needs W, centers and 1 <= K <= 1024");
    if (!std::isfinite(lambda3)) return fail(ESTP_ERR_INVALID_ARG, "lambda3 must be finite");
    if (!pooled || !targets || !loss_out) return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    estp_status st = set_device(ctx);
    if (st != ESTP_OK) return st;
    return launch_head_loss(ctx, pooled, B, D, *head, targets, lambda3, loss_out, grad_W,
                            grad_bias, grad_pooled, reinterpret_cast<cudaStream_t>(stream));
}

estp_status estp_lm_head_entropy(estp_ctx* ctx, const void* hidden, int64_t ldh, const void* W,
                                 int64_t ldw, estp_dtype dtype, int64_t n_rows, int64_t D,
                                 int64_t V, float* entropy_out, estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_lm_head_entropy");
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    if (dtype != ESTP_BF16) return fail(ESTP_ERR_UNSUPPORTED, "lm-head entropy: bf16 only");
    if (n_rows < 0 || D < 64 || D % 64 || V < 1)
        return fail(ESTP_ERR_INVALID_ARG, "need n_rows >= 0, D a positive multiple of 64, V >= 1");
    if (ldh < D || ldw < D || ldh % 8 || ldw % 8)
        return fail(ESTP_ERR_INVALID_ARG, "need ldh, ldw >= D and multiples of 8");
    if (n_rows > INT32_MAX || V > INT32_MAX) return fail(ESTP_ERR_INVALID_ARG, "n_rows, V < 2^31");
    if (n_rows == 0) return ESTP_OK;
    if (!hidden || !W || !entropy_out) return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    if (!aligned16(hidden) || !aligned16(W))
        return fail(ESTP_ERR_INVALID_ARG, "hidden and W must be 16-byte aligned");
    estp_status st = set_device(ctx);
    if (st != ESTP_OK) return st;
    return launch_lm_head_entropy(ctx, hidden, ldh, W, ldw, n_rows, D, V, entropy_out,
                                  reinterpret_cast<cudaStream_t>(stream));
}

static estp_status check_mlp(estp_ctx* ctx, const float* pooled, int32_t B, int64_t D,
                             const estp_mlp_head* head) {
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    if (B < 1 || D < 1) return fail(ESTP_ERR_INVALID_ARG, "need B >= 1 and D >= 1");
    if (!head || !head->W1 || !head->W2 || !head->centers || head->F < 1 || head->K < 1 ||
        head->K > 1024)
        return fail(ESTP_ERR_INVALID_ARG, "MLP head needs W1, W2, centers, F >= 1, 1 <= K <= 1024");
    if (!pooled) return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    return ESTP_OK;
}

estp_status estp_mlp_head_predict(estp_ctx* ctx, const float* pooled, int32_t B, int64_t D,
                                  const estp_mlp_head* head, float* pred_out, float* probs_out,
                                  estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_mlp_head_predict");
    estp_status st = check_mlp(ctx, pooled, B, D, head);
    if (st != ESTP_OK) return st;
    if (!pred_out) return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    st = set_device(ctx);
    if (st != ESTP_OK) return st;
    return launch_mlp_head_predict(ctx, pooled, B, D, *head, pred_out, probs_out,
                                   reinterpret_cast<cudaStream_t>(stream));
}

estp_status estp_mlp_head_loss(estp_ctx* ctx, const float* pooled, int32_t B, int64_t D,
                               const estp_mlp_head* head, const float* targets, float lambda3,
                               float* loss_out, const estp_mlp_grads* grads,
                               estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_mlp_head_loss");
    estp_status st = check_mlp(ctx, pooled, B, D, head);
    if (st != ESTP_OK) return st;
    if (!std::isfinite(lambda3)) return fail(ESTP_ERR_INVALID_ARG, "lambda3 must be finite");
    if (!targets || !loss_out) return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    st = set_device(ctx);
    if (st != ESTP_OK) return st;
    const estp_mlp_grads none = {nullptr, nullptr, nullptr, nullptr, nullptr};
    return launch_mlp_head_loss(ctx, pooled, B, D, *head, targets, lambda3, loss_out,
                                grads ? *grads : none, reinterpret_cast<cudaStream_t>(stream));
}

estp_status estp_misalignment(estp_ctx* ctx, const float* entropy, const float* importance,
                              const int32_t* cu_seqlens, int32_t B, int64_t sumT, int32_t pct,
                              int32_t* counts_out, estp_stream_t stream) {
    ESTP_NVTX_RANGE("estp_misalignment");
    if (!ctx) return fail(ESTP_ERR_INVALID_ARG, "ctx is NULL");
    if (B < 0 || sumT < 0 || sumT > INT32_MAX)
        return fail(ESTP_ERR_INVALID_ARG, "need B >= 0 and 0 <= sumT < 2^31");
    if (pct < 1 || pct > 50) return fail(ESTP_ERR_INVALID_ARG, "pct must be in 1..50");
    if (B == 0) return ESTP_OK;
    if (!cu_seqlens || !counts_out || (sumT > 0 && (!entropy || !importance)))
        return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    estp_status st = set_device(ctx);
    if (st != ESTP_OK) return st;
    return launch_misalignment(ctx, entropy, importance, cu_seqlens, B, sumT, pct, counts_out,
                               reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"
