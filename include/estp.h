/*
 * estp.h -- C ABI of the ESTP feature-extraction library (GB300, sm_103a).
 *
 * ESTP (Entropy-and-Semantic Token Pooling, arXiv 2608.15592) turns the
 * activations of one LLM prefill into a pooled per-prompt feature and a
 * predicted output length:
 *   (a) per-token next-token entropy H_i over the full vocabulary   (Eq. 2-1)
 *   (b) per-token attention importance S_j, the attention mass key j receives
 *       from the causal softmax rows of the selected layers/heads    (Eq. 2-0)
 *   (c) T_i = lambda1 S_i + lambda2 H_i, e_i = softmax_i(T_i / alpha),
 *       h = sum_i e_i h_i, and a linear length head y = sum_k p_k c_k
 *                                                   (Eqs. 2-2..2-4, 3-2)
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Batches are varlen-packed: B prompts, prompt b owns the global token rows
 *   cu_seqlens[b] .. cu_seqlens[b+1]-1, cu_seqlens is int32 [B+1] in DEVICE
 *   memory with cu_seqlens[0] = 0, non-decreasing, cu_seqlens[B] = sumT.
 *   Empty prompts (equal neighbours) are allowed.  There is no padding.
 * - Every tensor pointer is caller-owned DEVICE memory (on the context's device)
 *   unless a parameter says "host".  The library never frees caller memory.
 * - All work is enqueued asynchronously on `stream` (0 = legacy default stream).
 *   Arguments are validated on the host before any launch; a bad argument returns
 *   ESTP_ERR_INVALID_ARG (or ESTP_ERR_UNSUPPORTED) and enqueues nothing.
 * - Facts only the device can check (cu_seqlens contents, max_seqlen) and
 *   bounded-wait timeouts are recorded in a device status word of the context;
 *   estp_sync_status() synchronises the stream and returns (and clears) it.
 *   Kernels never trap: on such an error they skip their work and return.
 * - A context is not thread-safe; use one context per host thread / stream.
 *   Calls on one context must be ordered (same stream, or synchronised).
 * - Alignment: every tensor base address must be 16-byte aligned, and every row
 *   stride (ld, ldh) times the element size a multiple of 16 bytes.
 * - Results are deterministic: no floating-point atomics; every partial sum is
 *   reduced in a fixed order, so repeated calls give identical bits.
 */
#ifndef ESTP_H
#define ESTP_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* estp_stream_t; /* same type as cudaStream_t */

typedef enum {
    ESTP_OK = 0,
    ESTP_ERR_INVALID_ARG = 1,  /* bad size, pointer, alignment or varlen metadata */
    ESTP_ERR_UNSUPPORTED = 2,  /* valid request the library does not implement   */
    ESTP_ERR_CUDA = 3,         /* a CUDA runtime call failed (message in last_error) */
    ESTP_ERR_TIMEOUT = 4,      /* a device-side bounded wait gave up               */
    ESTP_ERR_WORKSPACE = 5,    /* workspace could not be (re)allocated             */
    ESTP_ERR_BOUNDS = 6        /* a device bounds check failed; only libraries built
                                  with -DESTP_CHECKS make these checks           */
} estp_status;

typedef enum { ESTP_F32 = 0, ESTP_BF16 = 1 } estp_dtype;

typedef struct estp_ctx estp_ctx;

/* Creates a context on CUDA device `device`: a device status word and an empty,
 * growable workspace.  *ctx receives the handle (NULL on failure). */
estp_status estp_create(estp_ctx** ctx, int device);

/* Frees the context's device memory.  Synchronises the device first.  NULL is a no-op. */
void estp_destroy(estp_ctx* ctx);

/* Human-readable message for the last non-OK status returned on this host thread
 * (ctx may be NULL).  The pointer stays valid until the next call on the thread. */
const char* estp_last_error(const estp_ctx* ctx);

/* Synchronises `stream`, then returns and clears the device status word
 * (ESTP_OK, ESTP_ERR_INVALID_ARG for bad varlen metadata, ESTP_ERR_TIMEOUT). */
estp_status estp_sync_status(estp_ctx* ctx, estp_stream_t stream);

/* Testing aid for the failure path; the paper has no counterpart.  Sets, for this
 * context's later calls, the limit in SM clock cycles of the abortable waits of the
 * tensor-core attention kernels (the row normalisers and column sums of
 * estp_attn_lse / estp_attn_importance on bf16 inputs, the fused prefill forward of
 * estp_attn_forward_importance) and of the output-projection kernel of
 * estp_lm_head_entropy.  cycles <= 0 restores the
 * default, about 2 s.  A limit far below a tile copy's latency makes those waits
 * expire: each CTA then records ESTP_ERR_TIMEOUT in the status word, skips the rest of
 * its work, and waits (with the full default limit) for the copies and MMAs it has
 * already issued before it frees its tensor memory and exits, so the context stays
 * usable.  The outputs of a call that timed out are undefined; estp_sync_status
 * returns ESTP_ERR_TIMEOUT.  Host-side only: nothing is enqueued. */
estp_status estp_set_wait_limit(estp_ctx* ctx, int64_t cycles);

/* ------------------------------------------------------------------ (a)
 * Token entropy, Eq. 2-1 (Sec. 3.2):
 *   entropy_out[r] = -sum_{v<V} p_rv ln p_rv,  p_r = softmax(logits[r, 0:V]),
 * in nats, for every row r < n_rows.  Row r is the next-token distribution that
 * the caller attributes to token r (aligning the prefill's shifted logits is the
 * caller's job).  Rows are independent, so the varlen packing needs no metadata.
 *   logits      : [n_rows, ld] row-major, dtype ESTP_BF16 or ESTP_F32; only the
 *                 first V columns are read.  Values must be finite.
 *   cu_seqlens  : optional (NULL allowed).  When given, the device checks that
 *                 cu_seqlens[B] == n_rows and records ESTP_ERR_INVALID_ARG otherwise.
 *   entropy_out : [n_rows] fp32.
 * n_rows = 0 is a no-op.  Requires V >= 1, ld >= V. */
estp_status estp_token_entropy(estp_ctx* ctx, const void* logits, estp_dtype dtype,
                               int64_t n_rows, int64_t V, int64_t ld,
                               const int32_t* cu_seqlens, int32_t B, float* entropy_out,
                               estp_stream_t stream);

/* Allocation-free token entropy.  The paper has no counterpart: this is a deployment
 * variant of estp_token_entropy for callers that cannot allocate device memory, such
 * as a serving engine whose allocator already owns all of HBM for its KV cache, or
 * code running where cudaMalloc is not allowed.  It computes the same entropy_out as
 * estp_token_entropy (same arguments, minus context and cu_seqlens) on the calling
 * thread's current device, allocating nothing: its scratch (per-piece (max, sum,
 * weighted sum) partials) is one file-scope static device array of 128 KiB (4096
 * partial pairs) that every GPU loading this library holds until the process exits.
 *   - The first call on a device looks up that array's device address (a one-time
 *     set-up); make the first call before any stream capture.
 *   - All calls share the array, and it keeps the last call's contents: calls that
 *     overlap on the GPU (different streams, or concurrent host threads) race on it.
 *     Order them on one stream.
 *   - The launch uses at most 4096 pieces (one per warp).  A GPU with more resident
 *     warps than that (more than ~170 SMs at the kernel's occupancy) runs with fewer,
 *     longer pieces: the result is the same, only the split differs.
 * Errors are reported as for estp_token_entropy; there is no device status word. */
estp_status estp_token_entropy_noalloc(const void* logits, estp_dtype dtype, int64_t n_rows,
                                       int64_t V, int64_t ld, float* entropy_out,
                                       estp_stream_t stream);

/* Token entropy with the logits formed on the GPU and never stored: Eq. 2-1 (Sec. 3.2)
 * of z_r = h_r W^T, where h_r is token r's final hidden state and W the model's output
 * projection (the LM head).  For a model with a large vocabulary the logits are the
 * largest tensor of the feature path; here they live only in tensor memory, one
 * 128 x 256 tile at a time.
 *   hidden      : bf16 [n_rows, ldh] row-major (first D columns used), 16-byte aligned
 *   ldh         : row stride in elements, >= D and a multiple of 8
 *   W           : bf16 [V, ldw] row-major: one row of D weights per vocabulary entry
 *                 (the usual lm_head.weight layout), 16-byte aligned
 *   ldw         : row stride in elements, >= D and a multiple of 8
 *   dtype       : ESTP_BF16 (anything else is ESTP_ERR_UNSUPPORTED)
 *   D           : hidden size, a positive multiple of 64
 *   V           : vocabulary size >= 1
 *   entropy_out : fp32 [n_rows], natural log
 * The products accumulate in fp32 on the tensor cores; the entropy is formed in fp32 from
 * the fp32 logits.  n_rows = 0 is a no-op.  Uses the context's workspace (12 bytes per row
 * and vocabulary split).  Repeated calls give identical bits. */
estp_status estp_lm_head_entropy(estp_ctx* ctx, const void* hidden, int64_t ldh, const void* W,
                                 int64_t ldw, estp_dtype dtype, int64_t n_rows, int64_t D,
                                 int64_t V, float* entropy_out, estp_stream_t stream);

/* ------------------------------------------------------------------ (b)
 * Attention layout for one layer (Sec. 3.1): Q is [sumT, Hq, head_dim] and K is
 * [sumT, Hkv, head_dim], row-major and contiguous, dtype ESTP_BF16 or ESTP_F32.
 * Query head h reads KV head h / (Hq / Hkv) (grouped-query attention).  Scores
 * are s_ij = softmax_scale * q_i . k_j for keys j <= i of the same prompt
 * (causal), and A^h_ij = exp(s_ij - lse_i) with lse_i = ln sum_{j<=i} exp(s_ij).
 * head_dim must be 64 or 128; Hq <= 256; max_seqlen >= every prompt length
 * (checked on the device).
 *
 * Row log-normalisers: lse_out[h * sumT + i] = lse^h_i for every query head h,
 * fp32 [Hq, sumT], natural log.  This is what a flash-attention prefill returns
 * as its LSE, so callers that kept it can skip this call. */
estp_status estp_attn_lse(estp_ctx* ctx, const void* Q, const void* K, estp_dtype dtype,
                          int32_t Hq, int32_t Hkv, int32_t head_dim, float softmax_scale,
                          const int32_t* cu_seqlens, int32_t B, int64_t sumT,
                          int32_t max_seqlen, float* lse_out, estp_stream_t stream);

/* Attention importance, Eq. 2-0 (Sec. 3.1), one layer per call:
 *   C_j (+)= sum_{h in heads} sum_{i >= j, i in prompt(j)} A^h_ij
 * into an fp32 [sumT] accumulator held by the context.  accumulate = 0 starts a
 * new accumulation (this layer only); accumulate = 1 adds this layer.  Every call
 * of one accumulation must use the same cu_seqlens, B, sumT and head count.
 *   lse   : fp32 [Hq, sumT] from estp_attn_lse / the prefill, or NULL to have
 *           the library compute it (into the workspace) first.
 *   heads : HOST int32 [n_heads] query-head indices in [0, Hq), or NULL = all Hq.
 *   flags : OR of
 *     ESTP_IMP_EXCLUDE_SELF  drop the diagonal term A_jj from C_j (the softmax rows keep
 *                            it); Sec. 3.1 speaks of attention from all *other* tokens.
 *     ESTP_IMP_DIV_CAUSAL    finalize divides C_j by the causal count n_j (the queries
 *                            whose terms enter C_j: N_b - j, or N_b - j - 1 with
 *                            ESTP_IMP_EXCLUDE_SELF; S_j = 0 where n_j = 0) instead of N_b.
 *     ESTP_IMP_DIV_NONE      finalize divides by nothing but the layer/head count: the
 *                            mean column sum, N_b times the S_j of Eq. 2-0.
 *           The two divisor flags are variants of Eq. 2-0's 1/N, not printed in the
 *           paper; at most one may be set.  They take effect in
 *           estp_attn_importance_finalize and are fixed by the call that opens the
 *           accumulation (accumulate = 0): later calls of it must pass the same divisor
 *           flags, and with ESTP_IMP_DIV_CAUSAL the same ESTP_IMP_EXCLUDE_SELF. */
#define ESTP_IMP_EXCLUDE_SELF 1u
#define ESTP_IMP_DIV_CAUSAL 2u
#define ESTP_IMP_DIV_NONE 4u
estp_status estp_attn_importance(estp_ctx* ctx, const void* Q, const void* K,
                                 estp_dtype dtype, const float* lse, int32_t Hq, int32_t Hkv,
                                 int32_t head_dim, float softmax_scale, const int32_t* heads,
                                 int32_t n_heads, const int32_t* cu_seqlens, int32_t B,
                                 int64_t sumT, int32_t max_seqlen, int accumulate,
                                 uint32_t flags, estp_stream_t stream);

/* The prefill's causal attention output with the importance column sums of the same
 * probabilities (Sec. 3.1: the attention maps of the prefill; Eq. 2-0), one layer per call:
 *   out[i, h, :] = sum_{j <= i, j in prompt(i)} A^h_ij V[j, h / (Hq / Hkv), :]
 *   C_j (+)= sum_{h < Hq} sum_{i >= j, i in prompt(j)} A^h_ij
 * with A^h_ij = exp(s_ij - lse_i) as in estp_attn_lse.  The importance side is that of
 * estp_attn_importance over all Hq heads (same accumulation, same flags, closed by
 * estp_attn_importance_finalize); the two entry points may be mixed within one
 * accumulation as long as every call covers all Hq heads.
 *   Q   : bf16 [sumT, Hq, 128];  K, V : bf16 [sumT, Hkv, 128] (device, 16-byte aligned)
 *   lse : fp32 [Hq, sumT] (the prefill's, or estp_attn_lse's), or NULL to have the library
 *         compute it first.
 *   out : bf16 [sumT, Hq, 128] (device, 16-byte aligned), written for every token.
 *   dtype must be ESTP_BF16 and head_dim 128 (else ESTP_ERR_UNSUPPORTED).
 * The probabilities enter O = A V rounded to bf16 (as a flash-attention forward does);
 * the column sums use them unrounded.  The workspace holds one fp32 row of 128 column sums
 * per (head, query tile, key tile <= query tile). */
estp_status estp_attn_forward_importance(estp_ctx* ctx, const void* Q, const void* K,
                                         const void* V, estp_dtype dtype, const float* lse,
                                         int32_t Hq, int32_t Hkv, int32_t head_dim,
                                         float softmax_scale, const int32_t* cu_seqlens,
                                         int32_t B, int64_t sumT, int32_t max_seqlen,
                                         int accumulate, uint32_t flags, void* out,
                                         estp_stream_t stream);

/* Ends an accumulation: importance_out[j] = C_j / (N_b * n_layers * n_heads), N_b
 * the length of the prompt holding token j (Eq. 2-0's 1/N, then the mean over the
 * selected layers and heads); N_b is replaced by the causal count n_j, or by 1, when
 * the accumulation was opened with ESTP_IMP_DIV_CAUSAL or ESTP_IMP_DIV_NONE.
 * n_layers = number of estp_attn_importance calls the caller means to average over
 * (normally the calls since accumulate = 0).
 *   importance_out : fp32 [sumT]. */
estp_status estp_attn_importance_finalize(estp_ctx* ctx, int32_t n_layers,
                                          float* importance_out, estp_stream_t stream);

/* ------------------------------------------------------------------ (c)
 * Mixing and pooling, Eqs. 2-2..2-4 (Sec. 3.2), then the length head, Eq. 3-2
 * (Sec. 3.3):
 *   T_i = lambda1 * S_i + lambda2 * H_i
 *   e_i = exp(T_i / alpha) / sum_{j in prompt} exp(T_j / alpha)
 *   pooled_b = sum_{i in prompt b} e_i h_i            (zero for an empty prompt)
 *   z = W pooled_b + bias,  p = softmax(z),  y_b = sum_k p_k centers_k
 * alpha > 0 is the temperature of Sec. 3.2 (alpha = 1 is the printed Eq. 2-3). */
typedef struct {
    float lambda1;  /* weight of the attention importance S (Eq. 2-2) */
    float lambda2;  /* weight of the entropy H (Eq. 2-2)              */
    float alpha;    /* softmax temperature (Sec. 3.2), > 0            */
} estp_mix_params;

typedef struct {
    const float* W;        /* device fp32 [K, D] row-major                */
    const float* bias;     /* device fp32 [K], or NULL for zero bias      */
    const float* centers;  /* device fp32 [K] bin centres c_k (Eq. 3-2)   */
    int32_t K;             /* number of length bins, 1..1024              */
} estp_head;

/*   hidden       : [sumT, ldh] row-major, dtype ESTP_BF16 or ESTP_F32, first D
 *                  columns used (the prefill's hidden states h_i)
 *   entropy      : fp32 [sumT] (H_i), importance : fp32 [sumT] (S_i)
 *   head         : HOST pointer to the head description, or NULL for pooling only
 *   pooled_out   : fp32 [B, D]
 *   pred_len_out : fp32 [B] predicted lengths y_b, or NULL (requires head != NULL) */
estp_status estp_pool(estp_ctx* ctx, const void* hidden, estp_dtype dtype, int64_t D,
                      int64_t ldh, const float* entropy, const float* importance,
                      const int32_t* cu_seqlens, int32_t B, int64_t sumT,
                      estp_mix_params mix, const estp_head* head, float* pooled_out,
                      float* pred_len_out, estp_stream_t stream);

/* ------------------------------------------------------------------ (d)
 * Training loss of the length head (Sec. 3.3), for fitting W and bias on pooled
 * features: the soft label of Eq. 3-1,
 *   p_bj = exp(-|j - i_b|) / sum_k exp(-|k - i_b|),
 * i_b the bin whose centre is nearest to the target y_b (the lower index on a tie),
 * the prediction of Eq. 3-2 through the linear head, and the loss of Eq. 3-3 averaged
 * over the B prompts:
 *   L = lambda3 * mean_b CE(p_b, p_hat_b) + (1 - lambda3) * mean_b (y_b - y_hat_b)^2,
 * with CE(p, q) = -sum_k p_k ln q_k, and the gradients of L.
 *   pooled      : fp32 [B, D] (estp_pool's pooled_out)
 *   head        : HOST pointer to the head description (W [K, D], bias or NULL, centers)
 *   targets     : fp32 [B] target lengths y_b
 *   lambda3     : weight of the cross-entropy term, finite
 *   loss_out    : fp32 [1]
 *   grad_W      : fp32 [K, D] dL/dW, or NULL
 *   grad_bias   : fp32 [K] dL/dbias, or NULL
 *   grad_pooled : fp32 [B, D] dL/dpooled, or NULL
 * B >= 1, D >= 1, 1 <= K <= 1024.  Every sum runs in a fixed order (no atomics), so
 * repeated calls give identical bits.  All arrays are caller-owned device memory. */
estp_status estp_head_loss(estp_ctx* ctx, const float* pooled, int32_t B, int64_t D,
                           const estp_head* head, const float* targets, float lambda3,
                           float* loss_out, float* grad_W, float* grad_bias,
                           float* grad_pooled, estp_stream_t stream);

/* The MLP predictor of Sec. 3.3 (Fig. 2 feeds the pooled representation to "an MLP
 * predictor"; its depth, width and activation are not given, and are read here as one
 * hidden layer of F ReLU units in front of the K-bin softmax projection of Eq. 3-2):
 *   u_b = max(W1 h_b + b1, 0),  z_b = W2 u_b + b2,  p_hat_b = softmax(z_b),
 *   y_hat_b = sum_k p_hat_bk c_k.
 * All arrays fp32, caller-owned device memory; the struct itself is a HOST pointer. */
typedef struct {
    const float* W1;       /* [F, D] */
    const float* b1;       /* [F] or NULL */
    const float* W2;       /* [K, F] */
    const float* b2;       /* [K] or NULL */
    const float* centers;  /* [K] bin centres c_k */
    int32_t F;             /* hidden units, >= 1 */
    int32_t K;             /* bins, 1..1024 */
} estp_mlp_head;

/* Gradients of estp_mlp_head_loss; every pointer may be NULL (not computed). */
typedef struct {
    float* W1;      /* [F, D] */
    float* b1;      /* [F] */
    float* W2;      /* [K, F] */
    float* b2;      /* [K] */
    float* pooled;  /* [B, D] */
} estp_mlp_grads;

/* Predicted lengths through the MLP predictor: pred_out [B] = y_hat_b, and, when
 * probs_out is not NULL, probs_out [B, K] = p_hat_b.  pooled: fp32 [B, D] (estp_pool's
 * pooled_out).  B >= 1, D >= 1. */
estp_status estp_mlp_head_predict(estp_ctx* ctx, const float* pooled, int32_t B, int64_t D,
                                  const estp_mlp_head* head, float* pred_out, float* probs_out,
                                  estp_stream_t stream);

/* The loss of Eq. 3-3 (soft labels of Eq. 3-1 around the bin nearest to y_b, ties to the
 * lower bin; batch mean, as estp_head_loss) through the MLP predictor, and its gradients:
 * the second layer as the linear head on u, then the chain rule through the ReLU (its
 * derivative at 0 taken as 0) and the first layer.
 *   targets  : fp32 [B] target lengths y_b;  lambda3: weight of the cross-entropy term
 *   loss_out : fp32 [1];  grads: HOST pointer, or NULL for the loss alone
 * Every sum runs in a fixed order (no atomics), so repeated calls give identical bits. */
estp_status estp_mlp_head_loss(estp_ctx* ctx, const float* pooled, int32_t B, int64_t D,
                               const estp_mlp_head* head, const float* targets, float lambda3,
                               float* loss_out, const estp_mlp_grads* grads,
                               estp_stream_t stream);

/* Entropy/importance misalignment, the diagnostic behind Fig. 1b and Sec. 3.1's
 * motivation (not part of the predictor).  Per prompt b, with k = floor(pct*T_b/100),
 * TopX and BotX are the k tokens with the largest and with the smallest X (ties: the
 * lower token index first) for X = entropy H and importance S:
 *   counts_out[b] = { k, |TopH ∩ BotS|, |BotH ∩ TopS| }
 * i.e. high-entropy tokens of low importance and low-entropy tokens of high importance.
 * The paper splits at the 60th percentile: pct = 40.
 *   entropy, importance : fp32 [sumT], finite
 *   pct                 : 1..50
 *   counts_out          : int32 [B, 3]
 * Bad cu_seqlens (not non-decreasing from 0 to sumT) record ESTP_ERR_INVALID_ARG in the
 * status word and write nothing. */
estp_status estp_misalignment(estp_ctx* ctx, const float* entropy, const float* importance,
                              const int32_t* cu_seqlens, int32_t B, int64_t sumT, int32_t pct,
                              int32_t* counts_out, estp_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* ESTP_H */
