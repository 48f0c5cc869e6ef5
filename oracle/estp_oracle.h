/*
 * ESTP fp64 CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * This is the plain, slow reference against which the CUDA path is checked.
 * Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
 * arm may load it.  It shares no code, header, table or helper with the CUDA
 * library under paper_2608_15592_gb300/csrc, and the product path never calls it.
 *
 * Every function follows the definition printed in the paper (arXiv 2608.15592,
 * "When Entropy Is Not Enough: Reclaiming Lost Semantics in LLM Output Length
 * Prediction"), evaluated in IEEE double precision:
 *   oracle_token_entropy       Eq. 2-1  (Sec. 3.2)
 *   oracle_lm_head_entropy     Eq. 2-1 of the logits h W^T of the output projection
 *   oracle_attn_lse            log-normaliser of the softmax rows of A (Sec. 3.1)
 *   oracle_attn_colsum         the column sums of A inside Eq. 2-0 (Sec. 3.1)
 *   oracle_attn_output         the attention output O = A V of the prefill (Sec. 3.1)
 *   oracle_importance          Eq. 2-0 (the 1/N scaling and the head/layer mean)
 *   oracle_importance_div      Eq. 2-0 with the causal-count or no divisor (variants)
 *   oracle_pool                Eqs. 2-2, 2-3, 2-4 (Sec. 3.2)
 *   oracle_length_head         Eq. 3-2 (Sec. 3.3), linear projection + softmax
 *   oracle_head_loss           Eqs. 3-1 and 3-3 (Sec. 3.3) and their gradients
 *   oracle_mlp_length_head     Eq. 3-2 behind a one-hidden-layer ReLU MLP (Sec. 3.3, Fig. 2)
 *   oracle_mlp_head_loss       Eqs. 3-1 and 3-3 through that MLP, and every gradient
 *
 * Parity status: every function is pinned by the CPU tests (closed forms,
 * invariants, brute force against independent library routines); none is
 * "parity unpinned".
 *
 * Element types of the input arrays: ORACLE_F32 (IEEE binary32) or ORACLE_BF16
 * (raw bfloat16 bits, uint16).  Both widen to double exactly.
 * Return value of every function: 0 on success, -1 on an invalid argument.
 * n_threads <= 0 means "one thread per online core".
 */
#ifndef ESTP_ORACLE_H
#define ESTP_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORACLE_F32 = 0, ORACLE_BF16 = 1 };

/* Eq. 2-1: H_r = -sum_v p_rv ln p_rv with p_r = softmax(logits row r), natural log.
 * logits: n_rows rows of V values, row stride ld elements.  H_out: [n_rows]. */
int oracle_token_entropy(const void* logits, int dtype, int64_t n_rows, int64_t V,
                         int64_t ld, double* H_out, int n_threads);

/* Eq. 2-1 of logits that are formed here from hidden states: z_rv = sum_k h_rk W_vk
 * (the model's output projection; W: V rows of D weights, row stride ldw), then
 * H_r = -sum_v p_rv ln p_rv with p_r = softmax(z_r).  hidden: n_rows rows of D values,
 * row stride ldh.  H_out: [n_rows]. */
int oracle_lm_head_entropy(const void* hidden, const void* W, int dtype, int64_t n_rows,
                           int64_t D, int64_t V, int64_t ldh, int64_t ldw, double* H_out,
                           int n_threads);

/* Row log-normaliser of causal attention for one layer:
 * lse_out[h * sumT + i] = ln sum_{j <= i, j in prompt(i)} exp(scale * q_i^h . k_j^{h/rep}).
 * Q: [sumT, Hq, d], K: [sumT, Hkv, d] row-major; cu_seqlens: [B+1] prompt offsets (host).
 * All Hq heads are computed.  lse_out: [Hq, sumT]. */
int oracle_attn_lse(const void* Q, const void* K, int dtype, int Hq, int Hkv, int d,
                    double scale, const int32_t* cu_seqlens, int B, double* lse_out,
                    int n_threads);

/* The output of causal attention for one layer (the prefill's own attention, whose softmax
 * rows A are those of Eq. 2-0): O[i, h, :] = sum_{j <= i, j in prompt(i)} A^h_ij V[j, h/rep, :].
 * Q: [sumT, Hq, d], K, V: [sumT, Hkv, d] row-major; O_out: [sumT, Hq, d]. */
int oracle_attn_output(const void* Q, const void* K, const void* V, int dtype, int Hq, int Hkv,
                       int d, double scale, const int32_t* cu_seqlens, int B, double* O_out,
                       int n_threads);

/* The same output for the query rows i >= row_from (prompt-local index) only; the rows
 * before are left as they are.  Used to check late rows of long prompts. */
int oracle_attn_output_rows(const void* Q, const void* K, const void* V, int dtype, int Hq,
                            int Hkv, int d, double scale, const int32_t* cu_seqlens, int B,
                            int64_t row_from, double* O_out, int n_threads);

/* Column sums of the causal softmax attention matrix of one layer, over a set of
 * query heads:  C_out[j] += sum_{h in heads} sum_{i >= j, i in prompt(j)} A^h_ij,
 * A^h_ij = softmax_j(scale * q_i^h . k_j^{h/rep}) over j <= i in the same prompt.
 * exclude_self != 0 drops the diagonal term i == j from the column sum (the row
 * softmax itself is unchanged).  C_out: [sumT], accumulated (caller zeroes it). */
int oracle_attn_colsum(const void* Q, const void* K, int dtype, int Hq, int Hkv, int d,
                       double scale, const int32_t* heads, int n_heads,
                       const int32_t* cu_seqlens, int B, int exclude_self, double* C_out,
                       int n_threads);

/* The same column sums formed from the rows i >= row_from (prompt-local index) only.
 * C_j depends only on rows i >= j, so C_out[j] is exact for every key j with local
 * index >= row_from; smaller j receive only part of their mass.  Used to check late
 * keys of prompts too long for the full O(T^2) evaluation. */
int oracle_attn_colsum_rows(const void* Q, const void* K, int dtype, int Hq, int Hkv, int d,
                            double scale, const int32_t* heads, int n_heads,
                            const int32_t* cu_seqlens, int B, int exclude_self,
                            int64_t row_from, double* C_out, int n_threads);

/* Eq. 2-0 with the head/layer mean: S_j = C_j / (N_b * n_layers * n_heads), where
 * N_b is the length of the prompt that holds token j.  S_out: [sumT]. */
int oracle_importance(const double* C, const int32_t* cu_seqlens, int B, int n_layers,
                      int n_heads, double* S_out);

/* Variants of Eq. 2-0's divisor (not printed in the paper):
 *   ORACLE_DIV_LENGTH  N_b (= oracle_importance)
 *   ORACLE_DIV_CAUSAL  the causal count n_j = N_b - j (N_b - j - 1 with exclude_self):
 *                      the queries whose terms enter C_j; S_j = 0 where n_j = 0
 *   ORACLE_DIV_NONE    1: S_j = C_j / (n_layers * n_heads), the mean column sum */
enum { ORACLE_DIV_LENGTH = 0, ORACLE_DIV_CAUSAL = 1, ORACLE_DIV_NONE = 2 };
int oracle_importance_div(const double* C, const int32_t* cu_seqlens, int B, int n_layers,
                          int n_heads, int divisor, int exclude_self, double* S_out);

/* Eqs. 2-2..2-4 per prompt b:  T_i = lambda1*S_i + lambda2*H_i,
 * e_i = exp(T_i/alpha) / sum_j exp(T_j/alpha) over the prompt's tokens,
 * pooled_b = sum_i e_i h_i.  hidden: [sumT, D] with row stride ldh elements.
 * A prompt with no tokens pools to the zero vector.
 * weights_out (may be NULL): [sumT] the e_i.  pooled_out: [B, D]. */
int oracle_pool(const void* hidden, int dtype, int64_t D, int64_t ldh, const double* H,
                const double* S, const int32_t* cu_seqlens, int B, double lambda1,
                double lambda2, double alpha, double* weights_out, double* pooled_out);

/* Eq. 3-2 with a linear projection: z = W h + bias, p = softmax(z), y = sum_k p_k c_k.
 * pooled: [B, D]; W: [K, D] fp32; bias, centers: [K] fp32 (bias may be NULL).
 * probs_out (may be NULL): [B, K].  yhat_out: [B]. */
int oracle_length_head(const double* pooled, int B, int64_t D, const float* W,
                       const float* bias, const float* centers, int K, double* probs_out,
                       double* yhat_out);

/* Eqs. 3-1 and 3-3 through the linear head of Eq. 3-2, averaged over the B prompts:
 *   L = lambda3 * mean_b CE(p_b, p_hat_b) + (1 - lambda3) * mean_b (y_b - y_hat_b)^2,
 * p_b the soft label of Eq. 3-1 around the bin whose centre is nearest to y_b (lower
 * index on a tie).  loss_out: [1]; the gradients of L (each may be NULL):
 * grad_W [K, D], grad_bias [K], grad_pooled [B, D]. */
int oracle_head_loss(const double* pooled, int B, int64_t D, const float* W, const float* bias,
                     const float* centers, int K, const float* y, double lambda3,
                     double* loss_out, double* grad_W, double* grad_bias, double* grad_pooled);

/* The MLP predictor of Sec. 3.3 (Fig. 2 names an MLP; its depth, width and activation are
 * not given, read here as one hidden layer of F ReLU units):
 *   u_b = max(W1 h_b + b1, 0),  z_b = W2 u_b + b2,  p_hat_b = softmax(z_b),
 *   y_hat_b = sum_k p_hat_bk c_k.
 * W1: [F, D] fp32, b1: [F] or NULL, W2: [K, F] fp32, b2: [K] or NULL.
 * oracle_mlp_length_head writes y_out [B] and, if probs_out != NULL, p_hat [B, K].
 * oracle_mlp_head_loss writes the loss of Eq. 3-3 (batch mean, as oracle_head_loss) and
 * each gradient whose pointer is not NULL: grad_W1 [F, D], grad_b1 [F], grad_W2 [K, F],
 * grad_b2 [K], grad_pooled [B, D].  The ReLU's derivative at a = 0 is taken as 0. */
int oracle_mlp_length_head(const double* pooled, int B, int64_t D, const float* W1, const float* b1,
                           int F, const float* W2, const float* b2, const float* centers, int K,
                           double* probs_out, double* y_out);
int oracle_mlp_head_loss(const double* pooled, int B, int64_t D, const float* W1, const float* b1,
                         int F, const float* W2, const float* b2, const float* centers, int K,
                         const float* y, double lambda3, double* loss_out, double* grad_W1,
                         double* grad_b1, double* grad_W2, double* grad_b2, double* grad_pooled);

#ifdef __cplusplus
}
#endif
#endif
