/*
 * ESTP fp64 CPU oracle -- TEST INFRASTRUCTURE ONLY (see estp_oracle.h).
 *
 * Plain loops in IEEE double.  Each function evaluates the paper's definition
 * directly: softmax rows are formed one at a time, the attention matrix is never
 * blocked or fused, and there is no algebraic rewrite of the entropy.  Threads
 * only split independent units (rows, or (prompt, head) pairs whose results are
 * summed afterwards in a fixed order), so every result is deterministic.
 *
 * Built with -ffp-contract=off so that x86 and Arm hosts give identical bits.
 */
#include "estp_oracle.h"

#include <math.h>
#include <pthread.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

/* ---------------------------------------------------------------- helpers */

static double load_elem(const void* base, int dtype, int64_t idx) {
    if (dtype == ORACLE_F32) return (double)((const float*)base)[idx];
    /* bfloat16 is the top half of a binary32: widen by a 16-bit shift (exact). */
    uint32_t bits = (uint32_t)((const uint16_t*)base)[idx] << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

static int resolve_threads(int n_threads) {
    if (n_threads > 0) return n_threads;
    long n = sysconf(_SC_NPROCESSORS_ONLN);
    return n > 0 ? (int)n : 1;
}

typedef void (*task_fn)(void* ctx, int64_t unit, double* scratch);

typedef struct {
    task_fn fn;
    void* ctx;
    int64_t n_units;
    int n_threads;
    int tid;
    size_t scratch_len;
} worker_arg;

/* Thread tid handles units tid, tid + n_threads, ...; each unit writes only its
 * own outputs, so the interleaving cannot change any value. */
static void* worker_main(void* p) {
    worker_arg* a = (worker_arg*)p;
    double* scratch = NULL;
    if (a->scratch_len) scratch = (double*)malloc(a->scratch_len * sizeof(double));
    for (int64_t u = a->tid; u < a->n_units; u += a->n_threads) a->fn(a->ctx, u, scratch);
    free(scratch);
    return NULL;
}

static void parallel_units(task_fn fn, void* ctx, int64_t n_units, size_t scratch_len,
                           int n_threads) {
    n_threads = resolve_threads(n_threads);
    if (n_threads > n_units) n_threads = (int)(n_units > 0 ? n_units : 1);
    pthread_t* th = (pthread_t*)malloc(sizeof(pthread_t) * n_threads);
    worker_arg* args = (worker_arg*)malloc(sizeof(worker_arg) * n_threads);
    for (int t = 0; t < n_threads; ++t) {
        args[t] = (worker_arg){fn, ctx, n_units, n_threads, t, scratch_len};
        if (t > 0) pthread_create(&th[t], NULL, worker_main, &args[t]);
    }
    worker_main(&args[0]);
    for (int t = 1; t < n_threads; ++t) pthread_join(th[t], NULL);
    free(th);
    free(args);
}

static int valid_dtype(int dtype) { return dtype == ORACLE_F32 || dtype == ORACLE_BF16; }

static int valid_cu(const int32_t* cu, int B) {
    if (!cu || B < 0 || cu[0] != 0) return 0;
    for (int b = 0; b < B; ++b)
        if (cu[b + 1] < cu[b]) return 0;
    return 1;
}

/* ------------------------------------------------------------ Eq. 2-1 */

typedef struct {
    const void* logits;
    int dtype;
    int64_t V, ld;
    double* H;
} entropy_ctx;

/* One row: p_v = exp(z_v - m) / sum_u exp(z_u - m) (m = max_v z_v only keeps exp
 * finite; it cancels in p), then H = -sum_v p_v ln p_v with 0 ln 0 = 0. */
static void entropy_unit(void* vctx, int64_t r, double* e) {
    entropy_ctx* c = (entropy_ctx*)vctx;
    int64_t off = r * c->ld;
    double m = -INFINITY;
    for (int64_t v = 0; v < c->V; ++v) {
        double z = load_elem(c->logits, c->dtype, off + v);
        if (z > m) m = z;
    }
    double s = 0.0;
    for (int64_t v = 0; v < c->V; ++v) {
        e[v] = exp(load_elem(c->logits, c->dtype, off + v) - m);
        s += e[v];
    }
    double H = 0.0;
    for (int64_t v = 0; v < c->V; ++v) {
        double p = e[v] / s;
        if (p > 0.0) H -= p * log(p);
    }
    c->H[r] = H;
}

int oracle_token_entropy(const void* logits, int dtype, int64_t n_rows, int64_t V,
                         int64_t ld, double* H_out, int n_threads) {
    if (!valid_dtype(dtype) || n_rows < 0 || V <= 0 || ld < V) return -1;
    if (n_rows == 0) return 0;
    if (!logits || !H_out) return -1;
    entropy_ctx c = {logits, dtype, V, ld, H_out};
    parallel_units(entropy_unit, &c, n_rows, (size_t)V, n_threads);
    return 0;
}

/* ------------------------------- Eq. 2-1 with the logits formed in place */

typedef struct {
    const void *hid, *W;
    int dtype;
    int64_t D, V, ldh, ldw;
    double* H;
} lm_head_ctx;

/* One row: the logits z_v = sum_k h_k W_vk of the output projection (W holds one row
 * of D weights per vocabulary entry), formed in double, then Eq. 2-1 of z exactly as
 * in entropy_unit.  scratch: [D + V] doubles. */
static void lm_head_entropy_unit(void* vctx, int64_t r, double* scratch) {
    lm_head_ctx* c = (lm_head_ctx*)vctx;
    double* h = scratch;
    double* z = scratch + c->D;
    for (int64_t k = 0; k < c->D; ++k) h[k] = load_elem(c->hid, c->dtype, r * c->ldh + k);
    for (int64_t v = 0; v < c->V; ++v) {
        double dot = 0.0;
        for (int64_t k = 0; k < c->D; ++k) dot += h[k] * load_elem(c->W, c->dtype, v * c->ldw + k);
        z[v] = dot;
    }
    double m = -INFINITY;
    for (int64_t v = 0; v < c->V; ++v)
        if (z[v] > m) m = z[v];
    double s = 0.0;
    for (int64_t v = 0; v < c->V; ++v) {
        z[v] = exp(z[v] - m);
        s += z[v];
    }
    double H = 0.0;
    for (int64_t v = 0; v < c->V; ++v) {
        double p = z[v] / s;
        if (p > 0.0) H += -p * log(p);
    }
    c->H[r] = H;
}

int oracle_lm_head_entropy(const void* hidden, const void* W, int dtype, int64_t n_rows,
                           int64_t D, int64_t V, int64_t ldh, int64_t ldw, double* H_out,
                           int n_threads) {
    if (!valid_dtype(dtype) || n_rows < 0 || D <= 0 || V <= 0 || ldh < D || ldw < D) return -1;
    if (n_rows == 0) return 0;
    if (!hidden || !W || !H_out) return -1;
    lm_head_ctx c = {hidden, W, dtype, D, V, ldh, ldw, H_out};
    parallel_units(lm_head_entropy_unit, &c, n_rows, (size_t)(D + V), n_threads);
    return 0;
}

/* ------------------------------------------- attention rows (Sec. 3.1) */

/* One (prompt, query head) pair: the prompt's q^h and k^{h/rep} rows widened to
 * double once, then every causal softmax row is formed from its definition. */
typedef struct {
    const void *Q, *K;
    int dtype, Hq, Hkv, d;
    double scale;
    const int32_t* heads; /* NULL: head index = unit's head slot */
    int n_heads;
    const int32_t* cu;
    int B;
    int exclude_self;
    double* out;      /* lse: [Hq, sumT];  colsum: [n_pairs, T_max] private rows */
    int64_t sumT;
    int64_t out_ld;   /* colsum: row length of the private buffers */
    int want_lse;
    int64_t row_from; /* first prompt-local query row formed */
} attn_ctx;

static void attn_unit(void* vctx, int64_t unit, double* scratch) {
    attn_ctx* c = (attn_ctx*)vctx;
    int b = (int)(unit / c->n_heads);
    int slot = (int)(unit % c->n_heads);
    int h = c->heads ? c->heads[slot] : slot;
    int g = h / (c->Hq / c->Hkv);
    int64_t t0 = c->cu[b], T = (int64_t)c->cu[b + 1] - c->cu[b];
    int d = c->d;
    if (T == 0) return;
    double* q = (double*)malloc(sizeof(double) * (size_t)(T * d));
    double* k = (double*)malloc(sizeof(double) * (size_t)(T * d));
    double* s = scratch; /* scores of one row, length >= T */
    for (int64_t t = 0; t < T; ++t)
        for (int x = 0; x < d; ++x) {
            if (t >= c->row_from)  /* query rows before row_from are never formed */
                q[t * d + x] = load_elem(c->Q, c->dtype, ((t0 + t) * c->Hq + h) * (int64_t)d + x);
            k[t * d + x] = load_elem(c->K, c->dtype, ((t0 + t) * c->Hkv + g) * (int64_t)d + x);
        }
    double* col = c->want_lse ? NULL : c->out + unit * c->out_ld;
    for (int64_t i = c->row_from; i < T; ++i) {
        /* s_ij = scale * q_i . k_j for the causal keys j <= i of the same prompt */
        double m = -INFINITY;
        for (int64_t j = 0; j <= i; ++j) {
            double dot = 0.0;
            for (int x = 0; x < d; ++x) dot += q[i * d + x] * k[j * d + x];
            s[j] = c->scale * dot;
            if (s[j] > m) m = s[j];
        }
        double Z = 0.0;
        for (int64_t j = 0; j <= i; ++j) Z += exp(s[j] - m);
        if (c->want_lse) {
            c->out[(int64_t)h * c->sumT + t0 + i] = m + log(Z);
        } else {
            /* A_ij = exp(s_ij - m) / Z; the column sum collects A_ij over rows i >= j */
            for (int64_t j = 0; j <= i; ++j) {
                if (c->exclude_self && j == i) continue;
                col[j] += exp(s[j] - m) / Z;
            }
        }
    }
    free(q);
    free(k);
}

static int64_t max_len(const int32_t* cu, int B) {
    int64_t mx = 0;
    for (int b = 0; b < B; ++b)
        if (cu[b + 1] - cu[b] > mx) mx = cu[b + 1] - cu[b];
    return mx;
}

/* ------------------------------- the attention output of the prefill (Sec. 3.1) */

typedef struct {
    const void *Q, *K, *V;
    int dtype, Hq, Hkv, d;
    double scale;
    const int32_t* cu;
    double* O;
    int64_t row_from; /* first prompt-local query row formed */
} attn_out_ctx;

/* One (prompt, query head) pair: for every query row i, the causal softmax row
 * A_ij = exp(s_ij - m) / Z over the keys j <= i, s_ij = scale * q_i . k_j, and the
 * attention output O_i = sum_j A_ij v_j (V read with K's head). scratch: >= T doubles. */
static void attn_out_unit(void* vctx, int64_t unit, double* s) {
    attn_out_ctx* c = (attn_out_ctx*)vctx;
    const int b = (int)(unit / c->Hq), h = (int)(unit % c->Hq), g = h / (c->Hq / c->Hkv);
    const int64_t t0 = c->cu[b], T = (int64_t)c->cu[b + 1] - c->cu[b];
    const int d = c->d;
    if (T == 0) return;
    double* q = (double*)malloc(sizeof(double) * (size_t)(T * d));
    double* k = (double*)malloc(sizeof(double) * (size_t)(T * d));
    double* v = (double*)malloc(sizeof(double) * (size_t)(T * d));
    for (int64_t t = 0; t < T; ++t) {
        const int64_t row_q = (t0 + t) * (int64_t)c->Hq + h;    /* token t, query head h */
        const int64_t row_kv = (t0 + t) * (int64_t)c->Hkv + g;  /* token t, its KV head */
        for (int x = 0; x < d; ++x) {
            q[t * d + x] = load_elem(c->Q, c->dtype, row_q * d + x);
            k[t * d + x] = load_elem(c->K, c->dtype, row_kv * d + x);
            v[t * d + x] = load_elem(c->V, c->dtype, row_kv * d + x);
        }
    }
    for (int64_t i = c->row_from; i < T; i++) {  /* output rows i >= row_from */
        double m = -INFINITY;
        for (int64_t j = 0; j <= i; ++j) {
            double dot = 0.0;
            for (int x = 0; x < d; ++x) dot += q[i * d + x] * k[j * d + x];
            s[j] = dot * c->scale;
            if (s[j] > m) m = s[j];
        }
        double Z = 0.0;
        for (int64_t j = 0; j <= i; ++j) Z += exp(s[j] - m);
        double* o = c->O + ((t0 + i) * c->Hq + h) * (int64_t)d;
        for (int x = 0; x < d; ++x) o[x] = 0.0;
        for (int64_t j = 0; j <= i; ++j) {
            const double a = exp(s[j] - m) / Z;
            for (int x = 0; x < d; ++x) o[x] += a * v[j * d + x];
        }
    }
    free(q);
    free(k);
    free(v);
}

int oracle_attn_output(const void* Q, const void* K, const void* V, int dtype, int Hq, int Hkv,
                       int d, double scale, const int32_t* cu_seqlens, int B, double* O_out,
                       int n_threads) {
    return oracle_attn_output_rows(Q, K, V, dtype, Hq, Hkv, d, scale, cu_seqlens, B, 0, O_out,
                                   n_threads);
}

int oracle_attn_output_rows(const void* Q, const void* K, const void* V, int dtype, int Hq,
                            int Hkv, int d, double scale, const int32_t* cu_seqlens, int B,
                            int64_t row_from, double* O_out, int n_threads) {
    if (row_from < 0) return -1;
    if (!valid_dtype(dtype) || Hq <= 0 || Hkv <= 0 || Hq % Hkv || d <= 0) return -1;
    if (!valid_cu(cu_seqlens, B)) return -1;
    const int64_t sumT = cu_seqlens[B];
    if (sumT == 0) return 0;
    if (!Q || !K || !V || !O_out) return -1;
    attn_out_ctx c = {Q, K, V, dtype, Hq, Hkv, d, scale, cu_seqlens, O_out, row_from};
    parallel_units(attn_out_unit, &c, (int64_t)B * Hq, (size_t)max_len(cu_seqlens, B), n_threads);
    return 0;
}

int oracle_attn_lse(const void* Q, const void* K, int dtype, int Hq, int Hkv, int d,
                    double scale, const int32_t* cu_seqlens, int B, double* lse_out,
                    int n_threads) {
    if (!valid_dtype(dtype) || Hq <= 0 || Hkv <= 0 || Hq % Hkv || d <= 0) return -1;
    if (!valid_cu(cu_seqlens, B)) return -1;
    int64_t sumT = cu_seqlens[B];
    if (sumT == 0) return 0;
    if (!Q || !K || !lse_out) return -1;
    attn_ctx c = {Q, K, dtype, Hq, Hkv, d, scale, NULL, Hq, cu_seqlens, B, 0,
                  lse_out, sumT, 0, 1, 0};
    parallel_units(attn_unit, &c, (int64_t)B * Hq, (size_t)max_len(cu_seqlens, B), n_threads);
    return 0;
}

int oracle_attn_colsum_rows(const void* Q, const void* K, int dtype, int Hq, int Hkv, int d,
                            double scale, const int32_t* heads, int n_heads,
                            const int32_t* cu_seqlens, int B, int exclude_self,
                            int64_t row_from, double* C_out, int n_threads) {
    if (row_from < 0) return -1;
    if (!valid_dtype(dtype) || Hq <= 0 || Hkv <= 0 || Hq % Hkv || d <= 0) return -1;
    if (!valid_cu(cu_seqlens, B)) return -1;
    if (heads) {
        if (n_heads <= 0) return -1;
        for (int s = 0; s < n_heads; ++s)
            if (heads[s] < 0 || heads[s] >= Hq) return -1;
    } else {
        n_heads = Hq;
    }
    int64_t sumT = cu_seqlens[B];
    if (sumT == 0) return 0;
    if (!Q || !K || !C_out) return -1;
    int64_t Tmax = max_len(cu_seqlens, B);
    int64_t n_units = (int64_t)B * n_heads;
    /* each (prompt, head) pair fills a private row; the rows are then added into
     * C_out in the fixed order (prompt, head slot) */
    double* priv = (double*)calloc((size_t)(n_units * Tmax), sizeof(double));
    if (!priv) return -1;
    attn_ctx c = {Q, K, dtype, Hq, Hkv, d, scale, heads, n_heads, cu_seqlens, B,
                  exclude_self, priv, sumT, Tmax, 0, row_from};
    parallel_units(attn_unit, &c, n_units, (size_t)Tmax, n_threads);
    for (int b = 0; b < B; ++b) {
        int64_t t0 = cu_seqlens[b], T = (int64_t)cu_seqlens[b + 1] - cu_seqlens[b];
        for (int s = 0; s < n_heads; ++s) {
            const double* row = priv + ((int64_t)b * n_heads + s) * Tmax;
            for (int64_t j = 0; j < T; ++j) C_out[t0 + j] += row[j];
        }
    }
    free(priv);
    return 0;
}

int oracle_attn_colsum(const void* Q, const void* K, int dtype, int Hq, int Hkv, int d,
                       double scale, const int32_t* heads, int n_heads,
                       const int32_t* cu_seqlens, int B, int exclude_self, double* C_out,
                       int n_threads) {
    return oracle_attn_colsum_rows(Q, K, dtype, Hq, Hkv, d, scale, heads, n_heads, cu_seqlens, B,
                                   exclude_self, 0, C_out, n_threads);
}

/* ------------------------------------------------------------ Eq. 2-0 */

int oracle_importance(const double* C, const int32_t* cu_seqlens, int B, int n_layers,
                      int n_heads, double* S_out) {
    return oracle_importance_div(C, cu_seqlens, B, n_layers, n_heads, ORACLE_DIV_LENGTH, 0, S_out);
}

/* Eq. 2-0 with the divisor of the column sum chosen: the prompt length N (the paper),
 * the number of queries whose terms enter C_j (rows i >= j, or i > j without the
 * diagonal; S_j = 0 when there are none), or 1. */
int oracle_importance_div(const double* C, const int32_t* cu_seqlens, int B, int n_layers,
                          int n_heads, int divisor, int exclude_self, double* S_out) {
    if (!valid_cu(cu_seqlens, B) || n_layers <= 0 || n_heads <= 0) return -1;
    if (divisor != ORACLE_DIV_LENGTH && divisor != ORACLE_DIV_CAUSAL && divisor != ORACLE_DIV_NONE)
        return -1;
    for (int b = 0; b < B; ++b) {
        int64_t t0 = cu_seqlens[b], N = (int64_t)cu_seqlens[b + 1] - cu_seqlens[b];
        for (int64_t j = 0; j < N; ++j) {
            double n;
            if (divisor == ORACLE_DIV_LENGTH) n = (double)N;
            else if (divisor == ORACLE_DIV_CAUSAL) n = (double)(N - j - (exclude_self ? 1 : 0));
            else n = 1.0;
            S_out[t0 + j] = n > 0.0 ? C[t0 + j] / (n * (double)n_layers * (double)n_heads) : 0.0;
        }
    }
    return 0;
}

/* -------------------------------------------------------- Eqs. 2-2..2-4 */

int oracle_pool(const void* hidden, int dtype, int64_t D, int64_t ldh, const double* H,
                const double* S, const int32_t* cu_seqlens, int B, double lambda1,
                double lambda2, double alpha, double* weights_out, double* pooled_out) {
    if (!valid_dtype(dtype) || D <= 0 || ldh < D || !(alpha > 0.0)) return -1;
    if (!valid_cu(cu_seqlens, B) || !pooled_out) return -1;
    for (int b = 0; b < B; ++b) {
        int64_t t0 = cu_seqlens[b], n = (int64_t)cu_seqlens[b + 1] - cu_seqlens[b];
        double* h = pooled_out + (int64_t)b * D;
        for (int64_t x = 0; x < D; ++x) h[x] = 0.0;
        if (n == 0) continue;
        /* Eq. 2-2 and the tempered softmax of Eq. 2-3 (max subtracted for range only) */
        double* w = (double*)malloc(sizeof(double) * (size_t)n);
        double M = -INFINITY;
        for (int64_t i = 0; i < n; ++i) {
            double T = lambda1 * S[t0 + i] + lambda2 * H[t0 + i];
            w[i] = T / alpha;
            if (w[i] > M) M = w[i];
        }
        double Z = 0.0;
        for (int64_t i = 0; i < n; ++i) Z += exp(w[i] - M);
        for (int64_t i = 0; i < n; ++i) {
            double e = exp(w[i] - M) / Z;
            if (weights_out) weights_out[t0 + i] = e;
            /* Eq. 2-4 */
            for (int64_t x = 0; x < D; ++x)
                h[x] += e * load_elem(hidden, dtype, (t0 + i) * ldh + x);
        }
        free(w);
    }
    return 0;
}

/* ------------------------------------------------------------ Eq. 3-2 */

int oracle_length_head(const double* pooled, int B, int64_t D, const float* W,
                       const float* bias, const float* centers, int K, double* probs_out,
                       double* yhat_out) {
    if (B < 0 || D <= 0 || K <= 0 || !W || !centers || !yhat_out) return -1;
    double* z = (double*)malloc(sizeof(double) * (size_t)K);
    for (int b = 0; b < B; ++b) {
        const double* h = pooled + (int64_t)b * D;
        double m = -INFINITY;
        for (int k = 0; k < K; ++k) {
            double acc = bias ? (double)bias[k] : 0.0;
            for (int64_t x = 0; x < D; ++x) acc += (double)W[(int64_t)k * D + x] * h[x];
            z[k] = acc;
            if (acc > m) m = acc;
        }
        double Z = 0.0;
        for (int k = 0; k < K; ++k) Z += exp(z[k] - m);
        double y = 0.0;
        for (int k = 0; k < K; ++k) {
            double p = exp(z[k] - m) / Z;
            if (probs_out) probs_out[(int64_t)b * K + k] = p;
            y += p * (double)centers[k];
        }
        yhat_out[b] = y;
    }
    free(z);
    return 0;
}

/* -------------------------------------------------------- Eqs. 3-1, 3-3 */

/* Soft label of Eq. 3-1: p_j = exp(-|j - i|) / sum_k exp(-|k - i|), i the bin whose
 * centre is nearest to y (the lower index on a tie). */
static int nearest_bin(const float* centers, int K, double y) {
    int best = 0;
    double d = fabs(y - (double)centers[0]);
    for (int k = 1; k < K; ++k) {
        double e = fabs(y - (double)centers[k]);
        if (e < d) { d = e; best = k; }
    }
    return best;
}

int oracle_head_loss(const double* pooled, int B, int64_t D, const float* W, const float* bias,
                     const float* centers, int K, const float* y, double lambda3,
                     double* loss_out, double* grad_W, double* grad_bias, double* grad_pooled) {
    if (B <= 0 || D <= 0 || K <= 0 || !pooled || !W || !centers || !y || !loss_out) return -1;
    double* ph = (double*)malloc(sizeof(double) * (size_t)B * K);
    double* yh = (double*)malloc(sizeof(double) * (size_t)B);
    double* dz = (double*)malloc(sizeof(double) * (size_t)K);
    if (oracle_length_head(pooled, B, D, W, bias, centers, K, ph, yh) != 0) {
        free(ph); free(yh); free(dz);
        return -1;
    }
    if (grad_W) for (int64_t q = 0; q < (int64_t)K * D; ++q) grad_W[q] = 0.0;
    if (grad_bias) for (int k = 0; k < K; ++k) grad_bias[k] = 0.0;
    double ce = 0.0, mse = 0.0;
    for (int b = 0; b < B; ++b) {
        const double* p_hat = ph + (int64_t)b * K;
        const int i = nearest_bin(centers, K, (double)y[b]);
        double norm = 0.0;
        for (int k = 0; k < K; ++k) norm += exp(-fabs((double)(k - i)));
        const double err = yh[b] - (double)y[b];
        for (int k = 0; k < K; ++k) {
            const double p = exp(-fabs((double)(k - i))) / norm;
            ce -= p * log(p_hat[k]);
            /* d/dz_k of the batch mean: CE term p_hat_k - p_k (sum_k p_k = 1); MSE term
             * 2 (y_hat - y) dy_hat/dz_k with dy_hat/dz_k = p_hat_k (c_k - y_hat) */
            dz[k] = (lambda3 * (p_hat[k] - p) +
                     (1.0 - lambda3) * 2.0 * err * p_hat[k] * ((double)centers[k] - yh[b])) / (double)B;
        }
        mse += err * err;
        const double* h = pooled + (int64_t)b * D;
        for (int k = 0; k < K; ++k) {
            double* gw = grad_W ? grad_W + (int64_t)k * D : NULL;  /* row k of dL/dW */
            if (grad_bias) grad_bias[k] += dz[k];
            if (gw)
                for (int64_t x = 0; x < D; ++x) gw[x] += dz[k] * h[x];
        }
        if (grad_pooled)
            for (int64_t x = 0; x < D; ++x) {
                double g = 0.0;
                for (int k = 0; k < K; ++k) {
                    const float* wk = W + (int64_t)k * D;  /* row k of the head */
                    g += (double)wk[x] * dz[k];
                }
                grad_pooled[(int64_t)b * D + x] = g;
            }
    }
    *loss_out = lambda3 * ce / (double)B + (1.0 - lambda3) * mse / (double)B;
    free(ph); free(yh); free(dz);
    return 0;
}


/* ---------------------------------------- the MLP predictor (Sec. 3.3, Fig. 2) */

/* Hidden layer of the MLP head: a_bf = sum_x W1_fx h_bx + b1_f, u_bf = max(a_bf, 0).
 * Returns a [B, F] array of u (caller frees), or NULL. */
static double* mlp_hidden(const double* pooled, int B, int64_t D, const float* W1, const float* b1,
                          int F) {
    double* u = (double*)malloc(sizeof(double) * (size_t)B * F);
    if (!u) return NULL;
    for (int b = 0; b < B; ++b)
        for (int f = 0; f < F; ++f) {
            double a = b1 ? (double)b1[f] : 0.0;
            for (int64_t x = 0; x < D; ++x) a += (double)W1[(int64_t)f * D + x] * pooled[(int64_t)b * D + x];
            u[(int64_t)b * F + f] = a > 0.0 ? a : 0.0;
        }
    return u;
}

int oracle_mlp_length_head(const double* pooled, int B, int64_t D, const float* W1, const float* b1,
                           int F, const float* W2, const float* b2, const float* centers, int K,
                           double* probs_out, double* y_out) {
    if (B <= 0 || D <= 0 || F <= 0 || !pooled || !W1 || !W2) return -1;
    double* u = mlp_hidden(pooled, B, D, W1, b1, F);
    if (!u) return -1;
    const int r = oracle_length_head(u, B, F, W2, b2, centers, K, probs_out, y_out);
    free(u);
    return r;
}

/* The loss of Eq. 3-3 through the MLP: the second layer is the linear head of Eq. 3-2 on u,
 * whose loss and gradients (dL/dW2, dL/db2, dL/du) come from oracle_head_loss; the chain
 * rule then goes through the ReLU (dL/da = dL/du where a > 0, else 0) and the first
 * layer: dL/dW1_fx = sum_b dL/da_bf h_bx, dL/db1_f = sum_b dL/da_bf,
 * dL/dh_bx = sum_f W1_fx dL/da_bf. */
int oracle_mlp_head_loss(const double* pooled, int B, int64_t D, const float* W1, const float* b1,
                         int F, const float* W2, const float* b2, const float* centers, int K,
                         const float* y, double lambda3, double* loss_out, double* grad_W1,
                         double* grad_b1, double* grad_W2, double* grad_b2, double* grad_pooled) {
    if (B <= 0 || D <= 0 || F <= 0 || !pooled || !W1 || !W2) return -1;
    double* u = mlp_hidden(pooled, B, D, W1, b1, F);
    double* du = (double*)malloc(sizeof(double) * (size_t)B * F);
    if (!u || !du) { free(u); free(du); return -1; }
    if (oracle_head_loss(u, B, F, W2, b2, centers, K, y, lambda3, loss_out, grad_W2, grad_b2, du) != 0) {
        free(u); free(du);
        return -1;
    }
    for (int64_t q = 0; q < (int64_t)B * F; ++q)
        if (!(u[q] > 0.0)) du[q] = 0.0;  /* dL/da: the ReLU passes the gradient where a > 0 */
    if (grad_W1)
        for (int f = 0; f < F; ++f)
            for (int64_t x = 0; x < D; ++x) {
                double g = 0.0;
                for (int b = 0; b < B; ++b) g += du[(int64_t)b * F + f] * pooled[(int64_t)b * D + x];
                grad_W1[(int64_t)f * D + x] = g;
            }
    if (grad_b1)
        for (int f = 0; f < F; ++f) {
            double g = 0.0;
            for (int b = 0; b < B; ++b) g += du[(int64_t)b * F + f];
            grad_b1[f] = g;
        }
    if (grad_pooled)
        for (int b = 0; b < B; ++b)
            for (int64_t x = 0; x < D; ++x) {
                double g = 0.0;
                for (int f = 0; f < F; ++f) g += (double)W1[(int64_t)f * D + x] * du[(int64_t)b * F + f];
                grad_pooled[(int64_t)b * D + x] = g;
            }
    free(u);
    free(du);
    return 0;
}
