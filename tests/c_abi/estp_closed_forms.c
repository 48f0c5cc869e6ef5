/*
 * The whole feature path through the C ABI alone (no Python, no torch): plain C11, CUDA
 * runtime for device memory, checked against closed forms that need no oracle.
 *
 *   entropy (Eq. 2-1)     : a row of equal logits gives ln V; one logit far above the
 *                           rest gives 0; k tied maxima far above the rest give ln k
 *   importance (Eq. 2-0)  : Q = 0 makes every causal row uniform, A_ij = 1 / (i + 1) for
 *                           j <= i (0-based), so C_j = sum_{i=j}^{T-1} 1 / (i + 1) and
 *                           S_j = C_j / T for every head and layer
 *   pooling (Eqs. 2-2..2-4): lambda1 = lambda2 = 0 gives equal weights, so the pooled
 *                           vector is the mean of the prompt's hidden rows
 *   head (Eq. 3-2)        : W = 0 and no bias give equal bin probabilities, so the
 *                           predicted length is the mean of the bin centres
 *
 * Exit status 0 and a last line "OK" when every check holds.
 */
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "estp.h"

static int failures = 0;

#define CUDA_OK(x)                                                                   \
    do {                                                                             \
        cudaError_t e_ = (x);                                                        \
        if (e_ != cudaSuccess) {                                                     \
            fprintf(stderr, "%s:%d %s: %s\n", __FILE__, __LINE__, #x,               \
                    cudaGetErrorString(e_));                                         \
            exit(2);                                                                 \
        }                                                                            \
    } while (0)

#define ESTP_OK_(ctx, x)                                                             \
    do {                                                                             \
        estp_status s_ = (x);                                                        \
        if (s_ != ESTP_OK) {                                                         \
            fprintf(stderr, "%s:%d %s: status %d: %s\n", __FILE__, __LINE__, #x,    \
                    (int)s_, estp_last_error(ctx));                                  \
            exit(3);                                                                 \
        }                                                                            \
    } while (0)

static void check(const char* what, double got, double want, double tol) {
    const double err = fabs(got - want);
    if (!(err <= tol)) {
        fprintf(stderr, "FAIL %s: got %.9g want %.9g (err %.3g > %.3g)\n", what, got, want, err, tol);
        ++failures;
    }
}

static void* dev_copy(const void* host, size_t bytes) {
    void* d = NULL;
    CUDA_OK(cudaMalloc(&d, bytes ? bytes : 16));
    if (bytes) CUDA_OK(cudaMemcpy(d, host, bytes, cudaMemcpyHostToDevice));
    return d;
}

/* bf16 bits of a float that bf16 holds exactly */
static uint16_t bf16(float x) {
    uint32_t u;
    memcpy(&u, &x, 4);
    return (uint16_t)(u >> 16);
}

int main(void) {
    estp_ctx* ctx = NULL;
    ESTP_OK_(NULL, estp_create(&ctx, 0));
    cudaStream_t stream;
    CUDA_OK(cudaStreamCreate(&stream));
    estp_stream_t st = (estp_stream_t)stream;

    /* ------------------------------------------------------------ entropy */
    {
        const int V = 1000, rows = 3;
        float* x = (float*)calloc((size_t)rows * V, sizeof(float));
        x[1 * V + 417] = 100.f;                                             /* one-hot */
        for (int k = 0; k < 4; ++k) x[2 * V + 3 + 250 * k] = 100.f;         /* 4 ties */
        float* dx = (float*)dev_copy(x, sizeof(float) * rows * V);
        float* dH = NULL;
        CUDA_OK(cudaMalloc((void**)&dH, sizeof(float) * rows));
        ESTP_OK_(ctx, estp_token_entropy(ctx, dx, ESTP_F32, rows, V, V, NULL, 0, dH, st));
        ESTP_OK_(ctx, estp_sync_status(ctx, st));
        float H[3];
        CUDA_OK(cudaMemcpy(H, dH, sizeof H, cudaMemcpyDeviceToHost));
        check("entropy of equal logits = ln V", H[0], log((double)V), 1e-3);
        check("entropy of one dominant logit = 0", H[1], 0.0, 1e-3);
        check("entropy of 4 tied maxima = ln 4", H[2], log(4.0), 1e-3);
        CUDA_OK(cudaFree(dx));
        CUDA_OK(cudaFree(dH));
        free(x);
    }

    /* ---------------------------------------- importance, pooling and the head */
    {
        const int B = 2, Hq = 4, Hkv = 2, d = 128, D = 64, K = 4, layers = 2;
        const int32_t lens[2] = {200, 77};
        const int32_t cu[3] = {0, lens[0], lens[0] + lens[1]};
        const int sumT = cu[2];
        /* Q = 0; K arbitrary (small integers, exact in bf16) */
        uint16_t* q = (uint16_t*)calloc((size_t)sumT * Hq * d, sizeof(uint16_t));
        uint16_t* k = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)sumT * Hkv * d);
        for (size_t i = 0; i < (size_t)sumT * Hkv * d; ++i) k[i] = bf16((float)((int)(i % 9) - 4));
        int32_t* dcu = (int32_t*)dev_copy(cu, sizeof cu);
        void* dq = dev_copy(q, sizeof(uint16_t) * (size_t)sumT * Hq * d);
        void* dk = dev_copy(k, sizeof(uint16_t) * (size_t)sumT * Hkv * d);
        float *dlse = NULL, *dS = NULL;
        CUDA_OK(cudaMalloc((void**)&dlse, sizeof(float) * (size_t)Hq * sumT));
        CUDA_OK(cudaMalloc((void**)&dS, sizeof(float) * (size_t)sumT));
        const float scale = 1.f / sqrtf((float)d);
        for (int l = 0; l < layers; ++l) {
            ESTP_OK_(ctx, estp_attn_lse(ctx, dq, dk, ESTP_BF16, Hq, Hkv, d, scale, dcu, B, sumT,
                                        lens[0], dlse, st));
            ESTP_OK_(ctx, estp_attn_importance(ctx, dq, dk, ESTP_BF16, dlse, Hq, Hkv, d, scale,
                                               NULL, 0, dcu, B, sumT, lens[0], l > 0, 0u, st));
        }
        ESTP_OK_(ctx, estp_attn_importance_finalize(ctx, layers, dS, st));
        ESTP_OK_(ctx, estp_sync_status(ctx, st));
        float* S = (float*)malloc(sizeof(float) * sumT);
        CUDA_OK(cudaMemcpy(S, dS, sizeof(float) * sumT, cudaMemcpyDeviceToHost));
        for (int b = 0; b < B; ++b) {
            const int T = lens[b];
            double tail = 0.0; /* sum_{i=j}^{T-1} 1 / (i + 1), built from j = T-1 down */
            double maxrel = 0.0, sum = 0.0;
            for (int j = T - 1; j >= 0; --j) {
                tail += 1.0 / (j + 1);
                const double want = tail / T, got = S[cu[b] + j];
                const double rel = fabs(got - want) / want;
                if (rel > maxrel) maxrel = rel;
                sum += got;
            }
            char what[96];
            snprintf(what, sizeof what, "prompt %d: importance of uniform attention, max rel err", b);
            check(what, maxrel, 0.0, 1e-2);
            snprintf(what, sizeof what, "prompt %d: importance sums to 1", b);
            check(what, sum, 1.0, 1e-3);
        }

        /* pooling with equal weights and a zero head */
        float* h = (float*)malloc(sizeof(float) * (size_t)sumT * D);
        for (int i = 0; i < sumT; ++i)
            for (int c = 0; c < D; ++c) h[(size_t)i * D + c] = (float)((i * 7 + c * 3) % 11) - 5.f;
        float* dh = (float*)dev_copy(h, sizeof(float) * (size_t)sumT * D);
        float* dH = NULL;
        CUDA_OK(cudaMalloc((void**)&dH, sizeof(float) * sumT));
        CUDA_OK(cudaMemset(dH, 0, sizeof(float) * sumT));
        float* W = (float*)calloc((size_t)K * D, sizeof(float));
        const float centers[4] = {128.f, 384.f, 640.f, 4000.f};
        float* dW = (float*)dev_copy(W, sizeof(float) * K * D);
        float* dc = (float*)dev_copy(centers, sizeof centers);
        float *dpooled = NULL, *dpred = NULL;
        CUDA_OK(cudaMalloc((void**)&dpooled, sizeof(float) * B * D));
        CUDA_OK(cudaMalloc((void**)&dpred, sizeof(float) * B));
        estp_mix_params mix = {0.f, 0.f, 1.f};
        estp_head head = {dW, NULL, dc, K};
        ESTP_OK_(ctx, estp_pool(ctx, dh, ESTP_F32, D, D, dH, dS, dcu, B, sumT, mix, &head, dpooled,
                                dpred, st));
        ESTP_OK_(ctx, estp_sync_status(ctx, st));
        float* pooled = (float*)malloc(sizeof(float) * B * D);
        float pred[2];
        CUDA_OK(cudaMemcpy(pooled, dpooled, sizeof(float) * B * D, cudaMemcpyDeviceToHost));
        CUDA_OK(cudaMemcpy(pred, dpred, sizeof pred, cudaMemcpyDeviceToHost));
        for (int b = 0; b < B; ++b) {
            double maxerr = 0.0, scale_b = 0.0;
            for (int c = 0; c < D; ++c) {
                double mean = 0.0;
                for (int i = cu[b]; i < cu[b + 1]; ++i) mean += h[(size_t)i * D + c];
                mean /= lens[b];
                const double err = fabs(pooled[b * D + c] - mean);
                if (err > maxerr) maxerr = err;
                if (fabs(mean) > scale_b) scale_b = fabs(mean);
            }
            char what[96];
            snprintf(what, sizeof what, "prompt %d: pooled = mean of hidden rows, max abs err", b);
            check(what, maxerr, 0.0, 2e-3 * scale_b + 1e-6);
            snprintf(what, sizeof what, "prompt %d: predicted length = mean of the centres", b);
            check(what, pred[b], (128.0 + 384.0 + 640.0 + 4000.0) / 4.0, 1.0);
        }
        cudaFree(dq); cudaFree(dk); cudaFree(dcu); cudaFree(dlse); cudaFree(dS); cudaFree(dh);
        cudaFree(dH); cudaFree(dW); cudaFree(dc); cudaFree(dpooled); cudaFree(dpred);
        free(q); free(k); free(S); free(h); free(W); free(pooled);
    }

    /* an argument the library must refuse before any launch */
    if (estp_token_entropy(ctx, (const void*)0x10, ESTP_F32, 4, 8, 4, NULL, 0, (float*)0x10, st) !=
        ESTP_ERR_INVALID_ARG) {
        fprintf(stderr, "FAIL ld < V accepted\n");
        ++failures;
    }

    CUDA_OK(cudaStreamDestroy(stream));
    estp_destroy(ctx);
    if (failures) {
        fprintf(stderr, "%d check(s) failed\n", failures);
        return 1;
    }
    printf("OK\n");
    return 0;
}
