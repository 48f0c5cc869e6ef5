// Device side of the seeded input generator (see synth/__init__.py for the
// definitions).  Holds none of ESTP's arithmetic; its only job is to write, on the
// GPU, the same bits that the numpy generator writes on the host.
//
// SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): output n of the stream seeded with
// key is mix64(key + (n+1) * GAMMA).  Normal draws: Irwin-Hall sum of twelve 16-bit
// uniforms, z = (sum + 6) / 2^16 - 6, exact in binary64.  Every binary64 step below
// is exact, so the single rounding to binary32 (and then to bf16) matches the host.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t word(uint64_t key, uint64_t n) { return mix64(key + (n + 1) * kGamma); }

__device__ __forceinline__ double normal(uint64_t key, uint64_t idx) {
    int64_t acc = 0;
#pragma unroll
    for (int k = 0; k < 3; ++k) {
        const uint64_t w = word(key, idx * 3 + k);
#pragma unroll
        for (int c = 0; c < 4; ++c) acc += (int64_t)((w >> (16 * c)) & 0xFFFF);
    }
    return __dsub_rn(__dmul_rn((double)(acc + 6), 1.0 / 65536.0), 6.0);
}

__device__ __forceinline__ void store(void* dst, int bf16, int64_t i, double x) {
    const float f = __double2float_rn(x);
    if (bf16) static_cast<__nv_bfloat16*>(dst)[i] = __float2bfloat16_rn(f);
    else static_cast<float*>(dst)[i] = f;
}

__global__ void fill_normal_kernel(void* dst, int bf16, uint64_t key, int64_t idx0, int64_t count,
                                   double scale) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count;
         i += (int64_t)gridDim.x * blockDim.x)
        store(dst, bf16, i, __dmul_rn(normal(key, (uint64_t)(idx0 + i)), scale));
}

__global__ void fill_logits_kernel(void* dst, int bf16, uint64_t key_vals, uint64_t key_rows,
                                   int64_t row0, int64_t n_rows, int64_t V, int64_t ld,
                                   double sigma_lo, double sigma_span, uint32_t spike_thr,
                                   double spike_val, float pad) {
    for (int64_t r = blockIdx.y; r < n_rows; r += gridDim.y) {
        const uint64_t gr = (uint64_t)(row0 + r);
        const double u = (double)(word(key_rows, 3 * gr) >> 40) * (1.0 / 16777216.0);
        const double sigma = __dadd_rn(sigma_lo, __dmul_rn(sigma_span, u));
        int64_t spike_pos = -1;
        if (spike_thr && (word(key_rows, 3 * gr + 1) >> 40) < spike_thr)
            spike_pos = (int64_t)(word(key_rows, 3 * gr + 2) % (uint64_t)V);
        for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < ld;
             v += (int64_t)gridDim.x * blockDim.x) {
            if (v >= V) {
                store(dst, bf16, r * ld + v, (double)pad);
                continue;
            }
            double x = __dmul_rn(normal(key_vals, gr * (uint64_t)V + (uint64_t)v), sigma);
            if (v == spike_pos) x = __dadd_rn(x, spike_val);
            store(dst, bf16, r * ld + v, x);
        }
    }
}

}  // namespace

extern "C" {

// dst[i] = round(normal(key, idx0 + i) * scale), i < count.  Returns a cudaError_t.
int synth_fill_normal(void* dst, int bf16, uint64_t key, int64_t idx0, int64_t count,
                      double scale, cudaStream_t stream) {
    if (count <= 0) return 0;
    int64_t blocks = (count + 255) / 256;
    if (blocks > 65536) blocks = 65536;
    fill_normal_kernel<<<(unsigned)blocks, 256, 0, stream>>>(dst, bf16, key, idx0, count, scale);
    return (int)cudaGetLastError();
}

// Rows row0 .. row0+n_rows-1 of the logit recipe into dst [n_rows, ld].
int synth_fill_logits(void* dst, int bf16, uint64_t key_vals, uint64_t key_rows, int64_t row0,
                      int64_t n_rows, int64_t V, int64_t ld, double sigma_lo, double sigma_span,
                      uint32_t spike_thr, double spike_val, float pad, cudaStream_t stream) {
    if (n_rows <= 0) return 0;
    dim3 grid((unsigned)((ld + 255) / 256 < 64 ? (ld + 255) / 256 : 64),
              (unsigned)(n_rows < 65535 ? n_rows : 65535));
    fill_logits_kernel<<<grid, 256, 0, stream>>>(dst, bf16, key_vals, key_rows, row0, n_rows, V,
                                                 ld, sigma_lo, sigma_span, spike_thr, spike_val, pad);
    return (int)cudaGetLastError();
}

}  // extern "C"
