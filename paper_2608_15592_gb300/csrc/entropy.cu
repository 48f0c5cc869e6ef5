// K-ENT: per-token entropy over the full vocabulary (Eq. 2-1, Sec. 3.2).
//
// For a row z of V logits, with y = z * log2(e), m = max y,
//   s = sum_v 2^(y_v - m),  t = sum_v 2^(y_v - m) (y_v - m)
// the entropy in nats is H = ln2 * (log2 s - t / s): p_v = 2^(y_v - m) / s and
// -sum p ln p = ln s - (ln2 / s) sum 2^(y_v - m)(y_v - m).  All three terms are
// built in one streaming pass, rescaling (s, t) whenever the running max grows:
//   m' > m:  f = 2^(m - m'),  t <- f (t + (m - m') s),  s <- f s.
//
// Work split: the logits are n_rows x nvec 16-byte units.  The flat unit range is
// cut into W equal pieces, one per warp, so every warp streams the same number of
// bytes whatever V and n_rows are.  A warp finishes the rows it covers whole; a row
// cut between warps leaves (m, s, t) partials that a second kernel merges in warp
// order (deterministic).
#include <mutex>

#include "estp_internal.cuh"

namespace estp {
namespace {

constexpr int kEntThreads = 256;
constexpr int kEntMinBlocks = 3;  // resident blocks per SM the registers are sized for
constexpr int kEntUnroll = 8;     // 16-byte loads per lane per batch
constexpr float kMaskedLogit = -1e30f;  // finite: 2^(masked - m) = 0 and 0 * d = 0

struct EntPart {
    float m, s, t, pad;
};

struct EntArgs {
    const char* base;
    int64_t ld_bytes;
    int64_t nvec;       // 16-byte units per row
    int64_t V;
    int64_t units;      // n_rows * nvec
    int64_t n_warps;
    float* H;
    EntPart* part;      // [n_warps][2]: slot 0 = first segment, slot 1 = last segment
    int* status;        // device status word, or nullptr (bounds checks of debug builds)
};

__device__ __forceinline__ int64_t warp_start(int64_t units, int64_t W, int64_t w) {
    return (units * w) / W;
}

// Largest warp whose range starts at or before unit u.
__device__ __forceinline__ int64_t unit_owner(int64_t units, int64_t W, int64_t u) {
    int64_t w = ((u + 1) * W - 1) / units;
    return w < W - 1 ? w : W - 1;
}


__device__ __forceinline__ void merge(float& m, float& s, float& t, float m2, float s2, float t2) {
    float mm = fmaxf(m, m2);
    float da = m - mm, db = m2 - mm;
    float fa = ex2(da), fb = ex2(db);
    t = fa * fmaf(da, s, t) + fb * fmaf(db, s2, t2);
    s = fa * s + fb * s2;
    m = mm;
}

__device__ __forceinline__ float entropy_of(float s, float t) {
    return kLn2 * (lg2(s) - __fdividef(t, s));
}

// Masks the elements at or past V in the row's last unit (bf16: 8 per unit).
__device__ __forceinline__ void mask_bf16(uint4& v, int valid) {
    uint32_t* w = reinterpret_cast<uint32_t*>(&v);
    const uint32_t neg = 0xF149u;  // bf16 bits of about -1e30
#pragma unroll
    for (int e = 0; e < 8; ++e)
        if (e >= valid) {
            uint32_t& word = w[e >> 1];
            word = (e & 1) ? ((word & 0x0000FFFFu) | (neg << 16)) : ((word & 0xFFFF0000u) | neg);
        }
}

__device__ __forceinline__ void mask_f32(uint4& v, int valid) {
    uint32_t* w = reinterpret_cast<uint32_t*>(&v);
#pragma unroll
    for (int e = 0; e < 4; ++e)
        if (e >= valid) w[e] = __float_as_uint(kMaskedLogit);
}

// Loads the units c, c + 32, .. c + 32 (kEntUnroll - 1) of a row segment ending at c1;
// units at or past c1 become masked logits (they contribute nothing).
template <bool kBf16>
__device__ __forceinline__ void load_batch(const char* row, int64_t c, int64_t c1, int64_t nvec,
                                           int tail_valid, uint4* v) {
    constexpr int kPerUnit = kBf16 ? 8 : 4;
#pragma unroll
    for (int k = 0; k < kEntUnroll; ++k) {
        const int64_t ck = c + 32 * k;
        if (ck < c1) {
            v[k] = ld_stream(row + ck * 16);
            if (ck == nvec - 1 && tail_valid < kPerUnit) {
                if (kBf16) mask_bf16(v[k], tail_valid); else mask_f32(v[k], tail_valid);
            }
        } else if (kBf16) {
            v[k] = make_uint4(0xF149F149u, 0xF149F149u, 0xF149F149u, 0xF149F149u);
        } else {
            const uint32_t n = __float_as_uint(kMaskedLogit);
            v[k] = make_uint4(n, n, n, n);
        }
    }
}

// Folds one batch of kEntUnroll units into the lane's running (m, s, t): one max and
// one rescale per batch, then two interleaved accumulator pairs to shorten the
// dependent add chains.
__device__ __forceinline__ void accum1(float x, float m, float& s, float& t) {
    const float d = fmaf(x, kLog2e, -m);  // y - m
    const float e = ex2(d);
    s += e;
    t = fmaf(e, d, t);
}

template <bool kBf16>
__device__ __forceinline__ void reduce_batch(const uint4* v, float& m, float2& s, float2& t,
                                             float2& s1, float2& t1) {
    float bm;
    if (kBf16) {  // tree max over the batch's bf16 pairs
        __nv_bfloat162 mx[kEntUnroll];
#pragma unroll
        for (int k = 0; k < kEntUnroll; ++k) {
            const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&v[k]);
            mx[k] = __hmax2(__hmax2(p[0], p[1]), __hmax2(p[2], p[3]));
        }
#pragma unroll
        for (int w = kEntUnroll / 2; w > 0; w >>= 1)
#pragma unroll
            for (int k = 0; k < w; ++k) mx[k] = __hmax2(mx[k], mx[k + w]);
        bm = fmaxf(__low2float(mx[0]), __high2float(mx[0]));
    } else {
        float mx[kEntUnroll];
#pragma unroll
        for (int k = 0; k < kEntUnroll; ++k)
            mx[k] = fmaxf(fmaxf(__uint_as_float(v[k].x), __uint_as_float(v[k].y)),
                          fmaxf(__uint_as_float(v[k].z), __uint_as_float(v[k].w)));
#pragma unroll
        for (int w = kEntUnroll / 2; w > 0; w >>= 1)
#pragma unroll
            for (int k = 0; k < w; ++k) mx[k] = fmaxf(mx[k], mx[k + w]);
        bm = mx[0];
    }
    const float new_m = fmaxf(m, bm * kLog2e);
    const float dm = m - new_m;  // <= 0
    const float f = ex2(dm);
    t = make_float2(f * fmaf(dm, s.x, t.x), f * fmaf(dm, s.y, t.y));
    t1 = make_float2(f * fmaf(dm, s1.x, t1.x), f * fmaf(dm, s1.y, t1.y));
    s = make_float2(s.x * f, s.y * f);
    s1 = make_float2(s1.x * f, s1.y * f);
    m = new_m;
#pragma unroll
    for (int k = 0; k < kEntUnroll; ++k) {
        if (kBf16) {  // four independent (s, t) chains
            accum1(bf16lo(v[k].x), m, s.x, t.x);
            accum1(bf16hi(v[k].x), m, s.y, t.y);
            accum1(bf16lo(v[k].y), m, s1.x, t1.x);
            accum1(bf16hi(v[k].y), m, s1.y, t1.y);
            accum1(bf16lo(v[k].z), m, s.x, t.x);
            accum1(bf16hi(v[k].z), m, s.y, t.y);
            accum1(bf16lo(v[k].w), m, s1.x, t1.x);
            accum1(bf16hi(v[k].w), m, s1.y, t1.y);
        } else {
            accum1(__uint_as_float(v[k].x), m, s.x, t.x);
            accum1(__uint_as_float(v[k].y), m, s.y, t.y);
            accum1(__uint_as_float(v[k].z), m, s1.x, t1.x);
            accum1(__uint_as_float(v[k].w), m, s1.y, t1.y);
        }
    }
}

// One lane's share of units [c0, c1) of one row (lane handles c0 + lane + 32k).
// Full batches run without bounds checks through a moving pointer; the ragged
// remainder and the row's partial last unit (when V is not a multiple of the
// unit width) go through the checked loader.
template <bool kBf16>
__device__ __forceinline__ void segment(const char* row, int64_t c0, int64_t c1, int64_t nvec,
                                        int tail_valid, float& m, float2& s, float2& t) {
    const int lane = threadIdx.x & 31;
    constexpr int kPerUnit = kBf16 ? 8 : 4;
    constexpr int64_t kStride = 32 * kEntUnroll;
    float2 s1 = make_float2(0.f, 0.f), t1 = make_float2(0.f, 0.f);
    // the unchecked range excludes a partial last unit of the row
    const int64_t c1m = (c1 == nvec && tail_valid < kPerUnit) ? c1 - 1 : c1;
    int64_t c = c0 + lane;
    const uint4* p = reinterpret_cast<const uint4*>(row) + c;
    for (; c + kStride - 32 < c1m; c += kStride, p += kStride) {
        uint4 v[kEntUnroll];
#pragma unroll
        for (int k = 0; k < kEntUnroll; ++k) v[k] = ld_stream(p + 32 * k);
        reduce_batch<kBf16>(v, m, s, t, s1, t1);
    }
    if (c < c1) {  // remainder: fewer than kEntUnroll units left for this lane
        uint4 v[kEntUnroll];
        load_batch<kBf16>(row, c, c1, nvec, tail_valid, v);
        reduce_batch<kBf16>(v, m, s, t, s1, t1);
    }
    s = make_float2(s.x + s1.x, s.y + s1.y);
    t = make_float2(t.x + t1.x, t.y + t1.y);
}

template <bool kBf16>
__global__ void __launch_bounds__(kEntThreads, kEntMinBlocks) entropy_kernel(EntArgs a) {
    const int lane = threadIdx.x & 31;
    const int64_t w = (int64_t)blockIdx.x * (kEntThreads / 32) + (threadIdx.x >> 5);
    if (w >= a.n_warps) return;
    constexpr int kPerUnit = kBf16 ? 8 : 4;
    const int tail_valid = (int)(a.V - (a.nvec - 1) * kPerUnit);
    const int64_t start = warp_start(a.units, a.n_warps, w);
    const int64_t end = warp_start(a.units, a.n_warps, w + 1);
    int64_t u = start;
    while (u < end) {
        const int64_t r = u / a.nvec;
        const int64_t row_u0 = r * a.nvec;
        const int64_t seg_end = min(end, row_u0 + a.nvec);
        const int64_t c0 = u - row_u0, c1 = seg_end - row_u0;
        if (!in_bounds(r < a.units / a.nvec && c0 >= 0 && c0 < c1 && c1 <= a.nvec, a.status))
            return;
        float m = kMaskedLogit;
        float2 s = make_float2(0.f, 0.f), t = make_float2(0.f, 0.f);
        segment<kBf16>(a.base + r * a.ld_bytes, c0, c1, a.nvec, tail_valid, m, s, t);
        float ss = s.x + s.y, tt = t.x + t.y;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            float m2 = __shfl_xor_sync(0xffffffffu, m, off);
            float s2 = __shfl_xor_sync(0xffffffffu, ss, off);
            float t2 = __shfl_xor_sync(0xffffffffu, tt, off);
            merge(m, ss, tt, m2, s2, t2);
        }
        if (lane == 0) {
            if (c0 == 0 && c1 == a.nvec) {
                a.H[r] = entropy_of(ss, tt);
            } else if (in_bounds(w < a.n_warps, a.status)) {
                a.part[w * 2 + (u == start ? 0 : 1)] = EntPart{m, ss, tt, 0.f};
            }
        }
        u = seg_end;
    }
}

// Rows cut between warps: merge the partials of the covering warps in warp order.
__global__ void entropy_merge_kernel(EntArgs a, int64_t n_rows, const int32_t* cu, int B,
                                     int* status) {
    const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (r == 0 && cu != nullptr && (int64_t)cu[B] != n_rows) report(status, ESTP_ERR_INVALID_ARG);
    if (r >= n_rows) return;
    const int64_t w_lo = unit_owner(a.units, a.n_warps, r * a.nvec);
    const int64_t w_hi = unit_owner(a.units, a.n_warps, (r + 1) * a.nvec - 1);
    if (w_lo == w_hi) return;  // one warp covered the whole row and wrote H[r]
    float m = kMaskedLogit, s = 0.f, t = 0.f;
    for (int64_t w = w_lo; w <= w_hi; ++w) {
        const int64_t st = warp_start(a.units, a.n_warps, w);
        if (st == warp_start(a.units, a.n_warps, w + 1)) continue;  // empty range
        if (!in_bounds(w >= 0 && w < a.n_warps, status)) return;
        const EntPart p = a.part[w * 2 + (st / a.nvec == r ? 0 : 1)];
        merge(m, s, t, p.m, p.s, p.t);
    }
    a.H[r] = entropy_of(s, t);
}

}  // namespace

estp_status launch_entropy(estp_ctx* ctx, const void* logits, estp_dtype dtype, int64_t n_rows,
                           int64_t V, int64_t ld, const int32_t* cu, int32_t B, float* H,
                           cudaStream_t st) {
    const int per_unit = dtype == ESTP_BF16 ? 8 : 4;
    EntArgs a;
    a.base = static_cast<const char*>(logits);
    a.ld_bytes = ld * esize(dtype);
    a.nvec = (V + per_unit - 1) / per_unit;
    a.V = V;
    a.units = n_rows * a.nvec;
    int occ = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &occ, dtype == ESTP_BF16 ? entropy_kernel<true> : entropy_kernel<false>, kEntThreads, 0);
    if (e != cudaSuccess) return cuda_fail(e, "occupancy query");
    int64_t max_warps = (int64_t)ctx->num_sms * (occ > 0 ? occ : 1) * (kEntThreads / 32);
    a.n_warps = a.units < max_warps ? a.units : max_warps;
    estp_status s = ws_reserve(ctx, sizeof(EntPart) * 2 * (size_t)a.n_warps);
    if (s != ESTP_OK) return s;
    a.part = static_cast<EntPart*>(ctx->ws);
    a.H = H;
    a.status = ctx->status;
    const int64_t blocks = (a.n_warps + kEntThreads / 32 - 1) / (kEntThreads / 32);
    if (dtype == ESTP_BF16) entropy_kernel<true><<<(unsigned)blocks, kEntThreads, 0, st>>>(a);
    else entropy_kernel<false><<<(unsigned)blocks, kEntThreads, 0, st>>>(a);
    const int64_t mblocks = (n_rows + 255) / 256;
    entropy_merge_kernel<<<(unsigned)mblocks, 256, 0, st>>>(a, n_rows, cu, B, ctx->status);
    e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "entropy launch");
}

// ------------------------------------------------ allocation-free variant
// Token entropy for callers that cannot allocate device memory: a serving engine whose
// allocator already owns all of HBM (for its KV cache), or code running where
// cudaMalloc is not allowed.  The per-piece partials that estp_token_entropy keeps in
// the context workspace live here in one file-scope device array instead, so this path
// needs no context and allocates nothing.  Every call shares the array: calls that
// overlap on the GPU race on it.  No slot needs clearing: each is written before it is
// read within a call.
constexpr int64_t kNoAllocPieces = 4096;  // partial pairs the static scratch holds (128 KiB)
static __device__ __align__(256) EntPart g_noalloc_part[2 * kNoAllocPieces];

namespace {
struct NoAllocDevice {
    bool ready = false;
    EntPart* part = nullptr;  // device address of g_noalloc_part on this device
    int num_sms = 0;
};
std::mutex g_noalloc_mu;
NoAllocDevice g_noalloc_devices[64];
}  // namespace

// Once per device, with that device current: the device address of the static scratch
// (the host-side name g_noalloc_part is only a stand-in) and the SM count.
static estp_status noalloc_setup(int dev, NoAllocDevice* out) {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (dev < 0 || dev >= 64) return fail(ESTP_ERR_UNSUPPORTED, "device ordinal %d >= 64", dev);
    NoAllocDevice& d = g_noalloc_devices[dev];
    if (!d.ready) {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_part);
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(entropy scratch)");
        e = cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
        d.part = static_cast<EntPart*>(p);
        d.ready = true;
    }
    *out = d;
    return ESTP_OK;
}

estp_status launch_entropy_noalloc(const void* logits, estp_dtype dtype, int64_t n_rows, int64_t V,
                                   int64_t ld, float* H, cudaStream_t st) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    NoAllocDevice d;
    estp_status s = noalloc_setup(dev, &d);
    if (s != ESTP_OK) return s;
    const int per_unit = dtype == ESTP_BF16 ? 8 : 4;
    EntArgs a;
    a.base = static_cast<const char*>(logits);
    a.ld_bytes = ld * esize(dtype);
    a.nvec = (V + per_unit - 1) / per_unit;
    a.V = V;
    a.units = n_rows * a.nvec;
    int occ = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &occ, dtype == ESTP_BF16 ? entropy_kernel<true> : entropy_kernel<false>, kEntThreads, 0);
    if (e != cudaSuccess) return cuda_fail(e, "occupancy query");
    // The flat unit split is exact for any piece count >= 1, so a GPU with more resident
    // warps than the scratch has pieces runs with fewer, longer pieces.
    int64_t max_warps = (int64_t)d.num_sms * (occ > 0 ? occ : 1) * (kEntThreads / 32);
    if (max_warps > kNoAllocPieces) max_warps = kNoAllocPieces;
    a.n_warps = a.units < max_warps ? a.units : max_warps;
    a.part = d.part;
    a.H = H;
    a.status = nullptr;
    const int64_t blocks = (a.n_warps + kEntThreads / 32 - 1) / (kEntThreads / 32);
    if (dtype == ESTP_BF16) entropy_kernel<true><<<(unsigned)blocks, kEntThreads, 0, st>>>(a);
    else entropy_kernel<false><<<(unsigned)blocks, kEntThreads, 0, st>>>(a);
    const int64_t mblocks = (n_rows + 255) / 256;
    entropy_merge_kernel<<<(unsigned)mblocks, 256, 0, st>>>(a, n_rows, nullptr, 0, nullptr);
    e = cudaGetLastError();
    return e == cudaSuccess ? ESTP_OK : cuda_fail(e, "entropy launch");
}

}  // namespace estp

extern "C" estp_status estp_token_entropy_noalloc(const void* logits, estp_dtype dtype,
                                                  int64_t n_rows, int64_t V, int64_t ld,
                                                  float* entropy_out, estp_stream_t stream) {
    using namespace estp;
    ESTP_NVTX_RANGE("estp_token_entropy_noalloc");
    if (dtype != ESTP_F32 && dtype != ESTP_BF16) return fail(ESTP_ERR_INVALID_ARG, "dtype");
    if (n_rows < 0 || V < 1 || ld < V)
        return fail(ESTP_ERR_INVALID_ARG, "need n_rows >= 0, V >= 1, ld >= V");
    if (n_rows == 0) return ESTP_OK;
    if (!logits || !entropy_out) return fail(ESTP_ERR_INVALID_ARG, "NULL tensor pointer");
    if (!aligned16(logits) || (ld * esize(dtype)) % 16)
        return fail(ESTP_ERR_INVALID_ARG, "logits base and row stride must be 16-byte aligned");
    return launch_entropy_noalloc(logits, dtype, n_rows, V, ld, entropy_out,
                                  reinterpret_cast<cudaStream_t>(stream));
}
