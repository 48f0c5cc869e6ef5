"""Seeded synthetic inputs shaped like the paper's workloads (host side).

This module holds none of ESTP's arithmetic.  It is the one piece shared by the
tests (which feed the oracle) and the bench / GPU tests (which feed the CUDA
library): the same counter-based generator is implemented here in numpy and in
``synth.cu`` for the device, and the two give bit-identical values.

Generator (published definitions, restated):
* SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): the n-th output (n >= 0) of the
  stream seeded with ``key`` is mix64(key + (n+1)*GAMMA) mod 2**64, with GAMMA =
  0x9E3779B97F4A7C15 and mix64 the variant-13 finaliser.
* Normal draws use the Irwin-Hall sum of twelve uniforms: the three words
  3n, 3n+1, 3n+2 give twelve 16-bit integers b_k, and
  z = (sum_k b_k + 6) / 2**16 - 6, exact in binary64 (mean 0, variance ~1).
* Uniforms on [0, 1) are (word >> 40) / 2**24, exact in binary64.
Values are formed exactly in binary64, rounded once to binary32 (RNE) and, for
bf16 tensors, rounded again from binary32 to bfloat16 (RNE).
"""
from __future__ import annotations

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 20

F32, BF16 = "f32", "bf16"


def mix64(z: np.ndarray) -> np.ndarray:
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def splitmix64(key, n) -> np.ndarray:
    """n-th output (vectorised over n) of SplitMix64 seeded with ``key``."""
    n = np.asarray(n, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return mix64(np.uint64(key) + (n + np.uint64(1)) * GAMMA)


def stream_key(seed: int, stream: int) -> int:
    """Key of an independent stream: output number ``stream`` of the seed's stream."""
    return int(splitmix64(np.uint64(seed), np.uint64(stream)))


def uniform24(key: int, n) -> np.ndarray:
    """Exact binary64 uniforms k / 2**24 from word n of the stream."""
    w = splitmix64(key, n)
    return (w >> np.uint64(40)).astype(np.float64) * (1.0 / (1 << 24))


def _splitmix64_inplace(key: int, n: np.ndarray) -> np.ndarray:
    """splitmix64(key, n) computed in the buffer n (uint64, overwritten)."""
    with np.errstate(over="ignore"):
        z = n
        z += np.uint64(1)
        z *= GAMMA
        z += np.uint64(key)
        z ^= z >> np.uint64(30)
        z *= _M1
        z ^= z >> np.uint64(27)
        z *= _M2
        z ^= z >> np.uint64(31)
    return z


def normal(key: int, idx) -> np.ndarray:
    """Irwin-Hall normal draws for element indices ``idx`` (exact binary64): the sum of
    the twelve 16-bit pieces of words 3 idx, 3 idx + 1 and 3 idx + 2."""
    idx = np.asarray(idx, dtype=np.uint64).reshape(-1)
    out = np.empty(idx.shape, dtype=np.float64)
    chunk = _CHUNK >> 2
    for s in range(0, idx.size, chunk):
        n3 = idx[s:s + chunk] * np.uint64(3)
        acc = np.zeros(n3.shape, dtype=np.int64)
        for k in range(3):
            w = _splitmix64_inplace(key, n3 + np.uint64(k))
            # the four 16-bit pieces of each word (their order does not matter for the sum)
            acc += w.view(np.uint16).reshape(-1, 4).sum(axis=1, dtype=np.int64)
        out[s:s + chunk] = (acc + 6).astype(np.float64) * (1.0 / 65536.0) - 6.0
    return out


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round binary32 to bfloat16 (nearest, ties to even); finite inputs."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))
    return (u >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_to(x64: np.ndarray, dtype: str) -> np.ndarray:
    """binary64 -> binary32 (RNE) -> bf16 bits (RNE) when dtype is bf16."""
    f = np.asarray(x64, dtype=np.float64).astype(np.float32)
    return f if dtype == F32 else f32_to_bf16_bits(f)


def as_float64(a: np.ndarray) -> np.ndarray:
    """Widen a generated array (f32, or uint16 bf16 bits) to float64 exactly."""
    if a.dtype == np.uint16:
        return bf16_bits_to_f32(a).astype(np.float64)
    return np.asarray(a, dtype=np.float64)


# ------------------------------------------------------------------ tensors

def normal_tensor(key: int, shape, dtype: str, idx0: int = 0, scale: float = 1.0) -> np.ndarray:
    """Tensor of N(0,1) draws (times ``scale`` in binary64) at flat indices idx0.."""
    count = int(np.prod(shape))
    z = normal(key, np.arange(idx0, idx0 + count, dtype=np.uint64))
    if scale != 1.0:
        z = z * scale
    return round_to(z, dtype).reshape(shape)


def logits_rows(key_vals: int, key_rows: int, rows, V: int, dtype: str, sigma_lo: float,
                sigma_hi: float, spike_prob: float = 0.0, spike_val: float = 0.0,
                ld: int | None = None, pad_val: float = 0.0) -> np.ndarray:
    """Logit rows (global row indices ``rows``) of the workload recipe:
    row r ~ N(0, sigma_r^2), sigma_r = lo + (hi - lo) u_r; with probability
    ``spike_prob`` one uniformly chosen vocabulary id gets ``spike_val`` added.
    Columns V..ld-1 hold ``pad_val`` (never part of the vocabulary)."""
    rows = np.asarray(rows, dtype=np.int64).reshape(-1)
    ld = V if ld is None else ld
    out = np.empty((rows.size, ld), dtype=np.float64)
    out[:, V:] = pad_val
    thr = spike_threshold(spike_prob)
    span = sigma_hi - sigma_lo
    for i, r in enumerate(rows):
        sigma = sigma_lo + span * float(uniform24(key_rows, 3 * int(r)))
        z = normal(key_vals, np.arange(int(r) * V, int(r) * V + V, dtype=np.uint64))
        x = z * sigma
        if thr:
            w1 = int(splitmix64(key_rows, 3 * int(r) + 1))
            if (w1 >> 40) < thr:
                pos = int(splitmix64(key_rows, 3 * int(r) + 2)) % V
                x[pos] = x[pos] + spike_val
        out[i, :V] = x
    return round_to(out, dtype)


def spike_threshold(p: float) -> int:
    return int(round(p * (1 << 24))) if p > 0 else 0
