"""The seeded generator on the host (CPU only)."""
import numpy as np
import torch

import synth
from synth import workloads as W


def test_splitmix64_published_outputs():
    # First outputs of SplitMix64 seeded with 0, as printed by the reference C
    # implementation of the generator (Steele, Lea & Flood 2014; Vigna's splitmix64.c).
    out = synth.splitmix64(0, np.arange(3))
    assert [int(x) for x in out] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_normal_moments_and_exactness():
    z = synth.normal(12345, np.arange(1 << 18))
    assert abs(z.mean()) < 0.01 and abs(z.var() - 1.0) < 0.01
    assert z.min() >= -6 and z.max() <= 6
    # values lie on the 2**-16 grid (integer-exact construction)
    assert np.all(z * 65536 == np.round(z * 65536))


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(100000) * rng.uniform(0.1, 100, 100000)).astype(np.float32)
    x[:4] = [1.0 + 2**-8, 1.0 + 3 * 2**-8, -(1.0 + 2**-8), 0.0]  # ties go to even
    ours = synth.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_workload_lengths_and_determinism():
    for w in W.ORDER:
        T = w.seqlens()
        assert len(T) == w.B and T.min() >= w.T_lo and T.max() <= w.T_hi
        assert np.array_equal(T, w.seqlens())
    cu = W.C2.cu_seqlens()
    assert 16 * 256 <= cu[-1] <= 16 * 2048
    a = W.host_logits(W.C2, [0, 5, 17])
    assert a.dtype == np.uint16 and a.shape == (3, W.C2.V)
    assert np.array_equal(a, W.host_logits(W.C2, [0, 5, 17]))
    assert np.array_equal(a[1], W.host_logits(W.C2, [5])[0])


def test_logit_recipe_structure():
    w = W.C2
    rows = np.arange(400)
    thr = synth.spike_threshold(w.spike_prob)
    spikes = [(int(synth.splitmix64(w.key(W.S_LOGIT_ROWS), 3 * r + 1)) >> 40) < thr for r in rows]
    assert 0 < sum(spikes) < 20  # ~1% of rows
    r = int(np.nonzero(spikes)[0][0])
    x = W.host_logits(w, [r])[0]
    pos = int(synth.splitmix64(w.key(W.S_LOGIT_ROWS), 3 * r + 2)) % w.V
    sigma = w.sigma_lo + (w.sigma_hi - w.sigma_lo) * float(synth.uniform24(w.key(W.S_LOGIT_ROWS), 3 * r))
    z = synth.normal(w.key(W.S_LOGIT_VALS), [r * w.V + pos, r * w.V + pos + 1])
    assert x[pos] == synth.round_to(np.asarray([z[0] * sigma + 12.0]), "bf16")[0]
    assert x[pos + 1] == synth.round_to(np.asarray([z[1] * sigma]), "bf16")[0]


def test_sinks_scaled():
    w = W.Workload("tiny", seed=9, B=2, T_lo=6, T_hi=6, dtype=synth.BF16, V=8,
                   n_layers_model=1, layers_used=1, Hq=2, Hkv=1, d=8, D=8, sinks=2)
    _, K = W.host_qk(w, 0)
    plain = synth.round_to(synth.normal(w.key_k(0), np.arange(12 * 8)), "bf16").reshape(12, 1, 8)
    Kf, Pf = synth.as_float64(K), synth.as_float64(plain)
    sink = [0, 1, 6, 7]
    assert np.array_equal(Kf[sink], 8 * Pf[sink])
    rest = [i for i in range(12) if i not in sink]
    assert np.array_equal(Kf[rest], Pf[rest])


def test_normal_matches_scalar_definition():
    # Irwin-Hall normal of index i: the twelve 16-bit pieces of SplitMix64 words 3i, 3i+1
    # and 3i+2, summed, plus 6, times 2**-16, minus 6 -- evaluated with Python integers.
    def word(key, n):
        z = (key + (n + 1) * 0x9E3779B97F4A7C15) & (2**64 - 1)
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & (2**64 - 1)
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & (2**64 - 1)
        return z ^ (z >> 31)

    key = synth.stream_key(5, 77)
    idx = [0, 1, 2, 1000, 123456789, (1 << 40) + 3]
    want = []
    for i in idx:
        acc = sum((word(key, 3 * i + k) >> (16 * c)) & 0xFFFF for k in range(3) for c in range(4))
        want.append((acc + 6) / 65536.0 - 6.0)
    assert list(synth.normal(key, idx)) == want
