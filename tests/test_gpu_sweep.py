"""Seeded random sweep of shapes against the oracle (GPU): combinations of ragged prompt
lengths (empty prompts included), GQA ratios, head dims, head subsets, vocabulary and
hidden sizes that the hand-picked cases of the other files do not cover one by one,
and the same for the fused prefill forward.
Tolerances are the parity bar's (tests/gpu_util.py)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import assert_entropy, assert_importance, assert_pooled
from synth import device as sd
from test_gpu_importance import _run, _wl

pytestmark = pytest.mark.gpu


def _lens(rng, B, hi):
    lens = rng.integers(0, hi, B)
    lens[rng.integers(0, B)] = max(1, int(lens.max()))  # at least one token
    return [int(x) for x in lens]


@pytest.mark.parametrize("seed", range(48))
def test_sweep_importance(cuda_lib, seed):
    """Random (lengths, Hq / Hkv, d, head subset, self term, divisor), bf16 on the tensor
    cores, two layers accumulated."""
    rng = np.random.default_rng(1000 + seed)
    Hkv = int(rng.choice([1, 2, 4]))
    Hq = Hkv * int(rng.choice([1, 2, 7]))
    d = int(rng.choice([64, 128]))
    lens = _lens(rng, int(rng.integers(1, 6)), int(rng.choice([40, 300, 900])))
    heads = None
    if rng.random() < 0.5 and Hq > 1:
        heads = sorted(int(h) for h in rng.choice(Hq, int(rng.integers(1, Hq + 1)), replace=False))
    exclude_self = bool(rng.random() < 0.3)
    divisor = str(rng.choice(["length", "causal", "none"]))
    w, cu = _wl(synth.BF16, lens, Hq, Hkv, d, seed=seed + 50)
    S, ref = _run(cuda_lib, w, cu, [0, 1], heads=heads, exclude_self=exclude_self,
                  divisor=divisor)
    assert_importance(S, ref)


@pytest.mark.parametrize("seed", range(24))
def test_sweep_entropy(cuda_lib, seed):
    """Random rows, vocabulary (not a multiple of anything) and row stride, bf16 and fp32."""
    rng = np.random.default_rng(2000 + seed)
    rows = int(rng.integers(1, 400))
    V = int(rng.integers(1, 70000))
    dtype = synth.BF16 if seed % 2 == 0 else synth.F32
    per16 = 8 if dtype == synth.BF16 else 4
    ld = V + int(rng.integers(0, 3)) * per16
    ld = (ld + per16 - 1) // per16 * per16  # 16-byte rows
    key = synth.stream_key(seed, 31)
    big = sd.normal(key, (rows, ld), dtype, scale=float(rng.choice([0.5, 3.0, 20.0])))
    ctx = cuda_lib.Context(0)
    H = ctx.token_entropy(big, V=V)
    ctx.sync_status()
    host = big.view(torch.int16).cpu().numpy().view(np.uint16) if dtype == synth.BF16 \
        else big.cpu().numpy()
    assert_entropy(H.cpu().numpy(), oracle.token_entropy(host, V=V))


@pytest.mark.parametrize("seed", range(24))
def test_sweep_pool(cuda_lib, seed):
    """Random lengths (empty prompts included), hidden size and mix, bf16, with the head."""
    rng = np.random.default_rng(3000 + seed)
    lens = _lens(rng, int(rng.integers(1, 9)), int(rng.choice([3, 200, 3000])))
    D = int(rng.choice([8, 64, 1000, 3584, 5000]))
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    sumT = int(cu[-1])
    hid = sd.normal(synth.stream_key(seed, 32), (sumT, D), synth.BF16)
    H = rng.uniform(0, 11, sumT).astype(np.float32)
    S = rng.uniform(0, 1, sumT).astype(np.float32)
    mix = (float(rng.uniform(0, 5)), float(rng.uniform(0, 2)), float(rng.choice([0.1, 1.0, 4.0])))
    K = int(rng.choice([1, 32, 300]))
    Wt = (rng.standard_normal((K, D)) / np.sqrt(D) * 10).astype(np.float32)
    b = rng.standard_normal(K).astype(np.float32)
    c = ((np.arange(K) + 0.5) * 64).astype(np.float32)
    ctx = cuda_lib.Context(0)
    head = cuda_lib.Head(torch.from_numpy(Wt).cuda(), torch.from_numpy(b).cuda(),
                         torch.from_numpy(c).cuda())
    pooled, pred = ctx.pool(hid, torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda(),
                            torch.as_tensor(cu, device="cuda"), *mix, head=head)
    ctx.sync_status()
    hb = hid.view(torch.int16).cpu().numpy().view(np.uint16)
    P_ref = oracle.pool(hb, H.astype(np.float64), S.astype(np.float64), cu, *mix)
    assert_pooled(pooled.cpu().numpy(), P_ref)
    y_ref = oracle.length_head(P_ref, Wt, b, c)
    assert np.max(np.abs(pred.cpu().numpy() - y_ref)) <= 1.0


@pytest.mark.parametrize("seed", range(24))
def test_sweep_lm_head(cuda_lib, seed):
    """Random rows, hidden size (a multiple of 64) and vocabulary for the entropy formed
    from hidden states."""
    rng = np.random.default_rng(4000 + seed)
    rows = int(rng.integers(1, 300))
    D = 64 * int(rng.integers(1, 17))
    V = int(rng.integers(1, 8000))
    spread = float(rng.choice([0.5, 3.0, 12.0]))
    h = sd.normal(synth.stream_key(seed, 33), (rows, D), synth.BF16)
    W = sd.normal(synth.stream_key(seed, 34), (V, D), synth.BF16, scale=spread / np.sqrt(D))
    ctx = cuda_lib.Context(0)
    H = ctx.lm_head_entropy(h, W)
    ctx.sync_status()
    bits = lambda t: t.view(torch.int16).cpu().numpy().view(np.uint16)
    assert_entropy(H.cpu().numpy(), oracle.lm_head_entropy(bits(h), bits(W)))


@pytest.mark.parametrize("seed", range(24))
def test_sweep_attn_forward(cuda_lib, seed):
    """Random lengths (empty prompts included), GQA ratio, self term, divisor, lse supplied
    or computed, one or two layers through the fused forward (bf16, d 128)."""
    from test_gpu_attn_forward import _run as _run_fwd
    rng = np.random.default_rng(5000 + seed)
    Hkv = int(rng.choice([1, 2, 4]))
    Hq = Hkv * int(rng.choice([1, 3, 7]))
    lens = _lens(rng, int(rng.integers(1, 7)), int(rng.choice([40, 300, 1500])))
    w, cu = _wl(synth.BF16, lens, Hq, Hkv, 128, seed=seed + 70)
    layers = [0] if rng.random() < 0.5 else [0, 1]
    S, ref = _run_fwd(cuda_lib, w, cu, layers, exclude_self=bool(rng.random() < 0.3),
                      supply_lse=bool(rng.random() < 0.5),
                      divisor=str(rng.choice(["length", "causal", "none"])))
    assert_importance(S, ref)
