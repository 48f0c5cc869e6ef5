"""Sizes at the edge of what the workloads reach (GPU): a 65 536-token prompt, a
256 000-entry vocabulary, 4096 prompts in one call, and the smallest shapes (a single
token, a single vocabulary entry), each against the oracle."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import assert_entropy, assert_importance, assert_pooled
from synth import device as sd
from synth import workloads as W

pytestmark = pytest.mark.gpu


def _bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def test_importance_65536_token_prompt(cuda_lib):
    """One 65 536-token prompt (256 key-tile pairs, the largest column-sum item counts),
    4 heads of 2 KV groups, sink keys: S sums to 1 and its last 8 keys match the oracle
    (C_j needs only the rows i >= j)."""
    T, R = 65536, 8
    w = W.Workload("long64k", seed=51, B=1, T_lo=T, T_hi=T, dtype=synth.BF16, V=8,
                   n_layers_model=1, layers_used=1, Hq=4, Hkv=2, d=128, D=64, sinks=4)
    ctx = cuda_lib.Context(0)
    Q, K = sd.qk(w, 0)
    ctx.attn_importance(Q, K, sd.cu_seqlens(w), T)
    S = ctx.attn_importance_finalize(1, T).cpu().numpy()
    ctx.sync_status()
    assert np.all(np.isfinite(S)) and np.all(S >= 0) and abs(S.sum() - 1.0) < 1e-4
    Qp = np.zeros((T, w.Hq, w.d), dtype=np.uint16)
    Qp[T - R:] = _bits(Q[T - R:])
    sub = np.asarray([0, T], dtype=np.int32)
    C = oracle.attn_colsum_rows(Qp, _bits(K), sub, w.scale, T - R)
    assert_importance(S[T - R:], oracle.importance(C, sub, 1, w.Hq)[T - R:])
    ctx.close()


@pytest.mark.parametrize("V", [256000, 1])
def test_entropy_vocab_extremes(cuda_lib, V):
    w = W.Workload("vocab", seed=52, B=1, T_lo=37, T_hi=37, dtype=synth.BF16, V=V,
                   n_layers_model=1, layers_used=1, Hq=1, Hkv=1, d=64, D=64, spike_prob=0.05)
    ld = (V + 7) // 8 * 8
    x = sd.logits(w, 0, 37, ld=ld)
    ctx = cuda_lib.Context(0)
    H = ctx.token_entropy(x, V=V).cpu().numpy()
    ctx.sync_status()
    assert_entropy(H, oracle.token_entropy(_bits(x), V=V))
    if V == 1:
        assert np.max(np.abs(H)) < 1e-6  # a one-entry vocabulary has zero entropy
    ctx.close()


def test_many_prompts_and_single_tokens(cuda_lib):
    """4096 prompts of 0 to 3 tokens in one call of every stage: importance (a single
    token gets S = 1), entropy and pooling with the head."""
    rng = np.random.default_rng(53)
    lens = rng.integers(0, 4, 4096)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    sumT = int(cu[-1])
    w = W.Workload("tiny4096", seed=53, B=4096, T_lo=0, T_hi=3, dtype=synth.BF16, V=300,
                   n_layers_model=1, layers_used=1, Hq=4, Hkv=2, d=128, D=256)
    Q = sd.normal(w.key_q(0), (sumT, w.Hq, w.d), synth.BF16)
    K = sd.normal(w.key_k(0), (sumT, w.Hkv, w.d), synth.BF16)
    cu_d = torch.as_tensor(cu, device="cuda")
    ctx = cuda_lib.Context(0)
    ctx.attn_importance(Q, K, cu_d, 3)
    S = ctx.attn_importance_finalize(1, sumT).cpu().numpy()
    x = sd.logits(w, 0, sumT, ld=304)  # 300 entries in rows of 304 (16-byte stride)
    H = ctx.token_entropy(x, V=w.V, cu_seqlens=cu_d).cpu().numpy()
    hid = sd.normal(w.key(4), (sumT, w.D), synth.BF16)
    pooled, _ = ctx.pool(hid, torch.as_tensor(H, device="cuda"), torch.as_tensor(S, device="cuda"),
                         cu_d, w.lambda1, w.lambda2, w.alpha)
    ctx.sync_status()
    C = oracle.attn_colsum(_bits(Q), _bits(K), cu, w.scale)
    assert_importance(S, oracle.importance(C, cu, 1, w.Hq))
    one = np.nonzero(lens == 1)[0]
    assert np.all(np.abs(S[cu[one]] - 1.0) < 1e-5)  # a one-token prompt puts all mass on itself
    assert_entropy(H, oracle.token_entropy(_bits(x), V=w.V))
    ref = oracle.pool(_bits(hid), H, S, cu, w.lambda1, w.lambda2, w.alpha)
    P = pooled.cpu().numpy()
    empty = lens == 0
    assert np.all(P[empty] == 0)
    assert_pooled(P[~empty], ref[~empty])
    ctx.close()
