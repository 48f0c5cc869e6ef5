"""Full-size importance, entropy, fused attention forward and pooling on the large
workloads (GPU).

The GPU runs the whole workload: every prompt, every selected layer and head, in
per-layer calls that accumulate, as a caller streaming one layer's Q/K at a time
would.  Checks: S is finite, non-negative and sums to 1 over every prompt (any size);
the last keys of one prompt match the oracle exactly, because C_j needs only the
rows i >= j; and every key of one whole long prompt (its sink keys included) matches
the oracle for one or two layers.  The oracle reads the inputs of a prompt back from
the device: the device generator writes the same bits as the host one
(test_gpu_synth), and host-side generation of these sizes would take minutes."""
import os

import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_entropy, assert_importance, assert_pooled, assert_pred
from synth import device as sd
from synth import workloads as W

pytestmark = pytest.mark.gpu


def _bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("w,R", [(W.C3, 8), (W.C4, 16), (W.C5, 4)], ids=lambda x: getattr(x, "name", str(x)))
def test_importance_full_size(cuda_lib, w, R):
    cu = w.cu_seqlens()
    sumT = int(cu[-1])
    lens = np.diff(cu)
    maxT = int(lens.max())
    b = int(np.argmax(lens)) if w.B > 8 else w.B - 1
    t0, t1 = int(cu[b]), int(cu[b + 1])
    T = t1 - t0
    ctx = cuda_lib.Context(0)
    cu_d = sd.cu_seqlens(w)
    C = np.zeros(T)
    sub = np.asarray([0, T], dtype=np.int32)
    for n, layer in enumerate(w.layers):
        Q, K = sd.qk(w, layer)
        ctx.attn_importance(Q, K, cu_d, maxT, accumulate=n > 0)
        Qp = np.zeros((T, w.Hq, w.d), dtype=np.uint16)
        Qp[T - R:] = _bits(Q[t1 - R:t1])
        Kp = _bits(K[t0:t1])
        oracle.attn_colsum_rows(Qp, Kp, sub, w.scale, T - R, out=C)
        del Q, K
    S = ctx.attn_importance_finalize(len(w.layers), sumT).cpu().numpy()
    ctx.sync_status()
    assert np.all(np.isfinite(S)) and np.all(S >= 0)
    sums = np.add.reduceat(S.astype(np.float64), cu[:-1])
    assert np.max(np.abs(sums - 1.0)) < 1e-4, sums
    ref = oracle.importance(C, sub, len(w.layers), w.Hq)[T - R:]
    assert_importance(S[t1 - R:t1], ref)


def _spread_heads(Hq: int, n: int) -> list[int]:
    """n query heads spread evenly over 0..Hq-1 (every KV group when n >= Hkv)."""
    return sorted({int(round(x)) for x in np.linspace(0, Hq - 1, min(n, Hq))})


@pytest.mark.parametrize("w,n_layers,all_heads", [(W.C3, 1, False), (W.C4, 2, True),
                                                  (W.C5, 2, False)],
                         ids=lambda x: getattr(x, "name", str(x)))
def test_importance_whole_long_prompt(cuda_lib, w, n_layers, all_heads):
    """Eq. 2-0 for EVERY key of one whole long prompt against the oracle, element by
    element: the last 32768-token prompt of the long-context batch, the longest prompt of
    the RL batch and the last 8192-token prompt of the 70B batch.  Their sink keys (K x 8,
    positions 0-3), which draw most of the attention mass, and the many column-sum chunks
    per key tile that only long prompts produce are compared like every other key.  The
    GPU runs the whole batch (every prompt) for the last n_layers layers; the heads are
    all Hq (RL batch, as the bench launches it) or one per host thread spread over every
    KV group (the oracle forms one (prompt, head) softmax per thread)."""
    cu = w.cu_seqlens()
    sumT = int(cu[-1])
    lens = np.diff(cu)
    maxT = int(lens.max())
    b = int(np.argmax(lens[::-1]))
    b = w.B - 1 - b  # the last of the longest prompts
    t0, t1 = int(cu[b]), int(cu[b + 1])
    T = t1 - t0
    heads = list(range(w.Hq)) if all_heads else _spread_heads(w.Hq, os.cpu_count() or 1)
    layers = w.layers[-n_layers:]
    ctx = cuda_lib.Context(0)
    cu_d = sd.cu_seqlens(w)
    C = np.zeros(T)
    sub = np.asarray([0, T], dtype=np.int32)
    for n, layer in enumerate(layers):
        Q, K = sd.qk(w, layer)
        ctx.attn_importance(Q, K, cu_d, maxT, heads=None if all_heads else heads,
                            accumulate=n > 0)
        Qp, Kp = _bits(Q[t0:t1]), _bits(K[t0:t1])
        del Q, K
        oracle.attn_colsum(Qp, Kp, sub, w.scale, heads=heads, out=C)
    S = ctx.attn_importance_finalize(len(layers), sumT).cpu().numpy()
    ctx.sync_status()
    assert np.all(np.isfinite(S)) and np.all(S >= 0)
    sums = np.add.reduceat(S.astype(np.float64), cu[:-1])
    assert np.max(np.abs(sums - 1.0)) < 1e-4, sums
    ref = oracle.importance(C, sub, len(layers), len(heads))
    assert_importance(S[t0:t1], ref)
    if w.sinks:  # the sink keys draw far more than a typical key's share
        assert np.max(ref[:w.sinks]) > 10 * np.median(ref)


@pytest.mark.parametrize("w", [W.C3, W.C4, W.C5], ids=lambda w: w.name)
def test_entropy_full_size(cuda_lib, w):
    """Eq. 2-1 over every row of the whole workload's logits in one call, as the bench
    launches it (40 / 136 / 17 GB of bf16 logits); 256 rows spread over the batch (first,
    last, evenly spaced and random) against the oracle, every row finite and within
    [0, ln V]."""
    sumT = int(w.cu_seqlens()[-1])
    ctx = cuda_lib.Context(0)
    x = sd.logits(w, 0, sumT)
    H = ctx.token_entropy(x, cu_seqlens=sd.cu_seqlens(w)).cpu().numpy()
    ctx.sync_status()
    assert np.all(np.isfinite(H)) and H.min() >= 0 and H.max() <= np.log(w.V) + 1e-3
    rng = np.random.default_rng(11)
    rows = np.unique(np.concatenate([[0, 1, sumT - 2, sumT - 1],
                                     np.linspace(0, sumT - 1, 124).round().astype(np.int64),
                                     rng.integers(0, sumT, 128)]))
    idx = torch.as_tensor(rows, device=x.device)
    xr = _bits(x.index_select(0, idx))
    del x
    assert_entropy(H[rows], oracle.token_entropy(xr))


@pytest.mark.parametrize("w,R", [(W.C2, 8), (W.C3, 4), (W.C4, 8), (W.C5, 4)],
                         ids=lambda x: getattr(x, "name", str(x)))
def test_forward_full_size(cuda_lib, w, R):
    """The fused forward (estp_attn_forward_importance) over every selected layer of the
    whole workload, row normalisers computed by the call, as the bench launches it. S is
    finite, non-negative and sums to 1 over every prompt; the last R query rows of one
    prompt (its O) and its last R keys (their importance) match the oracle."""
    from test_gpu_attn_forward import O_TOL
    import synth
    cu = w.cu_seqlens()
    sumT = int(cu[-1])
    lens = np.diff(cu)
    maxT = int(lens.max())
    b = int(np.argmax(lens))
    t0, t1 = int(cu[b]), int(cu[b + 1])
    T = t1 - t0
    ctx = cuda_lib.Context(0)
    cu_d = sd.cu_seqlens(w)
    C = np.zeros(T)
    sub = np.asarray([0, T], dtype=np.int32)
    for n, layer in enumerate(w.layers):
        Q, K = sd.qk(w, layer)
        V = sd.normal(w.key_v(layer), (sumT, w.Hkv, w.d), synth.BF16)
        O = ctx.attn_forward_importance(Q, K, V, cu_d, maxT, accumulate=n > 0)
        Qp = np.zeros((T, w.Hq, w.d), dtype=np.uint16)
        Qp[T - R:] = _bits(Q[t1 - R:t1])
        Kp, Vp = _bits(K[t0:t1]), _bits(V[t0:t1])
        oracle.attn_colsum_rows(Qp, Kp, sub, w.scale, T - R, out=C)
        if n == len(w.layers) - 1:
            O_ref = oracle.attn_output_rows(Qp, Kp, Vp, sub, w.scale, T - R)[T - R:]
            O_gpu = O[t1 - R:t1].float().cpu().numpy()
            vmax = float(np.max(np.abs(synth.bf16_bits_to_f32(Vp))))
            err = float(np.max(np.abs(O_gpu - O_ref)))
            assert err <= O_TOL * vmax, f"O max abs err {err:.3e} (max|V| {vmax:.3e})"
        del Q, K, V, O
    S = ctx.attn_importance_finalize(len(w.layers), sumT).cpu().numpy()
    ctx.sync_status()
    assert np.all(np.isfinite(S)) and np.all(S >= 0)
    sums = np.add.reduceat(S.astype(np.float64), cu[:-1])
    assert np.max(np.abs(sums - 1.0)) < 1e-4, sums
    ref = oracle.importance(C, sub, len(w.layers), w.Hq)[T - R:]
    assert_importance(S[t1 - R:t1], ref)


@pytest.mark.parametrize("w", [W.C3, W.C5], ids=lambda w: w.name)
def test_pool_full_size(cuda_lib, w):
    cu = w.cu_seqlens()
    sumT = int(cu[-1])
    rng = np.random.default_rng(4)
    H = rng.uniform(0, 12, sumT).astype(np.float32)
    S = (rng.uniform(0, 2, sumT) / np.repeat(np.diff(cu), np.diff(cu))).astype(np.float32)
    ctx = cuda_lib.Context(0)
    Wt, bias, c = w.head_params()
    head = cuda_lib.Head(torch.from_numpy(Wt).cuda(), torch.from_numpy(bias).cuda(),
                         torch.from_numpy(c).cuda())
    hid = sd.hidden(w)
    pooled, pred = ctx.pool(hid, torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda(),
                            sd.cu_seqlens(w), w.lambda1, w.lambda2, w.alpha, head=head)
    ctx.sync_status()
    for b in (0, w.B - 1):
        rows = slice(int(cu[b]), int(cu[b + 1]))
        sub = np.asarray([0, int(cu[b + 1] - cu[b])], dtype=np.int32)
        P = oracle.pool(_bits(hid[rows]), H[rows], S[rows], sub, w.lambda1, w.lambda2, w.alpha)
        assert_pooled(pooled[b:b + 1].cpu().numpy(), P)
        assert_pred(pred[b:b + 1].cpu().numpy(), oracle.length_head(P, Wt, bias, c))
