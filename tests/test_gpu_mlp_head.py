"""The MLP predictor of Sec. 3.3 (one ReLU hidden layer in front of the K-bin softmax
projection of Eq. 3-2): prediction, the loss of Eqs. 3-1 / 3-3 and every gradient, against
the oracle (GPU).

Tolerance: as for the linear head (fp32 against the fp64 oracle, dot products of length
D or F), 1e-4 relative to the largest reference magnitude of each output.  A hidden unit
whose pre-activation is within rounding of 0 could take the ReLU's other branch in fp32,
so the inputs are drawn with every |a| > 1e-5 (the fp32 error of a is ~1e-7 here)."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

RTOL = 1e-4


def _close(gpu, ref, what, rtol=RTOL):
    gpu, ref = np.asarray(gpu, np.float64), np.asarray(ref, np.float64)
    scale = max(float(np.max(np.abs(ref))), 1e-30)
    err = float(np.max(np.abs(gpu - ref))) if ref.size else 0.0
    assert err <= rtol * scale, f"{what}: max err {err:.3e} vs scale {scale:.3e}"


def _case(B, D, F, K, seed=3, bias=True, width=256.0, spread=4.0):
    """Inputs with no hidden pre-activation near the ReLU's kink (|a| > 1e-5)."""
    for s in range(seed, seed + 50):
        rng = np.random.default_rng(s)
        h = rng.standard_normal((B, D)).astype(np.float32)
        W1 = (rng.standard_normal((F, D)) / np.sqrt(D)).astype(np.float32)
        b1 = (rng.standard_normal(F) * 0.3).astype(np.float32) if bias else None
        a = h.astype(np.float64) @ W1.T.astype(np.float64) + (0 if b1 is None else b1)
        if np.min(np.abs(a)) > 1e-5:
            break
    W2 = (rng.standard_normal((K, F)) * spread / np.sqrt(F)).astype(np.float32)
    b2 = rng.standard_normal(K).astype(np.float32) if bias else None
    c = ((np.arange(K) + 0.5) * width).astype(np.float32)
    y = rng.uniform(0, K * width, B).astype(np.float32)
    return h, W1, b1, W2, b2, c, y


def _dev(cuda_lib, W1, b1, W2, b2, c):
    cu = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()
    return cuda_lib.MlpHead(cu(W1), cu(b1), cu(W2), cu(b2), cu(c))


@pytest.mark.parametrize("lam", [0.0, 0.5, 1.0])
@pytest.mark.parametrize("B,D,F,K", [(16, 3584, 1024, 32), (1, 512, 64, 32), (5, 64, 7, 1),
                                     (3, 33, 300, 1000), (9, 100, 1, 5), (19, 130, 37, 3),
                                     (2, 64, 13000, 4)])
def test_mlp_loss_against_oracle(cuda_lib, B, D, F, K, lam):
    h, W1, b1, W2, b2, c, y = _case(B, D, F, K)
    ctx = cuda_lib.Context(0)
    head = _dev(cuda_lib, W1, b1, W2, b2, c)
    out = ctx.mlp_head_loss(torch.from_numpy(h).cuda(), head, torch.from_numpy(y).cuda(), lam)
    ctx.sync_status()
    got = [t.cpu().numpy() for t in out]
    ref = oracle.mlp_head_loss(h.astype(np.float64), W1, b1, W2, b2, c, y, lam)
    _close(got[0], [ref[0]], "loss")
    for name, g, r in zip(("dL/dW1", "dL/db1", "dL/dW2", "dL/db2", "dL/dpooled"), got[1:], ref[1:]):
        _close(g, r, name)


@pytest.mark.parametrize("B,D,F,K,bias", [(16, 3584, 1024, 32, True), (4, 256, 40, 1000, False),
                                          (2, 64, 3, 1, True)])
def test_mlp_predict_against_oracle(cuda_lib, B, D, F, K, bias):
    h, W1, b1, W2, b2, c, _ = _case(B, D, F, K, seed=11, bias=bias)
    ctx = cuda_lib.Context(0)
    pred, probs = ctx.mlp_head_predict(torch.from_numpy(h).cuda(), _dev(cuda_lib, W1, b1, W2, b2, c),
                                       probs=True)
    ctx.sync_status()
    y_ref, p_ref = oracle.mlp_length_head(h.astype(np.float64), W1, b1, W2, b2, c, return_probs=True)
    assert np.max(np.abs(pred.cpu().numpy() - y_ref)) <= 1.0, "predicted length (tokens)"
    _close(probs.cpu().numpy(), p_ref, "p_hat")


def test_mlp_partial_grads_deterministic_and_checked(cuda_lib):
    """Only some gradients requested (the rest are not written); the loss alone; identical
    bits on repeated calls; bad arguments refused on the host."""
    h, W1, b1, W2, b2, c, y = _case(8, 1024, 128, 32, seed=21)
    ctx = cuda_lib.Context(0)
    head = _dev(cuda_lib, W1, b1, W2, b2, c)
    hd, yd = torch.from_numpy(h).cuda(), torch.from_numpy(y).cuda()
    full = [t.cpu().numpy() for t in ctx.mlp_head_loss(hd, head, yd, 0.5)]
    full2 = [t.cpu().numpy() for t in ctx.mlp_head_loss(hd, head, yd, 0.5)]
    for u, v in zip(full, full2):
        assert np.array_equal(u, v)
    part = ctx.mlp_head_loss(hd, head, yd, 0.5, grads={"W2", "pooled"})
    assert part[1] is None and part[2] is None and part[4] is None
    assert np.array_equal(part[3].cpu().numpy(), full[3])
    assert np.array_equal(part[5].cpu().numpy(), full[5])
    top = ctx.mlp_head_loss(hd, head, yd, 0.5, grads={"b2"})
    assert np.array_equal(top[4].cpu().numpy(), full[4])
    loss_only = ctx.mlp_head_loss(hd, head, yd, 0.5, grads=False)
    ctx.sync_status()
    assert loss_only.cpu().numpy()[0] == full[0][0]
    with pytest.raises(cuda_lib.EstpError):
        ctx.mlp_head_loss(hd, head, yd, float("inf"))
    with pytest.raises(cuda_lib.EstpError):  # B = 0
        ctx.mlp_head_loss(hd[:0], head, yd[:0], 0.5)
    big = _dev(cuda_lib, W1, None, np.zeros((1025, 128), np.float32), None, np.zeros(1025, np.float32))
    with pytest.raises(cuda_lib.EstpError):  # K > 1024
        ctx.mlp_head_predict(hd, big)
