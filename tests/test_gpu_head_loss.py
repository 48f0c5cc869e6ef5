"""Soft-label loss of the length head (Eqs. 3-1 to 3-3) and its gradients against the
oracle (GPU).

Tolerance: the kernels work in fp32 against the fp64 oracle.  The logits are fp32 dot
products of length D (relative error ~sqrt(D) * 2^-24, below 1e-5 for D <= 8192), the
softmax and the expectation add a few ulp, so the loss and every gradient are held to
1e-4 relative to the largest reference magnitude of that output."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

RTOL = 1e-4


def _close(gpu, ref, what):
    gpu, ref = np.asarray(gpu, np.float64), np.asarray(ref, np.float64)
    scale = max(float(np.max(np.abs(ref))), 1e-30)
    err = float(np.max(np.abs(gpu - ref))) if ref.size else 0.0
    assert err <= RTOL * scale, f"{what}: max err {err:.3e} vs scale {scale:.3e}"


def _case(B, D, K, seed=7, bias=True, width=256.0, spread=1.0):
    rng = np.random.default_rng(seed)
    pooled = rng.standard_normal((B, D)).astype(np.float32)
    W = (rng.standard_normal((K, D)) * spread / np.sqrt(D)).astype(np.float32)
    b = rng.standard_normal(K).astype(np.float32) if bias else None
    c = ((np.arange(K) + 0.5) * width).astype(np.float32)
    y = rng.uniform(0, K * width, B).astype(np.float32)
    return pooled, W, b, c, y


def _run(cuda_lib, pooled, W, b, c, y, lam, grads=True):
    ctx = cuda_lib.Context(0)
    cu = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()
    head = cuda_lib.Head(cu(W), cu(b), cu(c))
    out = ctx.head_loss(cu(pooled), head, cu(y), lam, grads=grads)
    ctx.sync_status()
    return [None if t is None else t.cpu().numpy() for t in (out if grads else (out,))]


@pytest.mark.parametrize("lam", [0.0, 0.5, 1.0])
@pytest.mark.parametrize("B,D,K", [(16, 3584, 32), (1, 1024, 32), (5, 4096, 1), (3, 33, 1000)])
def test_head_loss_against_oracle(cuda_lib, B, D, K, lam):
    pooled, W, b, c, y = _case(B, D, K, spread=20.0)
    loss, gW, gb, gp = _run(cuda_lib, pooled, W, b, c, y, lam)
    ref, rW, rb, rp = oracle.head_loss(pooled.astype(np.float64), W, b, c, y, lam)
    _close(loss, [ref], "loss")
    _close(gW, rW, "dL/dW")
    _close(gb, rb, "dL/dbias")
    _close(gp, rp, "dL/dpooled")


def test_head_loss_edge_cases(cuda_lib):
    """No bias; targets on a tie between two centres (the lower bin), below the first
    and beyond the last centre; only the loss requested (NULL gradients)."""
    pooled, W, _, c, _ = _case(4, 512, 16, seed=9, bias=False, width=10.0, spread=5.0)
    y = np.asarray([10.0, -3.0, 1e4, 70.0], np.float32)  # centres 5, 15, ...: 10 and 70 tie
    for lam in (0.2, 1.0):
        loss, gW, gb, gp = _run(cuda_lib, pooled, W, None, c, y, lam)
        ref, rW, rb, rp = oracle.head_loss(pooled.astype(np.float64), W, None, c, y, lam)
        _close(loss, [ref], "loss")
        _close(gW, rW, "dL/dW")
        _close(gb, rb, "dL/dbias")
        _close(gp, rp, "dL/dpooled")
        (loss_only,) = _run(cuda_lib, pooled, W, None, c, y, lam, grads=False)
        assert loss_only[0] == loss[0]


def test_head_loss_deterministic_and_checked(cuda_lib):
    """Fixed-order sums: two calls give identical bits.  Bad arguments are refused on
    the host before any launch."""
    pooled, W, b, c, y = _case(16, 3584, 32, seed=11)
    a = _run(cuda_lib, pooled, W, b, c, y, 0.5)
    a2 = _run(cuda_lib, pooled, W, b, c, y, 0.5)
    for u, v in zip(a, a2):
        assert np.array_equal(u, v)
    ctx = cuda_lib.Context(0)
    cu = lambda x: torch.from_numpy(x).cuda()
    head = cuda_lib.Head(cu(W), cu(b), cu(c))
    with pytest.raises(cuda_lib.EstpError):
        ctx.head_loss(cu(pooled), head, cu(y), float("nan"))
    with pytest.raises(cuda_lib.EstpError):  # B = 0
        ctx.head_loss(cu(pooled[:0]), head, cu(y[:0]), 0.5)
    big = cuda_lib.Head(cu(np.zeros((1025, 8), np.float32)), None, cu(np.zeros(1025, np.float32)))
    with pytest.raises(cuda_lib.EstpError):  # K > 1024
        ctx.head_loss(cu(np.zeros((2, 8), np.float32)), big, cu(np.zeros(2, np.float32)), 0.5)
