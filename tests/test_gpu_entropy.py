"""K-ENT against the oracle (GPU)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import assert_entropy
from synth import device as sd
from synth import workloads as W

pytestmark = pytest.mark.gpu


def _tiny(dtype, V, seed=11, spike=0.0):
    return W.Workload("ent", seed=seed, B=1, T_lo=1, T_hi=1, dtype=dtype, V=V, n_layers_model=1,
                      layers_used=1, Hq=1, Hkv=1, d=64, D=8, spike_prob=spike)


@pytest.mark.parametrize("dtype", [synth.BF16, synth.F32])
@pytest.mark.parametrize("V,rows", [(1, 3), (7, 5), (8, 1), (64, 37), (1000, 300), (32000, 64),
                                    (152064, 24), (128256, 9), (50257, 33)])
def test_entropy_shapes(cuda_lib, dtype, V, rows):
    w = _tiny(dtype, V, spike=0.2)
    per = 8 if dtype == synth.BF16 else 4
    ld = (V + per - 1) // per * per
    ctx = cuda_lib.Context(0)
    x = sd.logits(w, 17, rows, ld=ld, pad_val=1e4)  # padding would dominate if read
    H = ctx.token_entropy(x, V=V)
    ctx.sync_status()
    ref = oracle.token_entropy(W.host_logits(w, np.arange(17, 17 + rows), ld=ld), V=V)
    assert_entropy(H.cpu().numpy(), ref)


def test_entropy_padded_rows_and_determinism(cuda_lib):
    w = _tiny(synth.BF16, 4001, spike=0.5)
    ctx = cuda_lib.Context(0)
    x = sd.logits(w, 0, 257, ld=4096 + 64, pad_val=-7.0)
    a = ctx.token_entropy(x, V=4001)
    b = ctx.token_entropy(x, V=4001)
    ctx.sync_status()
    assert torch.equal(a, b)
    ref = oracle.token_entropy(W.host_logits(w, np.arange(257), ld=4096 + 64), V=4001)
    assert_entropy(a.cpu().numpy(), ref)


def test_entropy_closed_forms(cuda_lib):
    ctx = cuda_lib.Context(0)
    for dt in (torch.float32, torch.bfloat16):
        x = torch.zeros(4, 152064, dtype=dt, device="cuda")
        x[1, 5] = 1e4
        x[2, [3, 100, 5000]] = 60.0
        H = ctx.token_entropy(x).cpu().numpy()
        assert abs(H[0] - np.log(152064)) < 1e-3 and abs(H[3] - np.log(152064)) < 1e-3
        assert abs(H[1]) < 1e-3 and abs(H[2] - np.log(3)) < 1e-3


def test_entropy_empty_and_cu_check(cuda_lib):
    ctx = cuda_lib.Context(0)
    x = torch.zeros(0, 64, dtype=torch.bfloat16, device="cuda")
    assert ctx.token_entropy(x).numel() == 0
    y = torch.randn(10, 64, device="cuda").to(torch.bfloat16)
    cu_ok = torch.tensor([0, 4, 10], dtype=torch.int32, device="cuda")
    ctx.token_entropy(y, cu_seqlens=cu_ok)
    ctx.sync_status()
    cu_bad = torch.tensor([0, 4, 9], dtype=torch.int32, device="cuda")
    ctx.token_entropy(y, cu_seqlens=cu_bad)
    with pytest.raises(cuda_lib.EstpError) as e:
        ctx.sync_status()
    assert e.value.status == cuda_lib.ESTP_ERR_INVALID_ARG
    ctx.sync_status()  # cleared


@pytest.mark.parametrize("w", [W.C1, W.C2], ids=lambda w: w.name)
def test_entropy_workload_full(cuda_lib, w):
    """Whole workload on the GPU; oracle on every row of the small case, on a seeded
    sample of rows (first, last, random) for the full-size one."""
    sumT = int(w.cu_seqlens()[-1])
    ctx = cuda_lib.Context(0)
    x = sd.logits(w, 0, sumT)
    H = ctx.token_entropy(x, cu_seqlens=sd.cu_seqlens(w)).cpu().numpy()
    ctx.sync_status()
    if sumT <= 512:
        rows = np.arange(sumT)
    else:
        rng = np.random.default_rng(0)
        rows = np.unique(np.concatenate([[0, 1, sumT - 1], rng.integers(0, sumT, 96)]))
    ref = oracle.token_entropy(W.host_logits(w, rows))
    assert_entropy(H[rows], ref)


@pytest.mark.parametrize("w", [W.C3, W.C4, W.C5], ids=lambda w: w.name)
def test_entropy_workload_chunk(cuda_lib, w):
    """Large workloads process the logits in row chunks; check one 4096-row chunk at an
    offset deep inside the workload on sampled rows."""
    sumT = int(w.cu_seqlens()[-1])
    row0 = sumT - 4096 - 1234
    ctx = cuda_lib.Context(0)
    x = sd.logits(w, row0, 4096)
    H = ctx.token_entropy(x).cpu().numpy()
    rows = np.unique(np.random.default_rng(1).integers(0, 4096, 48))
    ref = oracle.token_entropy(W.host_logits(w, row0 + rows))
    assert_entropy(H[rows], ref)
