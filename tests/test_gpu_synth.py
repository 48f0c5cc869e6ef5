"""Device and host generators give identical bits (GPU)."""
import numpy as np
import pytest
import torch

import synth
from synth import device as sd
from synth import workloads as W

pytestmark = pytest.mark.gpu


def _bits(t):
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy()


@pytest.mark.parametrize("dtype", [synth.BF16, synth.F32])
def test_normal_bits(cuda_lib, dtype):
    key = synth.stream_key(5, 77)
    g = sd.normal(key, (3000,), dtype, idx0=123456789, scale=0.25)
    h = synth.round_to(synth.normal(key, np.arange(123456789, 123456789 + 3000)) * 0.25, dtype)
    assert np.array_equal(_bits(g), h)


@pytest.mark.parametrize("w", [W.C1, W.C2, W.C4], ids=lambda w: w.name)
def test_logit_rows_bits(cuda_lib, w):
    rows = [0, 3, 401, 499]
    ld = w.V + (8 if w.dtype == synth.BF16 else 4)
    g = sd.logits(w, 1000, 500, ld=ld)
    for r in rows:
        h = W.host_logits(w, [1000 + r], ld=ld)[0]
        assert np.array_equal(_bits(g[r]), h), r


def test_qk_and_hidden_bits(cuda_lib):
    w = W.Workload("t", seed=3, B=3, T_lo=5, T_hi=40, dtype=synth.BF16, V=8, n_layers_model=2,
                   layers_used=2, Hq=4, Hkv=2, d=64, D=96, sinks=2)
    Q, K = sd.qk(w, 1)
    Qh, Kh = W.host_qk(w, 1)
    assert np.array_equal(_bits(Q), Qh) and np.array_equal(_bits(K), Kh)
    sumT = int(w.cu_seqlens()[-1])
    assert np.array_equal(_bits(sd.hidden(w)), W.host_hidden(w, np.arange(sumT)))
