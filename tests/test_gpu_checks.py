"""The bounds-checked build (GPU).

libestp_checks.so is the library compiled with -DESTP_CHECKS: the kernels check the
indices of their global accesses and record ESTP_ERR_BOUNDS in the status word instead
of making an access outside a buffer.  On valid inputs no check may fire, and the checks
change no arithmetic: every output equals the release build's bit for bit.  The whole
feature path runs through it (entropy, row normalisers, column sums on both paths, the
fused forward, pooling with the head, the allocation-free entropy)."""
import ctypes

import numpy as np
import pytest
import torch

import synth
from synth import device as sd
from synth import workloads as W

pytestmark = pytest.mark.gpu


def _run(estp, library, w, dtype_q):
    cu = w.cu_seqlens()
    sumT, maxT = int(cu[-1]), int(np.diff(cu).max())
    ctx = estp.Context(0, library=library)
    cu_d = sd.cu_seqlens(w)
    ld = (w.V + 7) // 8 * 8 + 8  # padded rows, 16-byte row stride
    x = sd.logits(w, 0, sumT, ld=ld, pad_val=3.0)
    out = {"H": ctx.token_entropy(x, V=w.V, cu_seqlens=cu_d)}
    Q, K = sd.qk(w, w.layers[0])
    Q, K = Q.to(dtype_q), K.to(dtype_q)
    out["lse"] = ctx.attn_lse(Q, K, cu_d, maxT).clone()
    ctx.attn_importance(Q, K, cu_d, maxT, heads=[0, w.Hq - 1])  # row normalisers inside
    ctx.attn_importance(Q, K, cu_d, maxT, lse=out["lse"], heads=[0, w.Hq - 1], accumulate=True)
    out["S_subset"] = ctx.attn_importance_finalize(2, sumT)
    ctx.sync_status()
    ctx2 = estp.Context(0, library=library)
    ctx2.attn_importance(Q, K, cu_d, maxT, lse=out["lse"])
    out["S"] = ctx2.attn_importance_finalize(1, sumT)
    if dtype_q == torch.bfloat16 and w.d == 128:
        V = sd.normal(w.key_v(w.layers[0]), (sumT, w.Hkv, w.d), synth.BF16)
        out["O"] = ctx2.attn_forward_importance(Q, K, V, cu_d, maxT, lse=out["lse"])
        out["S_fwd"] = ctx2.attn_importance_finalize(1, sumT)
    Wt, b, c = sd.head(w)
    pooled, pred = ctx2.pool(sd.hidden(w), out["H"], out["S"], cu_d, w.lambda1, w.lambda2,
                             w.alpha, head=estp.Head(Wt, b, c))
    out["pooled"], out["pred"] = pooled, pred
    Hn = torch.full((sumT,), float("nan"), device="cuda")
    rc = library.estp_token_entropy_noalloc(ctypes.c_void_p(x.data_ptr()), estp.ESTP_BF16, sumT,
                                            w.V, ld, ctypes.c_void_p(Hn.data_ptr()), None)
    assert rc == estp.ESTP_OK
    out["H_noalloc"] = Hn
    ctx.sync_status()  # raises EstpError(ESTP_ERR_BOUNDS) if any check fired
    ctx2.sync_status()
    torch.cuda.synchronize()
    res = {k: v.cpu() for k, v in out.items() if v is not None}
    ctx.close()
    ctx2.close()
    return res


@pytest.mark.parametrize("dtype_q", [torch.bfloat16, torch.float32], ids=["tensor_cores", "fp32"])
def test_checked_build_matches_release_bitwise(cuda_lib, dtype_q):
    estp = cuda_lib
    checked = estp.load_library(estp.CHECKS_LIB_PATH)
    w = W.Workload("checks", seed=33, B=5, T_lo=0, T_hi=700, dtype=synth.BF16, V=3001,
                   n_layers_model=1, layers_used=1, Hq=8, Hkv=2, d=128, D=320, sinks=2)
    ref = _run(estp, estp.lib, w, dtype_q)
    got = _run(estp, checked, w, dtype_q)
    assert set(ref) == set(got)
    for k in ref:
        a, b = ref[k], got[k]
        if a.dtype == torch.bfloat16:
            a, b = a.view(torch.int16), b.view(torch.int16)
        assert torch.equal(a, b), k
