"""Failure detection on the GPU: a bounded wait that runs out (no fault, no hang).

estp_set_wait_limit lowers the limit of the tensor-core kernels' abortable waits (row
normalisers, column sums, the fused prefill forward, the entropy from hidden states) to
a few cycles, far below the latency of a tile copy, so they expire in every CTA.  The
call must then report ESTP_ERR_TIMEOUT through estp_sync_status (the kernels drain the
copies and MMAs they issued and free their tensor memory), and the next normal call on
the same context must match the oracle."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import assert_importance
from synth import device as sd
from synth import workloads as W

pytestmark = pytest.mark.gpu

WL = W.Workload("timeout", seed=21, B=3, T_lo=200, T_hi=900, dtype=synth.BF16, V=8,
                n_layers_model=1, layers_used=1, Hq=8, Hkv=2, d=128, D=64, sinks=2)


def _oracle_S(w):
    cu = w.cu_seqlens()
    Q, K = W.host_qk(w, w.layers[0])
    C = oracle.attn_colsum(Q, K, cu, w.scale)
    return oracle.importance(C, cu, 1, w.Hq)


@pytest.mark.parametrize("lse_given", [False, True], ids=["lse_computed", "lse_given"])
def test_wait_runs_out_then_context_recovers(cuda_lib, lse_given):
    w = WL
    cu = w.cu_seqlens()
    sumT, maxT = int(cu[-1]), int(np.diff(cu).max())
    Q, K = sd.qk(w, w.layers[0])
    cu_d = sd.cu_seqlens(w)
    ctx = cuda_lib.Context(0)
    lse = ctx.attn_lse(Q, K, cu_d, maxT) if lse_given else None
    ctx.sync_status()
    ctx.set_wait_limit(2)
    ctx.attn_importance(Q, K, cu_d, maxT, lse=lse)  # the row normalisers too when lse is None
    with pytest.raises(cuda_lib.EstpError) as err:
        ctx.sync_status()
    assert err.value.status == cuda_lib.ESTP_ERR_TIMEOUT
    ctx.sync_status()  # the status word was cleared by the read
    ctx.set_wait_limit(0)
    ctx.attn_importance(Q, K, cu_d, maxT, lse=lse)
    S = ctx.attn_importance_finalize(1, sumT).cpu().numpy()
    ctx.sync_status()
    assert_importance(S, _oracle_S(w))
    ctx.close()


@pytest.mark.parametrize("lse_given", [False, True], ids=["lse_computed", "lse_given"])
def test_forward_wait_runs_out_then_context_recovers(cuda_lib, lse_given):
    """The same for the fused prefill forward (O = A V with the column sums): its waits
    run out, the call reports ESTP_ERR_TIMEOUT, and the next call matches the oracle in
    both O and the importance."""
    w = WL
    cu = w.cu_seqlens()
    sumT, maxT = int(cu[-1]), int(np.diff(cu).max())
    layer = w.layers[0]
    Q, K = sd.qk(w, layer)
    Vh = synth.round_to(synth.normal(w.key_v(layer), np.arange(sumT * w.Hkv * w.d)),
                        w.dtype).reshape(sumT, w.Hkv, w.d)
    V = torch.from_numpy(Vh.view(np.int16)).view(torch.bfloat16).cuda()
    cu_d = sd.cu_seqlens(w)
    ctx = cuda_lib.Context(0)
    lse = ctx.attn_lse(Q, K, cu_d, maxT) if lse_given else None
    ctx.sync_status()
    ctx.set_wait_limit(2)
    ctx.attn_forward_importance(Q, K, V, cu_d, maxT, lse=lse)
    with pytest.raises(cuda_lib.EstpError) as err:
        ctx.sync_status()
    assert err.value.status == cuda_lib.ESTP_ERR_TIMEOUT
    ctx.sync_status()
    ctx.set_wait_limit(0)
    O = ctx.attn_forward_importance(Q, K, V, cu_d, maxT, lse=lse)
    S = ctx.attn_importance_finalize(1, sumT).cpu().numpy()
    ctx.sync_status()
    assert_importance(S, _oracle_S(w))
    Qh, Kh = W.host_qk(w, layer)
    O_ref = oracle.attn_output(Qh, Kh, Vh, cu, w.scale)
    vmax = float(np.max(np.abs(synth.bf16_bits_to_f32(Vh))))
    err = float(np.max(np.abs(O.float().cpu().numpy() - O_ref)))
    assert err <= 5e-3 * vmax, f"O max abs err {err:.3e}"
    ctx.close()


def test_lm_head_wait_runs_out_then_context_recovers(cuda_lib):
    """The same for the entropy with the logits formed from hidden states: its waits run
    out, the call reports ESTP_ERR_TIMEOUT, and the next call matches the oracle."""
    rows, D, V = 300, 192, 1000
    h = sd.normal(synth.stream_key(23, 7), (rows, D), synth.BF16)
    Wo = sd.normal(synth.stream_key(23, 8), (V, D), synth.BF16, scale=3.0 / np.sqrt(D))
    ctx = cuda_lib.Context(0)
    ctx.set_wait_limit(2)
    ctx.lm_head_entropy(h, Wo)
    with pytest.raises(cuda_lib.EstpError) as err:
        ctx.sync_status()
    assert err.value.status == cuda_lib.ESTP_ERR_TIMEOUT
    ctx.sync_status()
    ctx.set_wait_limit(0)
    H = ctx.lm_head_entropy(h, Wo).cpu().numpy()
    ctx.sync_status()
    bits = lambda t: t.view(torch.int16).cpu().numpy().view(np.uint16)
    ref = oracle.lm_head_entropy(bits(h), bits(Wo))
    assert np.max(np.abs(H - ref)) <= 1e-3
    ctx.close()


def test_wait_limit_rejects_null_context(cuda_lib):
    assert cuda_lib.lib.estp_set_wait_limit(None, 5) == cuda_lib.ESTP_ERR_INVALID_ARG
