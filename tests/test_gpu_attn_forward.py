"""The fused prefill attention forward (output O = A V and the importance column sums of
the same probabilities) against the oracle (GPU), through the C ABI."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import assert_importance
from test_gpu_importance import _qk, _wl

pytestmark = pytest.mark.gpu

# Tolerance of O, from the arithmetic.  P enters A V rounded to bf16 (relative error at
# most 2^-9 per term), so |dO_i| <= 2^-9 sum_j A_ij |V_j| <= 2^-9 max|V|; the bf16 output
# adds at most 2^-9 |O_i| <= 2^-9 max|V|.  Together 2^-8 = 3.9e-3 max|V|; ex2.approx and
# the fp32 row normaliser add below 1e-5 relative.
O_TOL = 5e-3


def _v(w, cu, layer):
    sumT = int(cu[-1])
    Vh = synth.round_to(synth.normal(w.key_v(layer), np.arange(sumT * w.Hkv * w.d)),
                        w.dtype).reshape(sumT, w.Hkv, w.d)
    Vd = torch.from_numpy(Vh.view(np.int16)).view(torch.bfloat16).cuda()
    return Vh, Vd


def _assert_o(O, O_ref, Vh):
    vmax = float(np.max(np.abs(synth.bf16_bits_to_f32(Vh)))) if Vh.size else 1.0
    err = float(np.max(np.abs(O.float().cpu().numpy() - O_ref))) if O_ref.size else 0.0
    assert err <= O_TOL * vmax, f"O max abs err {err:.3e} (max|V| {vmax:.3e})"


def _run(cuda_lib, w, cu, layers, exclude_self=False, supply_lse=False, divisor="length",
         mix_unfused=False):
    """Layers through the fused forward (layer 0 through estp_attn_importance when
    mix_unfused), one accumulation; returns S and the oracle's S."""
    ctx = cuda_lib.Context(0)
    cu_d = torch.as_tensor(cu, device="cuda")
    maxT = int(np.diff(cu).max())
    sumT = int(cu[-1])
    scale = 1 / math.sqrt(w.d)
    C = np.zeros(sumT)
    for n, layer in enumerate(layers):
        Qh, Kh, Qd, Kd = _qk(w, cu, layer)
        lse = None
        if supply_lse:
            lse = torch.as_tensor(oracle.attn_lse(Qh, Kh, cu, scale), dtype=torch.float32,
                                  device="cuda").contiguous()
        if mix_unfused and n == 0:
            ctx.attn_importance(Qd, Kd, cu_d, maxT, lse=lse, exclude_self=exclude_self,
                                divisor=divisor)
        else:
            Vh, Vd = _v(w, cu, layer)
            O = ctx.attn_forward_importance(Qd, Kd, Vd, cu_d, maxT, lse=lse, accumulate=n > 0,
                                            exclude_self=exclude_self, divisor=divisor)
            ctx.sync_status()
            _assert_o(O, oracle.attn_output(Qh, Kh, Vh, cu, scale), Vh)
        oracle.attn_colsum(Qh, Kh, cu, scale, exclude_self=exclude_self, out=C)
    S = ctx.attn_importance_finalize(len(layers), sumT)
    ctx.sync_status()
    ref = oracle.importance(C, cu, len(layers), w.Hq, divisor=divisor, exclude_self=exclude_self)
    return S.cpu().numpy(), ref


CASES = [
    # lens, Hq, Hkv
    ([1], 2, 1),
    ([5, 0, 130, 1], 4, 4),
    ([129, 300], 7, 1),
    ([0, 0, 200], 2, 2),
    ([257, 64, 63, 513], 28, 4),
    ([1100], 4, 2),
    ([300, 50, 129], 64, 1),   # GQA ratio 64: one KV head for every query head
]


@pytest.mark.parametrize("lens,Hq,Hkv", CASES)
def test_forward_output_and_importance(cuda_lib, lens, Hq, Hkv):
    w, cu = _wl(synth.BF16, lens, Hq, Hkv, 128, seed=61)
    S, ref = _run(cuda_lib, w, cu, [0])
    assert_importance(S, ref)


@pytest.mark.parametrize("exclude_self", [False, True])
@pytest.mark.parametrize("divisor", ["length", "causal", "none"])
def test_forward_flags_two_layers(cuda_lib, exclude_self, divisor):
    w, cu = _wl(synth.BF16, [300, 1, 129, 77], 8, 2, 128, seed=62)
    S, ref = _run(cuda_lib, w, cu, [0, 1], exclude_self=exclude_self, divisor=divisor)
    assert_importance(S, ref)


def test_forward_supplied_lse(cuda_lib):
    w, cu = _wl(synth.BF16, [640, 3, 255], 4, 1, 128, seed=63)
    S, ref = _run(cuda_lib, w, cu, [0, 1], supply_lse=True)
    assert_importance(S, ref)


def test_forward_mixed_with_importance_call(cuda_lib):
    """One accumulation: layer 0 by estp_attn_importance, layer 1 by the fused forward."""
    w, cu = _wl(synth.BF16, [400, 129], 4, 2, 128, seed=64)
    S, ref = _run(cuda_lib, w, cu, [0, 1], mix_unfused=True)
    assert_importance(S, ref)


def test_forward_sinks(cuda_lib):
    """Attention sinks: the first key rows of each prompt scaled up, so most of each row's
    mass sits on a few columns."""
    w, cu = _wl(synth.BF16, [700, 260], 4, 1, 128, seed=65, sinks=4)
    S, ref = _run(cuda_lib, w, cu, [0])
    assert_importance(S, ref)


def test_forward_long_prompt(cuda_lib):
    """One 4000-token prompt: 32 query tiles, so the dynamic scheduler, both ring stages
    and both P buffers wrap many times within one item."""
    w, cu = _wl(synth.BF16, [4000], 4, 1, 128, seed=66)
    S, ref = _run(cuda_lib, w, cu, [0])
    assert_importance(S, ref)


def test_forward_deterministic(cuda_lib):
    """Repeated calls give identical bits (fixed-order column sums, no atomics)."""
    w, cu = _wl(synth.BF16, [900, 33, 400], 8, 2, 128, seed=67)
    cu_d = torch.as_tensor(cu, device="cuda")
    Qh, Kh, Qd, Kd = _qk(w, cu, 0)
    Vh, Vd = _v(w, cu, 0)
    ctx = cuda_lib.Context(0)
    outs = []
    for _ in range(2):
        O = ctx.attn_forward_importance(Qd, Kd, Vd, cu_d, 900)
        S = ctx.attn_importance_finalize(1, int(cu[-1]))
        ctx.sync_status()
        outs.append((O.view(torch.int16).cpu().numpy(), S.cpu().numpy()))
    assert np.array_equal(outs[0][0], outs[1][0])
    assert np.array_equal(outs[0][1].view(np.int32), outs[1][1].view(np.int32))


def test_forward_rejects_unsupported(cuda_lib):
    ctx = cuda_lib.Context(0)
    cu = torch.tensor([0, 8], dtype=torch.int32, device="cuda")
    Q = torch.zeros(8, 2, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(cuda_lib.EstpError):
        ctx.attn_forward_importance(Q, Q, Q, cu, 8)          # head_dim 64
    Q32 = torch.zeros(8, 2, 128, dtype=torch.float32, device="cuda")
    with pytest.raises(cuda_lib.EstpError):
        ctx.attn_forward_importance(Q32, Q32, Q32, cu, 8)    # fp32


def test_forward_rejects_bad_arguments(cuda_lib):
    """Host-side validation, before any launch: misaligned V or output, a NULL V, and
    accumulate = 1 without an open accumulation."""
    ctx = cuda_lib.Context(0)
    cu = torch.tensor([0, 8], dtype=torch.int32, device="cuda")
    Q = torch.zeros(8, 2, 128, dtype=torch.bfloat16, device="cuda")
    K = torch.zeros(8, 1, 128, dtype=torch.bfloat16, device="cuda")
    flat = torch.zeros(8 * 128 + 8, dtype=torch.bfloat16, device="cuda")
    V_mis = flat[1:1 + 8 * 128].view(8, 1, 128)            # 2 bytes off a 16-byte boundary
    with pytest.raises(cuda_lib.EstpError):
        ctx.attn_forward_importance(Q, K, V_mis, cu, 8)
    out_flat = torch.zeros(8 * 2 * 128 + 8, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(cuda_lib.EstpError):
        ctx.attn_forward_importance(Q, K, K, cu, 8, out=out_flat[1:1 + 8 * 2 * 128].view(8, 2, 128))
    import ctypes
    lib = cuda_lib.lib
    rc = lib.estp_attn_forward_importance(ctx._h, Q.data_ptr(), K.data_ptr(), None, 1, None, 2, 1, 128,
                                          0.1, cu.data_ptr(), 1, 8, 8, 0, 0, Q.data_ptr(), None)
    assert rc != 0
    ctx2 = cuda_lib.Context(0)
    with pytest.raises(cuda_lib.EstpError):
        ctx2.attn_forward_importance(Q, K, K, cu, 8, accumulate=True)
    # a valid call still works on the same context afterwards
    O = ctx.attn_forward_importance(Q, K, K, cu, 8)
    ctx.sync_status()
    assert O.shape == (8, 2, 128)
