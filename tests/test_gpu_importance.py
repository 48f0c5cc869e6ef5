"""Attention importance (LSE + column sums + finalize) against the oracle (GPU)."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import assert_importance
from synth import device as sd
from synth import workloads as W

pytestmark = pytest.mark.gpu


def _wl(dtype, lens, Hq, Hkv, d, seed=21, sinks=0, layers=1):
    w = W.Workload("imp", seed=seed, B=len(lens), T_lo=1, T_hi=1, dtype=dtype, V=8,
                   n_layers_model=layers, layers_used=layers, Hq=Hq, Hkv=Hkv, d=d, D=8,
                   sinks=sinks)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    return w, cu


def _qk(w, cu, layer):
    """Q, K on the host (numpy) and device (torch) for explicit cu_seqlens."""
    sumT = int(cu[-1])
    rows = np.arange(sumT)
    key_q, key_k = w.key_q(layer), w.key_k(layer)
    Qh = synth.round_to(synth.normal(key_q, np.arange(sumT * w.Hq * w.d)), w.dtype).reshape(sumT, w.Hq, w.d)
    K64 = synth.normal(key_k, np.arange(sumT * w.Hkv * w.d)).reshape(sumT, w.Hkv, w.d)
    if w.sinks:
        for b in range(len(cu) - 1):
            K64[cu[b]:min(cu[b] + w.sinks, cu[b + 1])] *= w.sink_scale
    Kh = synth.round_to(K64, w.dtype).reshape(sumT, w.Hkv, w.d)
    tdt = torch.bfloat16 if w.dtype == synth.BF16 else torch.float32
    if w.dtype == synth.BF16:
        Qd = torch.from_numpy(Qh.view(np.int16)).view(tdt).cuda()
        Kd = torch.from_numpy(Kh.view(np.int16)).view(tdt).cuda()
    else:
        Qd, Kd = torch.from_numpy(Qh).cuda(), torch.from_numpy(Kh).cuda()
    return Qh, Kh, Qd, Kd


def _run(cuda_lib, w, cu, layers, heads=None, exclude_self=False, supply_lse=False,
         divisor="length"):
    ctx = cuda_lib.Context(0)
    cu_d = torch.as_tensor(cu, device="cuda")
    maxT = int(np.diff(cu).max())
    sumT = int(cu[-1])
    C = np.zeros(sumT)
    for n, layer in enumerate(layers):
        Qh, Kh, Qd, Kd = _qk(w, cu, layer)
        lse = None
        if supply_lse:
            lse = torch.as_tensor(oracle.attn_lse(Qh, Kh, cu, 1 / math.sqrt(w.d)),
                                  dtype=torch.float32, device="cuda").contiguous()
        ctx.attn_importance(Qd, Kd, cu_d, maxT, lse=lse, heads=heads, accumulate=n > 0,
                            exclude_self=exclude_self, divisor=divisor)
        oracle.attn_colsum(Qh, Kh, cu, 1 / math.sqrt(w.d), heads=heads,
                           exclude_self=exclude_self, out=C)
    S = ctx.attn_importance_finalize(len(layers), sumT)
    ctx.sync_status()
    nh = w.Hq if heads is None else len(heads)
    ref = oracle.importance(C, cu, len(layers), nh, divisor=divisor, exclude_self=exclude_self)
    return S.cpu().numpy(), ref


CASES = [
    # lens, Hq, Hkv, d
    ([1], 2, 1, 64),
    ([5, 0, 130, 1], 4, 4, 64),
    ([129, 300], 7, 1, 128),
    ([700], 8, 1, 128),
    ([257, 64, 63, 513], 28, 4, 128),
    ([1100], 4, 2, 64),
]


@pytest.mark.parametrize("dtype", [synth.BF16, synth.F32])
@pytest.mark.parametrize("lens,Hq,Hkv,d", CASES, ids=[f"c{i}" for i in range(len(CASES))])
def test_importance_cases(cuda_lib, dtype, lens, Hq, Hkv, d):
    w, cu = _wl(dtype, lens, Hq, Hkv, d)
    S, ref = _run(cuda_lib, w, cu, [0])
    assert_importance(S, ref)
    for b in range(len(lens)):
        if lens[b]:
            assert abs(S[cu[b]:cu[b + 1]].sum() - 1.0) < 1e-4


@pytest.mark.parametrize("dtype", [synth.BF16, synth.F32])
def test_importance_layers_heads_self(cuda_lib, dtype):
    w, cu = _wl(dtype, [300, 45, 200], 8, 2, 128, sinks=4, layers=3)
    S, ref = _run(cuda_lib, w, cu, [0, 1, 2])
    assert_importance(S, ref)
    S, ref = _run(cuda_lib, w, cu, [1], heads=[5, 0, 7])
    assert_importance(S, ref)
    S, ref = _run(cuda_lib, w, cu, [2], exclude_self=True)
    assert_importance(S, ref)
    S, ref = _run(cuda_lib, w, cu, [0, 2], supply_lse=True)
    assert_importance(S, ref)


def test_lse_against_oracle(cuda_lib):
    for dtype in (synth.BF16, synth.F32):
        w, cu = _wl(dtype, [1, 257, 90], 6, 2, 64, sinks=2)
        Qh, Kh, Qd, Kd = _qk(w, cu, 0)
        ctx = cuda_lib.Context(0)
        lse = ctx.attn_lse(Qd, Kd, torch.as_tensor(cu, device="cuda"), 257)
        ctx.sync_status()
        ref = oracle.attn_lse(Qh, Kh, cu, 1 / math.sqrt(64))
        err = np.max(np.abs(lse.cpu().numpy() - ref) / (1 + np.abs(ref)))
        assert err < 1e-5, err


def test_importance_deterministic(cuda_lib):
    w, cu = _wl(synth.BF16, [900, 333], 28, 4, 128)
    _, _, Qd, Kd = _qk(w, cu, 0)
    ctx = cuda_lib.Context(0)
    cu_d = torch.as_tensor(cu, device="cuda")
    outs = []
    for _ in range(2):
        ctx.attn_importance(Qd, Kd, cu_d, 900)
        outs.append(ctx.attn_importance_finalize(1, int(cu[-1])))
    ctx.sync_status()
    assert torch.equal(outs[0], outs[1])


def test_importance_device_checks(cuda_lib):
    w, cu = _wl(synth.BF16, [100, 50], 4, 2, 64)
    _, _, Qd, Kd = _qk(w, cu, 0)
    ctx = cuda_lib.Context(0)
    cu_d = torch.as_tensor(cu, device="cuda")
    ctx.attn_importance(Qd, Kd, cu_d, 99)  # max_seqlen below a prompt length
    with pytest.raises(cuda_lib.EstpError) as e:
        ctx.sync_status()
    assert e.value.status == cuda_lib.ESTP_ERR_INVALID_ARG
    with pytest.raises(cuda_lib.EstpError):
        ctx.attn_importance(Qd, Kd, cu_d, 100, heads=[4])  # head out of range
    fresh = cuda_lib.Context(0)
    with pytest.raises(cuda_lib.EstpError):
        fresh.attn_importance(Qd, Kd, cu_d, 100, accumulate=True)  # no open accumulation
    fresh.attn_importance(Qd, Kd, cu_d, 100)
    with pytest.raises(cuda_lib.EstpError):  # a different prompt set cannot join it
        fresh.attn_importance(Qd[:100], Kd[:100], cu_d[:2], 100, accumulate=True)


@pytest.mark.parametrize("divisor", ["causal", "none"])
@pytest.mark.parametrize("exclude_self", [False, True])
@pytest.mark.parametrize("dtype", [synth.BF16, synth.F32])
def test_importance_divisor_variants(cuda_lib, dtype, divisor, exclude_self):
    """The divisor variants of Eq. 2-0 (ESTP_IMP_DIV_CAUSAL / _NONE) against the oracle:
    1-token and empty prompts (a zero causal count without the diagonal), several tiles,
    a head subset and two layers."""
    w, cu = _wl(dtype, [1, 0, 257, 40, 130], 8, 2, 128 if dtype == synth.BF16 else 64, layers=3)
    S, ref = _run(cuda_lib, w, cu, [0, 2], heads=[1, 2, 5, 7], exclude_self=exclude_self,
                  divisor=divisor)
    assert_importance(S, ref)
    if exclude_self and divisor == "causal":  # the last token of every prompt has n_j = 0
        for b in range(len(cu) - 1):
            if cu[b + 1] > cu[b]:
                assert S[cu[b + 1] - 1] == 0.0


def test_importance_divisor_flags_checked(cuda_lib):
    """Both divisor flags at once, and a later call whose divisor (or, under the causal
    divisor, self-term) flags differ from the opening call's, are refused on the host."""
    w, cu = _wl(synth.BF16, [70, 30], 4, 2, 64)
    _, _, Qd, Kd = _qk(w, cu, 0)
    cu_d = torch.as_tensor(cu, device="cuda")
    ctx = cuda_lib.Context(0)
    lib = cuda_lib.lib
    rc = lib.estp_attn_importance(ctx._h, Qd.data_ptr(), Kd.data_ptr(), 1, None, 4, 2, 64, 0.125,
                                  None, 4, cu_d.data_ptr(), 2, 100, 70, 0,
                                  cuda_lib.ESTP_IMP_DIV_CAUSAL | cuda_lib.ESTP_IMP_DIV_NONE, None)
    assert rc == cuda_lib.ESTP_ERR_INVALID_ARG
    ctx.attn_importance(Qd, Kd, cu_d, 70, divisor="causal")
    with pytest.raises(cuda_lib.EstpError):
        ctx.attn_importance(Qd, Kd, cu_d, 70, accumulate=True)  # length divisor now
    with pytest.raises(cuda_lib.EstpError):
        ctx.attn_importance(Qd, Kd, cu_d, 70, accumulate=True, divisor="causal", exclude_self=True)
    ctx.attn_importance(Qd, Kd, cu_d, 70, accumulate=True, divisor="causal")
    plain = cuda_lib.Context(0)  # the length divisor lets the self term vary per layer
    plain.attn_importance(Qd, Kd, cu_d, 70)
    plain.attn_importance(Qd, Kd, cu_d, 70, accumulate=True, exclude_self=True)
    ctx.sync_status()
    plain.sync_status()


@pytest.mark.parametrize("w", [W.C1, W.C2], ids=lambda w: w.name)
def test_importance_workload(cuda_lib, w):
    """Whole workload, all selected layers and heads on the GPU (the bench's launch
    configuration), every prompt of the batch against the oracle element by element; S
    sums to 1 over every prompt.  The oracle reads the workload's Q and K back from the
    device (the device generator's bits equal the host one's, test_gpu_synth)."""
    cu = w.cu_seqlens()
    sumT = int(cu[-1])
    maxT = int(np.diff(cu).max())
    ctx = cuda_lib.Context(0)
    cu_d = sd.cu_seqlens(w)
    C = np.zeros(sumT)
    for n, layer in enumerate(w.layers):
        Q, K = sd.qk(w, layer)
        ctx.attn_importance(Q, K, cu_d, maxT, accumulate=n > 0)
        Qh = Q.contiguous().view(torch.int16).cpu().numpy().view(np.uint16) \
            if Q.dtype == torch.bfloat16 else Q.cpu().numpy()
        Kh = K.contiguous().view(torch.int16).cpu().numpy().view(np.uint16) \
            if K.dtype == torch.bfloat16 else K.cpu().numpy()
        oracle.attn_colsum(Qh, Kh, cu, w.scale, out=C)
        del Q, K
    S = ctx.attn_importance_finalize(len(w.layers), sumT).cpu().numpy()
    ctx.sync_status()
    for b in range(w.B):
        assert abs(S[cu[b]:cu[b + 1]].sum() - 1.0) < 1e-4
    assert_importance(S, oracle.importance(C, cu, len(w.layers), w.Hq))


@pytest.mark.parametrize("B,T,expect_qc", [(32, 2048, 4), (16, 4096, 8), (20, 4096, 16)])
def test_importance_chunk_sizes(cuda_lib, B, T, expect_qc):
    """Batches large enough that the column-sum items cover 4, 8 and 16 query-tile pairs
    (the host picks the largest that keeps ~16 items per SM): one head per KV group, every
    prompt against the oracle element by element."""
    w = W.Workload("chunks", seed=41 + B, B=B, T_lo=T, T_hi=T, dtype=synth.BF16, V=8,
                   n_layers_model=1, layers_used=1, Hq=32, Hkv=8, d=128, D=64, sinks=4)
    # the host's choice, restated: largest qc with B * groups * items(nt, qc) >= 16 * SMs
    def items_f(n, qc):
        a, r = n // qc, n % qc
        return qc * a * (a + 1) // 2 + r * (a + 1)
    n_sms = torch.cuda.get_device_properties(0).multi_processor_count
    nt = (T + 255) // 256
    picked = next((qc for qc in (16, 8, 4, 2) if B * w.Hkv * items_f(nt, qc) >= 16 * n_sms), 2)
    if picked != expect_qc:
        pytest.skip(f"{n_sms} SMs pick {picked} query-tile pairs per item, not {expect_qc}")
    cu = w.cu_seqlens()
    sumT = int(cu[-1])
    heads = list(range(0, w.Hq, w.Hq // w.Hkv))  # one per KV group
    ctx = cuda_lib.Context(0)
    Q, K = sd.qk(w, w.layers[0])
    ctx.attn_importance(Q, K, sd.cu_seqlens(w), T, heads=heads)
    S = ctx.attn_importance_finalize(1, sumT).cpu().numpy()
    ctx.sync_status()
    Qh = Q.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    Kh = K.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    C = oracle.attn_colsum(Qh, Kh, cu, w.scale, heads=heads)
    assert_importance(S, oracle.importance(C, cu, 1, len(heads)))
    ctx.close()
