"""Token entropy with the logits formed from hidden states on the tensor cores
(estp_lm_head_entropy) against the oracle (GPU).

Tolerance: the bf16 products are exact in fp32 and the tensor cores accumulate them in
fp32, so a logit of D terms carries an error of order sqrt(D) 2^-24 |z| (1e-5 for the
spreads here).  The entropy moves by at most max |dz| sum_v p_v |ln p_v + H| <= 2 H max |dz|,
far below the 1e-3 nats held for token entropy everywhere else."""
import numpy as np
import pytest
import torch

import oracle
import synth
from synth import device as sd

pytestmark = pytest.mark.gpu

TOL = 1e-3


def _bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def _inputs(rows, D, V, spread, seed=11, ldh=None, ldw=None):
    """hidden ~ N(0, 1) and W ~ N(0, (spread / sqrt(D))^2), so the logits have standard
    deviation ~spread; bf16, from the counter-based generator (host and device agree)."""
    ldh, ldw = ldh or D, ldw or D
    hk, wk = synth.stream_key(seed, 7), synth.stream_key(seed, 8)
    hbig = sd.normal(hk, (rows, ldh), synth.BF16)
    wbig = sd.normal(wk, (V, ldw), synth.BF16, scale=spread / np.sqrt(D))
    return hbig[:, :D], wbig[:, :D]


def _ref(h, W, rows_idx=None):
    hb, Wb = _bits(h.contiguous()), _bits(W.contiguous())
    if rows_idx is not None:
        hb = hb[rows_idx]
    return oracle.lm_head_entropy(hb, Wb)


@pytest.mark.parametrize("rows,D,V", [(1, 64, 1), (5, 64, 7), (128, 128, 256), (129, 64, 257),
                                      (300, 192, 1000), (257, 256, 513), (64, 512, 4096)])
@pytest.mark.parametrize("spread", [0.5, 3.0, 12.0])
def test_lm_head_entropy_cases(cuda_lib, rows, D, V, spread):
    """Several row blocks and vocabulary tiles with ragged ends, one vocabulary entry,
    flat to sharply peaked distributions."""
    h, W = _inputs(rows, D, V, spread)
    ctx = cuda_lib.Context(0)
    H = ctx.lm_head_entropy(h, W)
    ctx.sync_status()
    ref = _ref(h, W)
    err = np.abs(H.cpu().numpy().astype(np.float64) - ref)
    assert err.max() <= TOL, f"max err {err.max():.2e}"
    if V == 1:  # a single entry: H = 0 up to the rounding of the fp32 log2
        assert np.all(np.abs(H.cpu().numpy()) <= 1e-6)


def test_lm_head_entropy_strided_rows(cuda_lib):
    """Row strides wider than D for both operands (views of wider arrays)."""
    h, W = _inputs(200, 128, 700, 3.0, seed=12, ldh=136, ldw=192)
    assert h.stride(0) == 136 and W.stride(0) == 192
    ctx = cuda_lib.Context(0)
    H = ctx.lm_head_entropy(h, W)
    ctx.sync_status()
    assert np.abs(H.cpu().numpy() - _ref(h, W)).max() <= TOL


@pytest.mark.parametrize("rows", [2000, 21663])
def test_lm_head_entropy_qwen_shape(cuda_lib, rows):
    """The output projection of the 16-prompt batch: hidden size 3584, vocabulary 152064,
    2000 tokens (76 vocabulary splits) and the batch's 21663 tokens (170 row blocks, 8
    splits, the launch the bench times), the last row block ragged; sampled rows against
    the oracle, which forms each row's 152064 logits in double.  Two calls give identical
    bits."""
    D, V = 3584, 152064
    h, W = _inputs(rows, D, V, 3.0, seed=13)
    ctx = cuda_lib.Context(0)
    H = ctx.lm_head_entropy(h, W)
    H2 = ctx.lm_head_entropy(h, W)
    ctx.sync_status()
    Hn = H.cpu().numpy()
    assert np.array_equal(Hn, H2.cpu().numpy())
    pick = np.unique(np.asarray([0, 1, 127, 128, 1023, 1920, rows // 2, rows - 129, rows - 2, rows - 1]))
    ref = _ref(h, W, pick)
    err = np.abs(Hn[pick].astype(np.float64) - ref)
    assert err.max() <= TOL, f"max err {err.max():.2e} at rows {pick[np.argmax(err)]}"
    assert np.all(np.isfinite(Hn)) and np.all(Hn >= 0) and np.all(Hn <= np.log(V) + TOL)


def test_lm_head_entropy_checks(cuda_lib):
    """Bad arguments are refused on the host before any launch; zero rows is a no-op."""
    ctx = cuda_lib.Context(0)
    h, W = _inputs(4, 64, 16, 1.0)
    with pytest.raises(cuda_lib.EstpError) as ei:  # fp32 operands
        ctx.lm_head_entropy(h.float(), W.float())
    assert ei.value.status == cuda_lib.ESTP_ERR_UNSUPPORTED
    hb, Wb = _inputs(4, 96, 16, 1.0)
    with pytest.raises(cuda_lib.EstpError) as ei:  # D not a multiple of 64
        ctx.lm_head_entropy(hb[:, :80], Wb[:, :80])
    assert ei.value.status == cuda_lib.ESTP_ERR_INVALID_ARG
    big = sd.normal(synth.stream_key(3, 9), (4, 72), synth.BF16)
    with pytest.raises(cuda_lib.EstpError):  # row stride 68 elements: not 16-byte aligned
        ctx.lm_head_entropy(big.view(-1)[:4 * 68].view(4, 68)[:, :64], W)
    out = torch.full((0,), 7.0, device="cuda")
    assert ctx.lm_head_entropy(h[:0], W, out=out).numel() == 0
