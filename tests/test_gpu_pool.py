"""K-POOL + length head against the oracle (GPU)."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import assert_pooled, assert_pred
from synth import device as sd
from synth import workloads as W

pytestmark = pytest.mark.gpu


def _inputs(dtype, lens, D, ld=None, seed=31):
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    sumT = int(cu[-1])
    ld = D if ld is None else ld
    key = synth.stream_key(seed, 1)
    hid64 = synth.normal(key, np.arange(sumT * ld)).reshape(sumT, ld)
    hid = synth.round_to(hid64, dtype)
    rng = np.random.default_rng(seed)
    H = rng.uniform(0, 11, sumT).astype(np.float32)
    S = (rng.uniform(0, 2, sumT) / np.repeat(np.maximum(lens, 1), lens)).astype(np.float32)
    tdt = torch.bfloat16 if dtype == synth.BF16 else torch.float32
    hd = (torch.from_numpy(hid.view(np.int16)).view(tdt) if dtype == synth.BF16
          else torch.from_numpy(hid)).cuda()
    return cu, hid, H, S, hd


def _head(K, D, seed=5):
    rng = np.random.default_rng(seed)
    Wt = (rng.standard_normal((K, D)) / np.sqrt(D) * 40).astype(np.float32)
    b = rng.standard_normal(K).astype(np.float32)
    c = ((np.arange(K) + 0.5) * 256).astype(np.float32)
    return Wt, b, c


@pytest.mark.parametrize("dtype", [synth.BF16, synth.F32])
@pytest.mark.parametrize("lens,D,ld", [([128], 1024, None), ([1, 0, 64, 65, 300], 3584, None),
                                       ([2000, 7], 8192, None), ([100, 33], 100, 104),
                                       ([0], 16, None), ([5000], 4096, None)])
@pytest.mark.parametrize("mix", [(0.7, 0.3, 1.0), (0.0, 1.0, 0.5), (0.0, 0.0, 1.0),
                                 (5.0, 0.2, 0.05)])
def test_pool_cases(cuda_lib, dtype, lens, D, ld, mix):
    cu, hid, H, S, hd = _inputs(dtype, lens, D, ld)
    Wt, b, c = _head(32, D)
    ctx = cuda_lib.Context(0)
    head = cuda_lib.Head(torch.from_numpy(Wt).cuda(), torch.from_numpy(b).cuda(),
                         torch.from_numpy(c).cuda())
    pooled, pred = ctx.pool(hd, torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda(),
                            torch.as_tensor(cu, device="cuda"), *mix, head=head, D=D)
    ctx.sync_status()
    P_ref = oracle.pool(hid, H.astype(np.float64), S.astype(np.float64), cu, *mix, D=D)
    y_ref = oracle.length_head(P_ref, Wt, b, c)
    assert_pooled(pooled.cpu().numpy(), P_ref)
    assert_pred(pred.cpu().numpy(), y_ref)
    for k in np.nonzero(np.diff(cu) == 0)[0]:
        assert np.all(pooled[k].cpu().numpy() == 0)


def test_pool_mean_and_argmax(cuda_lib):
    cu, hid, H, S, hd = _inputs(synth.F32, [77, 200], 256)
    ctx = cuda_lib.Context(0)
    Hd, Sd, cud = (torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda(),
                   torch.as_tensor(cu, device="cuda"))
    pooled, _ = ctx.pool(hd, Hd, Sd, cud, 0.0, 0.0, 1.0)
    assert_pooled(pooled.cpu().numpy(), np.stack([hid[0:77].mean(0), hid[77:].mean(0)]))
    pooled, _ = ctx.pool(hd, Hd, Sd, cud, 0.0, 1.0, 1e-4)
    am = [int(np.argmax(H[0:77])), 77 + int(np.argmax(H[77:]))]
    assert_pooled(pooled.cpu().numpy(), hid[am])


@pytest.mark.parametrize("w", [W.C1, W.C2, W.C4], ids=lambda w: w.name)
def test_pool_workload(cuda_lib, w):
    """Full-size hidden states of the workload; entropy and importance stand-ins of the
    workload's scale; every prompt checked against the oracle."""
    cu = w.cu_seqlens()
    sumT = int(cu[-1])
    rng = np.random.default_rng(2)
    H = rng.uniform(0, 12, sumT).astype(np.float32)
    S = (rng.uniform(0, 2, sumT) / np.repeat(np.diff(cu), np.diff(cu))).astype(np.float32)
    ctx = cuda_lib.Context(0)
    Wt, b, c = w.head_params()
    head = cuda_lib.Head(torch.from_numpy(Wt).cuda(), torch.from_numpy(b).cuda(),
                         torch.from_numpy(c).cuda())
    hid = sd.hidden(w)
    pooled, pred = ctx.pool(hid, torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda(),
                            sd.cu_seqlens(w), w.lambda1, w.lambda2, w.alpha, head=head)
    ctx.sync_status()
    pick = range(w.B) if w.B <= 2 else np.random.default_rng(3).choice(w.B, 4, replace=False)
    for bb in pick:
        rows = np.arange(cu[bb], cu[bb + 1])
        sub = np.asarray([0, len(rows)], dtype=np.int32)
        P = oracle.pool(W.host_hidden(w, rows), H[rows], S[rows], sub, w.lambda1, w.lambda2,
                        w.alpha)
        assert_pooled(pooled[bb:bb + 1].cpu().numpy(), P)
        assert_pred(pred[bb:bb + 1].cpu().numpy(), oracle.length_head(P, Wt, b, c))


@pytest.mark.parametrize("K,with_bias", [(1, True), (7, False), (1024, True)])
def test_head_bins(cuda_lib, K, with_bias):
    """Length head at the bin-count limits, with and without a bias (Eq. 3-2)."""
    cu, hid, H, S, hd = _inputs(synth.BF16, [300, 0, 77, 1500], 3584)
    Wt, b, c = _head(K, 3584, seed=K)
    ctx = cuda_lib.Context(0)
    head = cuda_lib.Head(torch.from_numpy(Wt).cuda(),
                         torch.from_numpy(b).cuda() if with_bias else None,
                         torch.from_numpy(c).cuda())
    pooled, pred = ctx.pool(hd, torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda(),
                            torch.as_tensor(cu, device="cuda"), 0.7, 0.3, 1.0, head=head)
    ctx.sync_status()
    P_ref = oracle.pool(hid, H.astype(np.float64), S.astype(np.float64), cu, 0.7, 0.3, 1.0)
    assert_pooled(pooled.cpu().numpy(), P_ref)
    assert_pred(pred.cpu().numpy(), oracle.length_head(P_ref, Wt, b if with_bias else None, c))


def test_pool_bad_cu_then_good(cuda_lib):
    """Bad cu_seqlens (checked on the device): the call records ESTP_ERR_INVALID_ARG and
    writes nothing else, so the next call on the same context is exact."""
    cu, hid, H, S, hd = _inputs(synth.BF16, [300, 77, 1500, 9], 3584)
    Wt, b, c = _head(32, 3584)
    head = cuda_lib.Head(torch.from_numpy(Wt).cuda(), torch.from_numpy(b).cuda(),
                         torch.from_numpy(c).cuda())
    ctx = cuda_lib.Context(0)
    Hd, Sd = torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda()
    for bad in ([0, 300, 200, 1877, 1886],    # decreasing
                [0, 300, 377, 1877, 1885],    # cu[B] != sumT
                [5, 300, 377, 1877, 1886]):   # cu[0] != 0
        with pytest.raises(cuda_lib.EstpError) as ei:
            ctx.pool(hd, Hd, Sd, torch.as_tensor(np.asarray(bad, np.int32), device="cuda"),
                     0.7, 0.3, 1.0, head=head)
            ctx.sync_status()
        assert ei.value.status == cuda_lib.ESTP_ERR_INVALID_ARG
    pooled, pred = ctx.pool(hd, Hd, Sd, torch.as_tensor(cu, device="cuda"), 0.7, 0.3, 1.0, head=head)
    ctx.sync_status()
    P_ref = oracle.pool(hid, H.astype(np.float64), S.astype(np.float64), cu, 0.7, 0.3, 1.0)
    assert_pooled(pooled.cpu().numpy(), P_ref)
    assert_pred(pred.cpu().numpy(), oracle.length_head(P_ref, Wt, b, c))


def test_pool_deterministic_and_counters(cuda_lib):
    """Fixed-order merges: repeated calls give identical bits. The head's per-prompt
    arrival counters are back to zero after every call: a head-less call with several
    column slices, calls with the head, then a call of another shape on the same
    context, all exact."""
    cu, hid, H, S, hd = _inputs(synth.BF16, [2000, 7, 0, 300, 1], 8192)
    Wt, b, c = _head(32, 8192)
    head = cuda_lib.Head(torch.from_numpy(Wt).cuda(), torch.from_numpy(b).cuda(),
                         torch.from_numpy(c).cuda())
    ctx = cuda_lib.Context(0)
    Hd, Sd, cud = (torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda(),
                   torch.as_tensor(cu, device="cuda"))
    P_ref = oracle.pool(hid, H.astype(np.float64), S.astype(np.float64), cu, 0.7, 0.3, 1.0)
    pooled0, _ = ctx.pool(hd, Hd, Sd, cud, 0.7, 0.3, 1.0)
    ctx.sync_status()
    assert_pooled(pooled0.cpu().numpy(), P_ref)
    runs = []
    for _ in range(3):
        pooled, pred = ctx.pool(hd, Hd, Sd, cud, 0.7, 0.3, 1.0, head=head)
        ctx.sync_status()
        runs.append((pooled.cpu().numpy(), pred.cpu().numpy()))
    for p, y in runs[1:]:
        assert np.array_equal(p, runs[0][0]) and np.array_equal(y, runs[0][1])
    assert np.array_equal(runs[0][0], pooled0.cpu().numpy())
    assert_pred(runs[0][1], oracle.length_head(P_ref, Wt, b, c))
    cu2, hid2, H2, S2, hd2 = _inputs(synth.BF16, [50, 0, 700], 1024, seed=8)
    Wt2, b2, c2 = _head(32, 1024)
    head2 = cuda_lib.Head(torch.from_numpy(Wt2).cuda(), torch.from_numpy(b2).cuda(),
                          torch.from_numpy(c2).cuda())
    pooled2, pred2 = ctx.pool(hd2, torch.from_numpy(H2).cuda(), torch.from_numpy(S2).cuda(),
                              torch.as_tensor(cu2, device="cuda"), 0.7, 0.3, 1.0, head=head2)
    ctx.sync_status()
    P2 = oracle.pool(hid2, H2.astype(np.float64), S2.astype(np.float64), cu2, 0.7, 0.3, 1.0)
    assert_pooled(pooled2.cpu().numpy(), P2)
    assert_pred(pred2.cpu().numpy(), oracle.length_head(P2, Wt2, b2, c2))
