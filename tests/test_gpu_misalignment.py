"""Entropy/importance misalignment counts against the oracle (GPU): integer counts,
compared exactly."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def _inputs(lens, seed=3):
    rng = np.random.default_rng(seed)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    n = int(cu[-1])
    H = rng.uniform(0, 11, n).astype(np.float32)
    S = rng.exponential(1.0, n).astype(np.float32)
    # ties inside prompts, and both signed zeros
    if n > 40:
        H[5:25] = 2.5
        S[15:40] = 0.75
        H[30], H[31], S[32], S[33] = -0.0, 0.0, 0.0, -0.0
    return cu, H, S


@pytest.mark.parametrize("pct", [40, 25, 50, 1])
@pytest.mark.parametrize("lens", [[0, 1, 2, 3, 10, 257, 1000], [33000, 4096, 5]],
                         ids=["short", "long"])
def test_misalignment_against_oracle(cuda_lib, lens, pct):
    cu, H, S = _inputs(lens)
    ctx = cuda_lib.Context(0)
    got = ctx.misalignment(torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda(),
                           torch.from_numpy(cu).cuda(), pct)
    ctx.sync_status()
    ref = oracle.misalignment(H, S, cu, pct)
    assert np.array_equal(got.cpu().numpy().astype(np.int64), ref)


def test_misalignment_checks(cuda_lib):
    cu, H, S = _inputs([10, 20])
    ctx = cuda_lib.Context(0)
    Hd, Sd = torch.from_numpy(H).cuda(), torch.from_numpy(S).cuda()
    with pytest.raises(cuda_lib.EstpError):
        ctx.misalignment(Hd, Sd, torch.from_numpy(cu).cuda(), 51)
    bad = torch.tensor([0, 25, 20], dtype=torch.int32, device="cuda")  # decreasing
    ctx.misalignment(Hd, Sd, bad)
    with pytest.raises(cuda_lib.EstpError) as e:
        ctx.sync_status()
    assert e.value.status == cuda_lib.ESTP_ERR_INVALID_ARG
    good = ctx.misalignment(Hd, Sd, torch.from_numpy(cu).cuda())  # the context stays usable
    ctx.sync_status()
    assert np.array_equal(good.cpu().numpy().astype(np.int64), oracle.misalignment(H, S, cu))
