"""The allocation-free entropy entry point (GPU).

Some callers cannot allocate device memory: a serving engine whose allocator already
owns all of HBM for its KV cache, or code running where cudaMalloc is not allowed.
estp_token_entropy_noalloc serves them with the partials kept in a static device
array.  This test calls it through the C ABI and checks it against
estp_token_entropy on two calls in a row (the second call reuses the static array
with whatever the first call left in it), and against the fp64 oracle on the same
rows.  The file sorts last so that a run that stops at the first failure has already
run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from gpu_util import ENTROPY_ATOL, assert_entropy
from synth import device as sd
from synth import workloads as W

pytestmark = pytest.mark.gpu


def _noalloc(estp, x, V, ld, out):
    dt = estp.ESTP_BF16 if x.dtype == torch.bfloat16 else estp.ESTP_F32
    rc = estp.lib.estp_token_entropy_noalloc(ctypes.c_void_p(x.data_ptr()), dt, x.shape[0], V, ld,
                                             ctypes.c_void_p(out.data_ptr()),
                                             ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == estp.ESTP_OK, estp.lib.estp_last_error(None)


def test_noalloc_matches_entropy_twice(cuda_lib):
    estp = cuda_lib
    ctx = estp.Context(0)
    cases = [(W.C2, 700, W.C2.V, W.C2.V), (W.C1, 128, W.C1.V, W.C1.V), (W.C4, 65, 128250, 128256)]
    for w, rows, V, ld in cases:
        x = sd.logits(w, 3, rows, ld=ld, pad_val=1e4)
        ref = ctx.token_entropy(x, V=V)
        outs = []
        for _ in range(2):  # two calls in a row share the static scratch
            out = torch.full((rows,), float("nan"), device="cuda")
            _noalloc(estp, x, V, ld, out)
            torch.cuda.synchronize()
            outs.append(out.cpu().numpy())
        r = ref.cpu().numpy()
        if x.dtype == torch.bfloat16:
            xh = x.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        else:
            xh = x.cpu().numpy()
        exact = oracle.token_entropy(xh, V=V)
        for o in outs:
            assert np.all(np.isfinite(o))
            assert np.max(np.abs(o - r)) <= ENTROPY_ATOL
            assert_entropy(o, exact)
    ctx.close()


def test_noalloc_rejects_bad_arguments(cuda_lib):
    estp = cuda_lib
    x = torch.zeros(4, 10, dtype=torch.float32, device="cuda")
    out = torch.empty(4, device="cuda")
    rc = estp.lib.estp_token_entropy_noalloc(ctypes.c_void_p(x.data_ptr()), estp.ESTP_F32, 4, 11,
                                             10, ctypes.c_void_p(out.data_ptr()), None)
    assert rc == estp.ESTP_ERR_INVALID_ARG
