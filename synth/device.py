"""Device side of the seeded generator: the same values as the numpy functions in
``synth``, written straight into CUDA memory by ``synth.cu`` (no ESTP arithmetic)."""
from __future__ import annotations

import ctypes
import os

import torch

from . import BF16, F32, spike_threshold
from . import workloads as W

_SO = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_build", "libsynth.so")
_lib = None


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(_SO):
            raise ImportError(f"{_SO} missing: build it with paper_2608_15592_gb300.build.build_synth()")
        lib = ctypes.CDLL(_SO)
        P, I, I64, U64, D = (ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_uint64,
                             ctypes.c_double)
        lib.synth_fill_normal.argtypes = [P, I, U64, I64, I64, D, P]
        lib.synth_fill_logits.argtypes = [P, I, U64, U64, I64, I64, I64, I64, D, D, ctypes.c_uint32,
                                          D, ctypes.c_float, P]
        lib.synth_fill_normal.restype = I
        lib.synth_fill_logits.restype = I
        _lib = lib
    return _lib


def _tdtype(dtype: str):
    return torch.bfloat16 if dtype == BF16 else torch.float32


def _stream():
    return torch.cuda.current_stream().cuda_stream or None


def normal(key: int, shape, dtype: str, device="cuda", idx0: int = 0, scale: float = 1.0,
           out: torch.Tensor | None = None) -> torch.Tensor:
    out = torch.empty(shape, dtype=_tdtype(dtype), device=device) if out is None else out
    rc = _load().synth_fill_normal(out.data_ptr(), int(dtype == BF16), key, idx0, out.numel(),
                                   float(scale), _stream())
    if rc:
        raise RuntimeError(f"synth_fill_normal: cuda error {rc}")
    return out


def logits(w: W.Workload, row0: int, n_rows: int, ld: int | None = None, device="cuda",
           out: torch.Tensor | None = None, pad_val: float = 0.0) -> torch.Tensor:
    ld = w.V if ld is None else ld
    out = torch.empty(n_rows, ld, dtype=_tdtype(w.dtype), device=device) if out is None else out
    rc = _load().synth_fill_logits(out.data_ptr(), int(w.dtype == BF16), w.key(W.S_LOGIT_VALS),
                                   w.key(W.S_LOGIT_ROWS), row0, n_rows, w.V, ld, w.sigma_lo,
                                   w.sigma_hi - w.sigma_lo, spike_threshold(w.spike_prob),
                                   w.spike_val, pad_val, _stream())
    if rc:
        raise RuntimeError(f"synth_fill_logits: cuda error {rc}")
    return out


def hidden(w: W.Workload, device="cuda") -> torch.Tensor:
    sumT = int(w.cu_seqlens()[-1])
    return normal(w.key(W.S_HIDDEN), (sumT, w.D), w.dtype, device)


def qk(w: W.Workload, layer: int, device="cuda", out_q=None, out_k=None):
    """Q [sumT, Hq, d] and K [sumT, Hkv, d] of one layer, sink rows of K scaled."""
    sumT = int(w.cu_seqlens()[-1])
    Q = normal(w.key_q(layer), (sumT, w.Hq, w.d), w.dtype, device, out=out_q)
    K = normal(w.key_k(layer), (sumT, w.Hkv, w.d), w.dtype, device, out=out_k)
    sinks = w.sink_rows()
    if sinks.size:
        idx = torch.as_tensor(sinks, device=device)
        K[idx] = K[idx] * w.sink_scale  # power-of-two scaling: exact
    return Q, K


def cu_seqlens(w: W.Workload, device="cuda") -> torch.Tensor:
    return torch.as_tensor(w.cu_seqlens(), dtype=torch.int32, device=device)


def head(w: W.Workload, device="cuda"):
    Wt, b, c = w.head_params()
    return (torch.as_tensor(Wt, device=device), torch.as_tensor(b, device=device),
            torch.as_tensor(c, device=device))
