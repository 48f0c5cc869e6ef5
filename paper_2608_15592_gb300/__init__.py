"""ESTP feature extraction on GB300: Python binding of the C ABI in include/estp.h.

This module only marshals arguments: every step of the path runs in the CUDA
kernels of ``libestp.so`` (built in-tree by ``build.py``).  Importing it without
the built library raises ImportError; there is no CPU fallback.

The raw ctypes functions carry the C names (``lib.estp_token_entropy`` ...); the
``Context`` methods wrap them for torch CUDA tensors:

    ctx = Context(device=0)
    H   = ctx.token_entropy(logits)                       # Eq. 2-1
    lse = ctx.attn_lse(Q, K, cu_seqlens, max_seqlen)      # row normalisers of A
    ctx.attn_importance(Q, K, cu_seqlens, max_seqlen, lse=None, accumulate=False)
    S   = ctx.attn_importance_finalize(n_layers)          # Eq. 2-0
    pooled, y = ctx.pool(hidden, H, S, cu_seqlens, mix, head)   # Eqs. 2-2..2-4, 3-2
"""
from __future__ import annotations

import ctypes
import math
import os
from dataclasses import dataclass

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libestp.so")
# the same library built with -DESTP_CHECKS (device bounds checks), for tests and debugging
CHECKS_LIB_PATH = os.path.join(_HERE, "_build_checks", "libestp_checks.so")

ESTP_OK, ESTP_ERR_INVALID_ARG, ESTP_ERR_UNSUPPORTED = 0, 1, 2
ESTP_ERR_CUDA, ESTP_ERR_TIMEOUT, ESTP_ERR_WORKSPACE = 3, 4, 5
ESTP_ERR_BOUNDS = 6
ESTP_F32, ESTP_BF16 = 0, 1
ESTP_IMP_EXCLUDE_SELF = 1
ESTP_IMP_DIV_CAUSAL = 2
ESTP_IMP_DIV_NONE = 4
_DIVISOR_FLAGS = {"length": 0, "causal": ESTP_IMP_DIV_CAUSAL, "none": ESTP_IMP_DIV_NONE}

# every entry point declared in include/estp.h
EXPORTS = ("estp_create", "estp_destroy", "estp_last_error", "estp_sync_status",
           "estp_token_entropy", "estp_attn_lse", "estp_attn_importance",
           "estp_attn_importance_finalize", "estp_pool", "estp_token_entropy_noalloc",
           "estp_head_loss", "estp_misalignment", "estp_lm_head_entropy",
           "estp_mlp_head_predict", "estp_mlp_head_loss", "estp_attn_forward_importance",
           "estp_set_wait_limit")


class EstpError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"estp status {status}: {msg}")
        self.status = status


class MixParams(ctypes.Structure):
    """estp_mix_params: T_i = lambda1 S_i + lambda2 H_i, e = softmax(T / alpha)."""
    _fields_ = [("lambda1", ctypes.c_float), ("lambda2", ctypes.c_float),
                ("alpha", ctypes.c_float)]


class _Head(ctypes.Structure):
    _fields_ = [("W", ctypes.c_void_p), ("bias", ctypes.c_void_p),
                ("centers", ctypes.c_void_p), ("K", ctypes.c_int32)]


class _MlpHead(ctypes.Structure):
    _fields_ = [("W1", ctypes.c_void_p), ("b1", ctypes.c_void_p), ("W2", ctypes.c_void_p),
                ("b2", ctypes.c_void_p), ("centers", ctypes.c_void_p), ("F", ctypes.c_int32),
                ("K", ctypes.c_int32)]


class _MlpGrads(ctypes.Structure):
    _fields_ = [("W1", ctypes.c_void_p), ("b1", ctypes.c_void_p), ("W2", ctypes.c_void_p),
                ("b2", ctypes.c_void_p), ("pooled", ctypes.c_void_p)]


def load_library(path: str = LIB_PATH):
    """ctypes handle of a build of the C ABI with every entry point's signature set:
    libestp.so by default, or CHECKS_LIB_PATH for the bounds-checked build."""
    if not os.path.exists(path):
        raise ImportError(f"ESTP CUDA library not built ({path} missing): run "
                          "paper_2608_15592_gb300/build.py or __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    P, I32, I64, F, U32 = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float,
                           ctypes.c_uint32)
    sigs = {
        "estp_create": ([ctypes.POINTER(ctypes.c_void_p), ctypes.c_int], ctypes.c_int),
        "estp_destroy": ([P], None),
        "estp_last_error": ([P], ctypes.c_char_p),
        "estp_sync_status": ([P, P], ctypes.c_int),
        "estp_set_wait_limit": ([P, I64], ctypes.c_int),
        "estp_token_entropy": ([P, P, ctypes.c_int, I64, I64, I64, P, I32, P, P], ctypes.c_int),
        "estp_attn_lse": ([P, P, P, ctypes.c_int, I32, I32, I32, F, P, I32, I64, I32, P, P],
                          ctypes.c_int),
        "estp_attn_importance": ([P, P, P, ctypes.c_int, P, I32, I32, I32, F, P, I32, P, I32,
                                  I64, I32, ctypes.c_int, U32, P], ctypes.c_int),
        "estp_attn_importance_finalize": ([P, I32, P, P], ctypes.c_int),
        "estp_attn_forward_importance": ([P, P, P, P, ctypes.c_int, P, I32, I32, I32, F, P, I32,
                                          I64, I32, ctypes.c_int, U32, P, P], ctypes.c_int),
        "estp_token_entropy_noalloc": ([P, ctypes.c_int, I64, I64, I64, P, P], ctypes.c_int),
        "estp_pool": ([P, P, ctypes.c_int, I64, I64, P, P, P, I32, I64, MixParams,
                       ctypes.POINTER(_Head), P, P, P], ctypes.c_int),
        "estp_head_loss": ([P, P, I32, I64, ctypes.POINTER(_Head), P, F, P, P, P, P, P],
                           ctypes.c_int),
        "estp_misalignment": ([P, P, P, P, I32, I64, I32, P, P], ctypes.c_int),
        "estp_mlp_head_predict": ([P, P, I32, I64, ctypes.POINTER(_MlpHead), P, P, P],
                                  ctypes.c_int),
        "estp_mlp_head_loss": ([P, P, I32, I64, ctypes.POINTER(_MlpHead), P, F, P,
                                ctypes.POINTER(_MlpGrads), P], ctypes.c_int),
        "estp_lm_head_entropy": ([P, P, I64, P, I64, ctypes.c_int, I64, I64, I64, P, P],
                                 ctypes.c_int),
    }
    for name, (args, res) in sigs.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    return lib


lib = load_library()


def _check(status: int):
    if status != ESTP_OK:
        raise EstpError(status, lib.estp_last_error(None).decode())


def _dtype(t) -> int:
    import torch
    if t.dtype == torch.bfloat16:
        return ESTP_BF16
    if t.dtype == torch.float32:
        return ESTP_F32
    raise TypeError(f"tensors are bf16 or fp32, got {t.dtype}")


def _ptr(t) -> int | None:
    return None if t is None else t.data_ptr()


def _stream(stream) -> int | None:
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream or None


@dataclass
class Head:
    """Linear length head (Eq. 3-2): W [K, D], bias [K] or None, centers [K], fp32 CUDA."""
    W: "object"
    bias: "object"
    centers: "object"


@dataclass
class MlpHead:
    """MLP predictor (Sec. 3.3): u = relu(W1 h + b1), z = W2 u + b2, then Eq. 3-2.
    W1 [F, D], b1 [F] or None, W2 [K, F], b2 [K] or None, centers [K], fp32 CUDA."""
    W1: "object"
    b1: "object"
    W2: "object"
    b2: "object"
    centers: "object"


class Context:
    """One estp_ctx (status word + workspace) on a CUDA device, in `library` (the release
    build by default; load_library(CHECKS_LIB_PATH) for the bounds-checked one)."""

    def __init__(self, device: int = 0, library=None):
        self.device = device
        self._lib = lib if library is None else library
        h = ctypes.c_void_p()
        self._check(self._lib.estp_create(ctypes.byref(h), device))
        self._h = h

    def _check(self, status: int):
        if status != ESTP_OK:
            raise EstpError(status, self._lib.estp_last_error(None).decode())

    def close(self):
        if getattr(self, "_h", None):
            self._lib.estp_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def sync_status(self, stream=None):
        """estp_sync_status: synchronise the stream; raise on a device-side error."""
        self._check(self._lib.estp_sync_status(self._h, _stream(stream)))

    def set_wait_limit(self, cycles: int = 0):
        """estp_set_wait_limit: limit (SM cycles) of the attention kernels' abortable
        waits for later calls; 0 restores the default.  A testing aid."""
        self._check(self._lib.estp_set_wait_limit(self._h, int(cycles)))

    # ------------------------------------------------------------------ (a)
    def lm_head_entropy(self, hidden, W, out=None, stream=None):
        """estp_lm_head_entropy: entropy (nats) of softmax(hidden @ W^T) per row, the logits
        formed on the tensor cores and never stored.  hidden: bf16 [rows, D], W: bf16 [V, D]
        (row views of wider arrays allowed: stride(1) == 1)."""
        import torch
        assert hidden.dim() == 2 and W.dim() == 2 and hidden.shape[1] == W.shape[1]
        assert hidden.numel() == 0 or hidden.stride(1) == 1
        assert W.stride(1) == 1
        rows, D = hidden.shape
        V = W.shape[0]
        ldh = hidden.stride(0) if rows > 1 else D
        ldw = W.stride(0) if V > 1 else D
        out = torch.empty(rows, dtype=torch.float32, device=hidden.device) if out is None else out
        self._check(self._lib.estp_lm_head_entropy(self._h, _ptr(hidden), ldh, _ptr(W), ldw, _dtype(hidden),
                                        rows, D, V, _ptr(out), _stream(stream)))
        return out

    def token_entropy(self, logits, V: int | None = None, cu_seqlens=None, out=None,
                      stream=None):
        """estp_token_entropy on a 2-D [rows, ld] tensor (stride(1) == 1)."""
        import torch
        assert logits.dim() == 2 and (logits.numel() == 0 or logits.stride(1) == 1)
        rows, ld = logits.shape[0], logits.stride(0) if logits.shape[0] > 1 else logits.shape[1]
        V = logits.shape[1] if V is None else V
        out = torch.empty(rows, dtype=torch.float32, device=logits.device) if out is None else out
        B = 0 if cu_seqlens is None else cu_seqlens.numel() - 1
        self._check(self._lib.estp_token_entropy(self._h, _ptr(logits), _dtype(logits), rows, V, ld,
                                      _ptr(cu_seqlens), B, _ptr(out), _stream(stream)))
        return out

    # ------------------------------------------------------------------ (b)
    def attn_lse(self, Q, K, cu_seqlens, max_seqlen: int, scale: float | None = None,
                 out=None, stream=None):
        """estp_attn_lse: fp32 [Hq, sumT] row log-normalisers."""
        import torch
        sumT, Hq, d = Q.shape
        Hkv = K.shape[1]
        scale = 1.0 / math.sqrt(d) if scale is None else scale
        out = torch.empty(Hq, sumT, dtype=torch.float32, device=Q.device) if out is None else out
        self._check(self._lib.estp_attn_lse(self._h, _ptr(Q), _ptr(K), _dtype(Q), Hq, Hkv, d, scale,
                                 _ptr(cu_seqlens), cu_seqlens.numel() - 1, sumT, max_seqlen,
                                 _ptr(out), _stream(stream)))
        return out

    def attn_importance(self, Q, K, cu_seqlens, max_seqlen: int, lse=None,
                        scale: float | None = None, heads=None, accumulate: bool = False,
                        exclude_self: bool = False, divisor: str = "length", stream=None):
        """estp_attn_importance for one layer (column sums into the context).
        divisor: "length" (Eq. 2-0's 1/N), "causal" or "none" (ESTP_IMP_DIV_*), applied
        by attn_importance_finalize and fixed by the call that opens the accumulation."""
        sumT, Hq, d = Q.shape
        Hkv = K.shape[1]
        scale = 1.0 / math.sqrt(d) if scale is None else scale
        if heads is None:
            hp, nh = None, Hq
        else:
            arr = (ctypes.c_int32 * len(heads))(*[int(h) for h in heads])
            hp, nh = ctypes.cast(arr, ctypes.c_void_p), len(heads)
        self._check(self._lib.estp_attn_importance(self._h, _ptr(Q), _ptr(K), _dtype(Q), _ptr(lse), Hq,
                                        Hkv, d, scale, hp, nh, _ptr(cu_seqlens),
                                        cu_seqlens.numel() - 1, sumT, max_seqlen,
                                        1 if accumulate else 0,
                                        (ESTP_IMP_EXCLUDE_SELF if exclude_self else 0)
                                        | _DIVISOR_FLAGS[divisor],
                                        _stream(stream)))

    def attn_forward_importance(self, Q, K, V, cu_seqlens, max_seqlen: int, lse=None,
                                scale: float | None = None, accumulate: bool = False,
                                exclude_self: bool = False, divisor: str = "length", out=None,
                                stream=None):
        """estp_attn_forward_importance for one layer: returns the attention output bf16
        [sumT, Hq, 128] and adds the column sums of all Hq heads into the context's
        importance accumulation (same accumulation and flags as attn_importance)."""
        import torch
        sumT, Hq, d = Q.shape
        Hkv = K.shape[1]
        scale = 1.0 / math.sqrt(d) if scale is None else scale
        if out is None:
            out = torch.empty(sumT, Hq, d, dtype=Q.dtype, device=Q.device)
        self._check(self._lib.estp_attn_forward_importance(
            self._h, _ptr(Q), _ptr(K), _ptr(V), _dtype(Q), _ptr(lse), Hq, Hkv, d, scale,
            _ptr(cu_seqlens), cu_seqlens.numel() - 1, sumT, max_seqlen, 1 if accumulate else 0,
            (ESTP_IMP_EXCLUDE_SELF if exclude_self else 0) | _DIVISOR_FLAGS[divisor], _ptr(out),
            _stream(stream)))
        return out

    def attn_importance_finalize(self, n_layers: int, sumT: int, device=None, out=None,
                                 stream=None):
        """estp_attn_importance_finalize: S [sumT] (Eq. 2-0)."""
        import torch
        if out is None:
            out = torch.empty(sumT, dtype=torch.float32,
                              device=device if device is not None else f"cuda:{self.device}")
        self._check(self._lib.estp_attn_importance_finalize(self._h, n_layers, _ptr(out), _stream(stream)))
        return out

    # ------------------------------------------------------------------ (c)
    def misalignment(self, entropy, importance, cu_seqlens, pct: int = 40, out=None,
                     stream=None):
        """estp_misalignment: int32 [B, 3] = (k, |TopH & BotS|, |BotH & TopS|) per prompt."""
        import torch
        B = cu_seqlens.numel() - 1
        out = torch.empty(B, 3, dtype=torch.int32, device=entropy.device) if out is None else out
        self._check(self._lib.estp_misalignment(self._h, _ptr(entropy), _ptr(importance), _ptr(cu_seqlens),
                                     B, entropy.numel(), pct, _ptr(out), _stream(stream)))
        return out

    def head_loss(self, pooled, head: Head, targets, lambda3: float, grads: bool = True,
                  stream=None):
        """estp_head_loss (Eqs. 3-1 to 3-3): returns (loss [1], and if grads:
        dL/dW [K, D], dL/dbias [K], dL/dpooled [B, D]), fp32 CUDA tensors."""
        import torch
        B, D = pooled.shape
        K = head.W.shape[0]
        dev = pooled.device
        loss = torch.empty(1, dtype=torch.float32, device=dev)
        gW = torch.empty(K, D, dtype=torch.float32, device=dev) if grads else None
        gb = torch.empty(K, dtype=torch.float32, device=dev) if grads else None
        gp = torch.empty(B, D, dtype=torch.float32, device=dev) if grads else None
        hp = ctypes.pointer(_Head(_ptr(head.W), _ptr(head.bias), _ptr(head.centers), K))
        self._check(self._lib.estp_head_loss(self._h, _ptr(pooled), B, D, hp, _ptr(targets), lambda3,
                                  _ptr(loss), _ptr(gW), _ptr(gb), _ptr(gp), _stream(stream)))
        return (loss, gW, gb, gp) if grads else loss

    @staticmethod
    def _mlp(head: "MlpHead"):
        return ctypes.pointer(_MlpHead(_ptr(head.W1), _ptr(head.b1), _ptr(head.W2), _ptr(head.b2),
                                       _ptr(head.centers), head.W1.shape[0], head.W2.shape[0]))

    def mlp_head_predict(self, pooled, head: "MlpHead", probs: bool = False, stream=None):
        """estp_mlp_head_predict: predicted lengths [B] (and p_hat [B, K] if probs)."""
        import torch
        B, D = pooled.shape
        pred = torch.empty(B, dtype=torch.float32, device=pooled.device)
        p = torch.empty(B, head.W2.shape[0], dtype=torch.float32, device=pooled.device) if probs else None
        self._check(self._lib.estp_mlp_head_predict(self._h, _ptr(pooled), B, D, self._mlp(head), _ptr(pred),
                                         _ptr(p), _stream(stream)))
        return (pred, p) if probs else pred

    def mlp_head_loss(self, pooled, head: "MlpHead", targets, lambda3: float, grads=True,
                      stream=None):
        """estp_mlp_head_loss (Eqs. 3-1, 3-3 through the MLP predictor): returns loss [1]
        and, if grads, (dL/dW1 [F, D], dL/db1 [F], dL/dW2 [K, F], dL/db2 [K], dL/dpooled
        [B, D]).  grads may also be a set of those names to compute only some of them."""
        import torch
        B, D = pooled.shape
        F, K = head.W1.shape[0], head.W2.shape[0]
        dev = pooled.device
        shapes = {"W1": (F, D), "b1": (F,), "W2": (K, F), "b2": (K,), "pooled": (B, D)}
        want = set(shapes) if grads is True else (set(grads) if grads else set())
        out = {k: torch.empty(v, dtype=torch.float32, device=dev) if k in want else None
               for k, v in shapes.items()}
        loss = torch.empty(1, dtype=torch.float32, device=dev)
        gp = ctypes.pointer(_MlpGrads(*[_ptr(out[k]) for k in ("W1", "b1", "W2", "b2", "pooled")]))
        self._check(self._lib.estp_mlp_head_loss(self._h, _ptr(pooled), B, D, self._mlp(head), _ptr(targets),
                                      lambda3, _ptr(loss), gp if want else None, _stream(stream)))
        if not grads:
            return loss
        return (loss, *[out[k] for k in ("W1", "b1", "W2", "b2", "pooled")])

    def pool(self, hidden, entropy, importance, cu_seqlens, lambda1: float, lambda2: float,
             alpha: float, head: Head | None = None, D: int | None = None, pooled=None,
             pred=None, stream=None):
        """estp_pool: returns (pooled [B, D], predicted lengths [B] or None)."""
        import torch
        assert hidden.dim() == 2 and (hidden.numel() == 0 or hidden.stride(1) == 1)
        sumT = hidden.shape[0]
        ldh = hidden.stride(0) if sumT > 1 else hidden.shape[1]
        D = hidden.shape[1] if D is None else D
        B = cu_seqlens.numel() - 1
        dev = hidden.device
        pooled = torch.empty(B, D, dtype=torch.float32, device=dev) if pooled is None else pooled
        hp = None
        if head is not None:
            pred = torch.empty(B, dtype=torch.float32, device=dev) if pred is None else pred
            hp = ctypes.pointer(_Head(_ptr(head.W), _ptr(head.bias), _ptr(head.centers),
                                      head.W.shape[0]))
        mix = MixParams(lambda1, lambda2, alpha)
        self._check(self._lib.estp_pool(self._h, _ptr(hidden), _dtype(hidden), D, ldh, _ptr(entropy),
                             _ptr(importance), _ptr(cu_seqlens), B, sumT, mix, hp,
                             _ptr(pooled), _ptr(pred) if head is not None else None,
                             _stream(stream)))
        return pooled, (pred if head is not None else None)
