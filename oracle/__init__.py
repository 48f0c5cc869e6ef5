"""fp64 CPU oracle for the ESTP feature path -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s cpu_baseline /
reference arm may import this package.  It wraps ``liboracle.so`` (plain C in
``estp_oracle.c``), which shares no code with the CUDA library.

Functions and the paper passages they follow (arXiv 2608.15592):
  token_entropy   Eq. 2-1 (Sec. 3.2)
  lm_head_entropy Eq. 2-1 of the logits h W^T formed from hidden states
  attn_lse        the row normaliser of the causal softmax A (Sec. 3.1)
  attn_colsum     sum_i A_ij of Eq. 2-0 for one layer, summed over query heads
  attn_output     O = A V, the prefill's attention output (Sec. 3.1)
  attn_colsum_rows  the same from the rows i >= row_from only (exact for late keys)
  importance      Eq. 2-0: S_j = C_j / (N * layers * heads); divisor variants of its 1/N
  pool            Eqs. 2-2, 2-3, 2-4
  length_head     Eq. 3-2 with a linear projection
  head_loss       Eqs. 3-1, 3-3 (soft-label CE + MSE) and their gradients
  mlp_length_head Eq. 3-2 behind the one-hidden-layer ReLU MLP predictor
  mlp_head_loss   Eqs. 3-1, 3-3 through that MLP, and every gradient
  misalignment    the entropy/importance misalignment counts of Sec. 1 (Fig. 1b), numpy

bf16 arrays are passed as numpy uint16 holding the raw bfloat16 bits.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "_build", "liboracle.so")
F32, BF16 = 0, 1


def build(force: bool = False) -> str:
    """Compile estp_oracle.c with gcc (IEEE, no FMA contraction) into _build/."""
    src = os.path.join(_HERE, "estp_oracle.c")
    hdr = os.path.join(_HERE, "estp_oracle.h")
    if (not force and os.path.exists(_SO)
            and os.path.getmtime(_SO) >= max(os.path.getmtime(src), os.path.getmtime(hdr))):
        return _SO
    os.makedirs(os.path.dirname(_SO), exist_ok=True)
    tmp = _SO + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared",
                           "-D_DEFAULT_SOURCE", "-o", tmp, src, "-lm", "-lpthread"])
    os.replace(tmp, _SO)
    return _SO


class _Lib:
    """ctypes view of one build of the oracle library."""

    def __init__(self, path: str):
        lib = ctypes.CDLL(path)
        P, I, I64, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_double
        sig = {
            "oracle_token_entropy": [P, I, I64, I64, I64, P, I],
            "oracle_lm_head_entropy": [P, P, I, I64, I64, I64, I64, I64, P, I],
            "oracle_attn_lse": [P, P, I, I, I, I, D, P, I, P, I],
            "oracle_attn_output": [P, P, P, I, I, I, I, D, P, I, P, I],
            "oracle_attn_output_rows": [P, P, P, I, I, I, I, D, P, I, I64, P, I],
            "oracle_attn_colsum": [P, P, I, I, I, I, D, P, I, P, I, I, P, I],
            "oracle_attn_colsum_rows": [P, P, I, I, I, I, D, P, I, P, I, I, I64, P, I],
            "oracle_importance": [P, P, I, I, I, P],
            "oracle_importance_div": [P, P, I, I, I, I, I, P],
            "oracle_pool": [P, I, I64, I64, P, P, P, I, D, D, D, P, P],
            "oracle_length_head": [P, I, I64, P, P, P, I, P, P],
            "oracle_head_loss": [P, I, I64, P, P, P, I, P, D, P, P, P, P],
            "oracle_mlp_length_head": [P, I, I64, P, P, I, P, P, P, I, P, P],
            "oracle_mlp_head_loss": [P, I, I64, P, P, I, P, P, P, I, P, D, P, P, P, P, P, P],
        }
        for name, args in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
            setattr(self, name, fn)


_lib = None
_override = None


def _load():
    global _lib
    if _override is not None:
        return _override
    if _lib is None:
        _lib = _Lib(build())
    return _lib


class use_library:
    """Context manager: route the functions of this module through another build
    of the oracle (used by the tests that plant mistakes in a copy of the source)."""

    def __init__(self, path: str):
        self.lib = _Lib(path)

    def __enter__(self):
        global _override
        self._prev, _override = _override, self.lib
        return self

    def __exit__(self, *exc):
        global _override
        _override = self._prev
        return False


def compile_source(src_text: str, out_path: str) -> str:
    """Compile a (possibly modified) copy of estp_oracle.c with the oracle's flags."""
    d = os.path.dirname(out_path)
    os.makedirs(d, exist_ok=True)
    src = os.path.join(d, "estp_oracle_variant.c")
    with open(src, "w") as f:
        f.write(src_text)
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared",
                           "-D_DEFAULT_SOURCE", "-I", _HERE, "-o", out_path, src, "-lm",
                           "-lpthread"])
    return out_path


def source_text() -> str:
    with open(os.path.join(_HERE, "estp_oracle.c")) as f:
        return f.read()


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return F32
    if a.dtype == np.uint16:
        return BF16
    raise TypeError(f"oracle inputs are float32 or uint16 (bf16 bits), got {a.dtype}")


def _check(rc, name):
    if rc != 0:
        raise ValueError(f"{name}: invalid argument")


def _cu(cu):
    return np.ascontiguousarray(cu, dtype=np.int32)


def token_entropy(logits: np.ndarray, V: int | None = None, n_threads: int = 0) -> np.ndarray:
    """Eq. 2-1 per row of a 2-D [rows, ld] array (first V columns are the vocabulary)."""
    logits = np.ascontiguousarray(logits)
    rows, ld = logits.shape
    V = ld if V is None else V
    out = np.zeros(rows, dtype=np.float64)
    _check(_load().oracle_token_entropy(_ptr(logits), _dtype_code(logits), rows, V, ld,
                                        _ptr(out), n_threads), "token_entropy")
    return out


def lm_head_entropy(hidden: np.ndarray, W: np.ndarray, n_threads: int = 0) -> np.ndarray:
    """Eq. 2-1 per row of hidden [rows, D] with the logits hidden @ W^T, W [V, D] (same
    element type; bf16 as raw uint16 bits)."""
    hidden, W = np.ascontiguousarray(hidden), np.ascontiguousarray(W)
    assert hidden.dtype == W.dtype and hidden.ndim == 2 and W.ndim == 2
    rows, D = hidden.shape
    V, Dw = W.shape
    assert Dw == D
    out = np.zeros(rows, dtype=np.float64)
    _check(_load().oracle_lm_head_entropy(_ptr(hidden), _ptr(W), _dtype_code(hidden), rows, D,
                                          V, D, D, _ptr(out), n_threads), "lm_head_entropy")
    return out


def attn_output(Q, K, V, cu_seqlens, scale, n_threads: int = 0) -> np.ndarray:
    """O [sumT, Hq, d] = A V of the causal attention of one layer (V read with K's head)."""
    Q, K, V = np.ascontiguousarray(Q), np.ascontiguousarray(K), np.ascontiguousarray(V)
    cu = _cu(cu_seqlens)
    sumT, Hq, d = Q.shape
    Hkv = K.shape[1]
    assert K.shape == V.shape and K.dtype == Q.dtype == V.dtype
    out = np.zeros((sumT, Hq, d), dtype=np.float64)
    _check(_load().oracle_attn_output(_ptr(Q), _ptr(K), _ptr(V), _dtype_code(Q), Hq, Hkv, d,
                                      float(scale), _ptr(cu), len(cu) - 1, _ptr(out), n_threads),
           "attn_output")
    return out


def attn_output_rows(Q, K, V, cu_seqlens, scale, row_from: int, n_threads: int = 0) -> np.ndarray:
    """attn_output for the prompt-local query rows >= row_from; the other rows are 0."""
    Q, K, V = np.ascontiguousarray(Q), np.ascontiguousarray(K), np.ascontiguousarray(V)
    cu = _cu(cu_seqlens)
    sumT, Hq, d = Q.shape
    Hkv = K.shape[1]
    assert K.shape == V.shape and K.dtype == Q.dtype == V.dtype
    out = np.zeros((sumT, Hq, d), dtype=np.float64)
    _check(_load().oracle_attn_output_rows(_ptr(Q), _ptr(K), _ptr(V), _dtype_code(Q), Hq, Hkv,
                                           d, float(scale), _ptr(cu), len(cu) - 1,
                                           int(row_from), _ptr(out), n_threads),
           "attn_output_rows")
    return out


def attn_lse(Q, K, cu_seqlens, scale, n_threads: int = 0) -> np.ndarray:
    """Row log-normalisers [Hq, sumT] of the causal attention of one layer."""
    Q, K, cu = np.ascontiguousarray(Q), np.ascontiguousarray(K), _cu(cu_seqlens)
    sumT, Hq, d = Q.shape
    Hkv = K.shape[1]
    out = np.zeros((Hq, sumT), dtype=np.float64)
    _check(_load().oracle_attn_lse(_ptr(Q), _ptr(K), _dtype_code(Q), Hq, Hkv, d, float(scale),
                                   _ptr(cu), len(cu) - 1, _ptr(out), n_threads), "attn_lse")
    return out


def attn_colsum(Q, K, cu_seqlens, scale, heads=None, exclude_self=False,
                out: np.ndarray | None = None, n_threads: int = 0) -> np.ndarray:
    """sum_{h in heads} sum_{i>=j} A^h_ij for one layer, added into ``out`` ([sumT] f64)."""
    Q, K, cu = np.ascontiguousarray(Q), np.ascontiguousarray(K), _cu(cu_seqlens)
    sumT, Hq, d = Q.shape
    Hkv = K.shape[1]
    if out is None:
        out = np.zeros(sumT, dtype=np.float64)
    h = None if heads is None else np.ascontiguousarray(heads, dtype=np.int32)
    nh = Hq if h is None else len(h)
    _check(_load().oracle_attn_colsum(_ptr(Q), _ptr(K), _dtype_code(Q), Hq, Hkv, d,
                                      float(scale), _ptr(h), nh, _ptr(cu), len(cu) - 1,
                                      int(bool(exclude_self)), _ptr(out), n_threads),
           "attn_colsum")
    return out


def attn_colsum_rows(Q, K, cu_seqlens, scale, row_from: int, heads=None, exclude_self=False,
                     out: np.ndarray | None = None, n_threads: int = 0) -> np.ndarray:
    """attn_colsum formed from the rows i >= row_from of every prompt: exact for keys
    with prompt-local index >= row_from."""
    Q, K, cu = np.ascontiguousarray(Q), np.ascontiguousarray(K), _cu(cu_seqlens)
    sumT, Hq, d = Q.shape
    Hkv = K.shape[1]
    if out is None:
        out = np.zeros(sumT, dtype=np.float64)
    h = None if heads is None else np.ascontiguousarray(heads, dtype=np.int32)
    nh = Hq if h is None else len(h)
    _check(_load().oracle_attn_colsum_rows(_ptr(Q), _ptr(K), _dtype_code(Q), Hq, Hkv, d,
                                           float(scale), _ptr(h), nh, _ptr(cu), len(cu) - 1,
                                           int(bool(exclude_self)), int(row_from), _ptr(out),
                                           n_threads), "attn_colsum_rows")
    return out


DIVISORS = {"length": 0, "causal": 1, "none": 2}


def importance(C, cu_seqlens, n_layers: int, n_heads: int, divisor: str = "length",
               exclude_self: bool = False) -> np.ndarray:
    """Eq. 2-0 scaling of accumulated column sums. divisor: "length" (the paper's N),
    "causal" (the queries whose terms enter C_j) or "none" (mean column sum)."""
    C, cu = np.ascontiguousarray(C, dtype=np.float64), _cu(cu_seqlens)
    out = np.zeros_like(C)
    if divisor == "length":
        _check(_load().oracle_importance(_ptr(C), _ptr(cu), len(cu) - 1, n_layers, n_heads,
                                         _ptr(out)), "importance")
    else:
        _check(_load().oracle_importance_div(_ptr(C), _ptr(cu), len(cu) - 1, n_layers, n_heads,
                                             DIVISORS[divisor], int(bool(exclude_self)),
                                             _ptr(out)), "importance")
    return out


def pool(hidden, H, S, cu_seqlens, lambda1, lambda2, alpha, D: int | None = None,
         return_weights: bool = False):
    """Eqs. 2-2..2-4; returns pooled [B, D] (and the weights e_i if asked)."""
    hidden = np.ascontiguousarray(hidden)
    rows, ldh = hidden.shape
    D = ldh if D is None else D
    cu = _cu(cu_seqlens)
    B = len(cu) - 1
    H = np.ascontiguousarray(H, dtype=np.float64)
    S = np.ascontiguousarray(S, dtype=np.float64)
    pooled = np.zeros((B, D), dtype=np.float64)
    w = np.zeros(rows, dtype=np.float64) if return_weights else None
    _check(_load().oracle_pool(_ptr(hidden), _dtype_code(hidden), D, ldh, _ptr(H), _ptr(S),
                               _ptr(cu), B, float(lambda1), float(lambda2), float(alpha),
                               _ptr(w), _ptr(pooled)), "pool")
    return (pooled, w) if return_weights else pooled


def length_head(pooled, W, bias, centers, return_probs: bool = False):
    """Eq. 3-2: returns y_hat [B] (and p_hat [B, K] if asked)."""
    pooled = np.ascontiguousarray(pooled, dtype=np.float64)
    B, D = pooled.shape
    W = np.ascontiguousarray(W, dtype=np.float32)
    K = W.shape[0]
    bias = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    centers = np.ascontiguousarray(centers, dtype=np.float32)
    y = np.zeros(B, dtype=np.float64)
    p = np.zeros((B, K), dtype=np.float64) if return_probs else None
    _check(_load().oracle_length_head(_ptr(pooled), B, D, _ptr(W), _ptr(bias), _ptr(centers),
                                      K, _ptr(p), _ptr(y)), "length_head")
    return (y, p) if return_probs else y


def head_loss(pooled, W, bias, centers, y, lambda3: float, grads: bool = True):
    """Eqs. 3-1 and 3-3 through the linear head of Eq. 3-2, batch mean; returns the loss
    and, if asked, (grad_W [K, D], grad_bias [K], grad_pooled [B, D])."""
    pooled = np.ascontiguousarray(pooled, dtype=np.float64)
    B, D = pooled.shape
    W = np.ascontiguousarray(W, dtype=np.float32)
    K = W.shape[0]
    bias = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    centers = np.ascontiguousarray(centers, dtype=np.float32)
    y = np.ascontiguousarray(y, dtype=np.float32)
    loss = np.zeros(1, dtype=np.float64)
    gW = np.zeros((K, D)) if grads else None
    gb = np.zeros(K) if grads else None
    gp = np.zeros((B, D)) if grads else None
    _check(_load().oracle_head_loss(_ptr(pooled), B, D, _ptr(W), _ptr(bias), _ptr(centers), K,
                                    _ptr(y), float(lambda3), _ptr(loss), _ptr(gW), _ptr(gb),
                                    _ptr(gp)), "head_loss")
    return (float(loss[0]), gW, gb, gp) if grads else float(loss[0])


def _mlp_args(W1, b1, W2, b2, centers):
    W1 = np.ascontiguousarray(W1, dtype=np.float32)
    W2 = np.ascontiguousarray(W2, dtype=np.float32)
    b1 = None if b1 is None else np.ascontiguousarray(b1, dtype=np.float32)
    b2 = None if b2 is None else np.ascontiguousarray(b2, dtype=np.float32)
    return W1, b1, W2, b2, np.ascontiguousarray(centers, dtype=np.float32)


def mlp_length_head(pooled, W1, b1, W2, b2, centers, return_probs: bool = False):
    """Eq. 3-2 behind the MLP u = relu(W1 h + b1), z = W2 u + b2: y_hat [B] (and p_hat)."""
    pooled = np.ascontiguousarray(pooled, dtype=np.float64)
    B, D = pooled.shape
    W1, b1, W2, b2, centers = _mlp_args(W1, b1, W2, b2, centers)
    F, K = W1.shape[0], W2.shape[0]
    y = np.zeros(B)
    p = np.zeros((B, K)) if return_probs else None
    _check(_load().oracle_mlp_length_head(_ptr(pooled), B, D, _ptr(W1), _ptr(b1), F, _ptr(W2),
                                          _ptr(b2), _ptr(centers), K, _ptr(p), _ptr(y)),
           "mlp_length_head")
    return (y, p) if return_probs else y


def mlp_head_loss(pooled, W1, b1, W2, b2, centers, y, lambda3: float, grads: bool = True):
    """Eqs. 3-1, 3-3 through the MLP predictor; returns the loss and, if asked,
    (grad_W1 [F, D], grad_b1 [F], grad_W2 [K, F], grad_b2 [K], grad_pooled [B, D])."""
    pooled = np.ascontiguousarray(pooled, dtype=np.float64)
    B, D = pooled.shape
    W1, b1, W2, b2, centers = _mlp_args(W1, b1, W2, b2, centers)
    F, K = W1.shape[0], W2.shape[0]
    y = np.ascontiguousarray(y, dtype=np.float32)
    loss = np.zeros(1)
    g = [np.zeros((F, D)), np.zeros(F), np.zeros((K, F)), np.zeros(K), np.zeros((B, D))] if grads \
        else [None] * 5
    _check(_load().oracle_mlp_head_loss(_ptr(pooled), B, D, _ptr(W1), _ptr(b1), F, _ptr(W2),
                                        _ptr(b2), _ptr(centers), K, _ptr(y), float(lambda3),
                                        _ptr(loss), *[_ptr(x) for x in g]), "mlp_head_loss")
    return (float(loss[0]), *g) if grads else float(loss[0])


def misalignment(H, S, cu_seqlens, pct: int = 40) -> np.ndarray:
    """Per prompt b: k = floor(pct * T_b / 100); TopX / BotX the k tokens with the largest /
    smallest X (ties: the lower token index first), X in {H, S}. Returns int64 [B, 3]:
    (k, |TopH & BotS|, |BotH & TopS|) -- high-entropy tokens of low importance and
    low-entropy tokens of high importance (the paper splits at the 60th percentile:
    pct = 40)."""
    H = np.asarray(H, dtype=np.float64)
    S = np.asarray(S, dtype=np.float64)
    cu = _cu(cu_seqlens)
    if not 1 <= pct <= 50:
        raise ValueError("pct must be in 1..50")
    out = np.zeros((len(cu) - 1, 3), dtype=np.int64)
    for b in range(len(cu) - 1):
        t0, t1 = int(cu[b]), int(cu[b + 1])
        T = t1 - t0
        k = pct * T // 100
        out[b, 0] = k
        if k == 0:
            continue
        idx = np.arange(T)
        # sort by value, the lower index first among equal values (lexsort: last key primary)
        top = lambda x: set(np.lexsort((idx, -x))[:k].tolist())
        bot = lambda x: set(np.lexsort((idx, x))[:k].tolist())
        h, s = H[t0:t1], S[t0:t1]
        out[b, 1] = len(top(h) & bot(s))
        out[b, 2] = len(bot(h) & top(s))
    return out
