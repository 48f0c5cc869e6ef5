"""The five synthetic workloads, shaped like the paper's backbones and scenarios.

The paper evaluates on ForeLen (prompts from LongBench, ZeroSCROLLS, IFEval and
RL math/code sets) with Qwen2.5 and Llama backbones (Sec. 4.1).  None of that data
is used: these seeded recipes stand in for it with the same tensor shapes,
length mixes (short / medium / long prompt bins, Table 2; long-context reasoning)
and value structure (per-token logit temperature, rare confident spikes, attention
sinks).  Every array is drawn from the counter-based generator in ``synth``.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

from . import BF16, F32, normal, round_to, splitmix64, stream_key

# stream numbers of the generator (per workload seed)
S_LENGTHS = 1
S_LOGIT_VALS = 2
S_LOGIT_ROWS = 3
S_HIDDEN = 4
S_HEAD_W = 5
S_Q0 = 1000  # Q of layer l: S_Q0 + 2l, K of layer l: S_Q0 + 2l + 1
S_V0 = 3000  # V of layer l: S_V0 + l


@dataclass(frozen=True)
class Workload:
    name: str
    seed: int
    B: int
    T_lo: int
    T_hi: int
    dtype: str
    V: int
    n_layers_model: int
    layers_used: int          # importance from the last `layers_used` layers
    Hq: int
    Hkv: int
    d: int
    D: int
    sigma_lo: float = 0.5
    sigma_hi: float = 4.0
    spike_prob: float = 0.0
    spike_val: float = 12.0
    sinks: int = 0            # first `sinks` positions of each prompt: K rows x sink_scale
    sink_scale: float = 8.0
    K_bins: int = 32
    bin_width: float = 256.0
    lambda1: float = 0.7
    lambda2: float = 0.3
    alpha: float = 1.0
    note: str = field(default="", compare=False)

    # ---------------------------------------------------------- lengths
    def seqlens(self) -> np.ndarray:
        if self.T_lo == self.T_hi:
            return np.full(self.B, self.T_lo, dtype=np.int64)
        w = splitmix64(stream_key(self.seed, S_LENGTHS), np.arange(self.B, dtype=np.uint64))
        return self.T_lo + (w % np.uint64(self.T_hi - self.T_lo + 1)).astype(np.int64)

    def cu_seqlens(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.seqlens())]).astype(np.int32)

    @property
    def layers(self) -> list[int]:
        return list(range(self.n_layers_model - self.layers_used, self.n_layers_model))

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.d)

    # -------------------------------------------------------- stream keys
    def key(self, stream: int) -> int:
        return stream_key(self.seed, stream)

    def key_q(self, layer: int) -> int:
        return self.key(S_Q0 + 2 * layer)

    def key_k(self, layer: int) -> int:
        return self.key(S_Q0 + 2 * layer + 1)

    def key_v(self, layer: int) -> int:
        return self.key(S_V0 + layer)

    # ------------------------------------------------------- head params
    def head_params(self):
        """Random linear length head (W ~ N(0, 1/D), bias 0) and bin centres
        c_k = (k + 1/2) * bin_width; K = K_bins (fp32)."""
        K, D = self.K_bins, self.D
        z = normal(self.key(S_HEAD_W), np.arange(K * D, dtype=np.uint64))
        W = (z / math.sqrt(D)).astype(np.float32).reshape(K, D)
        bias = np.zeros(K, dtype=np.float32)
        centers = ((np.arange(K) + 0.5) * self.bin_width).astype(np.float32)
        return W, bias, centers

    def sink_rows(self) -> np.ndarray:
        """Global token indices whose K rows are scaled by sink_scale."""
        if not self.sinks:
            return np.zeros(0, dtype=np.int64)
        cu = self.cu_seqlens()
        r = [cu[b] + s for b in range(self.B) for s in range(self.sinks)
             if cu[b] + s < cu[b + 1]]
        return np.asarray(r, dtype=np.int64)


C1 = Workload("single_T128_f32", seed=0, B=1, T_lo=128, T_hi=128, dtype=F32, V=32000,
              n_layers_model=1, layers_used=1, Hq=8, Hkv=8, d=64, D=1024,
              note="single prompt, T=128, fp32")
C2 = Workload("qwen2.5-7b_varlen16", seed=1, B=16, T_lo=256, T_hi=2048, dtype=BF16,
              V=152064, n_layers_model=28, layers_used=4, Hq=28, Hkv=4, d=128, D=3584,
              spike_prob=0.01, spike_val=12.0,
              note="Qwen2.5-7B shape, 16 prompts T~U[256,2048], last 4 layers")
C3 = Workload("qwen2.5-7b_long4x32k", seed=2, B=4, T_lo=32768, T_hi=32768, dtype=BF16,
              V=152064, n_layers_model=28, layers_used=8, Hq=28, Hkv=4, d=128, D=3584,
              spike_prob=0.01, spike_val=12.0, sinks=4,
              note="long-context reasoning, 4 x 32768, last 8 layers, 4 sink keys")
C4 = Workload("llama3-8b_rl256", seed=3, B=256, T_lo=128, T_hi=4096, dtype=BF16,
              V=128256, n_layers_model=32, layers_used=32, Hq=32, Hkv=8, d=128, D=4096,
              note="RL rollout batch, 256 prompts T~U[128,4096], all 32 layers")
C5 = Workload("llama3-70b_8x8k", seed=4, B=8, T_lo=8192, T_hi=8192, dtype=BF16,
              V=128256, n_layers_model=80, layers_used=80, Hq=64, Hkv=8, d=128, D=8192,
              sinks=4, note="Llama-3-70B shape, 8 x 8192, all 80 layers, 4 sink keys")

WORKLOADS = {w.name: w for w in (C1, C2, C3, C4, C5)}
ORDER = [C1, C2, C3, C4, C5]


# ------------------------------------------------------- host tensors
def host_logits(w: Workload, rows, ld: int | None = None):
    from . import logits_rows
    return logits_rows(w.key(S_LOGIT_VALS), w.key(S_LOGIT_ROWS), rows, w.V, w.dtype,
                       w.sigma_lo, w.sigma_hi, w.spike_prob, w.spike_val, ld=ld)


def host_hidden(w: Workload, rows) -> np.ndarray:
    rows = np.asarray(rows, dtype=np.int64).reshape(-1)
    idx = (rows[:, None] * w.D + np.arange(w.D)[None, :]).reshape(-1)
    return round_to(normal(w.key(S_HIDDEN), idx), w.dtype).reshape(rows.size, w.D)


def _rows(w: Workload, rows):
    if rows is None:
        rows = np.arange(int(w.cu_seqlens()[-1]))
    return np.asarray(rows, dtype=np.int64).reshape(-1)


def host_q(w: Workload, layer: int, rows=None) -> np.ndarray:
    """Q [n, Hq, d] of one layer for global token rows (all by default)."""
    rows = _rows(w, rows)
    qi = (rows[:, None] * (w.Hq * w.d) + np.arange(w.Hq * w.d)[None, :]).reshape(-1)
    return round_to(normal(w.key_q(layer), qi), w.dtype).reshape(rows.size, w.Hq, w.d)


def host_k(w: Workload, layer: int, rows=None) -> np.ndarray:
    """K [n, Hkv, d] of one layer for global token rows (all by default), with the sink
    rows scaled."""
    rows = _rows(w, rows)
    ki = (rows[:, None] * (w.Hkv * w.d) + np.arange(w.Hkv * w.d)[None, :]).reshape(-1)
    K64 = normal(w.key_k(layer), ki).reshape(rows.size, w.Hkv, w.d)
    sink = np.isin(rows, w.sink_rows())
    K64[sink] *= w.sink_scale
    return round_to(K64, w.dtype).reshape(rows.size, w.Hkv, w.d)


def host_qk(w: Workload, layer: int, rows=None):
    """Q [n, Hq, d] and K [n, Hkv, d] of one layer for global token rows (all by default),
    with the sink rows of K scaled."""
    return host_q(w, layer, rows), host_k(w, layer, rows)
