"""Throughput of the ESTP feature path on GB300 (prompt tokens/s).

One step = the whole hot path over one batch of a workload.  The default is the
RL-rollout batch shaped like Llama-3-8B (256 varlen prompts, T ~ U[128, 4096],
531546 tokens, vocab 128256, all 32 layers, 32/8 heads, head_dim 128, hidden 4096,
bf16), the largest of the five workloads that runs on one GPU:
  token entropy over every row of the logits              (estp_token_entropy)
  per layer: row log-normalisers + causal column sums     (estp_attn_lse, estp_attn_importance)
  importance scaling                                      (estp_attn_importance_finalize)
  mixing, tempered softmax, pooling and the length head   (estp_pool)
Inputs are synthetic (seeded generator).  When every input of the step fits in HBM
(the other workloads) it is all resident before timing and the step is timed as one
region.  The RL batch's logits (136 GB) stay resident, but its 32 layers of Q and K
(174 GB) do not fit beside them: each layer's Q and K are generated into one buffer
before that layer's calls, as a prefill produces them layer by layer, and the step's
time is the sum of the CUDA-event times of its library calls (the generator runs
outside those events).  Every byte a timed call reads is distinct seeded data, and
the inputs are far larger than the 129 MB L2, so no flush is needed.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload NAME] [--prompts N]

--impl reference times the fp64 CPU oracle (the only other implementation of this
path) on a bounded sample of the same workload (--full: the whole batch, for the two
small workloads).  Under torchrun each rank runs its own batch (same shape,
rank-specific seed): prompts are independent, so there is no data-path collective and
the scaling is weak.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "prompt tokens/s through ESTP features (1 GB300)"
UNIT = "tokens/s"
DEFAULT_WORKLOAD = "llama3-8b_rl256"
HOST_POOL_BYTES = 32 << 30   # pinned host memory the end-to-end legs may hold (per process)
STREAM_FRACTION = 0.80       # stream Q/K per layer when resident inputs exceed this share of free HBM


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p["hbm_gbs"], p["bf16_tflops"], p.get("bf16_tflops_sustained"), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# --------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 50 ms. Each line is stamped
    with the host time at which it was read, and the summary keeps the lines that fall
    inside the window set by `window(t0, t1)` (the timed region)."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index, self.lines, self.proc = index, [], None
        self.t0, self.t1 = None, None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def window(self, t0: float, t1: float):
        self.t0, self.t1 = t0, t1

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
        return False

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        lines = self.lines
        widened = False
        if self.t0 is not None:
            # a line is read up to one sampling interval after the sample was taken
            inside = [x for x in lines if self.t0 <= x[0] <= self.t1 + 0.05]
            if not inside:
                # a timed region shorter than the sampling interval: the samples taken
                # within half a second of it
                inside = [x for x in lines if self.t0 - 0.5 <= x[0] <= self.t1 + 0.5]
                widened = True
            lines = inside
        for _, ln in lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        out = {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
               "samples": len(sm)}
        if widened:
            out["window"] = "timed region shorter than the 50 ms sampling: samples within 0.5 s of it"
        return out


# ------------------------------------------------------------------ workload
def workload_for_rank(rank: int, name: str | None = None, prompts: int = 0):
    """The named workload (default: the Llama-3-8B RL batch), optionally cut to its
    first `prompts` prompts (same lengths and bytes as in the full batch: the generator
    is counter-based); ranks > 0 draw their own batch of the same shape."""
    import dataclasses
    from synth import workloads as W
    w = W.WORKLOADS[name or DEFAULT_WORKLOAD]
    if prompts:
        w = dataclasses.replace(w, B=min(prompts, w.B), name=f"{w.name}[:{min(prompts, w.B)}]")
    if rank:
        w = dataclasses.replace(w, seed=w.seed + 1000 * rank)
    return w


def aggregate_ranks(ms: float, tokens: float, device=None):
    """Whole-job numbers from per-rank ones: the slowest rank's time (MAX) and the
    tokens of all ranks (SUM).  Prompts are independent, so this is the only
    cross-rank exchange; with one process it returns its inputs."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return ms, tokens
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    n = torch.tensor([tokens], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    return float(t.item()), float(n.item())


def esize(w) -> int:
    return 2 if w.dtype == "bf16" else 4


def layer_qk_bytes(w, sumT: int) -> int:
    return sumT * (w.Hq + w.Hkv) * w.d * esize(w)


def input_bytes(w, sumT: int) -> int:
    """Bytes of one step's inputs (logits, every selected layer's Q/K, hidden states)."""
    return sumT * w.V * esize(w) + len(w.layers) * layer_qk_bytes(w, sumT) + sumT * w.D * esize(w)


def l2_flush_buffer(w, sumT: int, device):
    """A buffer of twice the L2 size, written between timed steps when a step's inputs
    are smaller than that (else None: the inputs themselves push the previous step's
    lines out of L2)."""
    import torch
    l2 = torch.cuda.get_device_properties(device).L2_cache_size
    if input_bytes(w, sumT) >= 2 * l2:
        return None
    return torch.empty(2 * l2, dtype=torch.uint8, device=device)


def resident_bytes(w) -> int:
    """Device bytes of the step's inputs and outputs when every layer is resident."""
    sumT = int(w.cu_seqlens()[-1])
    return (sumT * w.V * esize(w) + len(w.layers) * layer_qk_bytes(w, sumT)
            + sumT * w.D * esize(w) + w.Hq * sumT * 4)


def algorithmic(w, cu):
    """Per-launch algorithmic work of each call of one step: the logits read once (and
    H written), one causal QK^T pass per layer for the row normalisers and one for the
    column sums, S read and written, and the hidden states read once by the pooling."""
    import numpy as np
    lens = np.diff(cu).astype(np.float64)
    sumT = float(lens.sum())
    attn_flops = float(w.Hq * 2 * w.d * np.sum(lens * (lens + 1) / 2))  # one QK^T pass
    return {
        "entropy": {"bytes": sumT * w.V * esize(w) + 4 * sumT},
        "lse": {"flops": attn_flops},
        "importance": {"flops": attn_flops},
        "finalize": {"bytes": 8 * sumT},
        "pool": {"bytes": sumT * w.D * esize(w) + 8 * sumT + w.B * w.D * 4},
    }


def source_hash(source: str) -> str:
    """First 16 hex digits of the SHA-256 of a kernel's translation unit followed by every
    header of the CUDA sources (sorted by name), so that a change to a shared header, too,
    marks a capture as stale."""
    csrc = os.path.join(ROOT, "paper_2608_15592_gb300", "csrc")
    h = hashlib.sha256(open(os.path.join(csrc, source), "rb").read())
    for name in sorted(os.listdir(csrc)):
        if name.endswith(".cuh"):
            h.update(open(os.path.join(csrc, name), "rb").read())
    return h.hexdigest()[:16]


def counters_for(kernel: str, workload: str):
    """The committed ncu record of a kernel (profiles/traffic.json: dram bytes per launch,
    and for the tensor-core kernels the tensor pipe's active share), if it was captured for
    this workload and the kernel's sources have not changed since the capture; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            t = json.load(f)[workload][kernel]
        return t if source_hash(t["source"]) == t["source_sha256_16"] else None
    except Exception:
        return None


def traffic_for(kernel: str, workload: str):
    """dram bytes per launch from the committed ncu record (counters_for), else None."""
    t = counters_for(kernel, workload)
    return t["dram_bytes_per_launch"] if t else None


def lib_launches(w) -> int:
    """Library launches per step: entropy 2 (kernel + merge); per layer, the row
    normaliser 2 (plan + kernel) and the column sums 3 (plan + kernel + reduce); the
    finalize 1; pooling 2 (stream + finish)."""
    return 2 + len(w.layers) * 5 + 1 + 2


class Step:
    """Device tensors of one batch plus the calls of one step.  With `stream_qk`, one
    layer's Q and K live in HBM at a time: `qk(n)` generates layer n into the buffer."""

    CALLS = ("entropy", "lse", "importance", "finalize", "pool")

    def __init__(self, estp, w, device, stream_qk: bool):
        import numpy as np
        import torch
        from synth import device as sd
        self.estp, self.w, self.device, self.stream_qk = estp, w, device, stream_qk
        self.cu_h = w.cu_seqlens()
        self.sumT = int(self.cu_h[-1])
        self.maxT = int(np.diff(self.cu_h).max())
        self.cu = sd.cu_seqlens(w, device)
        self.logits = sd.logits(w, 0, self.sumT, device=device)
        self.Q, self.K = [], []
        if stream_qk:
            self.Q.append(torch.empty(self.sumT, w.Hq, w.d, dtype=self.logits.dtype, device=device))
            self.K.append(torch.empty(self.sumT, w.Hkv, w.d, dtype=self.logits.dtype, device=device))
        else:
            for layer in w.layers:
                q, k = sd.qk(w, layer, device)
                self.Q.append(q)
                self.K.append(k)
        self.hidden = sd.hidden(w, device)
        Wt, b, c = sd.head(w, device)
        self.head = estp.Head(Wt, b, c)
        self.H = torch.empty(self.sumT, dtype=torch.float32, device=device)
        self.S = torch.empty(self.sumT, dtype=torch.float32, device=device)
        self.lse = torch.empty(w.Hq, self.sumT, dtype=torch.float32, device=device)
        self.pooled = torch.empty(w.B, w.D, dtype=torch.float32, device=device)
        self.pred = torch.empty(w.B, dtype=torch.float32, device=device)
        self.ctx = estp.Context(torch.cuda.current_device())
        self.n_layers = len(w.layers)

    def qk(self, n: int, slot: int = 0, Q=None, K=None):
        """Q and K of the n-th selected layer: the resident pair, or (streaming) the pair
        generated now into the given buffers, on the current stream."""
        from synth import device as sd
        if not self.stream_qk:
            return self.Q[n], self.K[n]
        Q = self.Q[slot] if Q is None else Q
        K = self.K[slot] if K is None else K
        sd.qk(self.w, self.w.layers[n], self.device, out_q=Q, out_k=K)
        return Q, K

    def run(self, ev=None):
        """One step on the current stream; ev: dict of per-call lists of (start, end)
        events, recorded around every library call."""
        w, c = self.w, self.ctx

        def timed(name, fn):
            if ev is None:
                return fn()
            import torch
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            out = fn()
            b.record()
            ev[name].append((a, b))
            return out

        timed("entropy", lambda: c.token_entropy(self.logits, cu_seqlens=self.cu, out=self.H))
        for n in range(self.n_layers):
            Q, K = self.qk(n)
            timed("lse", lambda: c.attn_lse(Q, K, self.cu, self.maxT, out=self.lse))
            timed("importance", lambda: c.attn_importance(Q, K, self.cu, self.maxT, lse=self.lse,
                                                          accumulate=n > 0))
        timed("finalize", lambda: c.attn_importance_finalize(self.n_layers, self.sumT, out=self.S))
        timed("pool", lambda: c.pool(self.hidden, self.H, self.S, self.cu, w.lambda1, w.lambda2,
                                     w.alpha, head=self.head, pooled=self.pooled, pred=self.pred))


# ------------------------------------------------------------------ our arm
def run_ours(args, rank, world, local_rank):
    import torch
    import paper_2608_15592_gb300 as estp

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = workload_for_rank(rank, args.workload, args.prompts)
    free = torch.cuda.mem_get_info(dev)[0]
    sumT = int(w.cu_seqlens()[-1])
    stream_qk = args.stream_qk or resident_bytes(w) > STREAM_FRACTION * free
    need = resident_bytes(w) - (len(w.layers) - 1) * layer_qk_bytes(w, sumT) if stream_qk \
        else resident_bytes(w)
    if need > STREAM_FRACTION * free:
        raise SystemExit(f"{w.name}: {need / 2**30:.1f} GiB of inputs exceed the free "
                         f"{free / 2**30:.1f} GiB even with one layer of Q/K at a time; "
                         "use --prompts to bench a slice of it")
    st = Step(estp, w, dev, stream_qk)
    torch.cuda.synchronize()

    for _ in range(args.warmup):
        st.run()
    st.ctx.sync_status()
    torch.cuda.synchronize()

    K = args.steps
    ev = {name: [] for name in Step.CALLS}
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    # small inputs: L2 written over between steps, each step timed on its own
    flush = None if stream_qk else l2_flush_buffer(w, sumT, dev)
    marks = []
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clk:
        time.sleep(0.3)  # nvidia-smi is sampling before the timed region starts
        t_host0 = time.time()
        start.record()
        for k in range(K):
            if flush is not None:
                flush.zero_()
                marks.append((torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)))
                marks[-1][0].record()
            st.run(ev)
            if flush is not None:
                marks[-1][1].record()
        end.record()
        torch.cuda.synchronize()
        clk.window(t_host0, time.time())
    if world > 1:
        torch.distributed.barrier()
    st.ctx.sync_status()
    region_ms = (sum(a.elapsed_time(b) for a, b in marks) if flush is not None
                 else start.elapsed_time(end))
    call_ms = {name: sum(a.elapsed_time(b) for a, b in ev[name]) for name in Step.CALLS}
    calls_total = sum(call_ms.values())
    # resident inputs: the whole region is library work; streamed Q/K: the calls only
    basis = calls_total if stream_qk else region_ms
    ms, tokens = aggregate_ranks(basis, float(st.sumT), dev)
    ms_per_step = ms / K
    value = tokens * K / (ms / 1e3)

    kern_ms = {name: call_ms[name] / len(ev[name]) for name in Step.CALLS}
    per_step = {name: len(ev[name]) // K for name in Step.CALLS}
    alg = algorithmic(w, st.cu_h)
    hbm, bf16, bf16_sus, peak_src = _peaks()
    kernels = {}
    for name, ms_k in kern_ms.items():
        a = alg[name]
        if name == "finalize":
            kernels[name] = {"ms": ms_k, "bound": "launch", "per_step": per_step[name]}
        elif "bytes" in a:
            achieved = a["bytes"] / (ms_k / 1e3) / 1e9
            kernels[name] = {"ms": ms_k, "bound": "hbm", "achieved": achieved, "unit": "GB/s",
                             "frac": achieved / hbm, "per_step": per_step[name],
                             "algorithmic_bytes": a["bytes"]}
        else:
            achieved = a["flops"] / (ms_k / 1e3) / 1e12
            kernels[name] = {"ms": ms_k, "bound": "tensor", "achieved": achieved,
                             "unit": "TFLOP/s", "frac": achieved / bf16_sus,
                             "per_step": per_step[name], "algorithmic_flops": a["flops"]}
    share = {k: kern_ms[k] * per_step[k] for k in kern_ms}
    dom = max(share, key=share.get)
    dk = kernels[dom]
    roofline = {"kernel": dom, "bound": dk["bound"], "achieved": dk["achieved"],
                "peak": hbm if dk["bound"] == "hbm" else bf16_sus, "unit": dk["unit"],
                "frac": dk["frac"], "traffic": traffic_for(dom, w.name),
                "peak_source": f"{peak_src} ({'hbm_gbs' if dk['bound'] == 'hbm' else 'bf16_tflops_sustained'})",
                "share_of_step": share[dom] / sum(share.values())}
    for name, rec in kernels.items():  # the committed ncu counters that still apply
        c = counters_for(name, w.name)
        if c:
            rec["ncu"] = {"dram_bytes_per_launch": c["dram_bytes_per_launch"]}
            if "tensor_pipe_active_pct" in c:
                rec["ncu"]["tensor_pipe_active_pct"] = c["tensor_pipe_active_pct"]
    if dk["bound"] == "tensor" and "ncu" in dk and "tensor_pipe_active_pct" in dk["ncu"]:
        roofline["tensor_pipe_active_pct"] = dk["ncu"]["tensor_pipe_active_pct"]
    clocks = clk.summary()

    # the library's outputs on the oracle's sample, taken while the step's inputs and
    # outputs are still those of the timed steps (the end-to-end legs overwrite them with
    # the host pool's data)
    sample = gpu_sample = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        sample = OracleSample(w)
        gpu_sample = sample.gpu_outputs(st)

    e2e = e2e_hidden = None
    if not args.no_e2e:
        pool = HostPool(st)
        e2e = run_e2e(args, st, pool, dev, world)
        e2e_hidden = run_e2e_from_hidden(args, st, pool, dev, world)
        del pool
    side = {}
    if not stream_qk:
        side["graph_replay"] = time_graph(st, K, flush)
    if not args.no_side:
        side["head_loss"] = time_head_loss(st, dev)
        side["misalignment"] = time_misalignment(st)
        side["lm_head_entropy"] = time_lm_head(st, bf16_sus)
        side["attn_forward_importance"] = time_attn_forward(st, bf16_sus, kern_ms)
    timing = ("one region (all inputs resident)" if not stream_qk else
              "sum of the CUDA-event times of the library calls; each layer's Q/K generated "
              "into one buffer before its calls, outside the events")
    out_cfg = {"workload": w.name, "B": w.B, "sum_tokens_per_gpu": st.sumT,
               "seq_len": f"U[{w.T_lo},{w.T_hi}]", "vocab": w.V, "layers": st.n_layers,
               "Hq": w.Hq, "Hkv": w.Hkv, "head_dim": w.d, "hidden": w.D,
               "mix": [w.lambda1, w.lambda2, w.alpha], "seed": w.seed,
               "parallelism": f"dp{world} (independent prompts)",
               "qk": "generated per layer (streamed)" if stream_qk else "resident",
               "timing": timing,
               "l2": (f"inputs larger than L2 ({(sumT * w.V * esize(w)) / 1e9:.1f} GB of logits "
                      "per step), no flush") if flush is None else
                     (f"inputs of {input_bytes(w, sumT) / 1e6:.1f} MB, under twice the L2: a "
                      f"{flush.numel() / 2**20:.0f} MiB buffer written between steps, outside "
                      "each step's events")}
    gen_per_step = (st.n_layers * (2 + (1 if w.sinks else 0))) if stream_qk else 0
    del st
    if rank != 0:
        return None
    cpu, parity = cpu_baseline(sample, gpu_sample) if sample is not None else (None, None)
    res = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
        "config": out_cfg, "roofline": roofline, "kernels": kernels, "cpu_baseline": cpu,
        "parity": parity,
        "e2e": e2e, "gpu_launches": lib_launches(w) * K, "clocks": clocks,
        "region_ms_per_step": region_ms / K, "calls_ms_per_step": calls_total / K,
        # context: a prefill's flash attention returns the row normalisers, and the path
        # then skips estp_attn_lse (the same metric without the lse calls' time)
        "value_lse_supplied": tokens * K / ((calls_total - call_ms["lse"]) / 1e3) if world == 1 else None,
        "generator_launches_per_step": gen_per_step,
        "e2e_from_hidden": e2e_hidden,
    }
    res.update(side)
    return res


# ------------------------------------------------------------- end to end
class HostPool:
    """Pinned host copies of the step's inputs for the end-to-end legs, at most budget()
    bytes in all: the hidden states, Q/K of the first Lp selected layers and the first R
    rows of the logits (all of them when they fit; one step of the RL batch needs 315 GB,
    more than a host may hold).  A step copies its FULL input size over the host link:
    layer n's Q/K from pool layer n mod Lp, logit row r from pool row r mod R."""

    @staticmethod
    def budget() -> int:
        """HOST_POOL_BYTES, or less: at most a third of the host's available memory shared
        by the processes of this node (torchrun's LOCAL_WORLD_SIZE)."""
        avail = None
        try:
            with open("/proc/meminfo") as f:
                for line in f:
                    if line.startswith("MemAvailable:"):
                        avail = int(line.split()[1]) * 1024
        except OSError:
            pass
        local = max(1, int(os.environ.get("LOCAL_WORLD_SIZE", os.environ.get("WORLD_SIZE", 1))))
        cap = HOST_POOL_BYTES if avail is None else min(HOST_POOL_BYTES, avail // (3 * local))
        return max(cap, 1 << 30)

    def __init__(self, st):
        import torch
        w = st.w
        self.st = st
        self.bytes = self.budget()
        self.hidden = self._pin(st.hidden)
        left = self.bytes - st.hidden.numel() * st.hidden.element_size()
        lb = layer_qk_bytes(w, st.sumT)
        self.Lp = max(1, min(st.n_layers, int(0.4 * max(left, 0)) // lb))
        self.q, self.k = [], []
        for n in range(self.Lp):
            Q, K = st.qk(n)
            self.q.append(self._pin(Q))
            self.k.append(self._pin(K))
        left -= self.Lp * lb
        row_bytes = st.logits.shape[1] * st.logits.element_size()
        self.R = max(1, min(st.sumT, max(left, 0) // row_bytes))
        self.logits = self._pin(st.logits[:self.R])
        self.pred = torch.empty(st.pred.shape, dtype=torch.float32, pin_memory=True)
        self.pooled = torch.empty(st.pooled.shape, dtype=torch.float32, pin_memory=True)
        torch.cuda.synchronize()

    @staticmethod
    def _pin(t):
        import torch
        h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        h.copy_(t)
        return h

    def copy_logits(self, dst, r0: int, r1: int) -> int:
        """dst rows [r0, r1) from the pool, on the current stream; returns bytes."""
        n = 0
        r = r0
        while r < r1:
            a = r % self.R
            m = min(r1 - r, self.R - a)
            dst[r:r + m].copy_(self.logits[a:a + m], non_blocking=True)
            n += m
            r += m
        return n * dst.shape[1] * dst.element_size()

    def describe(self) -> str:
        st = self.st
        if self.R == st.sumT and self.Lp == st.n_layers:
            return "pinned host copies of every input"
        return (f"pinned host pool of {self.bytes / 2**30:.1f} GiB: hidden states, Q/K of "
                f"{self.Lp} of {st.n_layers} layers (layer n from pool layer n mod {self.Lp}), "
                f"{self.R} of {st.sumT} logit rows (row r from pool row r mod {self.R}); "
                "every step copies its full input size over the host link")


def _qk_buffers(st):
    """Two device Q/K buffers for the pipelined legs (streamed workloads only)."""
    import torch
    if not hasattr(st, "Q2"):
        st.Q2 = torch.empty_like(st.Q[0])
        st.K2 = torch.empty_like(st.K[0])
    return [(st.Q[0], st.K[0]), (st.Q2, st.K2)]


def _blocks(step, st, world, dev, want_s: float = 2.0):
    """Warm up, then time blocks of steps with CUDA events and return (median tokens/s,
    all blocks, steps per block).  The host link is shared with other tenants of the
    machine, and single copies now and then run at a fraction of the link rate, so the
    median block is reported and every block listed."""
    import torch
    t = time.time()
    step()
    torch.cuda.synchronize()
    t1 = time.time() - t
    K = max(1, min(5, int(want_s / max(t1, 1e-3))))
    n_blocks = 5 if t1 < 0.25 else 3
    blocks = []
    for _ in range(n_blocks):
        if world > 1:
            torch.distributed.barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(K):
            step()
        b.record()
        torch.cuda.synchronize()
        ms, tokens = aggregate_ranks(a.elapsed_time(b), float(st.sumT), dev)
        blocks.append(tokens * K / (ms / 1e3))
    st.ctx.sync_status()
    return sorted(blocks)[len(blocks) // 2], blocks, K


def run_e2e(args, st, pool, dev, world):
    """Same metric through the public API with host buffers: every step copies all of
    its inputs from pinned host memory and reads the predictions and pooled features
    back.  The copies run on a copy stream: the hidden states, each layer's Q and K,
    then the logits in row chunks.  A layer's attention calls start when its Q and K
    have landed (streamed workloads: two device Q/K buffers in turn), and the entropy of
    each chunk runs as soon as that chunk is on the device, so the step costs about the
    host-to-device transfer time."""
    import torch
    w, c = st.w, st.ctx
    logit_bytes = st.logits.numel() * st.logits.element_size()
    n_chunks = max(8, int(math.ceil(logit_bytes / (8 << 30))))
    bounds = [st.sumT * i // n_chunks for i in range(n_chunks + 1)]
    copy_stream = torch.cuda.Stream(device=dev)
    L = st.n_layers
    bufs = _qk_buffers(st) if st.stream_qk else None
    ev_qk = [torch.cuda.Event() for _ in range(L)]
    ev_free = [torch.cuda.Event(), torch.cuda.Event()]
    ev_chunk = [torch.cuda.Event() for _ in range(n_chunks)]
    nbytes = {"h2d": 0}

    def step():
        h2d = 0
        main = torch.cuda.current_stream()
        copy_stream.wait_stream(main)  # the previous step has finished reading the buffers
        with torch.cuda.stream(copy_stream):
            st.hidden.copy_(pool.hidden, non_blocking=True)
        h2d += pool.hidden.numel() * pool.hidden.element_size()
        for n in range(L):
            Qd, Kd = bufs[n % 2] if bufs else (st.Q[n], st.K[n])
            with torch.cuda.stream(copy_stream):
                if bufs and n >= 2:
                    copy_stream.wait_event(ev_free[n % 2])
                Qd.copy_(pool.q[n % pool.Lp], non_blocking=True)
                Kd.copy_(pool.k[n % pool.Lp], non_blocking=True)
                ev_qk[n].record(copy_stream)
            h2d += (Qd.numel() + Kd.numel()) * Qd.element_size()
            main.wait_event(ev_qk[n])
            c.attn_lse(Qd, Kd, st.cu, st.maxT, out=st.lse)
            c.attn_importance(Qd, Kd, st.cu, st.maxT, lse=st.lse, accumulate=n > 0)
            if bufs:
                ev_free[n % 2].record(main)
        c.attn_importance_finalize(L, st.sumT, out=st.S)
        with torch.cuda.stream(copy_stream):
            for i in range(n_chunks):
                h2d += pool.copy_logits(st.logits, bounds[i], bounds[i + 1])
                ev_chunk[i].record(copy_stream)
        for i in range(n_chunks):
            r0, r1 = bounds[i], bounds[i + 1]
            main.wait_event(ev_chunk[i])
            c.token_entropy(st.logits[r0:r1], out=st.H[r0:r1])
        c.pool(st.hidden, st.H, st.S, st.cu, w.lambda1, w.lambda2, w.alpha,
               head=st.head, pooled=st.pooled, pred=st.pred)
        pool.pred.copy_(st.pred, non_blocking=True)
        pool.pooled.copy_(st.pooled, non_blocking=True)
        nbytes["h2d"] = h2d

    value, blocks, K = _blocks(step, st, world, dev)
    d2h = pool.pred.numel() * 4 + pool.pooled.numel() * 4
    return {"value": value, "unit": UNIT, "blocks": blocks,
            "h2d_bytes_per_step": nbytes["h2d"], "d2h_bytes_per_step": d2h, "steps": K,
            "host_inputs": pool.describe(),
            "pipeline": f"copy stream: hidden, Q/K per layer, then logits in {n_chunks} row "
                        "chunks; attention per layer after its Q/K land, entropy per chunk as "
                        "it lands"}


def run_e2e_from_hidden(args, st, pool, dev, world):
    """The step as a caller without materialised logits runs it: the output projection
    W [V, D] stays on the device (a model weight), and each step copies the hidden states
    and every layer's Q and K from pinned host memory.  The entropy is formed from the
    hidden states on the tensor cores (estp_lm_head_entropy) in one row slice per layer,
    each issued before the layer's attention: the main stream then never holds a layer's
    Q/K buffer for the whole projection, so the copy stream, which refills a buffer only
    after the attention of the layer two back, keeps the host link busy.  (One call over
    all rows ahead of the layers held the copies back for its ~0.33 s on the RL batch:
    4.7e5 against 6.2e5 tokens/s.)  Pooled features and predictions are copied back."""
    import numpy as np
    import torch
    import synth
    from synth import device as sd
    w, c = st.w, st.ctx
    if w.dtype != "bf16" or w.D % 64:
        return None
    W = sd.normal(synth.stream_key(w.seed, 101), (w.V, w.D), synth.BF16, scale=3.0 / np.sqrt(w.D))
    copy_stream = torch.cuda.Stream(device=dev)
    L = st.n_layers
    bufs = _qk_buffers(st) if st.stream_qk else None
    ev_h = torch.cuda.Event()
    ev_qk = [torch.cuda.Event() for _ in range(L)]
    ev_free = [torch.cuda.Event(), torch.cuda.Event()]
    nbytes = {"h2d": 0}

    n_slices = max(1, min(L, st.sumT))
    rows = [st.sumT * i // n_slices for i in range(n_slices + 1)]

    def step():
        h2d = 0
        main = torch.cuda.current_stream()
        copy_stream.wait_stream(main)
        with torch.cuda.stream(copy_stream):
            st.hidden.copy_(pool.hidden, non_blocking=True)
            ev_h.record(copy_stream)
        h2d += pool.hidden.numel() * pool.hidden.element_size()
        main.wait_event(ev_h)
        for n in range(L):
            Qd, Kd = bufs[n % 2] if bufs else (st.Q[n], st.K[n])
            with torch.cuda.stream(copy_stream):
                if bufs and n >= 2:
                    copy_stream.wait_event(ev_free[n % 2])
                Qd.copy_(pool.q[n % pool.Lp], non_blocking=True)
                Kd.copy_(pool.k[n % pool.Lp], non_blocking=True)
                ev_qk[n].record(copy_stream)
            h2d += (Qd.numel() + Kd.numel()) * Qd.element_size()
            if n < n_slices:  # this layer's slice of the entropy, while its Q/K land
                r0, r1 = rows[n], rows[n + 1]
                c.lm_head_entropy(st.hidden[r0:r1], W, out=st.H[r0:r1])
            main.wait_event(ev_qk[n])
            c.attn_lse(Qd, Kd, st.cu, st.maxT, out=st.lse)
            c.attn_importance(Qd, Kd, st.cu, st.maxT, lse=st.lse, accumulate=n > 0)
            if bufs:
                ev_free[n % 2].record(main)
        c.attn_importance_finalize(L, st.sumT, out=st.S)
        c.pool(st.hidden, st.H, st.S, st.cu, w.lambda1, w.lambda2, w.alpha,
               head=st.head, pooled=st.pooled, pred=st.pred)
        pool.pred.copy_(st.pred, non_blocking=True)
        pool.pooled.copy_(st.pooled, non_blocking=True)
        nbytes["h2d"] = h2d

    value, blocks, K = _blocks(step, st, world, dev)
    del W
    d2h = pool.pred.numel() * 4 + pool.pooled.numel() * 4
    return {"value": value, "unit": UNIT, "blocks": blocks,
            "h2d_bytes_per_step": nbytes["h2d"], "d2h_bytes_per_step": d2h, "steps": K,
            "host_inputs": pool.describe(),
            "pipeline": f"W resident; copy stream: hidden, then Q/K per layer; per layer, "
                        f"the entropy from hidden states of 1/{n_slices} of the rows (tensor "
                        "cores) while its Q/K land, then its attention; pooling"}


# ------------------------------------------------------- side measurements
def time_graph(st, K: int, flush):
    """The same step captured once in a CUDA graph and replayed K times (resident
    workloads only): the library calls enqueue nothing that a graph cannot hold (no
    allocation once the workspace has grown, no synchronisation), so a replay launches
    the step's kernels without the host's per-call work.  Each replay is timed with CUDA
    events, with the L2 written over in between when the inputs are small.  The outputs of
    a replay are checked bit for bit against the step run call by call."""
    import torch
    st.run()
    torch.cuda.synchronize()
    ref = [t.clone() for t in (st.H, st.S, st.pooled, st.pred)]
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        st.run()
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        st.run()
    for t in (st.H, st.S, st.pooled, st.pred):
        t.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    same = all(torch.equal(a, b) for a, b in zip(ref, (st.H, st.S, st.pooled, st.pred)))
    ms = []
    for _ in range(K):
        if flush is not None:
            flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        g.replay()
        b.record()
        ms.append((a, b))
    torch.cuda.synchronize()
    st.ctx.sync_status()
    per = sum(a.elapsed_time(b) for a, b in ms) / K
    del g
    return {"ms_per_step": per, "value": st.sumT / (per / 1e3), "unit": UNIT, "steps": K,
            "launches_per_step": lib_launches(st.w), "bit_equal_to_calls": same}


def _time_calls(fn, sync, min_warm_s: float = 0.5, want_s: float = 1.5, min_iters: int = 3):
    """CUDA-event time of one fn() after at least min_warm_s (and two calls) of warm-up;
    the number of timed calls targets want_s.  Returns ms per call."""
    import torch
    t_end = time.time() + min_warm_s
    n = 0
    t0 = time.time()
    while n < 2 or time.time() < t_end:
        fn()
        torch.cuda.synchronize()
        n += 1
    per = (time.time() - t0) / n
    iters = max(min_iters, min(50, int(want_s / max(per, 1e-4))))
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(iters):
        fn()
    b.record()
    torch.cuda.synchronize()
    sync()
    return a.elapsed_time(b) / iters


def time_head_loss(st, dev):
    """The training loss of the length head (Eqs. 3-1 to 3-3, estp_head_loss) on the
    step's pooled features with synthetic targets: not part of the step, timed on its
    own with CUDA events.  Its algorithmic bytes (W and the pooled features read by the
    forward and the gradient kernels, the three gradients written) are a few MB, so it
    is bound by launch latency, not by HBM."""
    import torch
    import paper_2608_15592_gb300 as estp
    B, D = st.pooled.shape
    K = st.head.W.shape[0]
    g = torch.Generator(device=dev).manual_seed(7)
    targets = torch.rand(B, generator=g, device=dev) * float(st.head.centers[-1] + st.head.centers[0])
    ms = _time_calls(lambda: st.ctx.head_loss(st.pooled, st.head, targets, 0.5),
                     st.ctx.sync_status, min_warm_s=0.05, want_s=0.05)
    nbytes = 4 * (2 * K * D + 2 * B * D + K * D + K + B * D + B * K)
    out = {"ms": ms, "B": B, "D": D, "K": K, "launches": 2, "bytes": nbytes,
           "achieved_gbs": nbytes / (ms / 1e3) / 1e9, "bound": "launch"}
    # the MLP predictor (one ReLU layer of F = 1024 units), its loss and all gradients
    F = 1024
    W1 = torch.randn(F, D, generator=g, device=dev) / D ** 0.5
    b1 = torch.randn(F, generator=g, device=dev) * 0.3
    W2 = torch.randn(K, F, generator=g, device=dev) * (3.0 / F ** 0.5)
    mlp = estp.MlpHead(W1, b1, W2, st.head.bias, st.head.centers)
    ms = _time_calls(lambda: st.ctx.mlp_head_loss(st.pooled, mlp, targets, 0.5),
                     st.ctx.sync_status, min_warm_s=0.05, want_s=0.05)
    # W1 read by the hidden layer and by both of its gradients, dL/dW1 written
    mbytes = 4 * (3 * F * D + F * D + 2 * K * F + 4 * B * D + 4 * B * F)
    out["mlp"] = {"ms": ms, "F": F, "launches": 5, "bytes": mbytes,
                  "achieved_gbs": mbytes / (ms / 1e3) / 1e9, "bound": "launch / L2"}
    return out


def time_lm_head(st, peak_tflops):
    """Token entropy with the logits formed from the step's hidden states and a seeded
    output projection W [V, D] (estp_lm_head_entropy): not part of the step, which
    reads materialised logits; timed on its own with CUDA events.  Algorithmic work is
    2 sumT D V flops of the projection; the logits it does not write and read back are
    2 sumT V bytes.  A call runs at full tensor rate, so the GPU settles under its power
    cap: at least 0.5 s of warm-up calls come first, and the figure is compared with the
    sustained bf16 peak."""
    import numpy as np
    import torch
    import synth
    from synth import device as sd
    w = st.w
    if w.dtype != "bf16" or w.D % 64:
        return None
    W = sd.normal(synth.stream_key(w.seed, 101), (w.V, w.D), synth.BF16, scale=3.0 / np.sqrt(w.D))
    H = torch.empty(st.sumT, dtype=torch.float32, device=W.device)
    ms = _time_calls(lambda: st.ctx.lm_head_entropy(st.hidden, W, out=H), st.ctx.sync_status)
    flops = 2.0 * st.sumT * w.D * w.V
    tf = flops / (ms / 1e3) / 1e12
    del W
    return {"ms": ms, "rows": st.sumT, "D": w.D, "V": w.V, "flops": flops, "launches": 2,
            "bound": "tensor", "achieved": tf, "unit": "TFLOP/s", "peak": peak_tflops,
            "frac": tf / peak_tflops, "tokens_per_s": st.sumT / (ms / 1e3),
            "logit_bytes_not_stored": 2 * st.sumT * w.V}


def time_attn_forward(st, peak_tflops, kern_ms, max_layers: int = 2):
    """The prefill's attention forward with the importance column sums of the same
    probabilities (estp_attn_forward_importance) with seeded V [sumT, Hkv, d]: not part
    of the step, which takes Q and K only; timed on its own with CUDA events over the
    first `max_layers` selected layers (every layer has the same shapes and work), with
    the row normalisers supplied (as a prefill provides them) and computed by the call.
    Algorithmic work: the causal pairs of every head, 2 d flops each for QK^T and for PV.
    For context, the same layers through torch's scaled_dot_product_attention (one
    causal call per prompt; no importance)."""
    import torch
    import synth
    from synth import device as sd
    w = st.w
    if w.dtype != "bf16" or w.d != 128:
        return None
    n_layers = min(max_layers, st.n_layers)
    bufs = _qk_buffers(st) if st.stream_qk else [(st.Q[n], st.K[n]) for n in range(n_layers)]
    QK = [st.qk(n, Q=bufs[n][0], K=bufs[n][1]) for n in range(n_layers)]
    V = [sd.normal(w.key_v(w.layers[n]), (st.sumT, w.Hkv, w.d), synth.BF16, device=st.device)
         for n in range(n_layers)]
    O = torch.empty(st.sumT, w.Hq, w.d, dtype=torch.bfloat16, device=st.device)
    alg = algorithmic(w, st.cu_h)["lse"]["flops"] * 2
    c = st.ctx
    lse = [c.attn_lse(Q, K, st.cu, st.maxT) for Q, K in QK]

    def fused_only():
        for n, (Q, K) in enumerate(QK):
            c.attn_forward_importance(Q, K, V[n], st.cu, st.maxT, lse=lse[n], accumulate=n > 0,
                                      out=O)

    def fused_internal():
        for n, (Q, K) in enumerate(QK):
            c.attn_forward_importance(Q, K, V[n], st.cu, st.maxT, lse=None, accumulate=n > 0,
                                      out=O)

    ms_fused = _time_calls(fused_only, c.sync_status) / n_layers
    ms_internal = _time_calls(fused_internal, c.sync_status) / n_layers
    tf = alg / (ms_fused / 1e3) / 1e12
    out = {"ms_per_layer": ms_fused, "ms_per_layer_with_lse": ms_internal,
           "layers_timed": n_layers, "flops_per_layer": alg, "bound": "tensor", "achieved": tf,
           "unit": "TFLOP/s", "peak": peak_tflops, "frac": tf / peak_tflops,
           "launches_per_layer": 3, "unfused_importance_ms_per_layer":
           kern_ms["lse"] + kern_ms["importance"]}
    try:
        import torch.nn.functional as F
        bounds = [(int(st.cu_h[b]), int(st.cu_h[b + 1])) for b in range(w.B)]

        def sdpa():
            for n, (Q, K) in enumerate(QK):
                for t0, t1 in bounds:
                    if t1 > t0:
                        q = Q[t0:t1].transpose(0, 1).unsqueeze(0)
                        k = K[t0:t1].transpose(0, 1).unsqueeze(0)
                        v = V[n][t0:t1].transpose(0, 1).unsqueeze(0)
                        F.scaled_dot_product_attention(q, k, v, is_causal=True, enable_gqa=True)

        out["torch_sdpa_ms_per_layer"] = _time_calls(sdpa, lambda: None) / n_layers
    except Exception as exc:  # context only
        out["torch_sdpa_ms_per_layer"] = None
        out["torch_sdpa_error"] = str(exc)[:200]
    del V, O
    return out


def time_misalignment(st):
    """The entropy/importance misalignment counts (estp_misalignment, pct = 40) on the
    step's H and S: a diagnostic, timed on its own.  One CTA per prompt runs four radix
    selections (8 passes each over the prompt's values, from L2) and a counting pass;
    its algorithmic bytes are the 8 bytes per token of H and S."""
    ms = _time_calls(lambda: st.ctx.misalignment(st.H, st.S, st.cu), st.ctx.sync_status,
                     min_warm_s=0.05, want_s=0.1)
    nbytes = 8 * st.sumT + 12 * st.w.B
    return {"ms": ms, "B": st.w.B, "tokens": st.sumT, "pct": 40, "launches": 1, "bytes": nbytes,
            "achieved_gbs": nbytes / (ms / 1e3) / 1e9, "bound": "latency (selection passes)"}


# ------------------------------------------------------------- CPU oracle arm
class OracleSample:
    """The bounded sample of a workload on which both CPU legs (this arm's cpu_baseline
    and --impl reference) time the fp64 oracle, extrapolated to the whole batch by
    algorithmic work:
      entropy   : 64 logit rows spread evenly over the batch (work: rows x V);
      importance: the prompt whose length T is nearest the batch median, the last selected
                  layer; all Hq heads when its T (T + 1) / 2 causal pairs per head allow,
                  else one head per host thread (evenly spaced) and only the last query
                  rows of the prompt (attn_colsum_rows).  Work: query-key pairs x heads,
                  scaled by sum_b T_b (T_b + 1) / 2 x layers x Hq;
      pooling   : that prompt's hidden states and the length head, scaled by tokens.
    The oracle parallelises over (prompt, head) units, so the head count keeps every
    host thread busy.  The inputs are generated once, outside the timing."""

    PAIR_BUDGET = 6e8  # query-key pairs x heads of the importance sample

    @classmethod
    def sizing(cls, w, n_threads: int):
        """(prompt b, heads, first query row, query-key pairs per head) of the sample."""
        import numpy as np
        lens = np.diff(w.cu_seqlens()).astype(np.int64)
        b = int(np.argmin(np.abs(lens - np.median(lens))))
        T = int(lens[b])
        full = T * (T + 1) // 2
        if full * w.Hq <= cls.PAIR_BUDGET:
            h, r0 = w.Hq, 0
        else:
            h = min(w.Hq, n_threads)
            # first row r0 with (T (T + 1) - r0 (r0 + 1)) / 2 pairs per head within budget
            per_head = cls.PAIR_BUDGET / h
            r0 = 0 if full <= per_head else int(math.ceil(
                (-1 + math.sqrt(1 + 4 * (T * (T + 1) - 2 * per_head))) / 2))
        heads = np.unique(np.linspace(0, w.Hq - 1, h).round().astype(np.int32))
        return b, heads, r0, (T * (T + 1) - r0 * (r0 + 1)) / 2.0

    def __init__(self, w):
        import numpy as np
        from synth import workloads as W
        self.w = w
        self.n_threads = os.cpu_count() or 1
        cu = w.cu_seqlens()
        lens = np.diff(cu).astype(np.int64)
        self.sumT = int(cu[-1])
        self.ent_rows = np.unique(np.linspace(0, self.sumT - 1, min(self.sumT, 64)).round()
                                  .astype(np.int64))
        self.x = W.host_logits(w, self.ent_rows)
        b, self.heads, r0, pairs = self.sizing(w, self.n_threads)
        self.rows = np.arange(cu[b], cu[b + 1])
        T = len(self.rows)
        self.row_from = r0
        # query rows before row_from are never read by the oracle: left zero
        layer = w.layers[-1]
        self.K = W.host_k(w, layer, self.rows)
        self.Q = np.zeros((T, w.Hq, w.d), dtype=self.K.dtype)
        self.Q[r0:] = W.host_q(w, layer, self.rows[r0:])
        self.sub = np.asarray([0, T], dtype=np.int32)
        # pooling and the head on (at most) the prompt's first 4096 tokens as one prompt
        Tp = min(T, 4096)
        self.hid = W.host_hidden(w, self.rows[:Tp])
        self.sub_pool = np.asarray([0, Tp], dtype=np.int32)
        self.head = w.head_params()
        self.ratio_ent = self.sumT / len(self.ent_rows)
        self.ratio_imp = (np.sum(lens * (lens + 1) / 2.0) * len(w.layers) * w.Hq
                          / (pairs * len(self.heads)))
        self.ratio_pool = self.sumT / Tp
        rows_txt = "all rows" if r0 == 0 else f"query rows {r0}..{T - 1}"
        self.b, self.T = b, T
        self.H = self.C = None
        self.desc = (f"entropy {len(self.ent_rows)} rows; importance: the {T}-token prompt "
                     f"(nearest the median), {rows_txt}, 1 layer x {len(self.heads)} of {w.Hq} "
                     f"heads; pooling + head on its first {min(T, 4096)} tokens; extrapolated by algorithmic work "
                     f"to the {self.sumT}-token batch of {len(w.layers)} layers")

    def run(self):
        """Times one pass of the sample; returns (wall seconds, extrapolated seconds per
        batch)."""
        import numpy as np
        import oracle
        w, n = self.w, self.n_threads
        t0 = time.perf_counter()
        H = oracle.token_entropy(self.x, n_threads=n)
        t1 = time.perf_counter()
        C = np.zeros(len(self.rows))
        oracle.attn_colsum_rows(self.Q, self.K, self.sub, w.scale, self.row_from,
                                heads=self.heads, out=C, n_threads=n)
        t2 = time.perf_counter()
        Tp = int(self.sub_pool[1])
        P = oracle.pool(self.hid, np.resize(H, Tp), C[:Tp], self.sub_pool, w.lambda1,
                        w.lambda2, w.alpha)
        oracle.length_head(P, *self.head)
        t3 = time.perf_counter()
        self.H, self.C = H, C
        batch = ((t1 - t0) * self.ratio_ent + (t2 - t1) * self.ratio_imp
                 + (t3 - t2) * self.ratio_pool)
        return t3 - t0, batch


    def gpu_outputs(self, st):
        """The library's results on the sample, for the parity record: the step's entropy
        of the sampled rows, and the importance of the sampled prompt alone (its rows of
        the last selected layer's Q and K, the sample's heads, one layer, lse computed by
        the call)."""
        import torch
        w = self.w
        H = st.H[torch.as_tensor(self.ent_rows, device=st.H.device)].cpu().numpy()
        Q, K = st.qk(len(w.layers) - 1)
        r0, r1 = int(self.rows[0]), int(self.rows[-1]) + 1
        cu = torch.as_tensor([0, self.T], dtype=torch.int32, device=Q.device)
        st.ctx.attn_importance(Q[r0:r1], K[r0:r1], cu, self.T, heads=[int(h) for h in self.heads])
        S = st.ctx.attn_importance_finalize(1, self.T).cpu().numpy()
        st.ctx.sync_status()
        return H, S

    def parity(self, gpu):
        """Largest errors of the library against the oracle on the sample: entropy (nats,
        absolute) on the sampled rows; importance (relative, element by element) on the keys
        the sample's query rows fix exactly (every key when the sample holds all rows)."""
        import numpy as np
        H_gpu, S_gpu = gpu
        S_ref = self.C / (self.T * len(self.heads))
        keys = np.arange(self.row_from, self.T)
        rel = np.abs(S_gpu[keys] - S_ref[keys]) / np.maximum(np.abs(S_ref[keys]), 1e-30)
        return {"entropy_max_abs_err_nats": float(np.max(np.abs(H_gpu - self.H))),
                "entropy_rows": int(len(self.ent_rows)),
                "importance_max_rel_err": float(rel.max()) if rel.size else 0.0,
                "importance_keys": int(len(keys)),
                "importance_sample": f"prompt {self.b} ({self.T} tokens), last selected layer, "
                                     f"{len(self.heads)} of {self.w.Hq} heads",
                "tolerance": {"entropy_nats": 1e-3, "importance_rel": 1e-2}}


def cpu_baseline(s, gpu=None, repeats: int = 3):
    """The oracle timed on the sample s (median of `repeats` passes), and, with the
    library's outputs on the same sample (OracleSample.gpu_outputs), the parity record."""
    runs = [s.run() for _ in range(repeats)]
    batch = statistics.median(r[1] for r in runs)
    cpu = {"value": s.sumT / batch, "unit": UNIT, "cores": s.n_threads, "kind": "oracle",
           "sample": s.desc + f"; median of {repeats} passes of "
                              f"{statistics.median(r[0] for r in runs):.1f} s",
           "extrapolated": True}
    return cpu, (s.parity(gpu) if gpu is not None else None)


def run_reference(args, rank, world):
    """The oracle as the comparison arm: each step is one pass of the bounded sample
    (OracleSample) of the same workload, extrapolated to tokens/s by algorithmic work;
    with --full, each step is the oracle over the whole batch (the two small
    workloads), measured, not extrapolated."""
    if rank != 0:
        return None
    import numpy as np
    w = workload_for_rank(0, args.workload, args.prompts)
    if args.full:
        step, desc, n = _full_oracle_step(w)
    else:
        s = OracleSample(w)
        step, desc, n = s.run, s.desc, s.n_threads
    walls, batches = [], []
    for i in range(args.warmup + args.steps):
        wall, batch = step()
        if i >= args.warmup:
            walls.append(wall)
            batches.append(batch)
    value = w.cu_seqlens()[-1] * len(batches) / sum(batches)
    ms_per_step = 1e3 * float(np.mean(walls))
    return {
        "impl": "reference", "metric": METRIC, "value": float(value), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "sum_tokens_per_gpu": int(w.cu_seqlens()[-1]),
                   "step": "the whole batch" if args.full else "one pass of the bounded sample",
                   "tokens_equivalent_per_step": float(value) * ms_per_step / 1e3},
        "cpu_baseline": {"value": float(value), "unit": UNIT, "cores": n, "kind": "oracle",
                         "sample": desc, "extrapolated": not args.full},
        "e2e": {"value": float(value), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def _full_inputs(w):
    """Every input of the batch on the host: drawn by the device generator and copied
    back when a GPU is present (the same bits as the host generator, which is far slower
    for the 3.3e9 logits of the Qwen batch), else by the host generator."""
    import numpy as np
    from synth import workloads as W
    sumT = int(w.cu_seqlens()[-1])
    try:
        import torch
        gpu = torch.cuda.is_available()
    except Exception:
        gpu = False
    if not gpu:
        rows = np.arange(sumT)
        return (W.host_logits(w, rows), [W.host_qk(w, layer) for layer in w.layers],
                W.host_hidden(w, rows))
    import __graft_entry__
    __graft_entry__._build_module().build_synth()  # the generator's device side only
    from synth import device as sd

    def host(t):
        if t.dtype == torch.bfloat16:
            return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        return t.cpu().numpy()

    x = host(sd.logits(w, 0, sumT))
    qk = []
    for layer in w.layers:
        Q, K = sd.qk(w, layer)
        qk.append((host(Q), host(K)))
    hid = host(sd.hidden(w))
    torch.cuda.empty_cache()
    return x, qk, hid


def _full_oracle_step(w):
    """The oracle over the whole batch: entropy of every row, importance of every
    selected layer and head, pooling and the head."""
    import numpy as np
    import oracle
    n = os.cpu_count() or 1
    cu = w.cu_seqlens()
    sumT = int(cu[-1])
    x, qk, hid = _full_inputs(w)
    head = w.head_params()

    def step():
        t0 = time.perf_counter()
        H = oracle.token_entropy(x, n_threads=n)
        C = np.zeros(sumT)
        for Q, K in qk:
            oracle.attn_colsum(Q, K, cu, w.scale, out=C, n_threads=n)
        S = oracle.importance(C, cu, len(w.layers), w.Hq)
        P = oracle.pool(hid, H, S, cu, w.lambda1, w.lambda2, w.alpha)
        oracle.length_head(P, *head)
        t = time.perf_counter() - t0
        return t, t

    return step, f"the whole {sumT}-token batch, every selected layer and head", n


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-side", action="store_true",
                    help="skip the side measurements (head losses, misalignment, entropy from "
                         "hidden states, fused attention forward)")
    ap.add_argument("--no-e2e", action="store_true",
                    help="skip the end-to-end legs with host buffers")
    ap.add_argument("--stream-qk", action="store_true",
                    help="generate each layer's Q/K before its calls even when all layers fit")
    ap.add_argument("--full", action="store_true",
                    help="--impl reference: run the oracle over the whole batch")
    ap.add_argument("--workload", default=None,
                    help=f"workload name (default {DEFAULT_WORKLOAD}); see synth/workloads.py")
    ap.add_argument("--prompts", type=int, default=0,
                    help="bench only the first N prompts of the workload")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local_rank = int(os.environ.get("LOCAL_RANK", 0))
    if args.impl == "reference":
        out = run_reference(args, rank, world)
        if out is not None:
            print(json.dumps(out), flush=True)
        return
    import __graft_entry__
    if rank == 0 or world == 1:
        __graft_entry__.build()
    import torch
    if world > 1:
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl")
        torch.distributed.barrier()
        if rank != 0:
            __graft_entry__.build()
    out = run_ours(args, rank, world, local_rank)
    if out is not None:
        print(json.dumps(out), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
