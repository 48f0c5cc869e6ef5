"""Host-side logic of bench.py (CPU): the oracle sample's extrapolation, the reference
arm's JSON line, the host pool's memory budget and the step's launch count."""
import json
import os
import subprocess
import sys

import numpy as np

import bench
from synth import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_oracle_sample_ratios_cover_the_batch():
    # one prompt, all heads, all rows: every ratio is exactly 1 (the sample is the batch)
    w = W.Workload("tiny", seed=5, B=1, T_lo=40, T_hi=40, dtype="bf16", V=50,
                   n_layers_model=1, layers_used=1, Hq=4, Hkv=2, d=64, D=32)
    s = bench.OracleSample(w)
    assert s.ratio_ent == 1.0 and s.ratio_pool == 1.0 and s.row_from == 0
    assert abs(s.ratio_imp - 1.0) < 1e-12 and list(s.heads) == [0, 1, 2, 3]
    wall, batch = s.run()
    assert wall > 0 and abs(batch - wall) <= 0.5 * wall + 1e-3


def test_parity_record_of_the_sample():
    # outputs equal to the oracle's give zero errors; a planted error in one sampled row
    # and one key shows up in the record with its size
    w = W.Workload("tiny", seed=6, B=2, T_lo=20, T_hi=40, dtype="bf16", V=50,
                   n_layers_model=1, layers_used=1, Hq=4, Hkv=2, d=64, D=32)
    s = bench.OracleSample(w)
    s.run()
    S = s.C / (s.T * len(s.heads))
    p = s.parity((s.H.copy(), S.copy()))
    assert p["entropy_max_abs_err_nats"] == 0.0 and p["importance_max_rel_err"] == 0.0
    assert p["importance_keys"] == s.T and p["entropy_rows"] == len(s.ent_rows)
    H_bad, S_bad = s.H.copy(), S.copy()
    H_bad[3] += 2e-3
    S_bad[s.T - 1] *= 1.05
    p = s.parity((H_bad, S_bad))
    assert abs(p["entropy_max_abs_err_nats"] - 2e-3) < 1e-9
    assert abs(p["importance_max_rel_err"] - 0.05) < 1e-6


def test_clock_summary_of_a_short_region():
    # a timed region shorter than the sampling interval holds no sample: the summary
    # takes the samples within half a second of it and says so
    c = bench.ClockSampler(0)
    c.lines = [(100.0, "0, 2070, 2070, 500.0, 0x0, Not Active, Not Active, Not Active, Not Active"),
               (100.3, "0, 2060, 2070, 510.0, 0x0, Not Active, Not Active, Not Active, Active"),
               (103.0, "0, 1000, 2070, 100.0, 0x0, Not Active, Not Active, Not Active, Not Active")]
    c.window(100.1, 100.11)
    out = c.summary()
    assert out["samples"] == 2 and out["sm_mhz"] == 2065.0 and out["reasons"] == ["sw_power_cap"]
    assert "window" in out
    c.window(99.9, 100.35)
    out = c.summary()
    assert out["samples"] == 2 and "window" not in out


def test_oracle_sample_long_prompt_uses_last_rows():
    # a 32768-token prompt exceeds the pair budget: one head per thread (8 here), its last
    # query rows only, the first row the one that keeps the pairs within budget
    w = W.C3
    T = 32768
    b, heads, r0, pairs = bench.OracleSample.sizing(w, 8)
    assert len(heads) == 8 and heads[0] == 0 and heads[-1] == w.Hq - 1
    per_head = bench.OracleSample.PAIR_BUDGET / 8
    assert 0 < r0 < T and pairs == (T * (T + 1) - r0 * (r0 + 1)) / 2
    assert pairs <= per_head < pairs + r0  # one row fewer would exceed the budget
    # a workload whose median prompt fits takes every head and every row
    b, heads, r0, pairs = bench.OracleSample.sizing(W.C4, 8)
    T4 = int(np.diff(W.C4.cu_seqlens())[b])
    assert len(heads) == W.C4.Hq and r0 == 0 and pairs == T4 * (T4 + 1) / 2


def test_reference_arm_json_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--workload", "single_T128_f32", "--steps", "2", "--warmup", "3"],
                         capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    d = json.loads(out.stdout.strip().splitlines()[-1])
    assert d["impl"] == "reference" and d["value"] > 0 and d["steps"] == 2 and d["warmup"] == 3
    assert d["config"]["workload"] == "single_T128_f32"
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]
    # the step is the timed sample: value = tokens-equivalent per step / step time
    eq = d["config"]["tokens_equivalent_per_step"]
    assert abs(eq / (d["ms_per_step"] / 1e3) - d["value"]) <= 1e-6 * d["value"]


def test_host_pool_budget_is_bounded(monkeypatch):
    monkeypatch.setenv("LOCAL_WORLD_SIZE", "8")
    b8 = bench.HostPool.budget()
    monkeypatch.setenv("LOCAL_WORLD_SIZE", "1")
    b1 = bench.HostPool.budget()
    assert (1 << 30) <= b8 <= b1 <= bench.HOST_POOL_BYTES


def test_step_launch_count():
    # entropy 2, per layer 2 + 3, finalize 1, pooling 2
    assert bench.lib_launches(W.C4) == 2 + 32 * 5 + 1 + 2
    assert bench.lib_launches(W.C2) == 2 + 4 * 5 + 1 + 2


def test_traffic_is_dropped_when_a_kernel_source_or_shared_header_changes(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2608_15592_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "profiles").mkdir()
    (csrc / "k.cu").write_text("kernel\n")
    (csrc / "h.cuh").write_text("header\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    rec = {"wl": {"k": {"source": "k.cu", "source_sha256_16": bench.source_hash("k.cu"),
                        "dram_bytes_per_launch": 123}}}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    assert bench.traffic_for("k", "wl") == 123
    assert bench.traffic_for("k", "other") is None and bench.traffic_for("x", "wl") is None
    (csrc / "h.cuh").write_text("header, changed\n")
    assert bench.traffic_for("k", "wl") is None
    (csrc / "h.cuh").write_text("header\n")
    assert bench.traffic_for("k", "wl") == 123
    (csrc / "k.cu").write_text("kernel, changed\n")
    assert bench.traffic_for("k", "wl") is None
