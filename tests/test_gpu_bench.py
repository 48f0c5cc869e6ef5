"""bench.py end to end on small workloads (GPU): the JSON line holds every key of the
contract, the library's outputs on the oracle's sample are within the parity bar (taken
before the end-to-end legs reuse the step's buffers), and a graph replay of the step
gives the call-by-call bits."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench(*args):
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--steps", "3",
                          "--warmup", "3", *args], capture_output=True, text=True, timeout=900,
                         cwd=ROOT)
    assert out.returncode == 0, out.stderr[-3000:]
    return json.loads(out.stdout.strip().splitlines()[-1])


@pytest.mark.parametrize("args", [["--workload", "single_T128_f32"],
                                  ["--workload", "qwen2.5-7b_varlen16", "--prompts", "2"]],
                         ids=["fp32_one_prompt", "bf16_two_prompts"])
def test_bench_line(args):
    d = _bench(*args)
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
              "roofline", "cpu_baseline", "e2e", "gpu_launches", "clocks", "parity"):
        assert k in d, k
    assert d["n_gpus"] == 1 and d["steps"] == 3 and d["warmup"] == 3 and d["value"] > 0
    r = d["roofline"]
    assert r["bound"] in ("hbm", "tensor") and r["achieved"] > 0 and r["peak"] > 0
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-9
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] > 0 and d["e2e"]["d2h_bytes_per_step"] > 0
    assert d["gpu_launches"] > 0
    assert d["clocks"] and d["clocks"]["sm_mhz"] > 0 and "reasons" in d["clocks"]
    p = d["parity"]
    assert p["entropy_max_abs_err_nats"] <= p["tolerance"]["entropy_nats"]
    assert p["importance_max_rel_err"] <= p["tolerance"]["importance_rel"]
    assert d["graph_replay"]["bit_equal_to_calls"] is True
