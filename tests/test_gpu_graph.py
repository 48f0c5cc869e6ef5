"""A whole step of the feature path captured in a CUDA graph and replayed (GPU).

The library's calls allocate nothing once their workspace has grown and never
synchronise, so a step (entropy, row normalisers and column sums of every layer,
finalize, pooling and the length head) can be captured once and replayed: the replay
launches the same kernels without the host's per-call work, which is what bounds the
small workloads.  A replay must give the same bits as the step run call by call, on two
replays in a row (the pooling kernel's arrival counters reset themselves, and the
column-sum accumulation reopens at the first layer of every replay)."""
import dataclasses

import pytest
import torch

import bench
from synth import workloads as W

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,B", [("single_T128_f32", 1), ("qwen2.5-7b_varlen16", 3)],
                         ids=["fp32_cuda_cores", "bf16_tensor_cores"])
def test_graph_replay_matches_calls(cuda_lib, name, B):
    w = dataclasses.replace(W.WORKLOADS[name], B=B)
    st = bench.Step(cuda_lib, w, torch.device("cuda", 0), stream_qk=False)
    outs = (st.H, st.S, st.pooled, st.pred)
    st.run()
    torch.cuda.synchronize()
    st.ctx.sync_status()
    ref = [t.clone() for t in outs]
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        st.run()
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        st.run()
    for _ in range(2):
        for t in outs:
            t.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        st.ctx.sync_status()
        for name_t, a, b in zip(("H", "S", "pooled", "pred"), ref, outs):
            assert torch.equal(a, b), f"{name_t} differs after a graph replay"
    del g
