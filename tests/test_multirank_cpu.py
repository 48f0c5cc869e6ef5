"""The N > 1 bench path on CPU with two gloo ranks: each rank draws its own batch of
the same shape (prompts are independent, no data-path collective) and the job's
numbers are the slowest rank's time and the sum of all ranks' tokens."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        w = bench.workload_for_rank(rank)
        lens = w.seqlens()
        ms, tokens = bench.aggregate_ranks(10.0 + 5.0 * rank, float(lens.sum()))
        out[rank] = (w.seed, w.B, w.d, int(lens.sum()), ms, tokens)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_prompts_and_aggregate():
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    os.environ["PYTHONPATH"] = root + os.pathsep + os.environ.get("PYTHONPATH", "")
    world, port = 2, _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    (s0, B0, d0, n0, ms0, t0), (s1, B1, d1, n1, ms1, t1) = res[0], res[1]
    assert s0 != s1 and (B0, d0) == (B1, d1)          # own batch, same shape
    assert ms0 == ms1 == 15.0                          # max over ranks
    assert t0 == t1 == float(n0 + n1)                  # all ranks' tokens
    import bench
    assert bench.aggregate_ranks(3.0, 7.0) == (3.0, 7.0)  # single process: unchanged
