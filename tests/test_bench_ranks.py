"""The replica path of bench.py on CPU with two gloo ranks: each rank gets its own
batch but the same weights, timings combine as the slowest rank's, and the
whole-job throughput counts every rank's tokens."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2607_02829_gb300 import synth


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, results):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        wl = synth.Workload("tiny", B=2, grid_h=4, grid_w=8, channels=3, patch=1, D=64, heads=1,
                            n1=1, n2=1, n3=0, keep_ratio=0.5, dtype="bf16", seed_index=3)
        x, ws = bench.rank_inputs(wl, rank)
        local_ms = 10.0 + 5.0 * rank                    # rank 1 is the slow one
        slowest = bench.max_over_ranks(local_ms, world, torch.device("cpu"))
        value = bench.job_tokens_per_s(wl.B * wl.L, world, slowest)
        gathered = [None] * world
        dist.all_gather_object(gathered, (x.float().sum().item(),
                                          sum(t.float().sum().item() for t in ws[0].values())))
        results[rank] = (slowest, value, gathered)
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas():
    world = 2
    mgr = mp.get_context("spawn").Manager()
    results = mgr.dict()
    mp.start_processes(_worker, args=(world, _free_port(), results), nprocs=world,
                       start_method="spawn")
    for rank in range(world):
        slowest, value, gathered = results[rank]
        assert slowest == 15.0                                  # the max over ranks
        assert value == pytest.approx(2 * 2 * 32 / 15e-3)      # both ranks' tokens
        (x0, w0), (x1, w1) = gathered
        assert x0 != x1                                          # own batch per rank
        assert w0 == w1                                          # same model weights


def test_single_rank_helpers_without_a_process_group():
    import bench
    assert bench.max_over_ranks(3.5, 1, torch.device("cpu")) == 3.5
    assert bench.job_tokens_per_s(1000, 1, 2.0) == pytest.approx(500000.0)
