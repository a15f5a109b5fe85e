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


def _run_bench(args, env_extra=None, timeout=300):
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ)
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        env.pop(k, None)
    env.update(env_extra or {})
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py")] + args, cwd=root, env=env,
                       capture_output=True, text=True, timeout=timeout)
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    return r.returncode, [json.loads(l) for l in lines]


def test_reference_arm_prints_the_contract_line():
    # the reference arm times the oracle on the host cores; on the small fp32
    # workload it finishes in seconds and needs no GPU
    rc, lines = _run_bench(["--impl", "reference", "--workload", "c1_5p625deg_f32",
                            "--steps", "1", "--warmup", "3"])
    assert rc == 0 and len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference"
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["value"] > 0 and d["steps"] == 1 and d["warmup"] >= 3 and d["higher_is_better"] is True
    assert d["config"]["workload"] == "c1_5p625deg_f32"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_reference_arm_other_ranks_exit_without_work():
    rc, lines = _run_bench(["--impl", "reference", "--workload", "c1_5p625deg_f32",
                            "--steps", "1", "--warmup", "3", "--gpus", "2"],
                           {"RANK": "1", "WORLD_SIZE": "2", "LOCAL_RANK": "1"}, timeout=120)
    assert rc == 0 and lines == []
