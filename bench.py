"""Throughput of the Sparse-Reslim routed encoder forward on GB300.

One step = one sr_forward over one batch of the 0.25 degree workload (B = 1,
720x1440 grid, patch 8 -> L = 16200 tokens, D = 1024, 16 heads, 24 blocks
split (4, 16, 4), keep ratio 0.25 -> K = 4050 routed tokens, bf16 storage,
fp32 accumulation), inputs resident in HBM.  Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the fp64 CPU oracle on the host cores

Multi-GPU (torchrun): every rank runs an independent replica on its own batch
(the forward has no cross-sample exchange), so scaling is weak.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "c4_0p25deg_bf16"
L2_FLUSH_BYTES = 512 << 20          # > 129 MB of L2

# DRAM bytes (read + write) per launch of a kernel kind, measured by ncu, are
# kept in a small text table under profiles/ together with a digest of the
# kernel's source files at the time of the capture.  The roofline reports them
# only while that digest matches the current sources; otherwise "traffic" is
# null and a warning names the stale capture.
TRAFFIC_TABLE = os.path.join(ROOT, "profiles", "dram_traffic_per_launch.txt")
KERNEL_SOURCES = {
    "attention": ("attention_tc.cu", "tc_ptx.cuh", "common.cuh", "kernels.h"),
    "gemm": ("gemm_tc.cu", "tc_ptx.cuh", "common.cuh", "kernels.h"),
}


def source_digest(kind):
    """sha256 (first 12 hex digits) over the CUDA sources a kernel kind is built from."""
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kind]:
        with open(os.path.join(ROOT, "paper_2607_02829_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:12]


def measured_traffic(kind, workload):
    """(bytes per launch, note) from the traffic table for this kernel kind and
    workload, or (None, reason)."""
    src = "gemm" if kind.startswith("gemm") else kind
    if src not in KERNEL_SOURCES:
        return None, f"no ncu traffic figure is kept for {kind}"
    try:
        lines = open(TRAFFIC_TABLE).read().splitlines()
    except OSError:
        return None, "no traffic table"
    want = source_digest(src)
    for line in lines:
        p = [c.strip() for c in line.strip().strip("|").split("|")]
        if len(p) >= 4 and p[0] == kind and p[1] == workload:
            if p[2] != want:
                msg = (f"the ncu traffic of {kind} on {workload} was captured on sources "
                       f"{p[2]}, the current ones are {want}: traffic reported as null")
                print("bench.py: " + msg, file=sys.stderr)
                return None, msg
            return float(p[3]) * 1e6, f"ncu capture of sources {p[2]}"
    return None, f"no ncu traffic figure for {kind} on {workload}"


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": p["hbm_gbs"], "bf16_tflops": p["bf16_tflops"],
                "bf16_tflops_sustained": p["bf16_tflops_sustained"],
                "sm_max_mhz": p.get("sm_max_mhz", 2070.0), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def _workload(name, split=None):
    from paper_2607_02829_gb300 import synth
    wl = synth.WORKLOADS.get(name)
    if wl is None:
        for w in synth.sweep_workloads():
            if w.name == name:
                wl = w
    if wl is None:
        raise SystemExit(f"unknown workload {name}")
    if split:
        n1, n2, n3 = (int(v) for v in split.split(","))
        wl = wl.with_(name=f"{wl.name}_split{n1}-{n2}-{n3}", n1=n1, n2=n2, n3=n3)
    return wl


def _describe(wl, K):
    return {"workload": wl.name, "grid": f"{wl.grid_h}x{wl.grid_w}", "channels": wl.channels,
            "patch": wl.patch, "B": wl.B, "L": wl.L, "D": wl.D, "heads": wl.heads,
            "split": [wl.n1, wl.n2, wl.n3], "keep_ratio": wl.keep_ratio, "K": K,
            "selector": wl.selector, "storage": wl.dtype}


class ClockSampler:
    """nvidia-smi clock / throttle-reason sampling during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index, keep_path=None):
        self.gpu = gpu_index
        self.proc = None
        self.path = None
        self.keep_path = keep_path       # raw samples are kept only when asked for

    def start(self):
        try:
            if self.keep_path:
                self.path = self.keep_path
            else:
                fd, self.path = tempfile.mkstemp(prefix="sr_clocks_", suffix=".csv")
                os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                p = [v.strip() for v in line.split(",")]
                if len(p) < 9:
                    continue
                try:
                    sm.append(float(p[1]))
                    smax = float(p[2])
                except ValueError:
                    continue
                for n, v in zip(names, p[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        if not self.keep_path:
            try:
                os.remove(self.path)
            except OSError:
                pass
        if not sm:
            return None
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


def rank_inputs(wl, rank):
    """One replica's inputs: its own batch (input seed offset by the rank) and the
    model's weights, the same on every rank.  CPU tensors in the storage dtype."""
    from paper_2607_02829_gb300 import synth
    xw = wl.with_(seed_index=wl.seed_index + 100 * rank) if rank else wl
    x = synth.to_storage(synth.make_tokens(xw), wl.dtype)
    ws = [{k: synth.to_storage(v, wl.dtype) for k, v in blk.items()}
          for blk in synth.make_weights(wl)]
    return x, ws


def max_over_ranks(value, world, device):
    """The largest value over all ranks (every rank gets it); the value itself at N=1."""
    if world == 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(tokens_per_rank, world, ms_slowest):
    """Whole-job throughput: every replica's tokens over the slowest rank's time."""
    return tokens_per_rank * world / (ms_slowest * 1e-3)


def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist
    from paper_2607_02829_gb300 import binding as b, synth

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    wl = _workload(args.workload, args.split)
    K = b.sr_keep_count(wl.L, wl.keep_ratio)
    cfg = b.make_config(wl.B, wl.L, wl.D, wl.heads, wl.n1, wl.n2, wl.n3, dtype=wl.dtype,
                        selector=wl.selector, grid_w=wl.grid_wp)
    enc = b.Encoder(cfg, max_keep_ratio=wl.keep_ratio)
    # each rank: its own batch (seeded by rank), shared weights
    x_cpu, w_cpu = rank_inputs(wl, rank)
    x = x_cpu.to(dev)
    wd = [{k: v.to(dev) for k, v in blk.items()} for blk in w_cpu]
    warr = b.weights_array(wd)
    out = torch.empty_like(x)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    seed = wl.select_seed

    def step(i):
        b.sr_forward(enc.handle, x.data_ptr(), warr, wl.keep_ratio, seed + i, out.data_ptr(),
                     None, stream.cuda_stream)

    def barrier():
        if world > 1:
            dist.barrier()

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()

    # ---- timed region: K steps, L2 flushed before each, events around each step
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    clocks = ClockSampler(local_rank, args.clocks_csv)
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for i in range(args.steps):
        flush.zero_()
        ev[i][0].record(stream)
        step(args.warmup + i)
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    barrier()
    wall = time.perf_counter() - t0
    clk = clocks.stop()
    ms = sum(a.elapsed_time(z) for a, z in ev) / args.steps
    ms = max_over_ranks(ms, world, dev)

    # ---- the same step captured into a CUDA graph and replayed K times (L2
    #      flushed before each replay); the seed is fixed in the graph
    graph = None
    try:
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            b.sr_forward(enc.handle, x.data_ptr(), warr, wl.keep_ratio, seed, out.data_ptr(),
                         None, side.cuda_stream)
        for _ in range(args.warmup):
            g.replay()
        torch.cuda.synchronize()
        gev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
        barrier()
        for i in range(args.steps):
            flush.zero_()
            gev[i][0].record()
            g.replay()
            gev[i][1].record()
        torch.cuda.synchronize()
        g_ms = max_over_ranks(sum(a.elapsed_time(z) for a, z in gev) / args.steps, world, dev)
        graph = {"ms_per_step": g_ms,
                 "value": job_tokens_per_s(wl.B * wl.L, world, g_ms), "unit": "tokens/s",
                 "note": "one sr_forward captured into a CUDA graph, replayed; L2 flushed before each"}
        del g
    except Exception as e:          # capture unsupported here: report why, keep the direct timing
        graph = {"unavailable": f"{type(e).__name__}: {e}"}

    # ---- per-kernel trace over K more steps (same launches, events around each)
    b.sr_trace_enable(enc.handle, True)
    b.sr_trace_read(enc.handle, reset=True)
    for i in range(args.steps):
        flush.zero_()
        step(args.warmup + i)
    torch.cuda.synchronize()
    trace = b.sr_trace_read(enc.handle, reset=True)
    b.sr_trace_enable(enc.handle, False)

    # ---- the sparse middle stage alone (split 0, n2, 0 on the same shapes and
    #      weights): select, gather, the n2 sparse blocks and the delta scatter
    segment = None
    if wl.n2 > 0 and wl.keep_ratio < 1.0:
        scfg = b.make_config(wl.B, wl.L, wl.D, wl.heads, 0, wl.n2, 0, dtype=wl.dtype,
                             selector=wl.selector, grid_w=wl.grid_wp)
        senc = b.Encoder(scfg, max_keep_ratio=wl.keep_ratio)
        sw = b.weights_array(wd[wl.n1:wl.n1 + wl.n2])
        for i in range(args.warmup):
            b.sr_forward(senc.handle, x.data_ptr(), sw, wl.keep_ratio, seed + i, out.data_ptr(),
                         None, stream.cuda_stream)
        sev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
        for i in range(args.steps):
            flush.zero_()
            sev[i][0].record(stream)
            b.sr_forward(senc.handle, x.data_ptr(), sw, wl.keep_ratio, seed + i, out.data_ptr(),
                         None, stream.cuda_stream)
            sev[i][1].record(stream)
        torch.cuda.synchronize()
        seg_ms = sum(a.elapsed_time(z) for a, z in sev) / args.steps
        rows = wl.B * K
        seg_flops = wl.n2 * (2.0 * rows * (3 * wl.D * wl.D + wl.D * wl.D + 2 * wl.mlp_hidden * wl.D)
                             + 4.0 * wl.B * K * K * wl.D)
        segment = {"ms": seg_ms, "gflop": seg_flops / 1e9,
                   "tflops": seg_flops / (seg_ms * 1e-3) / 1e12}
        # the segment traced: every FC2 here runs on the routed rows, so the last
        # one's extra time over a plain FC2 of the same shape is the scatter's
        b.sr_trace_enable(senc.handle, True)
        b.sr_trace_read(senc.handle, reset=True)
        for i in range(args.steps):
            flush.zero_()
            b.sr_forward(senc.handle, x.data_ptr(), sw, wl.keep_ratio, seed + i, out.data_ptr(),
                         None, stream.cuda_stream)
        torch.cuda.synchronize()
        segment["trace"] = b.sr_trace_read(senc.handle, reset=True)
        # the two stream copies the timed forward also runs (widen x, narrow the
        # output), from the traced steps, where each interval includes its launch
        cp = segment["trace"].get("copy", {})
        segment["copies_ms_traced"] = cp.get("ms", 0.0) / args.steps
        b.sr_trace_enable(senc.handle, False)
        senc.close()

    # ---- end to end through the C ABI from pinned host memory.  Every step copies
    # its input in and its result out; the copies run on their own streams, so
    # step i + 1's input and step i - 1's result move while step i computes
    # (two device and two pinned host buffers, ordered by events).
    xh = x_cpu.pin_memory()
    oh = [torch.empty_like(xh).pin_memory() for _ in range(2)]
    din = [torch.empty_like(x) for _ in range(2)]
    dout = [torch.empty_like(x) for _ in range(2)]
    bytes_io = x.numel() * x.element_size()
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    fwd_done = [torch.cuda.Event() for _ in range(2)]
    in_ready = [torch.cuda.Event() for _ in range(2)]
    out_read = [torch.cuda.Event() for _ in range(2)]

    def e2e_step(i):
        k = i % 2
        if i >= 2:
            s_in.wait_event(fwd_done[k])        # forward i - 2 has read din[k]
        with torch.cuda.stream(s_in):
            din[k].copy_(xh, non_blocking=True)
        in_ready[k].record(s_in)
        stream.wait_event(in_ready[k])
        if i >= 2:
            stream.wait_event(out_read[k])      # step i - 2's result has left dout[k]
        b.sr_forward(enc.handle, din[k].data_ptr(), warr, wl.keep_ratio, seed + i,
                     dout[k].data_ptr(), None, stream.cuda_stream)
        fwd_done[k].record(stream)
        s_out.wait_event(fwd_done[k])
        with torch.cuda.stream(s_out):
            oh[k].copy_(dout[k], non_blocking=True)
        out_read[k].record(s_out)

    for i in range(max(2, args.warmup // 2)):
        e2e_step(i)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    e0.record(s_in)
    for i in range(args.steps):
        e2e_step(i)
    e1.record(s_out)
    torch.cuda.synchronize()
    if not torch.equal(oh[(args.steps - 1) % 2], dout[(args.steps - 1) % 2].cpu()):
        raise RuntimeError("end-to-end result differs from the device result")
    e2e_ms = e0.elapsed_time(e1) / args.steps
    e2e_ms = max_over_ranks(e2e_ms, world, dev)
    enc.close()
    return wl, K, ms, wall, clk, trace, e2e_ms, bytes_io, segment, graph


def roofline(trace, peaks, steps, workload, fp32_alu=False):
    """The dominant kernel kind of the traced forward against its roofline.  A
    tensor-bound kind is divided by the burst bf16 peak (its launches last tens
    to hundreds of microseconds inside a step of about 12 ms); the sustained
    figure is given beside it."""
    kernels = {k: v for k, v in trace.items() if k != "copy" and v["launches"] > 0}
    dom = max(kernels, key=lambda k: kernels[k]["ms"])
    t = kernels[dom]
    per_launch_ms = t["ms"] / t["launches"]
    extra = {}
    if t["flops"] > 0 and fp32_alu:
        # CUDA-core fp32 kernels: 152 SMs x 128 FP32 lanes x 2 flops per FFMA at
        # the maximum SM clock
        achieved = t["flops"] / t["launches"] / (per_launch_ms * 1e-3) / 1e12
        peak = 152 * 128 * 2 * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
        bound, unit = "alu", "TFLOP/s"
        source = "derived from SM count, FP32 lanes and max clock"
    elif t["flops"] > 0:
        achieved = t["flops"] / t["launches"] / (per_launch_ms * 1e-3) / 1e12
        peak = peaks["bf16_tflops"]
        bound, unit = "tensor", "TFLOP/s"
        source = peaks["source"] + " burst"
        extra = {"peak_sustained": peaks["bf16_tflops_sustained"],
                 "frac_of_sustained": achieved / peaks["bf16_tflops_sustained"]}
    else:
        achieved = t["bytes"] / t["launches"] / (per_launch_ms * 1e-3) / 1e9
        peak = peaks["hbm_gbs"]
        bound, unit = "hbm", "GB/s"
        source = peaks["source"] + " copy bandwidth"
    traffic, traffic_note = measured_traffic(dom, workload)
    total_ms = sum(v["ms"] for v in kernels.values())
    detail = {}
    for k, v in kernels.items():
        d = {"launches_per_step": v["launches"] / steps, "ms_per_step": v["ms"] / steps,
             "share": v["ms"] / total_ms}
        if v["flops"] > 0:
            d["tflops"] = v["flops"] / (v["ms"] * 1e-3) / 1e12
        if v["bytes"] > 0:
            d["gbs"] = v["bytes"] / (v["ms"] * 1e-3) / 1e9
        detail[k] = d
    return (dict({"kernel": dom, "bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
                  "frac": achieved / peak, "peak_source": source}, **extra,
                 traffic=traffic, traffic_source=traffic_note,
                 algorithmic_bytes_per_launch=t["bytes"] / t["launches"]), detail)


def gather_scatter(wl, K, trace, segment, peaks):
    """GB/s and fraction of the measured HBM copy bandwidth of the gather (fused
    into the first sparse LN1) and of the delta scatter (fused into the last
    sparse FC2), with their algorithmic bytes per launch.
      gather : the selected fp32 stream rows read, h0 (fp32) and LN1 (storage
               dtype) written, plus the index set;
      scatter: x0 rows read and x' rows written (fp32 stream), plus the index
               set, over the time the scatter FC2 takes beyond a plain FC2 on
               the same routed rows (both from the sparse segment's trace)."""
    out = {}
    g = trace.get("gather", {})
    if g.get("launches"):
        gbs = g["bytes"] / (g["ms"] * 1e-3) / 1e9
        out["gather"] = {"bytes_per_launch": g["bytes"] / g["launches"],
                         "us_per_launch": g["ms"] / g["launches"] * 1e3,
                         "gbs": gbs, "frac_of_hbm": gbs / peaks["hbm_gbs"]}
    st = (segment or {}).get("trace") or {}
    fs, f = st.get("gemm_fc2_scatter", {}), st.get("gemm_fc2", {})
    if fs.get("launches") and f.get("launches"):
        extra_ms = fs["ms"] / fs["launches"] - f["ms"] / f["launches"]
        nbytes = 8.0 * wl.B * K * wl.D + 4.0 * wl.B * K
        rec = {"bytes_per_launch": nbytes, "us_fc2_scatter": fs["ms"] / fs["launches"] * 1e3,
               "us_fc2_plain": f["ms"] / f["launches"] * 1e3}
        if extra_ms > 0:
            gbs = nbytes / (extra_ms * 1e-3) / 1e9
            rec.update(gbs=gbs, frac_of_hbm=gbs / peaks["hbm_gbs"])
        else:
            rec["note"] = "the scatter FC2 was not slower than a plain FC2 of the same shape"
        out["scatter"] = rec
    return out


def cpu_baseline(wl, sparse_only=False):
    """The fp64 oracle, as it stands, on a bounded sample of the workload: one dense
    block over all L tokens and one sparse block over the K routed tokens of the
    same model; the full forward's time is those block times weighted by the
    block counts (selection and gather are negligible next to the blocks)."""
    import numpy as np
    from oracle import reslim as o
    from paper_2607_02829_gb300 import synth
    threads = len(os.sched_getaffinity(0))
    rng = np.random.Generator(np.random.PCG64(7))
    x = synth.stored_as_f64(synth.to_storage(synth.make_tokens(wl), wl.dtype))
    w = o.as_f64_weights([{k: synth.to_storage(v, wl.dtype) for k, v in
                           synth.make_block_weights(wl.D, wl.mlp_hidden, 1).items()}])[0]
    K = o.keep_count(wl.L, wl.keep_ratio)
    from concurrent.futures import ThreadPoolExecutor
    pool = ThreadPoolExecutor(threads)
    t_dense = 0.0
    if not sparse_only:
        t0 = time.perf_counter()
        o.block(x, w, wl.heads, pool=pool)
        t_dense = time.perf_counter() - t0
    idx = o.select_random(wl.B, wl.L, K, 1)
    h = x[np.arange(wl.B)[:, None], idx]
    t0 = time.perf_counter()
    o.block(h, w, wl.heads, pool=pool)
    t_sparse = time.perf_counter() - t0
    pool.shutdown()
    n_dense = wl.n1 + wl.n3 + (wl.n2 if wl.keep_ratio == 1.0 else 0)
    n_sparse = 0 if wl.keep_ratio == 1.0 else wl.n2
    est = n_dense * t_dense + n_sparse * t_sparse
    return {"value": wl.B * wl.L / est, "unit": "tokens/s", "cores": threads, "kind": "oracle",
            "sample": f"one dense block (T={wl.L}) + one sparse block (T={K}) of {wl.name}, "
                      f"{t_dense:.1f} s + {t_sparse:.1f} s fp64, weighted by {n_dense} dense "
                      f"+ {n_sparse} sparse blocks -> {est:.0f} s per forward",
            "sample_seconds": t_dense + t_sparse}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--split", default=None,
                    help="override the block split n1,n2,n3 (kernel studies and profiling)")
    ap.add_argument("--sweep", choices=["gather", "ensemble", "cross_attention"], default=None,
                    help="size sweep of one kernel (prints one JSON line per size)")
    ap.add_argument("--clocks-csv", default=None,
                    help="keep the raw nvidia-smi samples of the timed region in this file")
    ap.add_argument("--source-digest", choices=sorted(KERNEL_SOURCES), default=None,
                    help="print the digest of a kernel kind's CUDA sources and exit")
    args = ap.parse_args()
    if args.source_digest:
        print(source_digest(args.source_digest))
        return
    args.warmup = max(args.warmup, 3)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        return run_reference(args, rank, world)
    if args.sweep == "gather":
        return gather_sweep(args)
    if args.sweep == "ensemble":
        return ensemble_sweep(args)
    if args.sweep == "cross_attention":
        return cross_attention_sweep(args)

    import torch
    import torch.distributed as dist
    if world > 1:
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    # build once per node, then every rank loads the library
    if local_rank == 0:
        from paper_2607_02829_gb300 import build
        build.build()
    if world > 1:
        dist.barrier()

    wl, K, ms, wall, clk, trace, e2e_ms, bytes_io, segment, graph = run_ours(args, rank, world,
                                                                              local_rank)
    peaks = _peaks()
    tokens = wl.B * wl.L * world
    value = job_tokens_per_s(wl.B * wl.L, world, ms)
    roof, detail = roofline(trace, peaks, args.steps, wl.name, fp32_alu=wl.dtype == "f32")
    launches = sum(v["launches"] for v in trace.values())
    gs = gather_scatter(wl, K, trace, segment, peaks)
    if segment:
        segment.pop("trace", None)
    total_flops = sum(v["flops"] for v in trace.values()) / args.steps
    line = {
        "metric": "full-grid tokens/sec of routed encoder fwd",
        "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if wl.dtype == "bf16" else "f32",
        "data": "synthetic (seeded ERA5-shaped smooth fields, random-init weights)",
        "config": dict(_describe(wl, K), l2="flushed (512 MB write) before every timed step",
                       parallelism=f"replicas x{world}"),
        "roofline": roof,
        "forward_tflops": total_flops / (ms * 1e-3) / 1e12,
        "gather_scatter": gs,
        "sparse_segment": (dict(segment, frac_of_burst=segment["tflops"] / peaks["bf16_tflops"],
                                frac_of_sustained=segment["tflops"] /
                                peaks["bf16_tflops_sustained"],
                                note="a forward of the n2 sparse blocks alone (split 0,n2,0): "
                                     "select, gather, the sparse blocks and the delta scatter, "
                                     "plus the widen of x to the fp32 stream and the narrow of "
                                     "the output (copies_ms_traced); algorithmic flops of the "
                                     "sparse blocks")
                           if segment and wl.dtype == "bf16" else segment),
        "kernels": detail,
        "e2e": {"value": job_tokens_per_s(wl.B * wl.L, world, e2e_ms), "unit": "tokens/s",
                "h2d_bytes_per_step": bytes_io, "d2h_bytes_per_step": bytes_io},
        "graph": graph,
        "gpu_launches": int(launches),
        "wall_s_timed_region": wall,
        "clocks": clk,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def gather_sweep(args):
    """Gather GB/s from 33 MB to 530 MB of selected rows: one sparse block (split
    0,1,0) of the 0.25 deg model (L=16200, D=1024, r=0.25) at batch 1..16, L2
    flushed before every traced forward.  The gather of Eq. 8 runs fused with
    the first sparse block's LN1; its CUDA-event time and algorithmic bytes
    (selected rows read, h0 and LN1 written, index set) come from the trace."""
    import torch
    from paper_2607_02829_gb300 import binding as b, build, synth
    build.build()
    peaks = _peaks()
    L, D, H, r = 16200, 1024, 16, 0.25
    w = {k: synth.to_storage(v, "bf16").cuda()
         for k, v in synth.make_block_weights(D, 4 * D, 7).items()}
    warr = b.weights_array([w])
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    s = torch.cuda.current_stream()
    for B in (1, 2, 4, 8, 16):          # B*L*4D stays below the 2^31-element limit
        cfg = b.make_config(B, L, D, H, 0, 1, 0, dtype="bf16")
        enc = b.Encoder(cfg, max_keep_ratio=r)
        x = torch.randn(B, L, D, device="cuda").to(torch.bfloat16)
        out = torch.empty_like(x)
        for i in range(args.warmup):
            b.sr_forward(enc.handle, x.data_ptr(), warr, r, i, out.data_ptr(), None, s.cuda_stream)
        b.sr_trace_enable(enc.handle, True)
        b.sr_trace_read(enc.handle, reset=True)
        for i in range(args.steps):
            flush.zero_()
            b.sr_forward(enc.handle, x.data_ptr(), warr, r, 100 + i, out.data_ptr(), None,
                         s.cuda_stream)
        torch.cuda.synchronize()
        t = b.sr_trace_read(enc.handle, reset=True)["gather"]
        gbs = t["bytes"] / (t["ms"] * 1e-3) / 1e9
        print(json.dumps({"sweep": "gather", "B": B, "rows": B * b.sr_keep_count(L, r),
                          "bytes_per_launch": t["bytes"] / t["launches"],
                          "us_per_launch": t["ms"] / t["launches"] * 1e3, "gbs": gbs,
                          "frac_of_hbm": gbs / peaks["hbm_gbs"]}), flush=True)
        enc.close()
        del x, out
        torch.cuda.empty_cache()


def ensemble_sweep(args):
    """Implicit ensembling on the workload (default 0.25 deg): M = 1, 2, 4, 8
    members with different seeds through sr_forward_ensemble (dense-early blocks
    once) against M separate sr_forward calls; CUDA-event time per ensemble with
    L2 flushed before each, inputs resident in HBM."""
    import torch
    from paper_2607_02829_gb300 import binding as b, build
    build.build()
    wl = _workload(args.workload, args.split)
    x, ws = rank_inputs(wl, 0)
    cfg = b.make_config(wl.B, wl.L, wl.D, wl.heads, wl.n1, wl.n2, wl.n3, dtype=wl.dtype,
                        selector=wl.selector, grid_w=wl.grid_wp)
    enc = b.Encoder(cfg, max_keep_ratio=wl.keep_ratio)
    xd = x.cuda()
    warr = b.weights_array([{k: v.cuda() for k, v in blk.items()} for blk in ws])
    out = torch.empty_like(xd)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    s = torch.cuda.current_stream()

    def timed(fn):
        for _ in range(args.warmup):
            fn()
        tot = 0.0
        for _ in range(args.steps):
            flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(s)
            fn()
            e1.record(s)
            torch.cuda.synchronize()
            tot += e0.elapsed_time(e1)
        return tot / args.steps

    for M in (1, 2, 4, 8):
        seeds = [wl.select_seed + 17 * m for m in range(M)]
        ens_ms = timed(lambda: enc.forward_ensemble(xd, warr, wl.keep_ratio, seeds, out=out))

        def separate():
            for sd in seeds:
                b.sr_forward(enc.handle, xd.data_ptr(), warr, wl.keep_ratio, sd, out.data_ptr(),
                             None, s.cuda_stream)
        sep_ms = timed(separate)
        print(json.dumps({"sweep": "ensemble", "workload": wl.name, "members": M,
                          "ms_per_ensemble": ens_ms, "ms_separate_forwards": sep_ms,
                          "speedup_vs_separate": sep_ms / ens_ms,
                          "member_tokens_per_s": wl.B * wl.L * M / (ens_ms * 1e-3)}), flush=True)
    enc.close()


def cross_attention_sweep(args):
    """Asymmetric attention (queries from the routed tokens, keys/values from the
    full sequence) at the 0.25 deg shapes, 16 heads: CUDA-event time per call
    with L2 flushed before each, against the bf16 tensor peak."""
    import torch
    from paper_2607_02829_gb300 import binding as b, build
    build.build()
    peaks = _peaks()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    s = torch.cuda.current_stream()
    heads = 16
    D = 64 * heads
    for (B, Tq, Tkv) in [(1, 4050, 16200), (1, 16200, 16200), (1, 2025, 16200), (8, 512, 2048)]:
        q = torch.randn(B, Tq, D, device="cuda").to(torch.bfloat16)
        kv = torch.randn(B, Tkv, 2 * D, device="cuda").to(torch.bfloat16)
        out = torch.empty(B, Tq, D, dtype=torch.bfloat16, device="cuda")

        def call():
            b.sr_cross_attention(q.data_ptr(), kv.data_ptr(), B, Tq, Tkv, heads, out.data_ptr(),
                                 None, s.cuda_stream)
        for _ in range(args.warmup):
            call()
        tot = 0.0
        for _ in range(args.steps):
            flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(s)
            call()
            e1.record(s)
            torch.cuda.synchronize()
            tot += e0.elapsed_time(e1)
        ms = tot / args.steps
        tf = 4.0 * B * heads * Tq * Tkv * 64 / (ms * 1e-3) / 1e12
        print(json.dumps({"sweep": "cross_attention", "B": B, "Tq": Tq, "Tkv": Tkv, "heads": heads,
                          "ms": ms, "tflops": tf,
                          "frac_of_burst": tf / peaks["bf16_tflops"]}), flush=True)
        del q, kv, out


def run_reference(args, rank, world):
    """The oracle as the reference arm, on the host cores, rank 0 only."""
    if rank != 0:
        return
    wl = _workload(args.workload, args.split)
    from oracle import reslim as o
    K = o.keep_count(wl.L, wl.keep_ratio)
    vals = []
    base = None
    # untimed warm-up steps run the cheap half of the sample (one sparse block)
    for i in range(args.warmup):
        cpu_baseline(wl, sparse_only=True)
    for i in range(args.steps):
        base = cpu_baseline(wl)
        vals.append(base["value"])
    value = sum(vals) / len(vals)
    ms = wl.B * wl.L / value * 1e3
    line = {"impl": "reference", "metric": "full-grid tokens/sec of routed encoder fwd",
            "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded ERA5-shaped smooth fields, random-init weights)",
            "config": _describe(wl, K),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": base["cores"],
                             "kind": "oracle", "sample": base["sample"]},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
