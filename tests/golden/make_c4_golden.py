"""Writes tests/golden/c4_0p25deg_oracle_samples.npz: the fp64 oracle's output of
the 0.25 deg workload (B=1, L=16200, D=1024, 16 heads, 24 blocks (4,16,4),
r=0.25) at 32 sampled token rows, with the output's max |value| and a
checksum of the generated input tokens.  Calls only oracle/ and the seeded
input generator; run it on the machine whose generated inputs the GPU tests
will use (the input checksum is checked there):

    python tests/golden/make_c4_golden.py [output.npz]
"""
import hashlib
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import reslim as o                      # noqa: E402
from paper_2607_02829_gb300 import synth            # noqa: E402

OUT = os.path.join(ROOT, "tests", "golden", "c4_0p25deg_oracle_samples.npz")


def input_digest(x_storage) -> str:
    """sha256 of the stored bytes of a CPU torch tensor (bf16 viewed as int16)."""
    import torch
    t = x_storage.contiguous().view(-1)
    if t.dtype == torch.bfloat16:
        t = t.view(torch.int16)
    return hashlib.sha256(t.numpy().tobytes()).hexdigest()


def main(out_path=OUT):
    wl = synth.WORKLOADS["c4_0p25deg_bf16"]
    t0 = time.time()
    x, ws = synth.make_inputs(wl)
    digest = input_digest(x)
    out, idx = o.forward(synth.stored_as_f64(x), o.as_f64_weights(ws), wl.n1, wl.n2, wl.n3,
                         wl.heads, wl.keep_ratio, seed=wl.select_seed,
                         threads=len(os.sched_getaffinity(0)))
    rng = np.random.Generator(np.random.PCG64(4242))
    sel = np.sort(rng.choice(idx[0], 16, replace=False))
    uns = np.sort(rng.choice(np.setdiff1d(np.arange(wl.L), idx[0]), 16, replace=False))
    rows = np.sort(np.concatenate([sel, uns]))
    np.savez_compressed(out_path, rows=rows, out_rows=out[0, rows].astype(np.float32),
                        absmax=np.float64(np.abs(out).max()), input_sha256=np.array(digest),
                        workload=np.array(wl.name))
    print(f"wrote {out_path} in {time.time() - t0:.0f} s (absmax {np.abs(out).max():.4f})")


if __name__ == "__main__":
    main(sys.argv[1] if len(sys.argv) > 1 else OUT)
