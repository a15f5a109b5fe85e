"""Shared test helpers: build/load the library, move synthetic inputs to the GPU,
run the CUDA path through the C ABI, and compare with the oracle."""
from __future__ import annotations

import ctypes
import re
import os

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def built_lib():
    from paper_2607_02829_gb300 import build, binding
    build.build()
    return binding.lib()


def header_functions():
    """Function names declared in include/*.h."""
    names = []
    inc = os.path.join(ROOT, "include")
    for f in sorted(os.listdir(inc)):
        if not f.endswith(".h"):
            continue
        src = open(os.path.join(inc, f)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        src = re.sub(r"//[^\n]*", "", src)
        for m in re.finditer(r"^[A-Za-z_][\w \*]*?\b(sr_\w+)\s*\(", src, flags=re.M):
            if "typedef" not in m.group(0):
                names.append(m.group(1))
    return sorted(set(names))


def max_norm_rel(y, o):
    y = np.asarray(y, dtype=np.float64)
    o = np.asarray(o, dtype=np.float64)
    return float(np.abs(y - o).max() / max(np.abs(o).max(), 1e-300))


# (case, max-norm relative error, 99.9th percentile of |y - o| / max|o|, bar,
# elements compared, note), in test order; the session summary prints them
PARITY_RECORDS = []


def check_parity(case, y, o, tol, note=""):
    """Asserts max|y - o| / max|o| <= tol and records that error together with
    the elementwise 99.9th-percentile error |y - o| / max|o| (and a note)."""
    y = np.asarray(y, dtype=np.float64)
    o = np.asarray(o, dtype=np.float64)
    scale = max(float(np.abs(o).max()), 1e-300)
    e = np.abs(y - o).ravel() / scale
    err = float(e.max())
    p999 = float(np.quantile(e, 0.999))
    PARITY_RECORDS.append((case, err, p999, tol, int(e.size), note))
    assert err <= tol, f"{case}: max-norm relative error {err:.3e} exceeds {tol:.0e}"
    return err


def to_device(x, weights):
    xd = x.cuda()
    wd = [{k: v.cuda() for k, v in blk.items()} for blk in weights]
    return xd, wd


def gpu_forward(wl, x, weights, keep_ratio=None, seed=None, selector=None, shared=False,
                n_split=None, want_idx=True, inplace=False):
    """Runs sr_forward on CPU torch tensors (x, weights in storage dtype); returns
    (out as CPU torch tensor, idx as numpy int64 or None)."""
    import torch
    from paper_2607_02829_gb300 import binding as b
    n1, n2, n3 = n_split or (wl.n1, wl.n2, wl.n3)
    r = wl.keep_ratio if keep_ratio is None else keep_ratio
    cfg = b.make_config(wl.B, wl.L, wl.D, wl.heads, n1, n2, n3, dtype=wl.dtype,
                        selector=selector or wl.selector, shared=shared, grid_w=wl.grid_wp)
    enc = b.Encoder(cfg, max_keep_ratio=r)
    xd, wd = to_device(x, weights[:n1 + n2 + n3])
    warr = b.weights_array(wd)
    out = xd if inplace else None
    out, idx = enc.forward(xd, warr, r, wl.select_seed if seed is None else seed, out=out,
                           want_idx=want_idx)
    torch.cuda.synchronize()
    res = out.cpu(), (idx.cpu().numpy().astype(np.int64) if idx is not None else None)
    enc.close()
    return res
