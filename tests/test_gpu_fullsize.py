"""Parity at the workloads' full sizes, in the launch configuration bench.py times.

* 1.40625 deg (c3): the whole fp64 oracle forward, element by element.
* 0.25 deg (c4): 32 sampled output rows of the oracle forward stored in
  tests/golden/ (written by tests/golden/make_c4_golden.py, which calls only
  the oracle), plus the bit-exact index set and unselected-row passthrough.
* keep-ratio x selector sweep on the 1.40625 deg model: index sets for every
  point, r = 1 bitwise equal to the dense stack, oracle parity at r = 0.125.
"""
import os

import numpy as np
import pytest
import torch

from oracle import reslim as o
from paper_2607_02829_gb300 import synth
from tests._helpers import ROOT, built_lib, gpu_forward, max_norm_rel

pytestmark = pytest.mark.gpu
TOL = 2e-2
THREADS = len(os.sched_getaffinity(0))


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("CUDA GPU required for -m gpu tests")
    built_lib()


def _passthrough_ok(wl, x, ws, idx):
    """Unselected rows of the post-scatter stream equal the pre-routing stream."""
    post, _ = gpu_forward(wl, x, ws, n_split=(wl.n1, wl.n2, 0), want_idx=False)
    pre, _ = gpu_forward(wl, x, ws, n_split=(wl.n1, 0, 0), want_idx=False)
    sel = np.zeros((wl.B, wl.L), dtype=bool)
    sel[np.arange(wl.B)[:, None], idx] = True
    uns = torch.from_numpy(~sel)
    return torch.equal(post[uns], pre[uns]), pre


def test_c3_full_forward_matches_oracle():
    wl = synth.WORKLOADS["c3_1p40625deg_bf16"]
    x, ws = synth.make_inputs(wl)
    out, idx = gpu_forward(wl, x, ws)
    assert np.array_equal(idx, o.select_random(wl.B, wl.L, 512, wl.select_seed))
    ref, _ = o.forward(synth.stored_as_f64(x), o.as_f64_weights(ws), wl.n1, wl.n2, wl.n3,
                       wl.heads, wl.keep_ratio, seed=wl.select_seed, threads=THREADS)
    err = max_norm_rel(synth.stored_as_f64(out), ref)
    assert err <= TOL, err
    ok, _ = _passthrough_ok(wl, x, ws, idx)
    assert ok


def test_c4_sampled_rows_match_oracle():
    path = os.path.join(ROOT, "tests", "golden", "c4_0p25deg_oracle_samples.npz")
    g = np.load(path)
    wl = synth.WORKLOADS["c4_0p25deg_bf16"]
    x, ws = synth.make_inputs(wl)
    from tests.golden.make_c4_golden import input_digest
    assert input_digest(x) == str(g["input_sha256"]), "generated inputs differ from the golden's"
    out, idx = gpu_forward(wl, x, ws)
    assert np.array_equal(idx, o.select_random(1, wl.L, 4050, wl.select_seed))
    y = synth.stored_as_f64(out)[0, g["rows"]]
    err = float(np.abs(y - g["out_rows"]).max() / g["absmax"])
    assert err <= TOL, err
    ok, _ = _passthrough_ok(wl, x, ws, idx)
    assert ok


@pytest.fixture(scope="module")
def sweep_inputs():
    wl = synth.sweep_workloads()[0]
    return synth.make_inputs(wl)


@pytest.mark.parametrize("selector", ["random", "topk_l2"])
@pytest.mark.parametrize("r", [1.0, 0.5, 0.25, 0.125])
def test_sweep_index_sets_and_passthrough(sweep_inputs, selector, r):
    wl = [w for w in synth.sweep_workloads() if w.selector == selector and w.keep_ratio == r][0]
    x, ws = sweep_inputs
    if r == 1.0:
        a, _ = gpu_forward(wl, x, ws, want_idx=False)
        d, _ = gpu_forward(wl, x, ws, n_split=(wl.N, 0, 0), want_idx=False)
        assert torch.equal(a, d)
        return
    K = o.keep_count(wl.L, r)
    _, idx = gpu_forward(wl, x, ws, n_split=(wl.n1, wl.n2, 0))
    ok, pre = _passthrough_ok(wl, x, ws, idx)
    assert ok
    if selector == "random":
        assert np.array_equal(idx, o.select_random(wl.B, wl.L, K, wl.select_seed))
    else:
        # the GPU ranks the stored (bf16) block-n1 output; the oracle ranks the same
        # values in fp64: equal sets, or differences only inside the fp32 tie band
        x0 = synth.stored_as_f64(pre)
        s = o.token_sq_norms(x0)
        exp = o.select_topk_l2(x0, K)
        for b in range(wl.B):
            diff = set(idx[b].tolist()) ^ set(exp[b].tolist())
            kth = np.sort(s[b])[::-1][K - 1]
            assert all(abs(s[b, i] - kth) <= 1e-5 * kth for i in diff)


@pytest.mark.parametrize("selector", ["random", "topk_l2"])
def test_sweep_r0125_forward_matches_oracle(sweep_inputs, selector):
    wl = [w for w in synth.sweep_workloads() if w.selector == selector and w.keep_ratio == 0.125][0]
    x, ws = sweep_inputs
    out, idx = gpu_forward(wl, x, ws)
    ref, _ = o.forward(synth.stored_as_f64(x), o.as_f64_weights(ws), wl.n1, wl.n2, wl.n3,
                       wl.heads, wl.keep_ratio, seed=wl.select_seed, idx=idx, threads=THREADS)
    err = max_norm_rel(synth.stored_as_f64(out), ref)
    assert err <= TOL, err
