"""Failure detection on the GPU, in forms that fault, trap and hang nothing.

* Host-side injection (sr_debug_fail_enqueue): the n-th CUDA call of sr_forward
  reports an error instead of being made.  The call returns SR_ERR_CUDA with a
  message, attempts nothing after it, and the handle works normally afterwards.
* The bounded mbarrier wait of the tensor-core kernels, run on a barrier nothing
  arrives at with a 20 ms limit (sr_selftest_wait_timeout): it gives up, sets bit
  0 of the fault word and returns; the context stays usable.
* A canary-padded workspace: the library writes nothing outside the workspace
  it is given, and the fault word stays clear on every normal forward.
"""
import numpy as np
import pytest
import torch

from paper_2607_02829_gb300 import synth
from tests._helpers import built_lib

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("CUDA GPU required for -m gpu tests")
    built_lib()


def _tiny(dtype, split=(1, 2, 1), r=0.25, selector="random"):
    return synth.Workload(f"fail_{dtype}", B=2, grid_h=1, grid_w=200, channels=3, patch=1, D=128,
                          heads=2, n1=split[0], n2=split[1], n3=split[2], keep_ratio=r,
                          dtype=dtype, selector=selector, seed_index=91)


def _setup(wl, ws_bytes_extra=0):
    from paper_2607_02829_gb300 import binding as b
    x, ws = synth.make_inputs(wl)
    cfg = b.make_config(wl.B, wl.L, wl.D, wl.heads, wl.n1, wl.n2, wl.n3, dtype=wl.dtype,
                        selector=wl.selector)
    wd = [{k: v.cuda() for k, v in blk.items()} for blk in ws]
    return b, cfg, x.cuda(), wd, b.weights_array(wd)


@pytest.mark.parametrize("dtype,selector", [("bf16", "random"), ("bf16", "topk_l2"),
                                            ("f32", "random")])
def test_injected_failure_returns_cuda_error_and_enqueues_nothing_after(dtype, selector):
    wl = _tiny(dtype, selector=selector)
    b, cfg, x, wd, warr = _setup(wl)
    enc = b.Encoder(cfg, max_keep_ratio=wl.keep_ratio)
    s = torch.cuda.current_stream().cuda_stream
    try:
        ref = torch.empty_like(x)
        # the handle's first forward also clears its fault word: count the calls
        # of a later one
        b.sr_forward(enc.handle, x.data_ptr(), warr, wl.keep_ratio, 5, ref.data_ptr(), None, s)
        b.sr_debug_fail_enqueue(-1)
        b.sr_forward(enc.handle, x.data_ptr(), warr, wl.keep_ratio, 5, ref.data_ptr(), None, s)
        calls = b.sr_debug_enqueue_count()
        assert calls > 10
        torch.cuda.synchronize()
        for n in sorted({0, 1, 2, calls // 3, calls // 2, calls - 2, calls - 1}):
            out = torch.zeros_like(x)
            b.sr_debug_fail_enqueue(n)
            with pytest.raises(b.SRError) as e:
                b.sr_forward(enc.handle, x.data_ptr(), warr, wl.keep_ratio, 5, out.data_ptr(),
                             None, s)
            assert e.value.status == b.SR_ERR_CUDA
            assert "injected" in str(e.value)
            assert b.sr_debug_enqueue_count() == n + 1      # nothing attempted after the failure
            b.sr_debug_fail_enqueue(-1)
            torch.cuda.synchronize()
            if n == calls - 1:
                # the last call is the narrowing into out: nothing was written there
                assert not out.any()
        # the handle is intact: the next forward is bitwise the reference
        again = torch.empty_like(x)
        b.sr_forward(enc.handle, x.data_ptr(), warr, wl.keep_ratio, 5, again.data_ptr(), None, s)
        torch.cuda.synchronize()
        assert torch.equal(again, ref)
        assert b.sr_device_fault(enc.handle, False, s) == 0
    finally:
        b.sr_debug_fail_enqueue(-1)
        enc.close()


def test_bounded_wait_gives_up_and_sets_the_fault_bit():
    from paper_2607_02829_gb300 import binding as b
    fault = torch.zeros(1, dtype=torch.int32, device="cuda")
    waited = torch.zeros(1, dtype=torch.int64, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    b.sr_selftest_wait_timeout(fault.data_ptr(), 20000, waited.data_ptr(), s)
    torch.cuda.synchronize()
    assert int(fault.item()) == 1                # bit 0: gave up; bit 31 would mean it completed
    ns = int(waited.item())
    assert 20_000_000 <= ns < 1_000_000_000, ns
    # the context is still usable: a forward runs and gives the same result twice
    wl = _tiny("bf16")
    b_, cfg, x, wd, warr = _setup(wl)
    enc = b.Encoder(cfg, max_keep_ratio=wl.keep_ratio)
    o1, i1 = enc.forward(x, warr, wl.keep_ratio, 9, want_idx=True)
    o2, i2 = enc.forward(x, warr, wl.keep_ratio, 9, want_idx=True)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2) and torch.equal(i1, i2)
    assert b.sr_device_fault(enc.handle, False, s) == 0
    enc.close()


@pytest.mark.parametrize("wlname,r", [("tiny_bf16", 0.25), ("tiny_f32", 0.5), ("tiny_bf16", 1.0),
                                      ("c2_5p625deg_bf16", 0.25)])
def test_workspace_canaries_untouched(wlname, r):
    from paper_2607_02829_gb300 import binding as b
    if wlname.startswith("tiny"):
        wl = _tiny(wlname.split("_")[1], r=r, selector="topk_l2" if r == 0.25 else "random")
    else:
        wl = synth.WORKLOADS[wlname]
    b, cfg, x, wd, warr = _setup(wl)
    nbytes = b.sr_workspace_bytes(cfg, r)
    pad = 1 << 20
    buf = torch.empty(pad + nbytes + pad + 256, dtype=torch.uint8, device="cuda")
    pattern = (torch.arange(buf.numel(), device="cuda", dtype=torch.int64) * 7919 % 251).to(torch.uint8)
    buf.copy_(pattern)
    base = (buf.data_ptr() + pad + 255) // 256 * 256
    lo = base - buf.data_ptr()
    h = b.sr_create(cfg, base, nbytes)
    s = torch.cuda.current_stream().cuda_stream
    try:
        out = torch.empty_like(x)
        K = b.sr_keep_count(wl.L, r)
        idx = torch.empty(wl.B, K, dtype=torch.int32, device="cuda")
        for seed in (1, 2):
            b.sr_forward(h, x.data_ptr(), warr, r, seed, out.data_ptr(), idx.data_ptr(), s)
        torch.cuda.synchronize()
        assert torch.equal(buf[:lo], pattern[:lo]), "bytes before the workspace changed"
        assert torch.equal(buf[lo + nbytes:], pattern[lo + nbytes:]), "bytes after the workspace changed"
        assert b.sr_device_fault(h, False, s) == 0
        assert torch.isfinite(out.float()).all()
    finally:
        b.sr_destroy(h)
