"""GPU parity of the CUDA path (through the C ABI) against the fp64 oracle.

Bars: indices and the unselected-token passthrough bit-exact; outputs within a
max-norm relative error max|y - o| / max|o| of 1e-4 (fp32) or 2e-2 (bf16).
"""
import numpy as np
import pytest
import torch

from oracle import reslim as o
from paper_2607_02829_gb300 import synth
from tests._helpers import built_lib, check_parity, gpu_forward

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-4, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.fail("CUDA GPU required for -m gpu tests")
    built_lib()


def _oracle(wl, x, ws, keep_ratio=None, seed=None, selector=None, n_split=None, idx=None):
    n1, n2, n3 = n_split or (wl.n1, wl.n2, wl.n3)
    xf = synth.stored_as_f64(x)
    wf = o.as_f64_weights(ws[:n1 + n2 + n3])
    return o.forward(xf, wf, n1, n2, n3, wl.heads,
                     wl.keep_ratio if keep_ratio is None else keep_ratio,
                     seed=wl.select_seed if seed is None else seed,
                     selector=selector or wl.selector, idx=idx, threads=8, grid_w=wl.grid_wp)


def _tiny(dtype, B=2, L=200, heads=2, split=(1, 2, 1), r=0.25, selector="random"):
    return synth.Workload(f"tiny_{dtype}", B=B, grid_h=1, grid_w=L, channels=3, patch=1,
                          D=64 * heads, heads=heads, n1=split[0], n2=split[1], n3=split[2],
                          keep_ratio=r, dtype=dtype, selector=selector, seed_index=77)


# ------------------------------------------------------------ selection
@pytest.mark.parametrize("B,L,K,shared", [
    (1, 1, 1, False), (3, 10, 4, False), (2, 512, 128, False), (32, 512, 128, False),
    (8, 2048, 512, False), (8, 2048, 2048, False), (1, 16200, 4050, False),
    (4, 1000, 1, True), (2, 24576, 6144, False), (5, 777, 776, True)])
def test_select_random_bitexact(B, L, K, shared):
    from paper_2607_02829_gb300 import binding as b
    cfg = b.make_config(B, L, 64, 1, 0, 1, 0, dtype="bf16", shared=shared)
    for seed in (0, 3004, 2**64 - 1):
        enc = b.Encoder(cfg, max_keep_ratio=1.0)
        r = K / L
        assert b.sr_keep_count(L, r) == K
        idx = enc.select(None, r, seed).cpu().numpy()
        torch.cuda.synchronize()
        expect = o.select_random(B, L, K, seed, shared)
        assert np.array_equal(idx, expect)
        enc.close()


@pytest.mark.parametrize("B,L,D,K,dtype", [(2, 300, 64, 75, "bf16"), (8, 2048, 1024, 512, "bf16"),
                                           (1, 16200, 1024, 4050, "bf16"), (2, 512, 256, 128, "f32")])
def test_select_topk_l2(B, L, D, K, dtype):
    from paper_2607_02829_gb300 import binding as b
    g = torch.Generator().manual_seed(B * L + D)
    x = torch.randn(B, L, D, generator=g, dtype=torch.float64)
    x[:, 1::7] = x[:, 0::7][:, :x[:, 1::7].shape[1]]           # exact duplicate rows -> exact ties
    xs = x.to(synth.torch_dtype(dtype))
    cfg = b.make_config(B, L, D, D // 64, 0, 1, 0, dtype=dtype, selector="topk_l2")
    enc = b.Encoder(cfg, max_keep_ratio=1.0)
    idx = enc.select(xs.cuda(), K / L, 0).cpu().numpy()
    enc.close()
    xf = synth.stored_as_f64(xs)
    expect = o.select_topk_l2(xf, K)
    s = o.token_sq_norms(xf)
    for bb in range(B):
        assert np.all(np.diff(idx[bb]) > 0) and idx[bb].min() >= 0 and idx[bb].max() < L
        got, exp = set(idx[bb].tolist()), set(expect[bb].tolist())
        if got == exp:
            continue
        # the GPU ranks fp32 sums: a disagreement is only allowed inside the band of
        # fp32 rounding around the K-th score
        kth = np.sort(s[bb])[::-1][K - 1]
        for i in got ^ exp:
            assert abs(s[bb, i] - kth) <= 1e-5 * kth, (i, s[bb, i], kth)


# ------------------------------------------------- routing invariants (GPU)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_zero_sparse_blocks_give_exact_passthrough(dtype):
    # sparse blocks with all W and b zero add exactly 0: h == h0, delta == 0,
    # and x' == x0 everywhere -- checks gather and scatter addressing bit-exactly
    wl = _tiny(dtype, split=(1, 2, 0))
    x, ws = synth.make_inputs(wl)
    for i in (1, 2):
        ws[i] = {k: (v if k.endswith("_g") else torch.zeros_like(v)) for k, v in ws[i].items()}
    out, idx = gpu_forward(wl, x, ws)
    x0, _ = gpu_forward(wl, x, ws, n_split=(1, 0, 0), want_idx=False)
    assert torch.equal(out, x0)
    assert idx.shape == (wl.B, 50)


@pytest.mark.parametrize("wlname", ["c1_5p625deg_f32", "c2_5p625deg_bf16"])
def test_unselected_tokens_bitexact(wlname):
    wl = synth.WORKLOADS[wlname]
    x, ws = synth.make_inputs(wl)
    out, idx = gpu_forward(wl, x, ws, n_split=(wl.n1, wl.n2, 0))
    x0, _ = gpu_forward(wl, x, ws, n_split=(wl.n1, 0, 0), want_idx=False)
    assert np.array_equal(idx, o.select_random(wl.B, wl.L, wl.L // 4, wl.select_seed))
    sel = np.zeros((wl.B, wl.L), dtype=bool)
    sel[np.arange(wl.B)[:, None], idx] = True
    assert torch.equal(out[torch.from_numpy(~sel)], x0[torch.from_numpy(~sel)])
    changed = (out != x0).any(dim=-1)
    assert changed[torch.from_numpy(sel)].float().mean() > 0.99


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_r1_is_bitwise_the_dense_stack(dtype):
    wl = _tiny(dtype, split=(1, 2, 1))
    x, ws = synth.make_inputs(wl)
    a, _ = gpu_forward(wl, x, ws, keep_ratio=1.0, want_idx=False)
    d, _ = gpu_forward(wl, x, ws, keep_ratio=1.0, n_split=(4, 0, 0), want_idx=False)
    assert torch.equal(a, d)


def test_in_place_equals_out_of_place():
    wl = _tiny("bf16")
    x, ws = synth.make_inputs(wl)
    a, ia = gpu_forward(wl, x, ws)
    b_, ib = gpu_forward(wl, x, ws, inplace=True)
    assert torch.equal(a, b_) and np.array_equal(ia, ib)


# ------------------------------------------------------ end-to-end parity
@pytest.mark.parametrize("dtype,B,L,heads,split,r", [
    ("f32", 2, 200, 2, (1, 2, 1), 0.25),
    ("bf16", 2, 200, 2, (1, 2, 1), 0.25),
    ("bf16", 3, 333, 4, (1, 3, 1), 0.5),      # ragged tiles everywhere
    ("bf16", 1, 1, 1, (1, 1, 1), 1.0),        # a single token
    ("bf16", 2, 129, 2, (0, 2, 0), 0.125),    # K = 16, routing only
    ("f32", 1, 97, 1, (2, 1, 0), 0.5),
    ("bf16", 2, 129, 2, (1, 1, 1), 0.0078125),  # K = 1: one routed token per sample
])
def test_forward_parity_small(dtype, B, L, heads, split, r):
    wl = _tiny(dtype, B=B, L=L, heads=heads, split=split, r=r)
    x, ws = synth.make_inputs(wl)
    out, idx = gpu_forward(wl, x, ws, want_idx=r < 1.0)
    ref, ridx = _oracle(wl, x, ws)
    if r < 1.0:
        assert np.array_equal(idx, ridx)
    check_parity(f"small {dtype} B={B} L={L} H={heads} split={split} r={r}",
                 synth.stored_as_f64(out), ref, TOL[dtype])


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_forward_parity_shared_index_set(dtype):
    # one index set for the whole batch (the App. A.4 listing's reading)
    wl = _tiny(dtype, B=3, L=200, heads=2, split=(1, 2, 1), r=0.25)
    x, ws = synth.make_inputs(wl)
    out, idx = gpu_forward(wl, x, ws, shared=True)
    assert all(np.array_equal(idx[0], idx[i]) for i in range(wl.B))
    ref, ridx = o.forward(synth.stored_as_f64(x), o.as_f64_weights(ws), 1, 2, 1, wl.heads,
                          wl.keep_ratio, seed=wl.select_seed, shared_indices=True, threads=8)
    assert np.array_equal(idx, ridx)
    check_parity(f"small {dtype} shared index set", synth.stored_as_f64(out), ref, TOL[dtype])


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_forward_host_equals_device_forward(dtype):
    # the one-call host form: copy in, sr_forward in place, copy out
    from paper_2607_02829_gb300 import binding as b
    wl = _tiny(dtype, B=2, L=200, heads=2, split=(1, 2, 1), r=0.25)
    x, ws = synth.make_inputs(wl)
    ref, ridx = gpu_forward(wl, x, ws)
    cfg = b.make_config(wl.B, wl.L, wl.D, wl.heads, wl.n1, wl.n2, wl.n3, dtype=dtype)
    enc = b.Encoder(cfg, max_keep_ratio=wl.keep_ratio)
    wd = [{k: v.cuda() for k, v in blk.items()} for blk in ws[:wl.N]]
    warr = b.weights_array(wd)
    xh = x.pin_memory()
    oh = torch.empty_like(xh).pin_memory()
    dbuf = torch.empty_like(x, device="cuda")
    idx = torch.empty(wl.B, 50, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()
    b.sr_forward_host(enc.handle, xh.data_ptr(), warr, wl.keep_ratio, wl.select_seed,
                      dbuf.data_ptr(), oh.data_ptr(), idx.data_ptr(), stream.cuda_stream)
    torch.cuda.synchronize()
    assert torch.equal(oh, ref)
    assert np.array_equal(idx.cpu().numpy().astype(np.int64), ridx)
    enc.close()


@pytest.mark.parametrize("wlname", ["c1_5p625deg_f32", "c2_5p625deg_bf16"])
def test_forward_parity_workload(wlname):
    wl = synth.WORKLOADS[wlname]
    x, ws = synth.make_inputs(wl)
    out, idx = gpu_forward(wl, x, ws)
    ref, ridx = _oracle(wl, x, ws)
    assert np.array_equal(idx, ridx)
    check_parity(f"{wlname} (full output)", synth.stored_as_f64(out), ref, TOL[wl.dtype])


# bf16 with D = 128: the scores come from the dense-early block's FC2 epilogue;
# D = 192 (64-column GEMM tiles) and fp32 take the separate pass over the stream
@pytest.mark.parametrize("dtype,heads", [("bf16", 2), ("bf16", 3), ("f32", 2)])
def test_forward_parity_topk_selector_small(dtype, heads):
    wl = _tiny(dtype, B=2, L=256, heads=heads, split=(2, 2, 1), r=0.25, selector="topk_l2")
    x, ws = synth.make_inputs(wl)
    out, idx = gpu_forward(wl, x, ws)
    ref, ridx = _oracle(wl, x, ws, idx=idx)      # same indices on both sides
    check_parity(f"small top-K {dtype} H={heads}", synth.stored_as_f64(out), ref, TOL[dtype])
    x0, _ = gpu_forward(wl, x, ws, n_split=(2, 0, 0), want_idx=False)
    assert np.array_equal(idx, o.select_topk_l2(synth.stored_as_f64(x0), 64))
    again, idx2 = gpu_forward(wl, x, ws)
    assert torch.equal(out, again) and np.array_equal(idx, idx2)     # reproducible


# the Laplacian selector on a 2-D patch grid (8 x 24 tokens): the index set
# against the oracle's on the GPU's own pre-routing state, then the forward
# against the oracle given the GPU's indices
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_forward_parity_laplacian_selector_small(dtype):
    wl = synth.Workload(f"lap_{dtype}", B=2, grid_h=8, grid_w=24, channels=3, patch=1, D=128,
                        heads=2, n1=2, n2=2, n3=1, keep_ratio=0.25, dtype=dtype,
                        selector="laplacian", seed_index=78)
    x, ws = synth.make_inputs(wl)
    out, idx = gpu_forward(wl, x, ws)
    x0, _ = gpu_forward(wl, x, ws, n_split=(2, 0, 0), want_idx=False)
    xf = synth.stored_as_f64(x0)
    K = o.keep_count(wl.L, wl.keep_ratio)
    s = o.token_laplacian_scores(xf, wl.grid_wp)
    exp = o.select_topk_laplacian(xf, K, wl.grid_wp)
    for bb in range(wl.B):
        kth = np.sort(s[bb])[::-1][K - 1]
        diff = set(idx[bb].tolist()) ^ set(exp[bb].tolist())
        assert all(abs(s[bb, i] - kth) <= 1e-5 * kth for i in diff), sorted(diff)
    ref, _ = _oracle(wl, x, ws, idx=idx)
    check_parity(f"small Laplacian {dtype}", synth.stored_as_f64(out), ref, TOL[dtype])


@pytest.mark.parametrize("B,H,W,D,K", [(2, 8, 24, 64, 48), (1, 90, 180, 1024, 4050),
                                       (3, 5, 1, 64, 2), (1, 1, 7, 64, 3)])
def test_select_laplacian_integer_fields_exact(B, H, W, D, K):
    # small integer values: every score is an exact integer on both sides, so
    # the sets must be equal, ties included
    from paper_2607_02829_gb300 import binding as b
    g = torch.Generator().manual_seed(B * H * W + D)
    x = torch.randint(-3, 4, (B, H * W, D), generator=g).to(torch.bfloat16)
    cfg = b.make_config(B, H * W, D, D // 64, 0, 1, 0, dtype="bf16", selector="laplacian",
                        grid_w=W)
    enc = b.Encoder(cfg, max_keep_ratio=1.0)
    idx = enc.select(x.cuda(), K / (H * W), 0).cpu().numpy()
    enc.close()
    assert np.array_equal(idx, o.select_topk_laplacian(synth.stored_as_f64(x), K, W))


# ------------------------------------------------------------ implicit ensemble
@pytest.mark.parametrize("dtype,split,r", [("bf16", (1, 2, 1), 0.25), ("f32", (1, 2, 1), 0.5),
                                            ("bf16", (2, 1, 0), 0.25), ("bf16", (1, 2, 1), 1.0)])
def test_ensemble_members_bitwise_and_mean(dtype, split, r):
    from paper_2607_02829_gb300 import binding as b
    wl = _tiny(dtype, B=2, L=200, heads=2, split=split, r=r)
    x, ws = synth.make_inputs(wl)
    seeds = [3, 77, 2**63 + 5]
    n1, n2, n3 = split
    cfg = b.make_config(wl.B, wl.L, wl.D, wl.heads, n1, n2, n3, dtype=dtype)
    enc = b.Encoder(cfg, max_keep_ratio=r)
    xd = x.cuda()
    wd = [{k: v.cuda() for k, v in blk.items()} for blk in ws[:n1 + n2 + n3]]
    warr = b.weights_array(wd)
    mean, members, idx = enc.forward_ensemble(xd, warr, r, seeds, want_members=True, want_idx=r < 1.0)
    for m, s in enumerate(seeds):
        y, i1 = enc.forward(xd, warr, r, s, want_idx=r < 1.0)
        assert torch.equal(members[m], y)          # member m is exactly sr_forward(seed m)
        if r < 1.0:
            assert torch.equal(idx[m], i1)
    torch.cuda.synchronize()
    ref, _, ridx = o.forward_ensemble(synth.stored_as_f64(x), o.as_f64_weights(ws[:n1 + n2 + n3]),
                                      n1, n2, n3, wl.heads, r, seeds, threads=8)
    if r < 1.0:
        for m in range(len(seeds)):
            assert np.array_equal(idx[m].cpu().numpy(), ridx[m])
    check_parity(f"ensemble mean {dtype} split={split} r={r}", synth.stored_as_f64(mean.cpu()),
                 ref, TOL[dtype])
    enc.close()


# ------------------------------------------------------------ asymmetric attention
# the last three have more work items (sample, head, 256-query block) than the
# GPU has SMs and at most 16 key tiles: they run the persistent grid, whose CTAs
# take several items each (ragged queries and keys included)
@pytest.mark.parametrize("B,Tq,Tkv,heads", [(2, 300, 1000, 2), (1, 129, 77, 1), (3, 1, 5, 4),
                                            (1, 257, 256, 2), (2, 64, 1, 1),
                                            (64, 257, 129, 4), (48, 100, 300, 4),
                                            (40, 512, 2048, 8)])
def test_cross_attention_parity(B, Tq, Tkv, heads):
    from paper_2607_02829_gb300 import binding as b
    D = 64 * heads
    g = torch.Generator().manual_seed(B * 1000 + Tq + Tkv)
    q = torch.randn(B, Tq, D, generator=g).to(torch.bfloat16)
    kv = torch.randn(B, Tkv, 2 * D, generator=g).to(torch.bfloat16)
    out = torch.empty(B, Tq, D, dtype=torch.bfloat16, device="cuda")
    fault = torch.zeros(1, dtype=torch.int32, device="cuda")
    qd, kvd = q.cuda(), kv.cuda()
    b.sr_cross_attention(qd.data_ptr(), kvd.data_ptr(), B, Tq, Tkv, heads, out.data_ptr(),
                         fault.data_ptr(), torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    assert int(fault.item()) == 0
    ref = o.cross_attention(synth.stored_as_f64(q), synth.stored_as_f64(kv), heads)
    check_parity(f"cross-attention B={B} Tq={Tq} Tkv={Tkv} H={heads}",
                 synth.stored_as_f64(out.cpu()), ref, TOL["bf16"])


def test_cross_attention_routed_over_full_sequence_sampled():
    # the 0.25 deg shape of the EDM sparse stage: 4050 routed queries over the
    # 16200-token conditioning sequence, 16 heads; the oracle on sampled rows
    from paper_2607_02829_gb300 import binding as b
    B, Tq, Tkv, heads = 1, 4050, 16200, 16
    D = 64 * heads
    g = torch.Generator().manual_seed(4050)
    q = torch.randn(B, Tq, D, generator=g).to(torch.bfloat16)
    kv = torch.randn(B, Tkv, 2 * D, generator=g).to(torch.bfloat16)
    out = torch.empty(B, Tq, D, dtype=torch.bfloat16, device="cuda")
    fault = torch.zeros(1, dtype=torch.int32, device="cuda")
    b.sr_cross_attention(q.cuda().data_ptr(), kv.cuda().data_ptr(), B, Tq, Tkv, heads,
                         out.data_ptr(), fault.data_ptr(), torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    assert int(fault.item()) == 0
    rows = np.random.default_rng(0).choice(Tq, 48, replace=False)
    rows = np.concatenate([rows, [0, 255, 256, Tq - 1]])
    ref = o.cross_attention(synth.stored_as_f64(q)[:, rows], synth.stored_as_f64(kv), heads)
    got = synth.stored_as_f64(out.cpu())[:, rows]
    check_parity("cross-attention 4050 over 16200, 52 sampled rows", got, ref, TOL["bf16"])


# ------------------------------------------------------------ CUDA graphs
@pytest.mark.parametrize("dtype,selector", [("bf16", "random"), ("bf16", "topk_l2"), ("f32", "random")])
def test_forward_captured_in_a_cuda_graph_replays_bitwise(dtype, selector):
    # after a first (warm-up) call, sr_forward only enqueues work: captured into a
    # graph and replayed it gives bitwise the direct call's output, also after the
    # input changes in place
    from paper_2607_02829_gb300 import binding as b
    wl = _tiny(dtype, B=2, L=256, heads=2, split=(1, 2, 1), r=0.25, selector=selector)
    x, ws = synth.make_inputs(wl)
    cfg = b.make_config(wl.B, wl.L, wl.D, wl.heads, wl.n1, wl.n2, wl.n3, dtype=dtype,
                        selector=selector)
    enc = b.Encoder(cfg, max_keep_ratio=wl.keep_ratio)
    xd = x.cuda()
    wd = [{k: v.cuda() for k, v in blk.items()} for blk in ws]
    warr = b.weights_array(wd)
    ref, _ = enc.forward(xd, warr, wl.keep_ratio, 11)
    out = torch.zeros_like(xd)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        b.sr_forward(enc.handle, xd.data_ptr(), warr, wl.keep_ratio, 11, out.data_ptr(), None,
                     side.cuda_stream)
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(out, ref)
    xd.mul_(0.5)
    ref2, _ = enc.forward(xd, warr, wl.keep_ratio, 11)
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(out, ref2) and not torch.equal(ref2, ref)
    assert b.sr_device_fault(enc.handle, False, torch.cuda.current_stream().cuda_stream) == 0
    del g
    enc.close()
