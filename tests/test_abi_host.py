"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every function include/*.h declares, and rejects invalid arguments before any
CUDA call."""
import ctypes

import pytest

from tests._helpers import built_lib, header_functions


@pytest.fixture(scope="module")
def L():
    return built_lib()


def test_exports_every_declared_function(L):
    names = header_functions()
    assert "sr_forward" in names and "sr_create" in names
    for n in names:
        assert hasattr(L, n), f"{n} declared in include/ but not exported"


def test_keep_count(L):
    from paper_2607_02829_gb300 import binding as b
    assert b.sr_keep_count(16200, 0.25) == 4050
    assert b.sr_keep_count(8192, 0.25) == 2048
    assert b.sr_keep_count(2048, 0.125) == 256
    assert b.sr_keep_count(10, 0.0) == -1
    assert b.sr_keep_count(10, 1.5) == -1
    assert b.sr_keep_count(10, float("nan")) == -1
    assert b.sr_keep_count(0, 0.5) == -1
    assert b.sr_keep_count(3, 0.3) == 0


def test_invalid_configs_rejected(L):
    from paper_2607_02829_gb300 import binding as b
    good = b.make_config(2, 512, 256, 4, 2, 2, 2, dtype="f32")
    assert b.sr_workspace_bytes(good, 0.25) > 0
    lap = b.make_config(2, 512, 256, 4, 2, 2, 2, dtype="f32", selector="laplacian", grid_w=32)
    assert b.sr_workspace_bytes(lap, 0.25) > 0
    bad = [
        dict(D=250), dict(heads=3), dict(B=0), dict(L=0), dict(n1=-1),
        dict(n1=0, n2=0, n3=0), dict(dtype=7), dict(selector=5), dict(shared_indices=2),
        dict(ln_eps=0.0), dict(mlp_hidden=100), dict(L=100000),
        dict(selector=2), dict(selector=2, grid_w=7), dict(selector=2, grid_w=-64),
    ]
    for kw in bad:
        c = b.make_config(2, 512, 256, 4, 2, 2, 2, dtype="f32")
        for k, v in kw.items():
            setattr(c, k, v)
        assert b.sr_workspace_bytes(c, 0.25) == 0, kw


def _handle(b, cfg, nbytes):
    # a fake, 256-byte aligned device address: sr_create only records it
    return b.sr_create(cfg, 0x100000, nbytes)


def test_create_and_argument_errors(L):
    from paper_2607_02829_gb300 import binding as b
    cfg = b.make_config(2, 512, 256, 4, 2, 2, 2, dtype="f32")
    n = b.sr_workspace_bytes(cfg, 0.25)
    with pytest.raises(b.SRError) as e:
        b.sr_create(cfg, 0, n)
    assert e.value.status == b.SR_ERR_WORKSPACE
    with pytest.raises(b.SRError) as e:
        b.sr_create(cfg, 0x100001, n)
    assert e.value.status == b.SR_ERR_WORKSPACE
    with pytest.raises(b.SRError) as e:
        b.sr_create(cfg, 0x100000, 1000)
    assert e.value.status == b.SR_ERR_WORKSPACE
    h = _handle(b, cfg, n)
    try:
        w = (b.sr_block_weights * 6)()
        for i in range(6):
            for f in b.WEIGHT_FIELDS:
                setattr(w[i], f, 0x200000)
        X, O = 0x400000, 0x800000
        for r in (0.0, -1.0, 1.5, float("nan")):
            with pytest.raises(b.SRError) as e:
                b.sr_forward(h, X, w, r, 0, O, None, None)
            assert e.value.status == b.SR_ERR_INVALID_ARG
        # K = floor(512 * 0.001) = 0
        with pytest.raises(b.SRError) as e:
            b.sr_forward(h, X, w, 0.001, 0, O, None, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
        # beyond the workspace's routed capacity (sized for r <= 0.25)
        with pytest.raises(b.SRError) as e:
            b.sr_forward(h, X, w, 0.5, 0, O, None, None)
        assert e.value.status == b.SR_ERR_WORKSPACE
        # partial overlap of x and out
        with pytest.raises(b.SRError) as e:
            b.sr_forward(h, X, w, 0.25, 0, X + 1024, None, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
        # a NULL weight pointer
        w[3].w1 = None
        with pytest.raises(b.SRError) as e:
            b.sr_forward(h, X, w, 0.25, 0, O, None, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
        with pytest.raises(b.SRError) as e:
            b.sr_select(h, None, 0.0, 0, 0x300000, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
    finally:
        b.sr_destroy(h)


def test_status_strings(L):
    from paper_2607_02829_gb300 import binding as b
    for s in range(6):
        assert L.sr_status_string(s).decode().startswith("SR_")


def test_routed_only_workspace_is_smaller_and_rejects_the_dense_path(L):
    from paper_2607_02829_gb300 import binding as b
    cfg = b.make_config(2, 512, 256, 4, 0, 2, 0, dtype="f32")
    small = b.sr_workspace_bytes(cfg, 0.25)
    full = b.sr_workspace_bytes(cfg, 1.0)
    assert 0 < small < full
    h = _handle(b, cfg, small)
    try:
        w = (b.sr_block_weights * 2)()
        for i in range(2):
            for f in b.WEIGHT_FIELDS:
                setattr(w[i], f, 0x200000)
        with pytest.raises(b.SRError) as e:
            b.sr_forward(h, 0x400000, w, 1.0, 0, 0x800000, None, None)
        assert e.value.status == b.SR_ERR_WORKSPACE
    finally:
        b.sr_destroy(h)


def test_ensemble_workspace_and_argument_errors(L):
    from paper_2607_02829_gb300 import binding as b
    cfg = b.make_config(2, 512, 256, 4, 1, 2, 1, dtype="f32")
    ens = b.sr_ensemble_workspace_bytes(cfg, 2, 0.25)
    # the batch of M * B samples: at least its fp32 stream
    assert ens >= 2 * 2 * 512 * 256 * 4
    assert b.sr_ensemble_workspace_bytes(cfg, 3, 0.25) > ens
    bad = b.make_config(2, 512, 250, 4, 1, 2, 1, dtype="f32")
    assert b.sr_ensemble_workspace_bytes(bad, 2, 0.25) == 0
    assert b.sr_ensemble_workspace_bytes(cfg, 0, 0.25) == 0
    assert b.sr_ensemble_workspace_bytes(cfg, 2, 1.5) == 0
    big = b.make_config(64, 16200, 1024, 16, 4, 16, 4, dtype="bf16")
    assert b.sr_ensemble_workspace_bytes(big, 8, 0.25) == 0      # 2^31-element limit
    h = _handle(b, cfg, b.sr_workspace_bytes(cfg, 0.25))
    try:
        w = (b.sr_block_weights * 4)()
        for i in range(4):
            for f in b.WEIGHT_FIELDS:
                setattr(w[i], f, 0x200000)
        X, O, E = 0x400000, 0x800000, 0x1000000
        with pytest.raises(b.SRError) as e:          # no seeds
            b.sr_forward_ensemble(h, X, w, 0.25, [], E, ens, O, None, None, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
        with pytest.raises(b.SRError) as e:          # no ensemble workspace
            b.sr_forward_ensemble(h, X, w, 0.25, [1, 2], 0, ens, O, None, None, None)
        assert e.value.status == b.SR_ERR_WORKSPACE
        with pytest.raises(b.SRError) as e:          # short ensemble workspace
            b.sr_forward_ensemble(h, X, w, 0.25, [1, 2], E, ens - 256, O, None, None, None)
        assert e.value.status == b.SR_ERR_WORKSPACE
        with pytest.raises(b.SRError) as e:          # misaligned ensemble workspace
            b.sr_forward_ensemble(h, X, w, 0.25, [1, 2], E + 16, ens, O, None, None, None)
        assert e.value.status == b.SR_ERR_WORKSPACE
        with pytest.raises(b.SRError) as e:          # keep ratio out of range
            b.sr_forward_ensemble(h, X, w, 1.5, [1, 2], E, ens, O, None, None, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
        with pytest.raises(b.SRError) as e:          # members_out overlapping out
            b.sr_forward_ensemble(h, X, w, 0.25, [1, 2], E, ens, O, O + 4096, None, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
    finally:
        b.sr_destroy(h)


def test_cross_attention_argument_errors(L):
    from paper_2607_02829_gb300 import binding as b
    Q, KV, O = 0x400000, 0x800000, 0x2000000
    cases = [
        (dict(q=0), b.SR_ERR_INVALID_ARG), (dict(out=O + 8), b.SR_ERR_INVALID_ARG),
        (dict(B=0), b.SR_ERR_INVALID_ARG), (dict(Tq=0), b.SR_ERR_INVALID_ARG),
        (dict(Tkv=0), b.SR_ERR_INVALID_ARG), (dict(heads=0), b.SR_ERR_UNSUPPORTED),
        (dict(heads=33), b.SR_ERR_UNSUPPORTED), (dict(out=Q + 64), b.SR_ERR_INVALID_ARG),
        (dict(Tkv=1 << 22), b.SR_ERR_UNSUPPORTED),
    ]
    for kw, status in cases:
        a = dict(q=Q, kv=KV, B=2, Tq=100, Tkv=300, heads=2, out=O, fault=None, stream=None)
        a.update(kw)
        with pytest.raises(b.SRError) as e:
            b.sr_cross_attention(a["q"], a["kv"], a["B"], a["Tq"], a["Tkv"], a["heads"], a["out"],
                                 a["fault"], a["stream"])
        assert e.value.status == status, kw


def test_forward_host_rejects_arguments_before_any_copy(L):
    # every check runs on the host before the first copy is enqueued, so fake
    # addresses are never touched
    from paper_2607_02829_gb300 import binding as b
    cfg = b.make_config(2, 512, 256, 4, 1, 2, 1, dtype="bf16")
    h = _handle(b, cfg, b.sr_workspace_bytes(cfg, 0.25))
    try:
        w = (b.sr_block_weights * 4)()
        for i in range(4):
            for f in b.WEIGHT_FIELDS:
                setattr(w[i], f, 0x200000)
        XH, D, OH = 0x7000000, 0x400000, 0x8000000
        for args, status in [
            ((None, w, 0.25, D, OH), b.SR_ERR_INVALID_ARG),       # no host input
            ((XH, w, 0.25, None, OH), b.SR_ERR_INVALID_ARG),      # no device buffer
            ((XH, w, 0.25, D, None), b.SR_ERR_INVALID_ARG),       # no host output
            ((XH, w, 1.5, D, OH), b.SR_ERR_INVALID_ARG),          # keep ratio out of range
            ((XH, w, 0.5, D, OH), b.SR_ERR_WORKSPACE),            # beyond the routed capacity
            ((XH, w, 0.25, D + 8, OH), b.SR_ERR_INVALID_ARG),     # misaligned device buffer
        ]:
            x_host, ww, r, dev, out_host = args
            with pytest.raises(b.SRError) as e:
                b.sr_forward_host(h, x_host, ww, r, 0, dev, out_host, None, None)
            assert e.value.status == status, args
        w[2].w2 = None                                         # a NULL weight pointer
        with pytest.raises(b.SRError) as e:
            b.sr_forward_host(h, XH, w, 0.25, 0, D, OH, None, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
    finally:
        b.sr_destroy(h)


@pytest.mark.parametrize("lang", ["c", "c++"])
def test_header_compiles_as_plain_c_and_cpp(lang):
    # the boundary is a C header: it must stand alone in a C and a C++ unit
    import os
    import shutil
    import subprocess
    cc = shutil.which("gcc" if lang == "c" else "g++")
    if cc is None:
        pytest.skip("no host compiler")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([cc, "-fsyntax-only", "-Wall", "-Werror", "-x", lang,
                        os.path.join(root, "include", "sparse_reslim.h")],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_trace_fault_and_error_message_arguments(L):
    from paper_2607_02829_gb300 import binding as b
    assert L.sr_trace_enable(None, 1) == b.SR_ERR_INVALID_ARG
    assert L.sr_trace_read(None, None, 0) == b.SR_ERR_INVALID_ARG
    f = ctypes.c_uint32(7)
    assert L.sr_device_fault(None, ctypes.byref(f), 0, None) == b.SR_ERR_INVALID_ARG
    assert b"NULL" in L.sr_last_error_message()          # the message of that rejection
    cfg = b.make_config(2, 512, 256, 4, 1, 2, 1, dtype="bf16")
    h = _handle(b, cfg, b.sr_workspace_bytes(cfg, 0.25))
    try:
        # nothing traced yet: the read needs no device work and gives zeros
        assert L.sr_trace_enable(h, 1) == b.SR_OK
        buf = (b.sr_trace_entry * 10)()
        assert L.sr_trace_read(h, buf, 1) == b.SR_OK
        assert all(e.launches == 0 and e.ms == 0.0 and e.flops == 0.0 for e in buf)
        assert L.sr_trace_enable(h, 0) == b.SR_OK
        assert L.sr_device_fault(h, None, 0, None) == b.SR_ERR_INVALID_ARG
    finally:
        b.sr_destroy(h)


def test_static_topk_selector_rejects_arguments_before_any_launch(L):
    # x, B, L, D, dtype, keep_ratio, idx -> status; fake addresses are never touched
    from paper_2607_02829_gb300 import binding as b
    X, I = 0x400000, 0x800000
    good = dict(x=X, B=2, L=512, D=256, dtype=b.SR_BF16, r=0.25, idx=I)
    cases = [
        (dict(x=None), b.SR_ERR_INVALID_ARG), (dict(x=X + 8), b.SR_ERR_INVALID_ARG),
        (dict(idx=None), b.SR_ERR_INVALID_ARG), (dict(idx=I + 2), b.SR_ERR_INVALID_ARG),
        (dict(dtype=7), b.SR_ERR_INVALID_ARG), (dict(B=0), b.SR_ERR_INVALID_ARG),
        (dict(L=0), b.SR_ERR_INVALID_ARG), (dict(D=100), b.SR_ERR_UNSUPPORTED),
        (dict(D=4096), b.SR_ERR_UNSUPPORTED), (dict(D=2048, dtype=b.SR_F32), b.SR_ERR_UNSUPPORTED),
        (dict(B=65, L=16200), b.SR_ERR_UNSUPPORTED),        # B * L above the 1,048,576 scores
        (dict(r=0.0), b.SR_ERR_INVALID_ARG), (dict(r=1.5), b.SR_ERR_INVALID_ARG),
        (dict(r=float("nan")), b.SR_ERR_INVALID_ARG),
        (dict(L=10, r=0.05), b.SR_ERR_INVALID_ARG),         # K = floor(0.5) = 0
    ]
    for kw, status in cases:
        a = dict(good, **kw)
        k = ctypes.c_int32(-1)
        got = L.sr_select_topk_l2_static(a["x"], a["B"], a["L"], a["D"], a["dtype"], a["r"],
                                         a["idx"], ctypes.byref(k), None)
        assert got == status, (kw, got)
        assert k.value == -1                                # K_out untouched on a rejection


def test_injected_failure_stops_the_forward_at_its_first_call(L):
    # the host-side injection hook fails the first CUDA call sr_forward would
    # make: it returns SR_ERR_CUDA with a message naming that step, and attempts
    # no further call (no GPU is touched: every pointer here is a fake address)
    from paper_2607_02829_gb300 import binding as b
    cfg = b.make_config(2, 512, 256, 4, 2, 2, 2, dtype="f32")
    h = _handle(b, cfg, b.sr_workspace_bytes(cfg, 0.25))
    try:
        w = (b.sr_block_weights * 6)()
        for i in range(6):
            for f in b.WEIGHT_FIELDS:
                setattr(w[i], f, 0x200000)
        b.sr_debug_fail_enqueue(0)
        with pytest.raises(b.SRError) as e:
            b.sr_forward(h, 0x400000, w, 0.25, 0, 0x800000, None, None)
        assert e.value.status == b.SR_ERR_CUDA
        assert "injected" in str(e.value) and "clear fault word" in str(e.value)
        assert b.sr_debug_enqueue_count() == 1
        # an invalid argument is still rejected before any CUDA call is attempted
        b.sr_debug_fail_enqueue(0)
        with pytest.raises(b.SRError) as e:
            b.sr_forward(h, 0x400000, w, 0.0, 0, 0x800000, None, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
        assert b.sr_debug_enqueue_count() == 0
    finally:
        b.sr_debug_fail_enqueue(-1)
        b.sr_destroy(h)


def test_selftest_wait_timeout_rejects_bad_arguments(L):
    from paper_2607_02829_gb300 import binding as b
    for fault, limit, waited in [(0, 1000, 0x1000), (0x1001, 1000, 0x1000), (0x1000, 0, 0x1000),
                                 (0x1000, 2000000, 0x1000), (0x1000, 1000, 0), (0x1000, 1000, 0x1004)]:
        with pytest.raises(b.SRError) as e:
            b.sr_selftest_wait_timeout(fault, limit, waited, None)
        assert e.value.status == b.SR_ERR_INVALID_ARG
