"""Host-side logic that needs no GPU: the synthetic workloads against the
configurations they stand for, the input generator's documented structure, and
the measurement bookkeeping of bench.py (roofline, the ncu traffic row tied to
the kernel sources it was captured on, gather/scatter figures)."""
import os
import shutil

import numpy as np
import pytest

import bench
from oracle import reslim as o
from paper_2607_02829_gb300 import synth


# ---------------------------------------------------------------- workloads
# (B, L, D, heads, split, keep ratio, K, storage) of the five configurations
CONFIGS = {
    "c1_5p625deg_f32": (2, 512, 256, 4, (2, 2, 2), 0.25, 128, "f32"),
    "c2_5p625deg_bf16": (32, 512, 1024, 16, (2, 4, 2), 0.25, 128, "bf16"),
    "c3_1p40625deg_bf16": (8, 2048, 1024, 16, (4, 16, 4), 0.25, 512, "bf16"),
    "c4_0p25deg_bf16": (1, 16200, 1024, 16, (4, 16, 4), 0.25, 4050, "bf16"),
}


@pytest.mark.parametrize("name", sorted(CONFIGS))
def test_workloads_match_their_configurations(name):
    B, L, D, H, split, r, K, dt = CONFIGS[name]
    wl = synth.WORKLOADS[name]
    assert (wl.B, wl.L, wl.D, wl.heads, (wl.n1, wl.n2, wl.n3), wl.keep_ratio, wl.dtype) == \
        (B, L, D, H, split, r, dt)
    assert o.keep_count(wl.L, wl.keep_ratio) == K
    assert wl.mlp_hidden == 4 * D and wl.D == 64 * wl.heads
    assert wl.L == (wl.grid_h // wl.patch) * wl.grid_wp


def test_sweep_covers_ratios_and_selectors():
    sw = synth.sweep_workloads()
    got = {(w.selector, w.keep_ratio): o.keep_count(w.L, w.keep_ratio) for w in sw}
    for sel in ("random", "topk_l2", "laplacian"):
        assert [got[(sel, r)] for r in (1.0, 0.5, 0.25, 0.125)] == [2048, 1024, 512, 256]
    base = synth.WORKLOADS["c3_1p40625deg_bf16"]
    for w in sw:
        assert (w.B, w.L, w.D, w.n1, w.n2, w.n3) == (base.B, base.L, base.D, base.n1, base.n2, base.n3)


# ---------------------------------------------------------------- inputs
def test_smooth_fields_are_seeded_and_cropped():
    a = synth.smooth_fields(2, 3, 9, 16, seed=11)
    b = synth.smooth_fields(2, 3, 9, 16, seed=11)
    c = synth.smooth_fields(2, 3, 9, 16, seed=12)
    assert np.array_equal(a, b) and not np.array_equal(a, c)
    # crop_last_row draws on H + 1 latitudes (the last dropped): the kept rows
    # sit at the latitudes of the longer grid
    d = synth.smooth_fields(1, 1, 4, 8, seed=5, crop_last_row=True)
    assert d.shape == (1, 1, 4, 8)
    # signal amplitude: at most 8 terms of amplitude <= 1.5, plus N(0, 0.1) noise
    assert np.abs(a).max() < 8 * 1.5 + 1.0


def test_longitude_grid_spans_one_turn():
    # lam_i = 2 pi i / W: the same fields drawn at twice the resolution carry the
    # coarse grid's signal on their even columns (with integer wavenumbers k the
    # fields are then periodic in longitude).  The sinusoid parameters are drawn
    # before the noise, so both grids share them; column means over the
    # latitudes average the N(0, 0.1) noise down to about 0.0125.
    H, W = 64, 32
    f = synth.smooth_fields(1, 1, H, W, seed=3)[0, 0]
    g = synth.smooth_fields(1, 1, H, 2 * W, seed=3)[0, 0]
    assert np.abs(f.mean(axis=0) - g[:, ::2].mean(axis=0)).max() < 0.1
    # while a grid shifted by half a coarse column would not match
    assert np.abs(f.mean(axis=0) - g[:, 1::2].mean(axis=0)).max() > 0.1


def test_patchify_order_and_position_embedding():
    B, C, H, W, p = 1, 2, 4, 6, 2
    f = np.arange(B * C * H * W, dtype=np.float64).reshape(B, C, H, W)
    t = synth.patchify(f, p)
    assert t.shape == (B, (H // p) * (W // p), C * p * p)
    # token 1 is lat-patch 0, lon-patch 1; features ordered (c, dy, dx)
    for c in range(C):
        for dy in range(p):
            for dx in range(p):
                assert t[0, 1, c * p * p + dy * p + dx] == f[0, c, dy, p + dx]
    hp, wp, D = 3, 5, 16
    e = synth.sincos_pos_embed_2d(hp, wp, D)
    assert e.shape == (hp * wp, D)
    grid = e.reshape(hp, wp, D)
    # the first D/2 channels encode the latitude index, the rest the longitude
    assert np.allclose(grid[:, :, :D // 2], grid[:, :1, :D // 2])
    assert np.allclose(grid[:, :, D // 2:], grid[:1, :, D // 2:])


# ---------------------------------------------------------------- bench bookkeeping
PEAKS = {"hbm_gbs": 6784.5, "bf16_tflops": 1891.0, "bf16_tflops_sustained": 1708.9,
         "sm_max_mhz": 2070.0, "source": "measured"}


def _trace():
    return {
        "attention": {"launches": 4, "ms": 2.0, "flops": 2e12, "bytes": 4e8},
        "gemm_qkv": {"launches": 4, "ms": 0.5, "flops": 4e11, "bytes": 1e8},
        "layernorm": {"launches": 8, "ms": 0.2, "flops": 0.0, "bytes": 8e8},
        "copy": {"launches": 2, "ms": 5.0, "flops": 0.0, "bytes": 1e9},
    }


def test_roofline_takes_the_dominant_kernel_against_the_burst_peak(monkeypatch):
    monkeypatch.setattr(bench, "measured_traffic", lambda kind, wl: (None, "none"))
    rf, detail = bench.roofline(_trace(), PEAKS, steps=2, workload="w")
    # "copy" (widen / narrow) is left out of the roofline even though it is longest
    assert rf["kernel"] == "attention" and rf["bound"] == "tensor"
    achieved = (2e12 / 4) / (0.5e-3) / 1e12          # flops per launch / launch time
    assert rf["achieved"] == pytest.approx(achieved)
    assert rf["peak"] == PEAKS["bf16_tflops"]
    assert rf["frac"] == pytest.approx(achieved / 1891.0)
    assert rf["frac_of_sustained"] == pytest.approx(achieved / 1708.9)
    assert rf["algorithmic_bytes_per_launch"] == pytest.approx(1e8)
    assert detail["attention"]["launches_per_step"] == 2
    assert sum(d["share"] for d in detail.values()) == pytest.approx(1.0)


def test_roofline_of_a_bandwidth_bound_kernel(monkeypatch):
    monkeypatch.setattr(bench, "measured_traffic", lambda kind, wl: (None, "none"))
    tr = {"layernorm": {"launches": 2, "ms": 0.02, "flops": 0.0, "bytes": 2e8}}
    rf, _ = bench.roofline(tr, PEAKS, steps=1, workload="w")
    assert rf["bound"] == "hbm" and rf["unit"] == "GB/s"
    assert rf["achieved"] == pytest.approx(1e8 / 1e-5 / 1e9)
    assert rf["frac"] == pytest.approx(rf["achieved"] / PEAKS["hbm_gbs"])


def test_fp32_roofline_uses_the_ffma_peak(monkeypatch):
    monkeypatch.setattr(bench, "measured_traffic", lambda kind, wl: (None, "none"))
    tr = {"attention": {"launches": 1, "ms": 1.0, "flops": 1e10, "bytes": 1.0}}
    rf, _ = bench.roofline(tr, PEAKS, steps=1, workload="w", fp32_alu=True)
    assert rf["bound"] == "alu"
    assert rf["peak"] == pytest.approx(152 * 128 * 2 * 2070e6 / 1e12)


def test_traffic_row_counts_only_for_the_sources_it_was_captured_on(tmp_path, monkeypatch):
    digest = bench.source_digest("attention")
    table = tmp_path / "traffic.txt"
    table.write_text("| kind | workload | source digest | MB per launch | capture |\n"
                     f"| attention | wl_a | {digest} | 54.74 | note |\n"
                     "| attention | wl_b | 000000000000 | 60.00 | note |\n")
    monkeypatch.setattr(bench, "TRAFFIC_TABLE", str(table))
    val, note = bench.measured_traffic("attention", "wl_a")
    assert val == pytest.approx(54.74e6) and digest in note
    val, note = bench.measured_traffic("attention", "wl_b")
    assert val is None and "000000000000" in note and digest in note
    val, note = bench.measured_traffic("attention", "wl_c")
    assert val is None
    val, note = bench.measured_traffic("layernorm", "wl_a")
    assert val is None


def test_source_digest_follows_every_source_file(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2607_02829_gb300" / "csrc"
    csrc.mkdir(parents=True)
    real = os.path.join(bench.ROOT, "paper_2607_02829_gb300", "csrc")
    for f in bench.KERNEL_SOURCES["attention"]:
        shutil.copy(os.path.join(real, f), csrc / f)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    before = bench.source_digest("attention")
    assert before == bench.source_digest("attention")
    for f in bench.KERNEL_SOURCES["attention"]:
        p = csrc / f
        text = p.read_text()
        p.write_text(text + "\n")
        assert bench.source_digest("attention") != before, f
        p.write_text(text)
    assert bench.source_digest("attention") == before


def test_gather_and_scatter_figures():
    wl = synth.WORKLOADS["c4_0p25deg_bf16"]
    K = o.keep_count(wl.L, wl.keep_ratio)
    gbytes = 2 * 41.5e6
    trace = {"gather": {"launches": 2, "ms": 0.024, "bytes": gbytes}}
    seg = {"trace": {"gemm_fc2_scatter": {"launches": 2, "ms": 0.090},
                     "gemm_fc2": {"launches": 30, "ms": 1.050}}}
    out = bench.gather_scatter(wl, K, trace, seg, PEAKS)
    g = out["gather"]
    assert g["bytes_per_launch"] == pytest.approx(41.5e6)
    assert g["us_per_launch"] == pytest.approx(12.0)
    assert g["gbs"] == pytest.approx(gbytes / 0.024e-3 / 1e9)
    s = out["scatter"]
    nbytes = 8.0 * wl.B * K * wl.D + 4.0 * wl.B * K       # h0 / x0 read + x' written, fp32, + index
    assert s["bytes_per_launch"] == pytest.approx(nbytes)
    extra_s = (0.045 - 0.035) * 1e-3
    assert s["gbs"] == pytest.approx(nbytes / extra_s / 1e9)
    assert s["frac_of_hbm"] == pytest.approx(s["gbs"] / PEAKS["hbm_gbs"])
    # a scatter FC2 no slower than the plain one gives no bandwidth figure
    seg["trace"]["gemm_fc2_scatter"]["ms"] = 0.060
    out = bench.gather_scatter(wl, K, trace, seg, PEAKS)
    assert "gbs" not in out["scatter"] and "note" in out["scatter"]
