"""Seeded synthetic inputs shared by the CUDA path's tests/bench and by the oracle.

This module holds none of the routed encoder's arithmetic.  It produces:

* ERA5-shaped smooth lat-lon fields (ERA5 itself is not available; these stand
  in for it: a sum of 8 low-frequency sinusoids per channel plus N(0, 0.1^2)
  noise, on the 5.625 / 1.40625 / 0.25 degree grids),
* the token sequence x[B, L, D] that enters the first encoder block (linear
  patch embedding of the patchified fields plus a 2-D sin-cos position
  embedding; this replaces the paper's per-variable tokenizer, Sec. 3.1 Eq. 1,
  which needs learned weights),
* the per-block weights of the N pre-LN ViT blocks (random init),
* the named workload presets (5.625 deg / 1.40625 deg / 0.25 deg grids and the
  keep-ratio sweep).

All random numbers come from numpy's PCG64 seeded with documented integers, so
the oracle and the GPU path consume bit-identical inputs.  Storage rounding to
bf16 is done once here (round-to-nearest-even through torch's cast) so that
both sides see the same stored values.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List

import numpy as np

WEIGHT_NAMES = ("ln1_g", "ln1_b", "wqkv", "bqkv", "wo", "bo",
                "ln2_g", "ln2_b", "w1", "b1", "w2", "b2")


@dataclasses.dataclass(frozen=True)
class Workload:
    """One encoder workload: grid, tokenisation and the block stack."""
    name: str
    B: int
    grid_h: int          # latitude rows kept (after cropping)
    grid_w: int          # longitude columns
    channels: int
    patch: int
    D: int
    heads: int
    n1: int
    n2: int
    n3: int
    keep_ratio: float
    dtype: str           # "f32" or "bf16"
    selector: str = "random"   # "random", "topk_l2" or "laplacian"
    crop_last_row: bool = False  # generate grid_h + 1 latitudes, drop the last
    seed_index: int = 0

    @property
    def L(self) -> int:
        return (self.grid_h // self.patch) * (self.grid_w // self.patch)

    @property
    def grid_wp(self) -> int:
        """Tokens per latitude row of the patch grid."""
        return self.grid_w // self.patch

    @property
    def N(self) -> int:
        return self.n1 + self.n2 + self.n3

    @property
    def mlp_hidden(self) -> int:
        return 4 * self.D

    @property
    def input_seed(self) -> int:
        return 1000 + self.seed_index

    @property
    def weight_seed(self) -> int:
        return 2000 + self.seed_index

    @property
    def select_seed(self) -> int:
        return 3000 + self.seed_index

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads: 5.625 deg fp32 (small), 5.625 deg bf16 batch 32,
# 1.40625 deg bf16 batch 8, 0.25 deg bf16 batch 1, and the keep-ratio x selector
# sweep on the 1.40625 deg model.
WORKLOADS: Dict[str, Workload] = {
    "c1_5p625deg_f32": Workload("c1_5p625deg_f32", B=2, grid_h=32, grid_w=64, channels=48,
                                patch=2, D=256, heads=4, n1=2, n2=2, n3=2,
                                keep_ratio=0.25, dtype="f32", seed_index=1),
    "c2_5p625deg_bf16": Workload("c2_5p625deg_bf16", B=32, grid_h=32, grid_w=64, channels=48,
                                 patch=2, D=1024, heads=16, n1=2, n2=4, n3=2,
                                 keep_ratio=0.25, dtype="bf16", seed_index=2),
    "c3_1p40625deg_bf16": Workload("c3_1p40625deg_bf16", B=8, grid_h=128, grid_w=256,
                                   channels=48, patch=4, D=1024, heads=16, n1=4, n2=16,
                                   n3=4, keep_ratio=0.25, dtype="bf16", seed_index=3),
    "c4_0p25deg_bf16": Workload("c4_0p25deg_bf16", B=1, grid_h=720, grid_w=1440, channels=69,
                                patch=8, D=1024, heads=16, n1=4, n2=16, n3=4,
                                keep_ratio=0.25, dtype="bf16", crop_last_row=True,
                                seed_index=4),
}

SWEEP_RATIOS = (1.0, 0.5, 0.25, 0.125)
SWEEP_SELECTORS = ("random", "topk_l2", "laplacian")


def sweep_workloads() -> List[Workload]:
    """Keep-ratio x selector sweep on the 1.40625 deg / L=2048 / 24-block model."""
    base = WORKLOADS["c3_1p40625deg_bf16"]
    out = []
    for sel in SWEEP_SELECTORS:
        for r in SWEEP_RATIOS:
            out.append(base.with_(name=f"c5_{sel}_r{r}", keep_ratio=r, selector=sel,
                                  seed_index=5))
    return out


# --------------------------------------------------------------------------
# fields and tokens
# --------------------------------------------------------------------------

def smooth_fields(B: int, C: int, H: int, W: int, seed: int,
                  crop_last_row: bool = False) -> np.ndarray:
    """[B, C, H, W] float64 smooth fields on a regular lat-lon grid.

    f_c(phi, lam) = sum_{j=1..8} a_j sin(k_j lam + alpha_j) cos(m_j phi + beta_j) + eps,
    lam in [0, 2 pi) on W points, phi from +90 to -90 degrees on H points
    (H + 1 points with the last dropped when crop_last_row), k_j in {1..4},
    m_j in {0..3}, a_j ~ U(0.5, 1.5), alpha_j, beta_j ~ U(0, 2 pi), eps ~ N(0, 0.1^2).
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    Hg = H + 1 if crop_last_row else H
    lam = np.arange(W, dtype=np.float64) * (2.0 * np.pi / W)
    phi = np.deg2rad(np.linspace(90.0, -90.0, Hg, dtype=np.float64))[:H]
    out = np.empty((B, C, H, W), dtype=np.float64)
    for b in range(B):
        for c in range(C):
            k = rng.integers(1, 5, size=8)
            m = rng.integers(0, 4, size=8)
            a = rng.uniform(0.5, 1.5, size=8)
            al = rng.uniform(0.0, 2.0 * np.pi, size=8)
            be = rng.uniform(0.0, 2.0 * np.pi, size=8)
            lat_part = np.cos(np.outer(phi, m) + be) * a            # [H, 8]
            lon_part = np.sin(np.outer(k, lam) + al[:, None])        # [8, W]
            out[b, c] = lat_part @ lon_part
            out[b, c] += rng.normal(0.0, 0.1, size=(H, W))
    return out


def patchify(fields: np.ndarray, p: int) -> np.ndarray:
    """[B, C, H, W] -> [B, L, C*p*p]; tokens row-major over (lat-patch, lon-patch),
    features ordered (c, dy, dx)."""
    B, C, H, W = fields.shape
    hp, wp = H // p, W // p
    t = fields[:, :, :hp * p, :wp * p].reshape(B, C, hp, p, wp, p)
    t = t.transpose(0, 2, 4, 1, 3, 5)                               # B, hp, wp, C, p, p
    return t.reshape(B, hp * wp, C * p * p)


def sincos_pos_embed_2d(hp: int, wp: int, D: int) -> np.ndarray:
    """MAE-style 2-D sin-cos position embedding [hp*wp, D] (D/2 channels encode
    the lat-patch index, D/2 the lon-patch index; base 10000)."""
    assert D % 4 == 0
    def one_axis(pos, dim):
        omega = 1.0 / (10000.0 ** (np.arange(dim // 2, dtype=np.float64) / (dim / 2.0)))
        ang = np.outer(pos.astype(np.float64), omega)
        return np.concatenate([np.sin(ang), np.cos(ang)], axis=1)
    gy, gx = np.meshgrid(np.arange(hp), np.arange(wp), indexing="ij")
    emb_y = one_axis(gy.reshape(-1), D // 2)
    emb_x = one_axis(gx.reshape(-1), D // 2)
    return np.concatenate([emb_y, emb_x], axis=1)


def make_tokens(wl: Workload) -> np.ndarray:
    """x [B, L, D] float64: patch-embedded smooth fields + position embedding."""
    f = smooth_fields(wl.B, wl.channels, wl.grid_h, wl.grid_w, wl.input_seed,
                      crop_last_row=wl.crop_last_row)
    tok = patchify(f, wl.patch)
    del f
    rng = np.random.Generator(np.random.PCG64(wl.input_seed + 500_000))
    w_pe = rng.normal(0.0, 0.02, size=(wl.D, tok.shape[-1]))
    x = tok @ w_pe.T
    hp, wp = wl.grid_h // wl.patch, wl.grid_w // wl.patch
    x += sincos_pos_embed_2d(hp, wp, wl.D)[None]
    return x


def make_block_weights(D: int, hidden: int, seed: int) -> Dict[str, np.ndarray]:
    """One block's weights in nn.Linear layout ([out, in]); W, biases ~ N(0, 0.02^2),
    LayerNorm gamma = 1 + N(0, 0.02^2), beta ~ N(0, 0.02^2)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    s = 0.02
    return {
        "ln1_g": 1.0 + rng.normal(0.0, s, size=D),
        "ln1_b": rng.normal(0.0, s, size=D),
        "wqkv": rng.normal(0.0, s, size=(3 * D, D)),
        "bqkv": rng.normal(0.0, s, size=3 * D),
        "wo": rng.normal(0.0, s, size=(D, D)),
        "bo": rng.normal(0.0, s, size=D),
        "ln2_g": 1.0 + rng.normal(0.0, s, size=D),
        "ln2_b": rng.normal(0.0, s, size=D),
        "w1": rng.normal(0.0, s, size=(hidden, D)),
        "b1": rng.normal(0.0, s, size=hidden),
        "w2": rng.normal(0.0, s, size=(D, hidden)),
        "b2": rng.normal(0.0, s, size=D),
    }


def block_seed(weight_seed: int, block: int) -> int:
    return weight_seed * 1000 + block


def make_weights(wl: Workload) -> List[Dict[str, np.ndarray]]:
    return [make_block_weights(wl.D, wl.mlp_hidden, block_seed(wl.weight_seed, i))
            for i in range(wl.N)]


# --------------------------------------------------------------------------
# storage rounding (identical values for both sides)
# --------------------------------------------------------------------------

def torch_dtype(dtype: str):
    import torch
    return {"f32": torch.float32, "bf16": torch.bfloat16}[dtype]


def to_storage(a: np.ndarray, dtype: str):
    """float64 array -> CPU torch tensor in the storage dtype (RNE rounding)."""
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(torch_dtype(dtype))


def stored_as_f64(t) -> np.ndarray:
    """The exact stored values of a torch tensor, widened to float64."""
    import torch
    return t.detach().to("cpu").to(torch.float64).numpy()


def make_inputs(wl: Workload):
    """(x, weights) as CPU torch tensors in the workload's storage dtype."""
    x = to_storage(make_tokens(wl), wl.dtype)
    ws = [{k: to_storage(v, wl.dtype) for k, v in blk.items()} for blk in make_weights(wl)]
    return x, ws
