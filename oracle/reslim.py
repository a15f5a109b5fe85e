"""fp64 CPU oracle of the Sparse-Reslim routed encoder forward.

TEST INFRASTRUCTURE.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this module.  The
CUDA library never calls it, and it imports nothing from the CUDA path: it is
written from the paper alone, in float64, with numpy's matmul as the only
library primitive.

What it computes (arxiv 2607.02829):

* K = floor(L * r)                                   -- Sec. 3.2, Alg. 1
* the three-stage block partition (n1 dense, n2 sparse, n3 dense) -- Sec. 3.2 Eq. 7
* token selection, uniform without replacement, sorted ascending  -- Sec. 3.2
  (the paper draws it with torch.randperm, which cannot be reproduced
  independently; this oracle defines it through SplitMix64 keys, see
  ``random_keys``), and the activation-norm selector of App. B.2 Table 11
  (top-K by per-token L2 norm of the last dense-early block's output) and the
  gradient (Laplacian) selector of the same table (top-K by the squared norm
  of the 5-point Laplacian on the patch grid, see ``token_laplacian_scores``)
* gather h0 = x[:, I, :] and the sparse middle blocks on h      -- Sec. 3.2 Eq. 8
* the residual delta and scatter x' = x0 + Scatter(h - h0, I)   -- Sec. 3.2 Eq. 9
* the pre-LN block h <- h + Attn(LN h); h <- h + MLP(LN h)       -- Sec. 3.3 Eq. 11
  with LayerNorm (eps 1e-5, affine), multi-head softmax attention with
  scale 1/sqrt(head_dim) and no mask, exact-erf GELU, MLP ratio 4
  (App. A, Table "architecture specification")
* r = 1 is the plain dense stack                                -- Sec. 3.4, paragraph "Architecture-agnostic design"

Parity pins: every function here is pinned by the ``-m "not gpu"`` tests
(published SplitMix64 outputs, the K values the paper prints, brute-force
selection, PyTorch's own LayerNorm/GELU/TransformerEncoderLayer in float64,
closed-form special cases and the routing invariants).  Whole-model outputs
beyond those pins are "parity unpinned": the paper prints no activations.
"""
from __future__ import annotations

import math
from concurrent.futures import ThreadPoolExecutor
from typing import Dict, List, Optional, Sequence

import numpy as np
from scipy.special import erf

U64 = np.uint64
GOLDEN_GAMMA = 0x9E3779B97F4A7C15          # SplitMix64 increment (Steele, Lea, Flood 2014)


# ---------------------------------------------------------------- Sec. 3.2: K
def keep_count(L: int, r: float) -> int:
    """K = floor(L * r), the number of routed tokens (Sec. 3.2; App. A.4 writes
    int(r * L)).  The product is formed in double precision and truncated."""
    if not (0.0 < r <= 1.0):
        raise ValueError("keep ratio must lie in (0, 1]")
    return int(math.floor(float(r) * float(L)))


# ------------------------------------------------- Sec. 3.2: random selection
def splitmix64_mix(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function (Steele, Lea & Flood, OOPSLA 2014; the
    finaliser of Vigna's splitmix64.c), arithmetic mod 2^64."""
    z = np.asarray(z, dtype=U64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> U64(30))) * U64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> U64(27))) * U64(0x94D049BB133111EB)
        z = z ^ (z >> U64(31))
    return z


def random_keys(B: int, L: int, seed: int, shared: bool) -> np.ndarray:
    """[B, L] uint64 keys: key(b, i) = mix(seed + GAMMA * (1 + b' * L + i)),
    b' = b (one index set per sample, as Sec. 3.2 states) or b' = 0 (one set for
    the whole batch, as the listing of App. A.4 draws it).  Consecutive counters
    make key(0, i) the (i+1)-th output of a SplitMix64 generator seeded with
    ``seed``."""
    b = np.zeros(B, dtype=np.int64) if shared else np.arange(B, dtype=np.int64)
    ctr = (1 + b[:, None] * L + np.arange(L, dtype=np.int64)[None, :]).astype(U64)
    with np.errstate(over="ignore"):
        z = U64(seed % (1 << 64)) + U64(GOLDEN_GAMMA) * ctr
    return splitmix64_mix(z)


def select_random(B: int, L: int, K: int, seed: int, shared: bool = False) -> np.ndarray:
    """Index sets I[b] of K tokens drawn uniformly without replacement and sorted
    ascending (Sec. 3.2).  Ranking i.i.d. uniform keys and keeping the K smallest
    gives a uniformly random K-subset; equal keys rank by token index."""
    keys = random_keys(B, L, seed, shared)
    out = np.empty((B, K), dtype=np.int64)
    for b in range(B):
        order = np.lexsort((np.arange(L), keys[b]))   # primary: key, secondary: index
        out[b] = np.sort(order[:K])
    return out


# ------------------------------------------- App. B.2: activation-norm selector
def token_sq_norms(x: np.ndarray) -> np.ndarray:
    """[B, L] squared L2 norm of every token (ranks the same as the norm)."""
    x = np.asarray(x, dtype=np.float64)
    return np.einsum("bld,bld->bl", x, x)


def select_topk_l2(x: np.ndarray, K: int) -> np.ndarray:
    """K tokens with the largest L2 norm per sample (the activation-norm sampler
    of App. B.2 Table 11), ties to the lower token index, sorted ascending."""
    s = token_sq_norms(x)
    B, L = s.shape
    out = np.empty((B, K), dtype=np.int64)
    for b in range(B):
        order = np.lexsort((np.arange(L), -s[b]))     # primary: -score, secondary: index
        out[b] = np.sort(order[:K])
    return out


# ------------------------------------- App. B.2: gradient (Laplacian) selector
def token_laplacian_scores(x: np.ndarray, grid_w: int) -> np.ndarray:
    """[B, L] Laplacian score of every token (App. B.2 Table 11, "Gradient
    (Laplacian)"; the paper gives no formula, so this is a reading of it).

    Tokens lie on the patch grid row-major, grid_w tokens per latitude row and
    L / grid_w rows.  For the token at (i, j), the 5-point Laplacian of its
    feature vector is
        lap(i, j) = x(i-1, j) + x(i+1, j) + x(i, j-1) + x(i, j+1) - 4 x(i, j),
    with longitude periodic (j - 1 and j + 1 wrap around the row) and the first
    and last latitude rows reflected onto themselves (x(-1, j) = x(0, j),
    x(H, j) = x(H-1, j): a zero-flux boundary at the poles).  The score is the
    squared L2 norm over the features, sum_d lap(i, j)_d ** 2."""
    x = np.asarray(x, dtype=np.float64)
    B, L, D = x.shape
    if grid_w < 1 or L % grid_w != 0:
        raise ValueError("L must be a multiple of grid_w")
    H = L // grid_w
    g = x.reshape(B, H, grid_w, D)
    north = np.concatenate([g[:, :1], g[:, :-1]], axis=1)       # x(i-1, j), row 0 reflected
    south = np.concatenate([g[:, 1:], g[:, -1:]], axis=1)       # x(i+1, j), row H-1 reflected
    west = np.roll(g, 1, axis=2)                                 # x(i, j-1), periodic
    east = np.roll(g, -1, axis=2)                                # x(i, j+1), periodic
    lap = north + south + west + east - 4.0 * g
    return np.einsum("bhwd,bhwd->bhw", lap, lap).reshape(B, L)


def select_topk_laplacian(x: np.ndarray, K: int, grid_w: int) -> np.ndarray:
    """K tokens with the largest Laplacian score per sample, ties to the lower
    token index, sorted ascending (the gradient-based sampler of App. B.2)."""
    s = token_laplacian_scores(x, grid_w)
    B, L = s.shape
    out = np.empty((B, K), dtype=np.int64)
    for b in range(B):
        order = np.lexsort((np.arange(L), -s[b]))     # primary: -score, secondary: index
        out[b] = np.sort(order[:K])
    return out


# ------------------------------------------------------ Sec. 3.3: the block
def layer_norm(v: np.ndarray, g: np.ndarray, b: np.ndarray, eps: float) -> np.ndarray:
    """(v - mean) / sqrt(var + eps) * g + b over the last axis, biased variance."""
    mu = v.mean(axis=-1, keepdims=True)
    var = ((v - mu) ** 2).mean(axis=-1, keepdims=True)
    return (v - mu) / np.sqrt(var + eps) * g + b


def gelu(z: np.ndarray) -> np.ndarray:
    """Exact GELU: 0.5 z (1 + erf(z / sqrt 2))."""
    return 0.5 * z * (1.0 + erf(z / math.sqrt(2.0)))


def _attention_one_head(q: np.ndarray, k: np.ndarray, v: np.ndarray,
                        row_chunk: int = 1024) -> np.ndarray:
    """softmax(q k^T / sqrt(dh)) v for one (sample, head); q, k, v: [T, dh].
    Rows are processed in chunks only to bound memory; each row is the plain
    definition (subtract the row max, exponentiate, normalise)."""
    T, dh = q.shape
    scale = 1.0 / math.sqrt(dh)
    out = np.empty_like(q)
    for r0 in range(0, T, row_chunk):
        s = (q[r0:r0 + row_chunk] @ k.T) * scale
        s -= s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[r0:r0 + row_chunk] = p @ v
    return out


def attention(qkv: np.ndarray, heads: int, pool: Optional[ThreadPoolExecutor] = None) -> np.ndarray:
    """Multi-head self-attention core.  qkv: [B, T, 3D] with columns [0, D) = q,
    [D, 2D) = k, [2D, 3D) = v and head h owning columns [h dh, (h+1) dh) of each.
    Attention runs within each sample only.  Returns [B, T, D]."""
    B, T, D3 = qkv.shape
    D = D3 // 3
    dh = D // heads
    out = np.empty((B, T, D), dtype=np.float64)

    def one(bh):
        b, h = divmod(bh, heads)
        c = slice(h * dh, (h + 1) * dh)
        q = qkv[b, :, 0 * D:1 * D][:, c]
        k = qkv[b, :, 1 * D:2 * D][:, c]
        v = qkv[b, :, 2 * D:3 * D][:, c]
        out[b, :, c] = _attention_one_head(np.ascontiguousarray(q), np.ascontiguousarray(k),
                                           np.ascontiguousarray(v))

    if pool is None:
        for bh in range(B * heads):
            one(bh)
    else:
        list(pool.map(one, range(B * heads)))
    return out


def cross_attention(q: np.ndarray, kv: np.ndarray, heads: int,
                    pool: Optional[ThreadPoolExecutor] = None) -> np.ndarray:
    """Asymmetric attention (Sec. 3.4, "Integration with generative
    forecasting"; Alg. 2): queries from one token set, keys and values from
    another, within each sample.  q: [B, Tq, D]; kv: [B, Tkv, 2D] with columns
    [0, D) = k and [D, 2D) = v, head h owning columns [h dh, (h+1) dh) of each.
    Returns [B, Tq, D]."""
    B, Tq, D = q.shape
    dh = D // heads
    out = np.empty((B, Tq, D), dtype=np.float64)

    def one(bh):
        b, h = divmod(bh, heads)
        c = slice(h * dh, (h + 1) * dh)
        out[b, :, c] = _attention_one_head(np.ascontiguousarray(q[b][:, c]),
                                           np.ascontiguousarray(kv[b, :, :D][:, c]),
                                           np.ascontiguousarray(kv[b, :, D:][:, c]))

    if pool is None:
        for bh in range(B * heads):
            one(bh)
    else:
        list(pool.map(one, range(B * heads)))
    return out


def block(x: np.ndarray, w: Dict[str, np.ndarray], heads: int, eps: float = 1e-5,
          pool: Optional[ThreadPoolExecutor] = None) -> np.ndarray:
    """One pre-LN ViT block on x [B, T, D] (Sec. 3.3 Eq. 11):
    x <- x + (Attn(LN1 x) Wo^T + bo);  x <- x + (GELU(LN2 x W1^T + b1) W2^T + b2)."""
    B, T, D = x.shape
    a = layer_norm(x, w["ln1_g"], w["ln1_b"], eps)
    qkv = a.reshape(B * T, D) @ w["wqkv"].T + w["bqkv"]
    att = attention(qkv.reshape(B, T, 3 * D), heads, pool)
    x = x + (att.reshape(B * T, D) @ w["wo"].T + w["bo"]).reshape(B, T, D)
    m = layer_norm(x, w["ln2_g"], w["ln2_b"], eps)
    u = gelu(m.reshape(B * T, D) @ w["w1"].T + w["b1"])
    x = x + (u @ w["w2"].T + w["b2"]).reshape(B, T, D)
    return x


# ----------------------------------------------- Alg. 1: the routed encoder
def as_f64_weights(weights: Sequence[Dict[str, object]]) -> List[Dict[str, np.ndarray]]:
    out = []
    for blk in weights:
        d = {}
        for k, v in blk.items():
            if hasattr(v, "detach"):                     # a torch tensor
                import torch
                v = v.detach().to("cpu").to(torch.float64).numpy()
            d[k] = np.asarray(v, dtype=np.float64)
        out.append(d)
    return out


def forward(x: np.ndarray, weights: Sequence[Dict[str, np.ndarray]], n1: int, n2: int,
            n3: int, heads: int, keep_ratio: float, seed: int = 0,
            selector: str = "random", shared_indices: bool = False, eps: float = 1e-5,
            idx: Optional[np.ndarray] = None, bypass_dense: bool = True,
            threads: int = 0, return_stages: bool = False, grid_w: int = 0):
    """The routed encoder of Alg. 1 (dense early, sparse middle, dense late) in fp64.

    x: [B, L, D]; weights: N = n1 + n2 + n3 dicts of block weights.
    keep_ratio == 1 runs the plain dense stack (Sec. 3.4, "Architecture-agnostic design": r = 1 reverts to the
    dense baseline) unless ``bypass_dense`` is False, in which case the routed
    formulation runs with K = L (used only to check that the two agree).
    ``idx`` overrides the selector (used to re-run with given indices).
    Returns (out, idx) and, with return_stages, also the pre-routing state x0.
    """
    x = np.asarray(x, dtype=np.float64)
    B, L, D = x.shape
    assert len(weights) == n1 + n2 + n3
    pool = ThreadPoolExecutor(threads) if threads and threads > 1 else None
    try:
        for i in range(n1):                                       # stage 1: dense early
            x = block(x, weights[i], heads, eps, pool)
        x0 = x.copy()
        routed = n2 > 0 and not (keep_ratio == 1.0 and bypass_dense)
        if idx is None and n2 > 0 and not (keep_ratio == 1.0 and bypass_dense):
            K = keep_count(L, keep_ratio)
            if K < 1:
                raise ValueError("K = floor(L r) must be at least 1")
            if selector == "random":
                idx = select_random(B, L, K, seed, shared_indices)
            elif selector == "topk_l2":
                idx = select_topk_l2(x, K)
            elif selector == "laplacian":
                idx = select_topk_laplacian(x, K, grid_w)
            else:
                raise ValueError(selector)
        if routed:
            idx = np.asarray(idx, dtype=np.int64)
            bsel = np.arange(B)[:, None]
            h0 = x[bsel, idx]                                     # Gather(x, I)   [B, K, D]
            h = h0.copy()
            for i in range(n1, n1 + n2):                          # stage 2: sparse middle
                h = block(h, weights[i], heads, eps, pool)
            delta = h - h0                                        # Eq. 9
            x = x0.copy()
            x[bsel, idx] = x0[bsel, idx] + delta                  # x0 + Scatter(delta, I)
        else:
            for i in range(n1, n1 + n2):                          # r = 1: dense middle
                x = block(x, weights[i], heads, eps, pool)
        for i in range(n1 + n2, n1 + n2 + n3):                    # stage 3: dense late
            x = block(x, weights[i], heads, eps, pool)
    finally:
        if pool is not None:
            pool.shutdown()
    if return_stages:
        return x, idx, x0
    return x, idx


def forward_ensemble(x: np.ndarray, weights: Sequence[Dict[str, np.ndarray]], n1: int, n2: int,
                     n3: int, heads: int, keep_ratio: float, seeds: Sequence[int],
                     selector: str = "random", shared_indices: bool = False, eps: float = 1e-5,
                     threads: int = 0, grid_w: int = 0):
    """Implicit ensembling (Sec. 3, "Training and inference"; App. B): the mean
    of the routed forward over a set of selection seeds, each member a plain
    call of ``forward``.  Returns (mean, [member outputs], [member index sets]).
    """
    outs, idxs = [], []
    for seed in seeds:
        y, idx = forward(x, weights, n1, n2, n3, heads, keep_ratio, seed=seed, selector=selector,
                         shared_indices=shared_indices, eps=eps, threads=threads, grid_w=grid_w)
        outs.append(y)
        idxs.append(idx)
    return sum(outs) / float(len(outs)), outs, idxs


def dense_stack(x: np.ndarray, weights: Sequence[Dict[str, np.ndarray]], heads: int,
                eps: float = 1e-5, threads: int = 0) -> np.ndarray:
    """All blocks on all tokens: the dense baseline (routing disabled)."""
    pool = ThreadPoolExecutor(threads) if threads and threads > 1 else None
    try:
        x = np.asarray(x, dtype=np.float64)
        for w in weights:
            x = block(x, w, heads, eps, pool)
    finally:
        if pool is not None:
            pool.shutdown()
    return x
