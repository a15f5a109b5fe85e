"""Pins of the fp64 oracle against things other than itself.

Each test checks the oracle against a value the paper prints, a published
reference output, a library routine (PyTorch float64 CPU modules), a closed
form, brute force on tiny inputs, or an invariant the paper states.
"""
import math
import os

import numpy as np
import pytest
import torch

from oracle import reslim as o


def _read_rows(path):
    rows = []
    with open(path) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def _rand_weights(rng, D, hidden, scale=0.2):
    return {
        "ln1_g": 1.0 + scale * rng.standard_normal(D), "ln1_b": scale * rng.standard_normal(D),
        "wqkv": scale * rng.standard_normal((3 * D, D)), "bqkv": scale * rng.standard_normal(3 * D),
        "wo": scale * rng.standard_normal((D, D)), "bo": scale * rng.standard_normal(D),
        "ln2_g": 1.0 + scale * rng.standard_normal(D), "ln2_b": scale * rng.standard_normal(D),
        "w1": scale * rng.standard_normal((hidden, D)), "b1": scale * rng.standard_normal(hidden),
        "w2": scale * rng.standard_normal((D, hidden)), "b2": scale * rng.standard_normal(D),
    }


# ------------------------------------------------------------------ K
def test_keep_count_matches_paper(golden_dir):
    rows = _read_rows(os.path.join(golden_dir, "paper_keep_counts.txt"))
    assert rows
    for L, r, K in rows:
        assert o.keep_count(int(L), float(r)) == int(K)


def test_keep_count_workloads_and_bounds():
    # the five workloads: L = 512 / 512 / 2048 / 16200 at r = 0.25, and the sweep
    assert [o.keep_count(L, 0.25) for L in (512, 512, 2048, 16200)] == [128, 128, 512, 4050]
    assert [o.keep_count(2048, r) for r in (1.0, 0.5, 0.25, 0.125)] == [2048, 1024, 512, 256]
    assert o.keep_count(7, 0.5) == 3 and o.keep_count(3, 0.3) == 0
    for bad in (0.0, -0.1, 1.01):
        with pytest.raises(ValueError):
            o.keep_count(10, bad)


# ------------------------------------------------------- random selection
def test_splitmix64_published_outputs(golden_dir):
    rows = _read_rows(os.path.join(golden_dir, "splitmix64_published.txt"))
    assert len(rows) >= 2
    for row in rows:
        seed, outs = int(row[0]), [int(v) for v in row[1:]]
        keys = o.random_keys(1, len(outs), seed, shared=False)[0]
        assert [int(k) for k in keys] == outs


def test_random_keys_batch_counters():
    # sample b continues the counter sequence after sample b-1 (per-sample sets),
    # shared mode repeats sample 0's keys for every sample
    L = 7
    k = o.random_keys(3, L, 42, shared=False)
    flat = o.random_keys(1, 3 * L, 42, shared=False)[0]
    assert np.array_equal(k.reshape(-1), flat)
    ks = o.random_keys(3, L, 42, shared=True)
    assert all(np.array_equal(ks[b], k[0]) for b in range(3))


def test_random_select_bruteforce():
    for (B, L, K, seed) in [(3, 10, 4, 7), (2, 33, 33, 1), (1, 5, 1, 123456789), (4, 64, 16, 2**64 - 1)]:
        idx = o.select_random(B, L, K, seed)
        keys = o.random_keys(B, L, seed, shared=False)
        for b in range(B):
            pairs = sorted((int(keys[b, i]), i) for i in range(L))
            expect = sorted(i for _, i in pairs[:K])
            assert idx[b].tolist() == expect


def test_random_select_invariants():
    B, L, K = 5, 300, 75
    idx = o.select_random(B, L, K, 99)
    assert idx.shape == (B, K)
    for b in range(B):
        assert np.all(np.diff(idx[b]) > 0)          # strictly increasing => unique and sorted
        assert idx[b].min() >= 0 and idx[b].max() < L
    assert not np.array_equal(idx[0], idx[1])      # per-sample sets differ
    sh = o.select_random(B, L, K, 99, shared=True)
    assert all(np.array_equal(sh[b], sh[0]) for b in range(B))
    assert np.array_equal(sh[0], idx[0])
    assert not np.array_equal(o.select_random(1, L, K, 100), idx[:1])


def test_random_select_uniform_inclusion():
    # "drawn uniformly without replacement": every token is included with
    # probability K/L; chi-square over many seeds (Sec. 3.2).
    L, K, S = 48, 12, 3000
    counts = np.zeros(L)
    for s in range(S):
        counts[o.select_random(1, L, K, s)[0]] += 1
    expected = S * K / L
    chi2 = ((counts - expected) ** 2 / expected).sum()
    # dof = L - 1 = 47; P(chi2 > 100) < 1e-5
    assert chi2 < 100.0, chi2
    # pairs are uniform too: two fixed tokens are jointly selected with prob K(K-1)/(L(L-1))
    both = sum(1 for s in range(S) if {0, 1} <= set(o.select_random(1, L, K, s)[0].tolist()))
    p = K * (K - 1) / (L * (L - 1))
    assert abs(both - S * p) < 5 * math.sqrt(S * p * (1 - p))


# -------------------------------------------------------------- top-K L2
def test_topk_bruteforce_with_ties():
    rng = np.random.default_rng(3)
    x = rng.integers(-2, 3, size=(3, 20, 4)).astype(np.float64)   # many equal norms
    for K in (1, 5, 11, 20):
        idx = o.select_topk_l2(x, K)
        for b in range(3):
            norms = [sum(v * v for v in x[b, i]) for i in range(20)]
            order = sorted(range(20), key=lambda i: (-norms[i], i))
            assert idx[b].tolist() == sorted(order[:K])


# ----------------------------------------- Laplacian selector (App. B.2)
def _lap_scores_bruteforce(x, grid_w):
    """Pure-Python 5-point Laplacian score: clamp the latitude index to the grid
    (the poles reflected onto themselves), wrap the longitude index."""
    B, L, D = x.shape
    H = L // grid_w
    s = np.zeros((B, L))
    for b in range(B):
        for i in range(H):
            for j in range(grid_w):
                def at(ii, jj):
                    return x[b, min(max(ii, 0), H - 1) * grid_w + jj % grid_w]
                lap = at(i - 1, j) + at(i + 1, j) + at(i, j - 1) + at(i, j + 1) - 4.0 * at(i, j)
                s[b, i * grid_w + j] = sum(float(v) * float(v) for v in lap)
    return s


def test_laplacian_scores_closed_forms():
    H, W, D = 6, 8, 3
    a = np.array([0.5, -1.25, 2.0])
    # a constant field has no curvature
    assert np.all(o.token_laplacian_scores(np.full((2, H * W, D), 3.7), W) == 0.0)
    # quadratic in latitude, x = a i^2: interior rows 4 |a|^2; the first row
    # sees x(1) - x(0) = a, the last x(H-2) - x(H-1) = -(2H - 3) a
    i = np.repeat(np.arange(H), W).astype(np.float64)
    x = (i[:, None] ** 2 * a[None, :])[None]
    s = o.token_laplacian_scores(x, W).reshape(H, W)
    na = float(np.dot(a, a))
    assert np.allclose(s[1:-1], 4.0 * na, rtol=0, atol=1e-12)
    assert np.allclose(s[0], na, rtol=0, atol=1e-12)
    assert np.allclose(s[-1], (2 * H - 3) ** 2 * na, rtol=0, atol=1e-9)
    # a longitude wave, x = c cos(2 pi k j / W), is an eigenfunction of the
    # periodic second difference: lap = 2 (cos(2 pi k / W) - 1) x
    for k in (1, 3):
        j = np.tile(np.arange(W), H).astype(np.float64)
        c = np.array([1.0, -0.5, 0.25])
        cw = np.cos(2 * np.pi * k * j / W)
        x = (cw[:, None] * c[None, :])[None]
        expect = 4.0 * (np.cos(2 * np.pi * k / W) - 1.0) ** 2 * cw ** 2 * float(np.dot(c, c))
        assert np.allclose(o.token_laplacian_scores(x, W)[0], expect, rtol=0, atol=1e-12)


def test_laplacian_scores_bruteforce():
    rng = np.random.default_rng(11)
    for (B, H, W, D) in [(2, 5, 7, 4), (1, 1, 6, 3), (1, 4, 1, 2), (3, 3, 3, 5)]:
        x = rng.standard_normal((B, H * W, D))
        assert np.allclose(o.token_laplacian_scores(x, W), _lap_scores_bruteforce(x, W),
                           rtol=1e-13, atol=1e-13)


def test_laplacian_scores_against_scipy_ndimage():
    # scipy's discrete Laplacian over the two grid axes, latitude edges repeated
    # ("nearest": x(-1) = x(0)) and longitude periodic ("wrap"), squared and
    # summed over the features
    ndimage = pytest.importorskip("scipy.ndimage")
    rng = np.random.default_rng(23)
    for (B, H, W, D) in [(2, 6, 9, 5), (1, 90, 180, 4), (1, 3, 2, 3)]:
        x = rng.standard_normal((B, H * W, D))
        for b in range(B):
            lap = ndimage.laplace(x[b].reshape(H, W, D), mode=["nearest", "wrap"], axes=(0, 1))
            expect = (lap ** 2).sum(axis=-1).reshape(-1)
            assert np.allclose(o.token_laplacian_scores(x[b:b + 1], W)[0], expect,
                               rtol=1e-12, atol=1e-12)


def test_laplacian_topk_bruteforce_with_ties():
    rng = np.random.default_rng(5)
    H, W = 4, 5
    x = rng.integers(-1, 2, size=(2, H * W, 3)).astype(np.float64)   # many equal scores
    s = _lap_scores_bruteforce(x, W)
    for K in (1, 4, 9, 20):
        idx = o.select_topk_laplacian(x, K, W)
        for b in range(2):
            order = sorted(range(H * W), key=lambda t: (-s[b, t], t))
            assert idx[b].tolist() == sorted(order[:K])


# ---------------------------------------------------- block ingredients
def test_layer_norm_closed_form_and_torch():
    v = np.array([1.0, 2.0, 3.0, 4.0])
    y = o.layer_norm(v, np.ones(4), np.zeros(4), 0.0)
    assert np.allclose(y, (v - 2.5) / math.sqrt(1.25), rtol=0, atol=1e-15)
    rng = np.random.default_rng(0)
    x = rng.standard_normal((6, 40)) * 3 + 1
    g, b = rng.standard_normal(40), rng.standard_normal(40)
    ref = torch.nn.functional.layer_norm(torch.from_numpy(x), (40,), torch.from_numpy(g),
                                         torch.from_numpy(b), eps=1e-5).numpy()
    assert np.allclose(o.layer_norm(x, g, b, 1e-5), ref, rtol=0, atol=1e-13)
    z = o.layer_norm(x, np.ones(40), np.full(40, 0.5), 1e-5)
    assert np.allclose(z.mean(axis=1), 0.5, atol=1e-13)
    assert np.allclose(z.var(axis=1), 1.0, atol=1e-5)


def test_gelu_known_values_and_torch():
    # GELU(z) = z * Phi(z); Phi(1) = 0.8413447460685429, Phi(2) = 0.9772498680518208
    assert o.gelu(np.array([0.0]))[0] == 0.0
    assert abs(o.gelu(np.array([1.0]))[0] - 0.8413447460685429) < 1e-15
    assert abs(o.gelu(np.array([-1.0]))[0] + 0.15865525393145707) < 1e-15
    assert abs(o.gelu(np.array([2.0]))[0] - 2 * 0.9772498680518208) < 1e-15
    assert abs(o.gelu(np.array([30.0]))[0] - 30.0) < 1e-12
    z = np.linspace(-6, 6, 101)
    ref = torch.nn.functional.gelu(torch.from_numpy(z)).numpy()
    assert np.allclose(o.gelu(z), ref, rtol=0, atol=1e-15)


def test_attention_against_torch_sdpa_and_bruteforce():
    rng = np.random.default_rng(1)
    B, T, H, dh = 2, 9, 3, 8
    D = H * dh
    qkv = rng.standard_normal((B, T, 3 * D))
    out = o.attention(qkv, H)
    q = torch.from_numpy(qkv[..., :D]).reshape(B, T, H, dh).transpose(1, 2)
    k = torch.from_numpy(qkv[..., D:2 * D]).reshape(B, T, H, dh).transpose(1, 2)
    v = torch.from_numpy(qkv[..., 2 * D:]).reshape(B, T, H, dh).transpose(1, 2)
    ref = torch.nn.functional.scaled_dot_product_attention(q, k, v).transpose(1, 2).reshape(B, T, D)
    assert np.allclose(out, ref.numpy(), rtol=0, atol=1e-13)
    # pure-Python brute force of one output element
    b, h, t, c = 1, 2, 4, 5
    s = [sum(qkv[b, t, h * dh + j] * qkv[b, u, D + h * dh + j] for j in range(dh)) / math.sqrt(dh)
         for u in range(T)]
    m = max(s)
    e = [math.exp(v_ - m) for v_ in s]
    val = sum(e[u] * qkv[b, u, 2 * D + h * dh + c] for u in range(T)) / sum(e)
    assert abs(out[b, t, h * dh + c] - val) < 1e-13
    # chunking over query rows must not change anything
    one = o._attention_one_head(q[0, 0].numpy().copy(), k[0, 0].numpy().copy(), v[0, 0].numpy().copy(), row_chunk=2)
    assert np.allclose(one, out[0, :, :dh], rtol=0, atol=1e-14)


def test_single_key_attention_returns_value():
    qkv = np.random.default_rng(2).standard_normal((1, 1, 3 * 16))
    out = o.attention(qkv, 2)
    assert np.allclose(out[0, 0], qkv[0, 0, 32:], rtol=0, atol=0)


def _torch_block(w, D, H, hidden):
    layer = torch.nn.TransformerEncoderLayer(d_model=D, nhead=H, dim_feedforward=hidden, dropout=0.0,
                                             activation="gelu", layer_norm_eps=1e-5, batch_first=True,
                                             norm_first=True, dtype=torch.float64)
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    with torch.no_grad():
        layer.norm1.weight.copy_(t(w["ln1_g"])); layer.norm1.bias.copy_(t(w["ln1_b"]))
        layer.self_attn.in_proj_weight.copy_(t(w["wqkv"])); layer.self_attn.in_proj_bias.copy_(t(w["bqkv"]))
        layer.self_attn.out_proj.weight.copy_(t(w["wo"])); layer.self_attn.out_proj.bias.copy_(t(w["bo"]))
        layer.norm2.weight.copy_(t(w["ln2_g"])); layer.norm2.bias.copy_(t(w["ln2_b"]))
        layer.linear1.weight.copy_(t(w["w1"])); layer.linear1.bias.copy_(t(w["b1"]))
        layer.linear2.weight.copy_(t(w["w2"])); layer.linear2.bias.copy_(t(w["b2"]))
    return layer.eval()


def test_block_against_torch_prenorm_encoder_layer():
    # PyTorch's TransformerEncoderLayer with norm_first=True is the pre-LN block
    # of Eq. 11 (packed q/k/v in_proj, per-head column groups, 1/sqrt(dh) scale).
    rng = np.random.default_rng(5)
    B, T, D, H = 2, 11, 32, 4
    w = _rand_weights(rng, D, 4 * D)
    x = rng.standard_normal((B, T, D))
    layer = _torch_block(w, D, H, 4 * D)
    with torch.no_grad():
        ref = layer(torch.from_numpy(x)).numpy()
    out = o.block(x, w, H, 1e-5)
    assert np.allclose(out, ref, rtol=0, atol=1e-12), np.abs(out - ref).max()


def test_block_zero_weights_is_identity():
    rng = np.random.default_rng(6)
    D = 16
    w = {k: np.zeros_like(v) for k, v in _rand_weights(rng, D, 4 * D).items()}
    w["ln1_g"] = rng.standard_normal(D)
    w["ln2_g"] = rng.standard_normal(D)
    x = rng.standard_normal((2, 5, D))
    assert np.array_equal(o.block(x, w, 2), x)


def test_block_uniform_attention_closed_form():
    # Wqkv = 0, bqkv = (0, 0, bv): every score is 0, every softmax row uniform,
    # the attention output is bv for every token; with W1 = 0 the MLP adds
    # GELU(b1) W2^T + b2 to every token.
    rng = np.random.default_rng(7)
    D, hidden = 16, 64
    w = _rand_weights(rng, D, hidden)
    w["wqkv"] = np.zeros((3 * D, D))
    bv = rng.standard_normal(D)
    w["bqkv"] = np.concatenate([np.zeros(2 * D), bv])
    w["w1"] = np.zeros((hidden, D))
    x = rng.standard_normal((3, 7, D))
    expect = x + (w["wo"] @ bv + w["bo"]) + (w["w2"] @ o.gelu(w["b1"]) + w["b2"])
    assert np.allclose(o.block(x, w, 4), expect, rtol=0, atol=1e-13)


# ------------------------------------------------------ routing invariants
def _tiny_model(seed=11, B=2, L=24, D=16, N=4):
    rng = np.random.default_rng(seed)
    ws = [_rand_weights(rng, D, 4 * D) for _ in range(N)]
    x = rng.standard_normal((B, L, D))
    return x, ws


def test_r1_is_exactly_the_dense_stack():
    x, ws = _tiny_model()
    out, idx = o.forward(x, ws, 1, 2, 1, heads=2, keep_ratio=1.0, seed=3)
    assert idx is None
    assert np.array_equal(out, o.dense_stack(x, ws, heads=2))
    # the routed formulation with K = L reaches the same result up to rounding
    out2, idx2 = o.forward(x, ws, 1, 2, 1, heads=2, keep_ratio=1.0, seed=3, bypass_dense=False)
    assert idx2.shape == (2, 24) and np.array_equal(idx2[0], np.arange(24))
    assert np.allclose(out2, out, rtol=0, atol=1e-12)


def test_unselected_tokens_keep_pre_routing_values_exactly():
    x, ws = _tiny_model(N=3)
    out, idx, x0 = o.forward(x, ws, 1, 2, 0, heads=2, keep_ratio=0.25, seed=9, return_stages=True)
    B, L, _ = x.shape
    assert np.array_equal(x0, o.dense_stack(x, ws[:1], heads=2))
    for b in range(B):
        sel = set(idx[b].tolist())
        for i in range(L):
            if i not in sel:
                assert np.array_equal(out[b, i], x0[b, i])
            else:
                assert not np.array_equal(out[b, i], x0[b, i])


def test_routed_block_equals_block_on_extracted_subsequence():
    # attention only among the selected tokens of the same sample (Sec. 3.2 Eq. 8)
    x, ws = _tiny_model(N=2)
    out, idx = o.forward(x, ws, 0, 2, 0, heads=2, keep_ratio=0.5, seed=21)
    for b in range(x.shape[0]):
        sub = x[b:b + 1, idx[b]]
        for w in ws:
            sub = o.block(sub, w, 2)
        expect = x[b].copy()
        expect[idx[b]] = x[b, idx[b]] + (sub[0] - x[b, idx[b]])
        assert np.allclose(out[b], expect, rtol=0, atol=1e-13)


def test_zero_routed_blocks_leave_everything_bitwise():
    x, ws = _tiny_model(N=4)
    for i in (1, 2):
        ws[i] = {k: (np.ones_like(v) if k.endswith("_g") else np.zeros_like(v)) for k, v in ws[i].items()}
    out, idx, x0 = o.forward(x, ws, 1, 2, 1, heads=2, keep_ratio=0.5, seed=4, return_stages=True)
    # delta is exactly zero, so x' == x0 and the late block sees x0
    expect = o.dense_stack(x0, ws[3:], heads=2)
    assert np.array_equal(out, expect)


def test_topk_selector_in_forward_uses_post_dense_state():
    x, ws = _tiny_model(N=3)
    out, idx, x0 = o.forward(x, ws, 1, 1, 1, heads=2, keep_ratio=0.25, selector="topk_l2",
                             return_stages=True)
    assert np.array_equal(idx, o.select_topk_l2(x0, 6))


def test_laplacian_selector_in_forward_uses_post_dense_state():
    x, ws = _tiny_model(N=3)                 # L = 24 tokens on a 6 x 4 patch grid
    out, idx, x0 = o.forward(x, ws, 1, 1, 1, heads=2, keep_ratio=0.25, selector="laplacian",
                             return_stages=True, grid_w=4)
    assert np.array_equal(idx, o.select_topk_laplacian(x0, 6, 4))


# ------------------------------------------------------------------ implicit ensemble
def test_ensemble_of_the_dense_path_is_the_dense_stack():
    # r = 1 routes nothing, so every member is the dense stack and their mean
    # (four equal terms, an exact division by 4) is too
    x, ws = _tiny_model()
    mean, members, idxs = o.forward_ensemble(x, ws, 1, 2, 1, heads=2, keep_ratio=1.0,
                                             seeds=[1, 2, 3, 4])
    assert np.array_equal(mean, o.dense_stack(x, ws, heads=2))
    assert all(i is None for i in idxs)


def test_ensemble_members_and_mean():
    x, ws = _tiny_model(N=3)
    seeds = [5, 11, 2**64 - 3]
    mean, members, idxs = o.forward_ensemble(x, ws, 1, 1, 1, heads=2, keep_ratio=0.25, seeds=seeds)
    for s, y, idx in zip(seeds, members, idxs):
        y1, idx1 = o.forward(x, ws, 1, 1, 1, heads=2, keep_ratio=0.25, seed=s)
        assert np.array_equal(y, y1) and np.array_equal(idx, idx1)
    assert np.allclose(mean, (members[0] + members[1] + members[2]) / 3.0, rtol=0, atol=1e-15)
    assert not np.array_equal(idxs[0], idxs[1])


def test_ensemble_passthrough_tokens():
    # with no late blocks, a token no member selects keeps its pre-routing value
    # exactly in the mean, and a token one of two members selects is the
    # average of that member's value and the pre-routing value
    x, ws = _tiny_model(N=2)
    mean, members, idxs = o.forward_ensemble(x, ws, 1, 1, 0, heads=2, keep_ratio=0.25, seeds=[7, 8])
    _, _, x0 = o.forward(x, ws, 1, 1, 0, heads=2, keep_ratio=0.25, seed=7, return_stages=True)
    B, L, _ = x.shape
    for b in range(B):
        s0, s1 = set(idxs[0][b].tolist()), set(idxs[1][b].tolist())
        for i in range(L):
            if i not in s0 and i not in s1:
                assert np.array_equal(mean[b, i], x0[b, i])
            elif (i in s0) != (i in s1):
                m = 0 if i in s0 else 1
                assert np.allclose(mean[b, i], 0.5 * (members[m][b, i] + x0[b, i]), rtol=0, atol=1e-15)


# ------------------------------------------------------------------ asymmetric attention
def test_cross_attention_against_torch_sdpa_and_bruteforce():
    # queries and keys/values of different lengths (Sec. 3.4: Q from the K routed
    # tokens, K and V from the L-token conditioning sequence)
    rng = np.random.default_rng(5)
    B, Tq, Tkv, H, dh = 2, 7, 13, 3, 8
    D = H * dh
    q = rng.standard_normal((B, Tq, D))
    kv = rng.standard_normal((B, Tkv, 2 * D))
    out = o.cross_attention(q, kv, H)
    tq = torch.from_numpy(q).reshape(B, Tq, H, dh).transpose(1, 2)
    tk = torch.from_numpy(kv[..., :D]).reshape(B, Tkv, H, dh).transpose(1, 2)
    tv = torch.from_numpy(kv[..., D:]).reshape(B, Tkv, H, dh).transpose(1, 2)
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv).transpose(1, 2).reshape(B, Tq, D)
    assert np.allclose(out, ref.numpy(), rtol=0, atol=1e-13)
    b, h, t, c = 1, 2, 6, 3
    s = [sum(q[b, t, h * dh + j] * kv[b, u, h * dh + j] for j in range(dh)) / math.sqrt(dh)
         for u in range(Tkv)]
    m = max(s)
    e = [math.exp(v_ - m) for v_ in s]
    val = sum(e[u] * kv[b, u, D + h * dh + c] for u in range(Tkv)) / sum(e)
    assert abs(out[b, t, h * dh + c] - val) < 1e-13


def test_cross_attention_on_the_same_tokens_is_self_attention():
    rng = np.random.default_rng(6)
    B, T, H, dh = 2, 11, 2, 8
    D = H * dh
    qkv = rng.standard_normal((B, T, 3 * D))
    assert np.array_equal(o.cross_attention(qkv[..., :D], qkv[..., D:], H), o.attention(qkv, H))


def test_cross_attention_single_key_returns_its_value():
    rng = np.random.default_rng(7)
    B, Tq, H, dh = 2, 5, 2, 8
    D = H * dh
    q = rng.standard_normal((B, Tq, D))
    kv = rng.standard_normal((B, 1, 2 * D))
    out = o.cross_attention(q, kv, H)
    assert np.allclose(out, np.broadcast_to(kv[:, :, D:], out.shape), rtol=0, atol=1e-15)
