"""The oracle's pins catch plausible mistakes.

Each case plants one mistake in the oracle (a replacement for one of its
functions, on the CPU only): a dropped term, a wrong sign, index, axis or
scale, a transposed or swapped operand, a wrong tie-break.  It then runs the
pins of tests/test_oracle_pins.py that cover that function and requires at
least one of them to fail.  A mistake no pin catches would be a hole in the
parity evidence.
"""
import math
import os

import numpy as np
import pytest

from oracle import reslim as o
from tests import test_oracle_pins as pins

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


# ------------------------------------------------------------ planted mistakes
def m_keep_count_round(L, r):
    return int(round(float(r) * float(L)))


def m_random_keys_from_zero(B, L, seed, shared):
    b = np.zeros(B, dtype=np.int64) if shared else np.arange(B, dtype=np.int64)
    ctr = (b[:, None] * L + np.arange(L, dtype=np.int64)[None, :]).astype(o.U64)   # counter 0, not 1
    with np.errstate(over="ignore"):
        z = o.U64(seed % (1 << 64)) + o.U64(o.GOLDEN_GAMMA) * ctr
    return o.splitmix64_mix(z)


def m_random_keys_interleaved(B, L, seed, shared):
    b = np.zeros(B, dtype=np.int64) if shared else np.arange(B, dtype=np.int64)
    ctr = (1 + b[:, None] + np.arange(L, dtype=np.int64)[None, :] * B).astype(o.U64)
    with np.errstate(over="ignore"):
        z = o.U64(seed % (1 << 64)) + o.U64(o.GOLDEN_GAMMA) * ctr
    return o.splitmix64_mix(z)


def m_select_random_largest(B, L, K, seed, shared=False):
    keys = o.random_keys(B, L, seed, shared)
    out = np.empty((B, K), dtype=np.int64)
    for b in range(B):
        order = np.lexsort((np.arange(L), keys[b]))[::-1]
        out[b] = np.sort(order[:K])
    return out


def m_select_random_unsorted(B, L, K, seed, shared=False):
    keys = o.random_keys(B, L, seed, shared)
    out = np.empty((B, K), dtype=np.int64)
    for b in range(B):
        out[b] = np.lexsort((np.arange(L), keys[b]))[:K]
    return out


def m_topk_ties_high(x, K):
    s = o.token_sq_norms(x)
    B, L = s.shape
    out = np.empty((B, K), dtype=np.int64)
    for b in range(B):
        order = np.lexsort((-np.arange(L), -s[b]))
        out[b] = np.sort(order[:K])
    return out


def m_topk_smallest(x, K):
    s = o.token_sq_norms(x)
    B, L = s.shape
    out = np.empty((B, K), dtype=np.int64)
    for b in range(B):
        order = np.lexsort((np.arange(L), s[b]))
        out[b] = np.sort(order[:K])
    return out


def _lap(x, grid_w, *, lat="reflect", lon="periodic", centre=4.0, transpose=False):
    x = np.asarray(x, dtype=np.float64)
    B, L, D = x.shape
    H = L // grid_w
    g = x.reshape(B, grid_w, H, D).transpose(0, 2, 1, 3) if transpose else x.reshape(B, H, grid_w, D)
    if lat == "reflect":
        north = np.concatenate([g[:, :1], g[:, :-1]], axis=1)
        south = np.concatenate([g[:, 1:], g[:, -1:]], axis=1)
    elif lat == "periodic":
        north, south = np.roll(g, 1, axis=1), np.roll(g, -1, axis=1)
    else:                                      # zero outside the grid
        z = np.zeros_like(g[:, :1])
        north = np.concatenate([z, g[:, :-1]], axis=1)
        south = np.concatenate([g[:, 1:], z], axis=1)
    if lon == "periodic":
        west, east = np.roll(g, 1, axis=2), np.roll(g, -1, axis=2)
    else:                                      # reflected at the first and last column
        west = np.concatenate([g[:, :, :1], g[:, :, :-1]], axis=2)
        east = np.concatenate([g[:, :, 1:], g[:, :, -1:]], axis=2)
    lap = north + south + west + east - centre * g
    s = np.einsum("bhwd,bhwd->bhw", lap, lap)
    return (s.transpose(0, 2, 1) if transpose else s).reshape(B, L)


def m_lap_lat_periodic(x, grid_w):
    return _lap(x, grid_w, lat="periodic")


def m_lap_lat_zero(x, grid_w):
    return _lap(x, grid_w, lat="zero")


def m_lap_lon_reflected(x, grid_w):
    return _lap(x, grid_w, lon="reflect")


def m_lap_centre_two(x, grid_w):
    return _lap(x, grid_w, centre=2.0)


def m_lap_grid_transposed(x, grid_w):
    return _lap(x, grid_w, transpose=True)


def m_lap_topk_ties_high(x, K, grid_w):
    s = o.token_laplacian_scores(x, grid_w)
    B, L = s.shape
    out = np.empty((B, K), dtype=np.int64)
    for b in range(B):
        out[b] = np.sort(np.lexsort((-np.arange(L), -s[b]))[:K])
    return out


def m_ln_unbiased(v, g, b, eps):
    mu = v.mean(axis=-1, keepdims=True)
    var = v.var(axis=-1, ddof=1, keepdims=True)
    return (v - mu) / np.sqrt(var + eps) * g + b


def m_ln_eps_outside(v, g, b, eps):
    mu = v.mean(axis=-1, keepdims=True)
    var = ((v - mu) ** 2).mean(axis=-1, keepdims=True)
    return (v - mu) / (np.sqrt(var) + eps) * g + b


def m_gelu_tanh(z):
    return 0.5 * z * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (z + 0.044715 * z ** 3)))


def m_gelu_no_half(z):
    return z * (1.0 + o.erf(z / math.sqrt(2.0)))


def _head(q, k, v, scale, axis=1):
    s = (q @ k.T) * scale
    s = s - s.max(axis=axis, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=axis, keepdims=True)
    return p @ v


def m_head_scale_dh(q, k, v, row_chunk=1024):
    return _head(q, k, v, 1.0 / q.shape[1])


def m_head_kv_swapped(q, k, v, row_chunk=1024):
    return _head(q, v, k, 1.0 / math.sqrt(q.shape[1]))


def m_head_softmax_axis0(q, k, v, row_chunk=1024):
    return _head(q, k, v, 1.0 / math.sqrt(q.shape[1]), axis=0)


def m_attention_interleaved_heads(qkv, heads, pool=None):
    B, T, D3 = qkv.shape
    D = D3 // 3
    out = np.empty((B, T, D))
    for b in range(B):
        for h in range(heads):
            c = slice(h, D, heads)                    # head h takes every heads-th column
            out[b, :, c] = o._attention_one_head(np.ascontiguousarray(qkv[b, :, :D][:, c]),
                                                 np.ascontiguousarray(qkv[b, :, D:2 * D][:, c]),
                                                 np.ascontiguousarray(qkv[b, :, 2 * D:][:, c]))
    return out


def _block(x, w, heads, eps, *, out_bias=True, post_ln=False, ln2_from_ln1=False, mlp_residual=True):
    B, T, D = x.shape
    g2, b2 = (w["ln1_g"], w["ln1_b"]) if ln2_from_ln1 else (w["ln2_g"], w["ln2_b"])
    a = x if post_ln else o.layer_norm(x, w["ln1_g"], w["ln1_b"], eps)
    qkv = a.reshape(B * T, D) @ w["wqkv"].T + w["bqkv"]
    att = o.attention(qkv.reshape(B, T, 3 * D), heads)
    x = x + (att.reshape(B * T, D) @ w["wo"].T + (w["bo"] if out_bias else 0.0)).reshape(B, T, D)
    if post_ln:
        x = o.layer_norm(x, w["ln1_g"], w["ln1_b"], eps)
    m = x if post_ln else o.layer_norm(x, g2, b2, eps)
    u = o.gelu(m.reshape(B * T, D) @ w["w1"].T + w["b1"])
    y = (u @ w["w2"].T + w["b2"]).reshape(B, T, D)
    x = x + y if mlp_residual else y
    if post_ln:
        x = o.layer_norm(x, g2, b2, eps)
    return x


def m_block_no_out_bias(x, w, heads, eps=1e-5, pool=None):
    return _block(x, w, heads, eps, out_bias=False)


def m_block_post_ln(x, w, heads, eps=1e-5, pool=None):
    return _block(x, w, heads, eps, post_ln=True)


def m_block_ln1_for_ln2(x, w, heads, eps=1e-5, pool=None):
    return _block(x, w, heads, eps, ln2_from_ln1=True)


def m_block_no_mlp_residual(x, w, heads, eps=1e-5, pool=None):
    return _block(x, w, heads, eps, mlp_residual=False)


def _routed_forward(x, weights, n1, n2, n3, heads, keep_ratio, seed=0, selector="random",
                    shared_indices=False, eps=1e-5, idx=None, bypass_dense=True, threads=0,
                    return_stages=False, grid_w=0, *, scatter_sample0=False, no_gather=False,
                    skip_late=False, topk_on_input=False):
    x_in = np.asarray(x, dtype=np.float64)
    x = x_in
    B, L, D = x.shape
    for i in range(n1):
        x = o.block(x, weights[i], heads, eps)
    x0 = x.copy()
    routed = n2 > 0 and not (keep_ratio == 1.0 and bypass_dense)
    if idx is None and routed:
        K = o.keep_count(L, keep_ratio)
        xs = x_in if topk_on_input else x
        idx = (o.select_random(B, L, K, seed, shared_indices) if selector == "random"
               else o.select_topk_laplacian(xs, K, grid_w) if selector == "laplacian"
               else o.select_topk_l2(xs, K))
    if routed:
        bsel = np.zeros((B, 1), dtype=np.int64) if scatter_sample0 else np.arange(B)[:, None]
        if no_gather:
            h = x0.copy()
            for i in range(n1, n1 + n2):
                h = o.block(h, weights[i], heads, eps)
            x = x0.copy()
            x[np.arange(B)[:, None], idx] = h[np.arange(B)[:, None], idx]
        else:
            h0 = x[np.arange(B)[:, None], idx]
            h = h0.copy()
            for i in range(n1, n1 + n2):
                h = o.block(h, weights[i], heads, eps)
            x = x0.copy()
            x[bsel, idx] = x0[bsel, idx] + (h - h0)
    else:
        for i in range(n1, n1 + n2):
            x = o.block(x, weights[i], heads, eps)
    if not skip_late:
        for i in range(n1 + n2, n1 + n2 + n3):
            x = o.block(x, weights[i], heads, eps)
    if return_stages:
        return x, idx, x0
    return x, idx


def _fwd_variant(**kw):
    def f(*a, **k):
        return _routed_forward(*a, **k, **kw)
    return f


def m_cross_kv_swapped(q, kv, heads, pool=None):
    D = q.shape[2]
    return _cross(q, np.concatenate([kv[..., D:], kv[..., :D]], axis=-1), heads)


def _cross(q, kv, heads):
    B, Tq, D = q.shape
    dh = D // heads
    out = np.empty((B, Tq, D))
    for b in range(B):
        for h in range(heads):
            c = slice(h * dh, (h + 1) * dh)
            out[b, :, c] = o._attention_one_head(np.ascontiguousarray(q[b][:, c]),
                                                 np.ascontiguousarray(kv[b, :, :D][:, c]),
                                                 np.ascontiguousarray(kv[b, :, D:][:, c]))
    return out


def m_ensemble_sum(x, weights, n1, n2, n3, heads, keep_ratio, seeds, selector="random",
                   shared_indices=False, eps=1e-5, threads=0):
    outs, idxs = [], []
    for seed in seeds:
        y, idx = o.forward(x, weights, n1, n2, n3, heads, keep_ratio, seed=seed, selector=selector,
                           shared_indices=shared_indices, eps=eps, threads=threads)
        outs.append(y)
        idxs.append(idx)
    return sum(outs), outs, idxs


# (name, {oracle attribute: replacement}, pins that should notice)
CASES = [
    ("K rounded instead of truncated", {"keep_count": m_keep_count_round},
     ["test_keep_count_matches_paper", "test_keep_count_workloads_and_bounds"]),
    ("random keys: counter starts at 0", {"random_keys": m_random_keys_from_zero},
     ["test_splitmix64_published_outputs", "test_random_keys_batch_counters"]),
    ("random keys: samples interleaved", {"random_keys": m_random_keys_interleaved},
     ["test_splitmix64_published_outputs", "test_random_keys_batch_counters"]),
    ("random selection keeps the largest keys", {"select_random": m_select_random_largest},
     ["test_random_select_bruteforce"]),
    ("random selection not sorted", {"select_random": m_select_random_unsorted},
     ["test_random_select_bruteforce", "test_random_select_invariants"]),
    ("top-K ties to the higher index", {"select_topk_l2": m_topk_ties_high},
     ["test_topk_bruteforce_with_ties"]),
    ("top-K keeps the smallest norms", {"select_topk_l2": m_topk_smallest},
     ["test_topk_bruteforce_with_ties"]),
    ("Laplacian: latitude wraps around", {"token_laplacian_scores": m_lap_lat_periodic},
     ["test_laplacian_scores_closed_forms", "test_laplacian_scores_bruteforce",
      "test_laplacian_scores_against_scipy_ndimage"]),
    ("Laplacian: zero outside the poles", {"token_laplacian_scores": m_lap_lat_zero},
     ["test_laplacian_scores_closed_forms", "test_laplacian_scores_bruteforce",
      "test_laplacian_scores_against_scipy_ndimage"]),
    ("Laplacian: longitude reflected, not periodic", {"token_laplacian_scores": m_lap_lon_reflected},
     ["test_laplacian_scores_closed_forms", "test_laplacian_scores_bruteforce",
      "test_laplacian_scores_against_scipy_ndimage"]),
    ("Laplacian: centre weight 2", {"token_laplacian_scores": m_lap_centre_two},
     ["test_laplacian_scores_closed_forms", "test_laplacian_scores_bruteforce",
      "test_laplacian_scores_against_scipy_ndimage"]),
    ("Laplacian: grid rows and columns swapped", {"token_laplacian_scores": m_lap_grid_transposed},
     ["test_laplacian_scores_closed_forms", "test_laplacian_scores_bruteforce",
      "test_laplacian_scores_against_scipy_ndimage"]),
    ("Laplacian top-K ties to the higher index", {"select_topk_laplacian": m_lap_topk_ties_high},
     ["test_laplacian_topk_bruteforce_with_ties"]),
    ("LayerNorm with the unbiased variance", {"layer_norm": m_ln_unbiased},
     ["test_layer_norm_closed_form_and_torch"]),
    ("LayerNorm eps outside the square root", {"layer_norm": m_ln_eps_outside},
     ["test_layer_norm_closed_form_and_torch"]),
    ("GELU as the tanh approximation", {"gelu": m_gelu_tanh}, ["test_gelu_known_values_and_torch"]),
    ("GELU without the factor 1/2", {"gelu": m_gelu_no_half}, ["test_gelu_known_values_and_torch"]),
    ("attention scaled by 1/dh", {"_attention_one_head": m_head_scale_dh},
     ["test_attention_against_torch_sdpa_and_bruteforce"]),
    ("attention with k and v swapped", {"_attention_one_head": m_head_kv_swapped},
     ["test_attention_against_torch_sdpa_and_bruteforce", "test_single_key_attention_returns_value"]),
    ("softmax over the queries", {"_attention_one_head": m_head_softmax_axis0},
     ["test_attention_against_torch_sdpa_and_bruteforce"]),
    ("heads take interleaved columns", {"attention": m_attention_interleaved_heads},
     ["test_attention_against_torch_sdpa_and_bruteforce"]),
    ("block drops the out-projection bias", {"block": m_block_no_out_bias},
     ["test_block_against_torch_prenorm_encoder_layer", "test_block_uniform_attention_closed_form"]),
    ("block is post-LN", {"block": m_block_post_ln},
     ["test_block_against_torch_prenorm_encoder_layer", "test_block_zero_weights_is_identity"]),
    ("block reuses LN1's parameters for LN2", {"block": m_block_ln1_for_ln2},
     ["test_block_against_torch_prenorm_encoder_layer"]),
    ("block drops the MLP residual", {"block": m_block_no_mlp_residual},
     ["test_block_against_torch_prenorm_encoder_layer", "test_block_zero_weights_is_identity"]),
    ("scatter into sample 0's rows", {"forward": _fwd_variant(scatter_sample0=True)},
     ["test_unselected_tokens_keep_pre_routing_values_exactly",
      "test_routed_block_equals_block_on_extracted_subsequence"]),
    ("sparse blocks see every token", {"forward": _fwd_variant(no_gather=True)},
     ["test_routed_block_equals_block_on_extracted_subsequence"]),
    ("dense-late blocks skipped", {"forward": _fwd_variant(skip_late=True)},
     ["test_r1_is_exactly_the_dense_stack", "test_zero_routed_blocks_leave_everything_bitwise"]),
    ("top-K scored on the input, not the block-n1 output", {"forward": _fwd_variant(topk_on_input=True)},
     ["test_topk_selector_in_forward_uses_post_dense_state",
      "test_laplacian_selector_in_forward_uses_post_dense_state"]),
    ("cross-attention with k and v swapped", {"cross_attention": m_cross_kv_swapped},
     ["test_cross_attention_against_torch_sdpa_and_bruteforce",
      "test_cross_attention_single_key_returns_its_value"]),
    ("ensemble sums instead of averaging", {"forward_ensemble": m_ensemble_sum},
     ["test_ensemble_of_the_dense_path_is_the_dense_stack", "test_ensemble_members_and_mean"]),
]


def _run_pin(name):
    fn = getattr(pins, name)
    if "golden_dir" in fn.__code__.co_varnames[:fn.__code__.co_argcount]:
        fn(GOLDEN)
    else:
        fn()


def test_pins_pass_on_the_unchanged_oracle():
    for _, _, names in CASES:
        for n in names:
            _run_pin(n)


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_a_planted_mistake_fails_a_pin(case, monkeypatch):
    name, patches, names = case
    for attr, repl in patches.items():
        assert hasattr(o, attr), attr
        monkeypatch.setattr(o, attr, repl)
    failed = []
    for n in names:
        try:
            _run_pin(n)
        except Exception:       # an assertion, or the mistake breaking a shape or an invariant
            failed.append(n)
    assert failed, f"no pin noticed: {name}"


# controls: the restatements above with no mistake planted pass the same pins,
# so a failure in a case comes from its planted mistake
CONTROLS = [
    ("head restatement", {"_attention_one_head": lambda q, k, v, row_chunk=1024:
                          _head(q, k, v, 1.0 / math.sqrt(q.shape[1]))},
     ["test_attention_against_torch_sdpa_and_bruteforce", "test_single_key_attention_returns_value"]),
    ("block restatement", {"block": lambda x, w, heads, eps=1e-5, pool=None: _block(x, w, heads, eps)},
     ["test_block_against_torch_prenorm_encoder_layer", "test_block_zero_weights_is_identity",
      "test_block_uniform_attention_closed_form"]),
    ("forward restatement", {"forward": _fwd_variant()},
     ["test_unselected_tokens_keep_pre_routing_values_exactly",
      "test_routed_block_equals_block_on_extracted_subsequence", "test_r1_is_exactly_the_dense_stack",
      "test_zero_routed_blocks_leave_everything_bitwise",
      "test_topk_selector_in_forward_uses_post_dense_state",
      "test_laplacian_selector_in_forward_uses_post_dense_state"]),
    ("cross-attention restatement", {"cross_attention": lambda q, kv, heads, pool=None: _cross(q, kv, heads)},
     ["test_cross_attention_against_torch_sdpa_and_bruteforce",
      "test_cross_attention_single_key_returns_its_value",
      "test_cross_attention_on_the_same_tokens_is_self_attention"]),
]


@pytest.mark.parametrize("case", CONTROLS, ids=[c[0] for c in CONTROLS])
def test_restatements_without_a_mistake_pass(case, monkeypatch):
    _, patches, names = case
    for attr, repl in patches.items():
        monkeypatch.setattr(o, attr, repl)
    for n in names:
        _run_pin(n)
