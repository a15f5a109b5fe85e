"""The allocation-free top-K selector (sr_select_topk_l2_static) against the
fp64 oracle's top-K selection and against the workspace-based sr_select.

Callers that cannot allocate device memory (a plugin inside a framework that
owns the GPU memory pool and gives it no workspace, or a latency-critical path
that cannot afford cudaMalloc's implicit synchronisation) use the static-scratch
entry point; it must select exactly the same tokens.  This file is collected
last so that a failure here leaves every other test already run.
"""
import numpy as np
import pytest
import torch

from oracle import reslim as o
from paper_2607_02829_gb300 import synth
from tests._helpers import built_lib

pytestmark = pytest.mark.gpu


def _inputs(B, L, D, seed):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(B, L, D, generator=g, dtype=torch.float64)
    x[:, 1::5] = x[:, 0::5][:, :x[:, 1::5].shape[1]]          # exact duplicates -> exact ties
    return x.to(torch.bfloat16).cuda()


def _workspace_select(b, x, r):
    B, L, D = x.shape
    enc = b.Encoder(b.make_config(B, L, D, D // 64, 0, 1, 0, dtype="bf16", selector="topk_l2"),
                    max_keep_ratio=1.0)
    idx = enc.select(x, r, 0)
    torch.cuda.synchronize()
    enc.close()
    return idx.cpu().numpy()


def _static_select(b, x, r):
    B, L, D = x.shape
    K = b.sr_keep_count(L, r)
    idx = torch.full((B, K), -1, dtype=torch.int32, device="cuda")
    got_K = b.sr_select_topk_l2_static(x.data_ptr(), B, L, D, b.SR_BF16, r, idx.data_ptr(),
                                       torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    assert got_K == K
    return idx.cpu().numpy()


def test_static_scratch_topk_matches_workspace_select_twice():
    if not torch.cuda.is_available():
        pytest.fail("CUDA GPU required")
    built_lib()
    from paper_2607_02829_gb300 import binding as b
    # two calls in a row on the same device: the second reuses the static array
    # (holding the first call's scores) with a different shape
    for (B, L, D, r, seed) in [(8, 2048, 1024, 0.25, 1), (1, 16200, 1024, 0.25, 2)]:
        x = _inputs(B, L, D, seed)
        ref = _workspace_select(b, x, r)
        got = _static_select(b, x, r)
        assert np.array_equal(got, ref)
        assert np.all(np.diff(got, axis=1) > 0)
        # against the oracle on the same stored values: equal sets, or differences
        # only inside the fp32 rounding band around the K-th score (the GPU sums
        # squares in fp32, the oracle in fp64; exact ties are exact on both sides)
        K = got.shape[1]
        xf = synth.stored_as_f64(x.cpu())
        exp = o.select_topk_l2(xf, K)
        s = o.token_sq_norms(xf)
        for bb in range(B):
            kth = np.sort(s[bb])[::-1][K - 1]
            diff = set(got[bb].tolist()) ^ set(exp[bb].tolist())
            assert all(abs(s[bb, i] - kth) <= 1e-5 * kth for i in diff), (bb, sorted(diff)[:8])


def test_static_scratch_rejects_oversize_before_launch():
    built_lib()
    from paper_2607_02829_gb300 import binding as b
    with pytest.raises(b.SRError) as e:
        b.sr_select_topk_l2_static(0x1000, 65, 16200, 1024, b.SR_BF16, 0.25, 0x2000, None)
    assert e.value.status == b.SR_ERR_UNSUPPORTED
    assert "1048576" in str(e.value)
