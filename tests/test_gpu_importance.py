"""GPU parity of the visual-token importance (Eq. 2) and top-r selection
against the fp64 oracle: importances within f32 summation error; the kept
positions exactly equal to the oracle's selection applied to the kernel's own
f32 importances (the decision taken in the kernel's precision), and equal to
the exact selection wherever no near-tie straddles the cut."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dreams():
    import paper_2606_00535_gb300 as d
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    d._lib()
    return d


def _attn(B, H, Q, K, v0, n_vis, seed, dtype):
    """Causal softmax attention with a per-visual-token salience bias."""
    g = torch.Generator(device="cuda").manual_seed(seed)
    s = torch.randn((B, H, Q, K), device="cuda", generator=g)
    s[..., v0:v0 + n_vis] += 1.5 * torch.randn((B, 1, 1, n_vis), device="cuda", generator=g)
    qpos = torch.arange(Q, device="cuda")[:, None] + (K - Q)
    mask = torch.arange(K, device="cuda")[None, :] <= qpos
    a = torch.softmax(s.masked_fill(~mask, float("-inf")), dim=-1)
    return a.to(dtype).contiguous()


def _check(a, v0, n_vis, r, imp, keep):
    bf16 = a.dtype == torch.bfloat16
    ref_imp, ref_keep = oracle.visual_importance(W.bits(a.cpu()) if bf16 else a.cpu().numpy(), v0, n_vis, r,
                                                 bf16_bits=bf16)
    g = imp.cpu().numpy().astype(np.float64)
    rel = np.abs(g - ref_imp) / np.maximum(np.abs(ref_imp), 1e-12)
    assert rel.max() < 1e-4, rel.max()
    k = keep.cpu().numpy()
    np.testing.assert_array_equal(k, oracle.top_r(imp.cpu().numpy(), r, v0))  # the kernel's own decision
    return (k == ref_keep).mean()


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("B,H,Q,K,v0,n_vis,r", [
    (1, 8, 256, 256, 16, 200, 40),     # one column block, aligned
    (2, 4, 100, 300, 3, 290, 1),       # unaligned visual start: scalar loads
    (1, 2, 64, 4200, 40, 4100, 4100),  # two column blocks, keep everything
    (3, 1, 1, 50, 0, 50, 25),          # one query row
])
def test_importance_matches_oracle(dreams, dtype, B, H, Q, K, v0, n_vis, r):
    a = _attn(B, H, Q, K, v0, n_vis, seed=B * 31 + K, dtype=dtype)
    imp, keep = dreams.visual_importance(a, v0, n_vis, r)
    torch.cuda.synchronize()
    agree = _check(a, v0, n_vis, r, imp, keep)
    assert agree > 0.98


def test_importance_ties_and_repeat(dreams):
    """Equal importances: the lower positions are kept; a second call on the
    same workspace gives the same result."""
    B, H, Q, K = 1, 2, 8, 64
    a = torch.full((B, H, Q, K), 1.0 / K, device="cuda")
    ws = torch.zeros(dreams._lib().dreams_visual_importance_workspace_size(B, H, Q, K), dtype=torch.uint8,
                     device="cuda")
    for _ in range(2):
        imp, keep = dreams.visual_importance(a, 0, K, 10, workspace=ws)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(keep.cpu().numpy(), [list(range(10))])


def test_importance_llava_shape(dreams):
    """LLaVA-7B-shaped prefill: 32 heads, 3392 positions, 2880 visual tokens
    after a 35-token prompt, keep 576."""
    B, H, Q, K, v0, n_vis, r = 1, 32, 3392, 3392, 35, 2880, 576
    a = _attn(B, H, Q, K, v0, n_vis, seed=7, dtype=torch.bfloat16)
    imp, keep = dreams.visual_importance(a, v0, n_vis, r)
    torch.cuda.synchronize()
    agree = _check(a, v0, n_vis, r, imp, keep)
    assert agree > 0.99
