"""Pins for the oracle's visual-token importance (Eq. 2) and top-r selection,
CPU only: uniform attention (a closed form), one-hot attention rows (counts by
numpy's bincount), rows that sum to one (the importances over all K columns sum
to one), the bf16 widening, and the selection's tie rule."""
import numpy as np

import oracle
import workloads as W


def test_uniform_attention_closed_form():
    B, H, Q, K = 2, 3, 5, 40
    a = np.full((B, H, Q, K), 1.0 / K, np.float32)
    imp, keep = oracle.visual_importance(a, 4, 30, 7)
    np.testing.assert_allclose(imp, np.float32(1.0 / K), rtol=1e-12)
    np.testing.assert_array_equal(keep, np.tile(np.arange(4, 11), (B, 1)))  # ties: lowest positions


def test_one_hot_rows_count_attention():
    rng = np.random.default_rng(1)
    B, H, Q, K = 2, 4, 50, 64
    tgt = rng.integers(0, K, (B, H, Q))
    a = np.zeros((B, H, Q, K), np.float32)
    np.put_along_axis(a, tgt[..., None], 1.0, axis=3)
    imp, keep = oracle.visual_importance(a, 0, K, 5)
    for b in range(B):
        cnt = np.bincount(tgt[b].ravel(), minlength=K) / (H * Q)
        np.testing.assert_allclose(imp[b], cnt, rtol=0, atol=1e-15)
        order = sorted(range(K), key=lambda j: (-cnt[j], j))[:5]
        np.testing.assert_array_equal(keep[b], sorted(order))


def test_softmax_rows_sum_to_one_and_bf16():
    import torch
    rng = np.random.default_rng(2)
    B, H, Q, K = 1, 2, 30, 30
    s = torch.from_numpy(rng.standard_normal((B, H, Q, K)).astype(np.float32))
    causal = torch.ones(Q, K, dtype=torch.bool).tril()
    a = torch.softmax(s.masked_fill(~causal, float("-inf")), dim=-1)
    imp, _ = oracle.visual_importance(a.numpy(), 0, K, 3)
    assert abs(imp.sum() - 1.0) < 1e-6  # every row of A sums to one
    b = W.bf16(a.numpy())
    imp_b, _ = oracle.visual_importance(W.bits(b), 0, K, 3, bf16_bits=True)
    np.testing.assert_allclose(imp_b, oracle.visual_importance(b.float().numpy(), 0, K, 3)[0], rtol=1e-12)


def test_top_r_ties_and_nan():
    v = np.array([[0.5, 0.7, 0.7, 0.1, 0.7, np.nan]])
    np.testing.assert_array_equal(oracle.top_r(v, 1), [[5]])          # NaN above everything
    np.testing.assert_array_equal(oracle.top_r(v, 3), [[1, 2, 5]])    # equal values: lower positions
    np.testing.assert_array_equal(oracle.top_r(v, 4, v0=10), [[11, 12, 14, 15]])
