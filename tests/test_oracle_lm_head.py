"""Pins for the oracle's LM-head argmax (fp64 H W^T, then the argmax), CPU only:
one-hot hidden rows reduce it to numpy's argmax of one weight column, brute
force dot products on a tiny case, a planted winner, and the bf16 widening."""
import numpy as np

import oracle
import workloads as W


def _bits(x):
    return W.bits(W.bf16(np.asarray(x, np.float32)))


def test_one_hot_rows_pick_a_weight_column():
    rng = np.random.default_rng(1)
    V, K = 300, 64
    w = rng.standard_normal((V, K)).astype(np.float32)
    ks = [0, 5, 63, 17]
    h = np.zeros((len(ks), K), np.float32)
    h[np.arange(len(ks)), ks] = 1.0
    idx, mx, _ = oracle.lm_head_argmax(_bits(h), _bits(w))
    wb = W.bf16(w).float().numpy()
    np.testing.assert_array_equal(idx, [int(np.argmax(wb[:, k])) for k in ks])
    np.testing.assert_allclose(mx, [wb[:, k].max() for k in ks])


def test_brute_force_dot_products():
    rng = np.random.default_rng(2)
    rows, V, K = 3, 11, 8
    h = W.bf16(rng.standard_normal((rows, K)).astype(np.float32)).float().numpy()
    w = W.bf16(rng.standard_normal((V, K)).astype(np.float32)).float().numpy()
    idx, mx, logits = oracle.lm_head_argmax(W.bits(W.bf16(h)), W.bits(W.bf16(w)))
    for r in range(rows):
        vals = [sum(float(h[r, k]) * float(w[v, k]) for k in range(K)) for v in range(V)]
        best = max(range(V), key=lambda v: (vals[v], -v))
        assert idx[r] == best
        np.testing.assert_allclose(logits[r], vals, rtol=0, atol=1e-12)


def test_planted_winner_and_ties_to_lowest_index():
    rng = np.random.default_rng(3)
    V, K = 50, 32
    w = rng.standard_normal((V, K)).astype(np.float32) * 0.1
    h = rng.standard_normal((4, K)).astype(np.float32)
    w[7] = h[0] * 2.0      # row 0 aligns with token 7
    w[9] = h[1] * 2.0      # rows 1 and 2 tie between 9 and 30 (the same weight row)
    w[30] = h[1] * 2.0
    h[2] = h[1]
    idx, _, _ = oracle.lm_head_argmax(_bits(h), _bits(w))
    assert idx[0] == 7 and idx[1] == 9 and idx[2] == 9
