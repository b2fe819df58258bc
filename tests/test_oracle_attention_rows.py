"""Pins for the oracle's attention without a tree and its row entropy (CPU):
torch's scaled_dot_product_attention (no mask, and is_causal) for the output,
scipy's entropy of the softmax row for the entropy, and closed forms (equal
scores give the mean of V and entropy ln n)."""
import numpy as np
import scipy.special
import scipy.stats
import torch

import oracle


def _data(rng, B, T, Hq, Hkv, D, cap):
    q = rng.standard_normal((B, T, Hq, D))
    k = rng.standard_normal((B, cap, Hkv, D))
    v = rng.standard_normal((B, cap, Hkv, D))
    return q, k, v


def test_full_matches_sdpa_and_entropy():
    rng = np.random.default_rng(1)
    B, T, Hq, Hkv, D, cap = 2, 5, 4, 2, 16, 40
    q, k, v = _data(rng, B, T, Hq, Hkv, D, cap)
    kv_len = np.array([40, 17])
    sel = [(b, t, h) for b in range(B) for t in range(T) for h in range(Hq)]
    out, lse, ent = oracle.attention_rows(q, k, v, [T, T], kv_len, 0.25, False, sel)
    for i, (b, t, h) in enumerate(sel):
        n, g = kv_len[b], h // 2
        qt = torch.from_numpy(q[b, t, h])[None, None, None]
        kt = torch.from_numpy(k[b, :n, g])[None, None]
        vt = torch.from_numpy(v[b, :n, g])[None, None]
        ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, scale=0.25)[0, 0, 0].numpy()
        np.testing.assert_allclose(out[i], ref, rtol=1e-10, atol=1e-12)
        srow = 0.25 * (k[b, :n, g] @ q[b, t, h])
        np.testing.assert_allclose(lse[i], scipy.special.logsumexp(srow), rtol=1e-12)
        np.testing.assert_allclose(ent[i], scipy.stats.entropy(scipy.special.softmax(srow)), rtol=1e-10)


def test_causal_matches_sdpa_is_causal():
    rng = np.random.default_rng(2)
    B, T, H, D = 1, 12, 2, 8
    q, k, v = _data(rng, B, T, H, H, D, T)
    sel = [(0, t, h) for t in range(T) for h in range(H)]
    out, _, ent = oracle.attention_rows(q, k, v, [T], [0], 0.3, True, sel)
    qt = torch.from_numpy(q).transpose(1, 2)
    kt = torch.from_numpy(k).transpose(1, 2)
    vt = torch.from_numpy(v).transpose(1, 2)
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True, scale=0.3)
    ref = ref.transpose(1, 2).numpy()
    for i, (b, t, h) in enumerate(sel):
        np.testing.assert_allclose(out[i], ref[b, t, h], rtol=1e-10, atol=1e-12)
    assert ent[0] == 0.0  # the first row sees one key


def test_equal_scores_closed_form():
    rng = np.random.default_rng(3)
    q = np.zeros((1, 3, 1, 8))
    k = rng.standard_normal((1, 50, 1, 8))
    v = rng.standard_normal((1, 50, 1, 8))
    out, lse, ent = oracle.attention_rows(q, k, v, [3], [50], 1.0, False, [(0, t, 0) for t in range(3)])
    np.testing.assert_allclose(out, np.tile(v[0, :, 0].mean(axis=0), (3, 1)), rtol=1e-12)
    np.testing.assert_allclose(ent, np.log(50.0), rtol=1e-12)
    np.testing.assert_allclose(lse, np.log(50.0), rtol=1e-12)
