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


def _prefix_causal_mask(L, T):
    """[T, L+T] boolean: every prefix slot, then query slot s only for s <= t."""
    m = np.zeros((T, L + T), dtype=bool)
    m[:, :L] = True
    m[:, L:] = np.tril(np.ones((T, T), dtype=bool))
    return m


def test_causal_with_prefix_matches_sdpa_explicit_mask():
    """Causal rows after a committed prefix (Sec. 3.3: a layer's prefill with
    tokens already cached) against torch's SDPA in float64 with an explicit
    [T, L+T] mask built from the definition: all L prefix slots, then the query
    slots up to the row's own. Several prefix lengths, one beyond a 128-key
    tile, one with two KV heads per group. A reading that drops the prefix
    (n = t + 1) or the row's own slot (n = L + t) fails here."""
    rng = np.random.default_rng(4)
    for L, T, Hq, Hkv in ((1, 6, 2, 2), (37, 9, 4, 2), (150, 7, 2, 1), (300, 4, 2, 2)):
        D = 8
        q, k, v = _data(rng, 2, T, Hq, Hkv, D, L + T)
        kv_len = [L, L]
        sel = [(b, t, h) for b in range(2) for t in range(T) for h in range(Hq)]
        out, lse, ent = oracle.attention_rows(q, k, v, [T, T], kv_len, 0.35, True, sel)
        mask = torch.from_numpy(_prefix_causal_mask(L, T))
        G = Hq // Hkv
        for i, (b, t, h) in enumerate(sel):
            g = h // G
            qt = torch.from_numpy(q[b, :, h])[None, None]
            kt = torch.from_numpy(k[b, :L + T, g])[None, None]
            vt = torch.from_numpy(v[b, :L + T, g])[None, None]
            ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask,
                                                                   scale=0.35)[0, 0, t].numpy()
            np.testing.assert_allclose(out[i], ref, rtol=1e-10, atol=1e-12)
            srow = 0.35 * (k[b, :L + T, g] @ q[b, t, h])
            srow = np.where(mask[t].numpy(), srow, -np.inf)
            np.testing.assert_allclose(lse[i], scipy.special.logsumexp(srow), rtol=1e-12)
            pr = scipy.special.softmax(srow)
            np.testing.assert_allclose(ent[i], scipy.stats.entropy(pr[pr > 0]), rtol=1e-10, atol=1e-14)


def test_causal_with_prefix_equal_scores_closed_form():
    """Q = 0 makes every allowed score equal: row t after a prefix of L slots
    sees exactly L + t + 1 keys, so out = the mean of V over slots 0 .. L+t and
    lse = entropy = ln(L + t + 1)."""
    rng = np.random.default_rng(5)
    for L in (0, 3, 129, 200):
        T = 5
        q = np.zeros((1, T, 1, 4))
        k = rng.standard_normal((1, L + T, 1, 4))
        v = rng.standard_normal((1, L + T, 1, 4))
        sel = [(0, t, 0) for t in range(T)]
        out, lse, ent = oracle.attention_rows(q, k, v, [T], [L], 0.7, True, sel)
        for t in range(T):
            n = L + t + 1
            np.testing.assert_allclose(out[t], v[0, :n, 0].mean(axis=0), rtol=1e-12, atol=1e-14)
            np.testing.assert_allclose(lse[t], np.log(n), rtol=1e-12, atol=1e-14)
            np.testing.assert_allclose(ent[t], np.log(n), rtol=1e-12, atol=1e-14)
