"""Pins for the oracle's tree-masked attention (CPU only).

Each test checks the oracle against something other than itself: a library
routine on the special case where the tree mask is causal (chains), an
ancestor relation built by matrix transitive closure, the Q = 0 closed form,
a hand-worked fixture, and invariances the definition implies.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import workloads as W


def _rand_bf16(rng, shape, scale=1.0):
    return W.bf16(rng.standard_normal(shape, dtype=np.float32) * np.float32(scale))


def _as_f64(t):
    return t.to(torch.float64).numpy()


def _run(q, k, v, parent, tree_len, kv_len, Hq, scale, layout):
    out, lse, sel, st = oracle.tree_attention(
        W.bits(q), W.bits(k), W.bits(v), layout, parent, tree_len, kv_len, Hq, scale)
    assert st == 0
    return out, lse, sel


def _closure_mask(parent):
    """Ancestor-or-self relation by boolean matrix powers of the parent
    adjacency (independent of walking parent links)."""
    T = len(parent)
    A = np.zeros((T, T), dtype=np.int64)
    for i in range(1, T):
        A[i, parent[i]] = 1
    R = np.eye(T, dtype=np.int64)
    P = np.eye(T, dtype=np.int64)
    for _ in range(T):
        P = (P @ A > 0).astype(np.int64)
        R = R | P
    return R.astype(bool)


def _dense_reference(q, k, v, parent, L, T, Hq, Hkv, scale, use_sdpa):
    """Full-sequence attention over [prefix; tree slots] with a boolean mask,
    via numpy fp64 or torch SDPA in fp64. q: [T, Hq, D]; k, v: [L+T, Hkv, D]."""
    tree = _closure_mask(parent[:T])
    mask = np.zeros((T, L + T), dtype=bool)
    mask[:, :L] = True
    mask[:, L:] = tree
    G = Hq // Hkv
    kk = np.repeat(k, G, axis=1)  # [S, Hq, D]
    vv = np.repeat(v, G, axis=1)
    if use_sdpa:
        qt = torch.from_numpy(q).permute(1, 0, 2)  # [Hq, T, D]
        kt = torch.from_numpy(kk).permute(1, 0, 2)
        vt = torch.from_numpy(vv).permute(1, 0, 2)
        o = torch.nn.functional.scaled_dot_product_attention(
            qt, kt, vt, attn_mask=torch.from_numpy(mask), scale=scale)
        s = torch.einsum("htd,hsd->hts", qt, kt) * scale
        s = s.masked_fill(~torch.from_numpy(mask), float("-inf"))
        lse = torch.logsumexp(s, dim=-1)
        return o.permute(1, 0, 2).numpy(), lse.permute(1, 0).numpy()
    s = np.einsum("thd,shd->ths", q, kk) * scale
    s = np.where(mask[:, None, :], s, -np.inf)
    m = s.max(axis=-1, keepdims=True)
    w = np.exp(s - m)
    den = w.sum(axis=-1, keepdims=True)
    o = np.einsum("ths,shd->thd", w / den, vv)
    return o, (m + np.log(den))[..., 0]


@pytest.mark.parametrize("use_sdpa", [False, True])
@pytest.mark.parametrize("L,T,Hq,Hkv,D", [(20, 8, 2, 2, 16), (0, 5, 4, 2, 8), (37, 12, 6, 3, 32)])
def test_chain_matches_causal_library_attention(use_sdpa, L, T, Hq, Hkv, D):
    """On a chain the ancestor mask is causal: compare with dense causal
    attention (numpy fp64 and torch SDPA fp64 with a boolean mask)."""
    rng = np.random.default_rng(1 + L + T)
    q = _rand_bf16(rng, (1, T, Hq, D))
    k = _rand_bf16(rng, (1, L + T, Hkv, D))
    v = _rand_bf16(rng, (1, L + T, Hkv, D))
    parent = W.chain_parent(T)
    scale = 1.0 / math.sqrt(D)
    lay = oracle.KVLayout(L + T, Hkv, D)
    out, lse, sel = _run(q, k, v, parent[None], [T], [L], Hq, scale, lay)
    ro, rl = _dense_reference(_as_f64(q[0]), _as_f64(k[0]), _as_f64(v[0]), parent, L, T, Hq, Hkv,
                              scale, use_sdpa)
    # causal check by construction
    assert (_closure_mask(parent) == np.tril(np.ones((T, T), bool))).all()
    for n, (b, t, h) in enumerate(sel):
        np.testing.assert_allclose(out[n], ro[t, h], rtol=0, atol=1e-12)
        assert abs(lse[n] - rl[t, h]) < 1e-12


@pytest.mark.parametrize("seed", range(4))
def test_random_tree_matches_masked_sdpa(seed):
    """Random trees: oracle vs SDPA with the transitive-closure ancestor mask."""
    rng = np.random.default_rng(100 + seed)
    L, T, Hq, Hkv, D = int(rng.integers(0, 40)), int(rng.integers(1, 20)), 4, 2, 16
    q = _rand_bf16(rng, (1, T, Hq, D))
    k = _rand_bf16(rng, (1, L + T, Hkv, D), scale=2.0)
    v = _rand_bf16(rng, (1, L + T, Hkv, D))
    parent = W.random_tree(rng, T)
    scale = 0.37
    out, lse, sel = _run(q, k, v, parent[None], [T], [L], Hq, scale, oracle.KVLayout(L + T, Hkv, D))
    ro, rl = _dense_reference(_as_f64(q[0]), _as_f64(k[0]), _as_f64(v[0]), parent, L, T, Hq, Hkv,
                              scale, True)
    for n, (b, t, h) in enumerate(sel):
        np.testing.assert_allclose(out[n], ro[t, h], rtol=0, atol=1e-12)
        assert abs(lse[n] - rl[t, h]) < 1e-12


def test_ancestor_mask_matches_closure():
    rng = np.random.default_rng(7)
    for T in [1, 2, 5, 17, 64]:
        parent = W.random_tree(rng, T)
        assert (oracle.ancestor_mask(parent).astype(bool) == _closure_mask(parent)).all()


def test_q_zero_closed_form():
    """Q = 0: equal scores, so out = mean of the visible V rows and
    lse = log(#visible keys)."""
    rng = np.random.default_rng(3)
    L, T, Hq, Hkv, D = 13, 9, 3, 1, 8
    parent = W.random_tree(rng, T)
    q = torch.zeros((1, T, Hq, D), dtype=torch.bfloat16)
    k = _rand_bf16(rng, (1, L + T, Hkv, D))
    v = _rand_bf16(rng, (1, L + T, Hkv, D))
    out, lse, sel = _run(q, k, v, parent[None], [T], [L], Hq, 0.125, oracle.KVLayout(L + T, Hkv, D))
    vv = _as_f64(v[0, :, 0])
    for n, (b, t, h) in enumerate(sel):
        anc = []
        a = t
        while a >= 0:
            anc.append(a)
            a = parent[a]
        rows = list(range(L)) + [L + a for a in anc]
        np.testing.assert_allclose(out[n], vv[rows].mean(axis=0), rtol=0, atol=1e-13)
        assert abs(lse[n] - math.log(len(rows))) < 1e-13


def test_golden_five_node_tree(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "five_node_tree.json")))
    parent = np.array(g["parent"], np.int32)
    mask = oracle.ancestor_mask(parent)
    assert ["".join(str(int(x)) for x in row) for row in mask] == g["ancestor_mask"]
    z = g["attention_q_zero"]
    T, D, L = len(parent), 2, z["kv_len"]
    q = torch.zeros((1, T, 1, D), dtype=torch.bfloat16)
    k = torch.zeros((1, L + T, 1, D), dtype=torch.bfloat16)
    v = torch.tensor(z["v_rows"], dtype=torch.float32).to(torch.bfloat16).reshape(1, T, 1, D)
    out, lse, sel = _run(q, k, v, parent[None], [T], [L], 1, 1.0, oracle.KVLayout(L + T, 1, D))
    np.testing.assert_allclose(out, np.array(z["out"]), rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, np.array(z["lse"]), rtol=0, atol=1e-12)


def test_single_key():
    """kv_len 0 and a root-only tree: the root sees only itself."""
    rng = np.random.default_rng(5)
    q = _rand_bf16(rng, (1, 1, 2, 8))
    k = _rand_bf16(rng, (1, 1, 2, 8))
    v = _rand_bf16(rng, (1, 1, 2, 8))
    out, lse, sel = _run(q, k, v, np.array([[-1]], np.int32), [1], [0], 2, 0.5,
                         oracle.KVLayout(1, 2, 8))
    for n, (b, t, h) in enumerate(sel):
        np.testing.assert_array_equal(out[n], _as_f64(v[0, 0, h]))
        s = 0.5 * float((_as_f64(q[0, 0, h]) * _as_f64(k[0, 0, h])).sum())
        assert abs(lse[n] - s) < 1e-12


def test_prefix_permutation_invariance():
    """Softmax attention is a set function of the visible keys: permuting the
    prefix slots (K and V together) leaves every output unchanged."""
    rng = np.random.default_rng(11)
    L, T, Hq, Hkv, D = 50, 10, 2, 2, 16
    parent = W.random_tree(rng, T)
    q = _rand_bf16(rng, (1, T, Hq, D))
    k = _rand_bf16(rng, (1, L + T, Hkv, D))
    v = _rand_bf16(rng, (1, L + T, Hkv, D))
    lay = oracle.KVLayout(L + T, Hkv, D)
    o1, l1, _ = _run(q, k, v, parent[None], [T], [L], Hq, 0.25, lay)
    perm = torch.from_numpy(np.concatenate([rng.permutation(L), np.arange(L, L + T)]))
    o2, l2, _ = _run(q, k[:, perm], v[:, perm], parent[None], [T], [L], Hq, 0.25, lay)
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-12)


def test_gqa_equals_mha_with_repeated_kv():
    """A GQA query head h uses KV head h // G: identical to MHA on K/V heads
    repeated G times."""
    rng = np.random.default_rng(12)
    L, T, Hq, Hkv, D = 30, 7, 6, 2, 16
    parent = W.random_tree(rng, T)
    q = _rand_bf16(rng, (1, T, Hq, D))
    k = _rand_bf16(rng, (1, L + T, Hkv, D))
    v = _rand_bf16(rng, (1, L + T, Hkv, D))
    o1, l1, _ = _run(q, k, v, parent[None], [T], [L], Hq, 0.3, oracle.KVLayout(L + T, Hkv, D))
    kr = k.repeat_interleave(Hq // Hkv, dim=2)
    vr = v.repeat_interleave(Hq // Hkv, dim=2)
    o2, l2, _ = _run(q, kr, vr, parent[None], [T], [L], Hq, 0.3, oracle.KVLayout(L + T, Hq, D))
    np.testing.assert_array_equal(o1, o2)
    np.testing.assert_array_equal(l1, l2)


def test_paged_equals_contiguous():
    """The same per-sequence data placed in shuffled 64-token pages."""
    rng = np.random.default_rng(13)
    B, Hq, Hkv, D, T_max, page = 3, 4, 2, 8, 6, 64
    L_b = np.array([100, 0, 200], np.int32)
    T_b = np.array([6, 3, 5], np.int32)
    cap = 320
    parent = np.full((B, T_max), -1, np.int32)
    for b in range(B):
        parent[b, :T_b[b]] = W.random_tree(rng, int(T_b[b]))
    q = _rand_bf16(rng, (B, T_max, Hq, D))
    k = _rand_bf16(rng, (B, cap, Hkv, D))
    v = _rand_bf16(rng, (B, cap, Hkv, D))
    o1, l1, s1 = _run(q, k, v, parent, T_b, L_b, Hq, 0.35, oracle.KVLayout(cap, Hkv, D))
    pps = cap // page
    perm = rng.permutation(B * pps).astype(np.int32)
    table = perm.reshape(B, pps)
    kp = torch.empty((B * pps, page, Hkv, D), dtype=torch.bfloat16)
    vp = torch.empty_like(kp)
    for b in range(B):
        for j in range(pps):
            kp[table[b, j]] = k[b, j * page:(j + 1) * page]
            vp[table[b, j]] = v[b, j * page:(j + 1) * page]
    lay = oracle.KVLayout(cap, Hkv, D, page_table=table, page_size=page, num_pages=B * pps)
    o2, l2, s2 = _run(q, kp, vp, parent, T_b, L_b, Hq, 0.35, lay)
    np.testing.assert_array_equal(s1, s2)
    np.testing.assert_array_equal(o1, o2)
    np.testing.assert_array_equal(l1, l2)


def test_bad_data_reported():
    rng = np.random.default_rng(14)
    q = _rand_bf16(rng, (1, 3, 1, 8))
    k = _rand_bf16(rng, (1, 8, 1, 8))
    lay = oracle.KVLayout(8, 1, 8)
    _, _, _, st = oracle.tree_attention(W.bits(q), W.bits(k), W.bits(k), lay,
                                        np.array([[-1, 1, 0]]), [3], [2], 1, 1.0)
    assert st & oracle.BAD_PARENT
    _, _, _, st = oracle.tree_attention(W.bits(q), W.bits(k), W.bits(k), lay,
                                        np.array([[-1, 0, 0]]), [3], [6], 1, 1.0)
    assert st & oracle.BAD_KV_LEN
