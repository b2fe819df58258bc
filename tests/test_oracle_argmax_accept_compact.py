"""Pins for the oracle's argmax, acceptance walk and KV compaction (CPU only)."""
import itertools
import json
import os

import numpy as np
import pytest
import torch

import oracle
import workloads as W


# ---------------------------------------------------------------- argmax
@pytest.mark.parametrize("V", [1, 7, 1024, 4097])
def test_argmax_f32_matches_numpy(V):
    rng = np.random.default_rng(V)
    x = rng.standard_normal((33, V)).astype(np.float32)
    np.testing.assert_array_equal(oracle.argmax(x), np.argmax(x, axis=1))


def test_argmax_bf16_matches_numpy():
    rng = np.random.default_rng(2)
    t = W.bf16(rng.standard_normal((20, 3000), dtype=np.float32))
    np.testing.assert_array_equal(oracle.argmax(W.bits(t), bf16_bits=True),
                                  np.argmax(t.float().numpy(), axis=1))


def test_argmax_ties_nan_and_signed_zero():
    nan, inf = np.nan, np.inf
    rows = np.array([
        [1, 3, 3, 2],           # tie -> first
        [5, 5, 5, 5],           # all equal -> 0
        [-0.0, 0.0, -1, -2],    # +0 == -0 -> first
        [-1, -0.0, 0.0, -2],
        [1, nan, 9, nan],       # NaN beats numbers, first NaN
        [-inf, -inf, -inf, -inf],
        [-inf, inf, inf, 3],
        [nan, nan, 1, 2],
    ], dtype=np.float32)
    expect = [1, 0, 0, 1, 1, 0, 1, 0]
    np.testing.assert_array_equal(oracle.argmax(rows), expect)
    np.testing.assert_array_equal(np.argmax(rows, axis=1), expect)
    np.testing.assert_array_equal(torch.argmax(torch.from_numpy(rows), dim=1).numpy(), expect)
    b = W.bf16(rows)
    np.testing.assert_array_equal(oracle.argmax(W.bits(b), bf16_bits=True), expect)


def test_argmax_row_stride():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((10, 64)).astype(np.float32)
    x[:, 40:] = 100.0  # padding beyond V must be ignored
    np.testing.assert_array_equal(oracle.argmax(x, V=40), np.argmax(x[:, :40], axis=1))


# ---------------------------------------------------------------- acceptance
def _one(parent, tokens, am, L=0, max_path=None):
    parent = np.asarray(parent, np.int32)[None]
    T = parent.shape[1]
    r = oracle.accept_path(np.asarray(am, np.int32)[None], parent,
                           np.asarray(tokens, np.int32)[None], [T], [L],
                           max_path or T + 1)
    n = int(r["accept_len"][0])
    return {"accept_len": n, "path": list(r["path"][0, :n]), "out_tokens": list(r["out_tokens"][0, :n]),
            "new_kv_len": int(r["new_kv_len"][0]), "status": r["status"],
            "path_row": r["path"][0], "tok_row": r["out_tokens"][0]}


def test_golden_five_node_walk(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "five_node_tree.json")))
    r = _one(g["parent"], g["tokens"], g["am"], L=g["kv_len"])
    e = g["expect"]
    assert r["path"] == e["path"] and r["out_tokens"] == e["out_tokens"]
    assert r["accept_len"] == e["accept_len"] and r["new_kv_len"] == e["new_kv_len"]
    assert (r["path_row"][e["accept_len"]:] == -1).all()
    for var in g["variants"]:
        r = _one(g["parent"], var["tokens"], var["am"])
        assert r["path"] == var["expect"]["path"], var["why"]
        assert r["out_tokens"] == var["expect"]["out_tokens"], var["why"]
        assert r["accept_len"] == var["expect"]["accept_len"], var["why"]


def test_paper_chain_rule(golden_dir):
    """Sec. 2: first mismatch at i -> (t_1..t_(i-1), t'_i); all accepted ->
    gamma drafts plus the target's next token."""
    g = json.load(open(os.path.join(golden_dir, "chain_gamma6.json")))
    parent = W.chain_parent(g["gamma"] + 1)
    for c in g["cases"]:
        r = _one(parent, g["tokens"], c["am"])
        assert r["out_tokens"] == c["out_tokens"] and r["accept_len"] == c["accept_len"]
    # every mismatch position of the gamma = 6 chain
    toks = np.array(g["tokens"])
    for i in range(1, g["gamma"] + 2):
        am = list(toks[1:]) + [999]
        if i <= g["gamma"]:
            am[i - 1] = 5000 + i
        r = _one(parent, toks, am)
        assert r["accept_len"] == min(i, g["gamma"] + 1)
        assert r["out_tokens"][:-1] == list(toks[1:r["accept_len"]])


def test_tau_bounds_from_paper_tables(golden_dir):
    """Every mean acceptance length in Table 6 is at most gamma + 1, and some
    exceed gamma (gamma = 4, 5, 6 on MMT-Bench), which is only possible when
    the accepted length counts the target's own token."""
    g = json.load(open(os.path.join(golden_dir, "chain_gamma6.json")))
    above = 0
    for col in ("table6_mmt_tau", "table6_seed_tau"):
        for gamma, tau in g[col].items():
            if gamma == "source":
                continue
            assert tau <= int(gamma) + 1
            above += tau > int(gamma)
    assert above >= 3
    # the walk reaches gamma + 1 exactly when every draft matches
    parent = W.chain_parent(7)
    r = _one(parent, g["tokens"], g["cases"][2]["am"])
    assert r["accept_len"] == g["gamma"] + 1


def _brute_force(parent, tokens, am, max_path):
    """Enumerate every root path by DFS, keep the matching ones, take the
    longest (cut to max_path - 1 drafts), ties to the smallest sequence."""
    T = len(parent)
    kids = [[c for c in range(T) if parent[c] == a] for a in range(T)]
    paths = []

    def dfs(p):
        paths.append(list(p))
        for c in kids[p[-1]]:
            if tokens[c] == am[p[-1]]:
                dfs(p + [c])
    dfs([0])
    n = min(max(len(p) for p in paths) - 1, max_path - 1)
    best = min(p[:n + 1] for p in paths if len(p) >= n + 1)
    return best, [tokens[c] for c in best[1:]] + [am[best[-1]]]


@pytest.mark.parametrize("seed", range(300))
def test_walk_brute_force_small_trees(seed):
    rng = np.random.default_rng(seed)
    T = int(rng.integers(1, 9))
    parent = W.random_tree(rng, T)
    vocab = int(rng.integers(1, 4))  # tiny vocab: many duplicate sibling tokens
    tokens = rng.integers(0, vocab, T)
    am = rng.integers(0, vocab, T)
    max_path = int(rng.integers(1, T + 2))
    path, toks = _brute_force(list(parent), list(tokens), list(am), max_path)
    r = _one(parent, tokens, am, L=5, max_path=max_path)
    assert r["path"] == path and r["out_tokens"] == toks
    assert r["new_kv_len"] == 5 + len(path)


def _first_match_walk(parent, tokens, am):
    """The plain sequential walk: from the root, step to the first child
    carrying the target's token. Equals the longest path when siblings carry
    distinct tokens."""
    cur, path = 0, [0]
    while True:
        nxt = [c for c in range(len(parent)) if parent[c] == cur and tokens[c] == am[cur]]
        if not nxt:
            return path
        cur = nxt[0]
        path.append(cur)


@pytest.mark.parametrize("seed", range(50))
def test_walk_equals_sequential_walk_with_distinct_siblings(seed):
    rng = np.random.default_rng(1000 + seed)
    T = int(rng.integers(2, 65))
    parent = W.random_tree(rng, T)
    tokens = rng.permutation(10 * T)[:T]  # all distinct
    am = np.where(rng.random(T) < 0.8, 0, -1)
    for a in range(T):  # predict one child's token w.p. 0.8
        kids = [c for c in range(T) if parent[c] == a]
        am[a] = tokens[kids[int(rng.integers(len(kids)))]] if kids and am[a] == 0 else 10 * T + 1
    r = _one(parent, tokens, am)
    assert r["path"] == _first_match_walk(parent, tokens, am)
    # invariants
    depth = W.tree_depth(parent, T)
    p = r["path"]
    assert r["accept_len"] <= depth + 1
    assert all(p[i] < p[i + 1] and parent[p[i + 1]] == p[i] for i in range(len(p) - 1))
    assert all(tokens[p[i + 1]] == am[p[i]] for i in range(len(p) - 1))


def test_chain_acceptance_statistics():
    """Chain of depth d, each prediction equal to the next draft w.p. p
    independently: E[accept_len] = sum_{k=0..d} p^k."""
    rng = np.random.default_rng(77)
    d, p, n = 6, 0.75, 20000
    T = d + 1
    parent = np.tile(W.chain_parent(T), (n, 1))
    tokens = rng.integers(0, 1000, (n, T)).astype(np.int32)
    hit = rng.random((n, T)) < p
    am = np.where(hit, np.roll(tokens, -1, axis=1), 1000 + np.arange(T)[None])
    r = oracle.accept_path(am, parent, tokens, np.full(n, T), np.zeros(n), T + 1)
    mean = r["accept_len"].mean()
    expect = sum(p ** k for k in range(d + 1))
    sd = r["accept_len"].std() / np.sqrt(n)
    assert abs(mean - expect) < 5 * sd


def test_walk_bad_trees():
    r = oracle.accept_path(np.zeros((3, 4), np.int32),
                           np.array([[-1, 0, 2, 1], [0, 0, 1, 2], [-1, 0, 0, 0]], np.int32),
                           np.zeros((3, 4), np.int32), [4, 4, 5], [3, 3, 3], 4)
    assert r["status"] & oracle.BAD_PARENT and r["status"] & oracle.BAD_TREE_LEN
    assert list(r["accept_len"]) == [0, 0, 0] and list(r["new_kv_len"]) == [3, 3, 3]
    assert (r["path"] == -1).all() and (r["out_tokens"] == -1).all()


# ---------------------------------------------------------------- compaction
def _paged(k, page, rng):
    B, cap = k.shape[:2]
    pps = cap // page
    table = rng.permutation(B * pps).astype(np.int32).reshape(B, pps)
    kp = np.empty((B * pps, page) + k.shape[2:], k.dtype)
    for b in range(B):
        for j in range(pps):
            kp[table[b, j]] = k[b, j * page:(j + 1) * page]
    return kp, table


@pytest.mark.parametrize("paged", [False, True])
def test_compaction_equals_gather(paged):
    """Slots [L, L+A) become the gather of slots L + path; every other byte
    of every layer stays as it was."""
    rng = np.random.default_rng(21)
    B, cap, Hkv, D, n_layers, page = 4, 128, 2, 8, 3, 64
    k = rng.integers(0, 65536, (n_layers, B, cap, Hkv, D), dtype=np.uint16)
    v = rng.integers(0, 65536, (n_layers, B, cap, Hkv, D), dtype=np.uint16)
    L = np.array([10, 0, 60, 100], np.int32)
    max_path = 6
    path = np.full((B, max_path), -1, np.int32)
    acc = np.array([3, 1, 5, 0], np.int32)
    path[0, :3] = [0, 2, 3]   # in place: slot L+2 is read then overwritten
    path[1, :1] = [0]
    path[2, :5] = [0, 1, 5, 7, 9]  # crosses the page boundary at slot 64
    if paged:
        kl, table = zip(*[_paged(k[i], page, np.random.default_rng(5)) for i in range(n_layers)])
        kin, vin = np.stack(kl), np.stack([_paged(v[i], page, np.random.default_rng(5))[0]
                                            for i in range(n_layers)])
        table = table[0]
        lay = oracle.KVLayout(cap, Hkv, D, page_table=table, page_size=page, num_pages=B * cap // page)
    else:
        kin, vin = k, v
        lay = oracle.KVLayout(cap, Hkv, D)
    stride = kin[0].size
    ko, vo, st = oracle.kv_compact(kin, vin, lay, L, acc, path, n_layers=n_layers, layer_stride=stride)
    assert st == 0
    if paged:  # back to logical order
        def unpage(x):
            out = np.empty_like(k)
            for i in range(n_layers):
                for b in range(B):
                    for j in range(cap // page):
                        out[i, b, j * page:(j + 1) * page] = x[i, table[b, j]]
            return out
        ko, vo = unpage(ko), unpage(vo)
    for src, out in ((k, ko), (v, vo)):
        expect = src.copy()
        for b in range(B):
            for x in range(acc[b]):
                expect[:, b, L[b] + x] = src[:, b, L[b] + path[b, x]]
        np.testing.assert_array_equal(out, expect)


def test_compaction_bad_path_untouched():
    k = np.arange(2 * 16 * 1 * 4, dtype=np.uint16).reshape(2, 16, 1, 4)
    lay = oracle.KVLayout(16, 1, 4)
    path = np.array([[0, 9, -1], [0, 1, -1]], np.int32)
    ko, vo, st = oracle.kv_compact(k, k, lay, np.array([10, 3]), np.array([2, 2]), path)
    assert st & oracle.BAD_KV_LEN
    np.testing.assert_array_equal(ko[0], k[0])
    np.testing.assert_array_equal(ko[1, 4], k[1, 4])
    for bad_path in ([1, 2, -1], [0, 2, 2], [0, 3, 1]):
        ko, _, st = oracle.kv_compact(k, k, lay, np.array([2, 2]), np.array([3, 0]),
                                      np.array([bad_path, [0, 1, 2]], np.int32))
        assert st == oracle.BAD_PATH
        np.testing.assert_array_equal(ko, k)
