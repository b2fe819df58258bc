"""GPU parity of the speculative-sampling verification tail
(dreams_verify_step_speculative) against the fp64 oracle: a draft is accepted
with probability min(1, r/q) against the current residual r (the target p at
first), a rejection renormalises max(0, r - q), and the bonus is drawn from
what is left (Leviathan et al.'s rule, cited in Sec. 1; verification at T = 1,
Table 2).

Every decision compares a uniform with a number the kernel computes in f32
and the oracle in fp64. A uniform closer to its threshold than MARGIN could
go either way within rounding, so the tests redraw the uniforms of such
sequences (the oracle reports each sequence's smallest distance) and then
require bit-identical walks, outputs and compacted caches. The defining
property, that the first emitted token is distributed as the target whatever
the draft, is also checked on the kernel's own outputs by sampling."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import layout, to_gpu

pytestmark = pytest.mark.gpu

MARGIN = 1e-4  # probability (draws) or ratio (acceptance tests) units


@pytest.fixture(scope="module")
def dreams():
    import paper_2606_00535_gb300 as d
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    d._lib()
    return d


def _status():
    return torch.zeros(1, dtype=torch.int32, device="cuda")


def _softmax(x, tau):
    x = np.asarray(x, np.float64) / tau
    w = np.exp(x - x.max(axis=-1, keepdims=True))
    return w / w.sum(axis=-1, keepdims=True)


def _oracle_clean(tgt_np, drf_np, par, tok, tl, kl, max_path, tau, rng, bf16=False, tries=30):
    """Uniforms for which no decision of the oracle lies within MARGIN of its
    threshold, and the oracle's result on them."""
    B, T = par.shape
    u_acc = rng.random((B, T), dtype=np.float32)
    u_res = rng.random((B, T), dtype=np.float32)
    for _ in range(tries):
        ref = oracle.spec_path(tgt_np, drf_np, par, tok, tl, kl, max_path, tau, u_acc, u_res, bf16_bits=bf16)
        close = ref["margin"] < MARGIN
        if not close.any():
            return u_acc, u_res, ref
        u_acc[close] = rng.random((int(close.sum()), T), dtype=np.float32)
        u_res[close] = rng.random((int(close.sum()), T), dtype=np.float32)
    raise AssertionError("could not draw uniforms away from every threshold")


def _draft_tokens(rng, drf, par, tl, tau):
    """Children's tokens drawn i.i.d. from their parent's draft distribution,
    as a drafter would produce them."""
    B, T = par.shape
    tok = np.zeros((B, T), np.int32)
    for b in range(B):
        for c in range(1, int(tl[b])):
            q = _softmax(drf[b, par[b, c]], tau)
            tok[b, c] = rng.choice(q.shape[-1], p=q)
    return tok


def _run(dreams, tgt, drf, par, tok, tl, kl, k, v, max_path, tau, u_acc, u_res, page_table=None):
    kv = dreams.KVCache(k, v, page_table)
    tree = dreams.Tree(torch.from_numpy(par).cuda(), torch.from_numpy(tok).cuda(), torch.from_numpy(tl).cuda(),
                       torch.from_numpy(kl).cuda())
    st = _status()
    r = dreams.verify_step_speculative(tgt, drf, tree, kv, max_path, tau, torch.from_numpy(u_acc).cuda(),
                                       torch.from_numpy(u_res).cuda(), status=st)
    torch.cuda.synchronize()
    return r, int(st.item())


def _compare(r, ref):
    for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
        np.testing.assert_array_equal(r[key].cpu().numpy(), ref[key], err_msg=key)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("V", [777, 3000])
def test_speculative_matches_oracle(dreams, dtype, V):
    """Random trees of ragged lengths, drafts drawn from the draft
    distribution (draft logits = target + noise), a max_path that cuts some
    walks; V spans one ragged segment or several with a ragged tail."""
    rng = np.random.default_rng(V + (7 if dtype == "bf16" else 0))
    B, T, Hkv, D, cap, tau, max_path = 48, 24, 2, 64, 128, 1.0, 6
    par = np.full((B, T), -1, np.int32)
    tl = rng.integers(1, T + 1, B).astype(np.int32)
    tl[:4] = T
    for b in range(B):
        par[b, :tl[b]] = W.random_tree(rng, int(tl[b]))
    kl = rng.integers(0, cap - T + 1, B).astype(np.int32)
    tgt32 = (2.0 * rng.standard_normal((B, T, V))).astype(np.float32)
    drf32 = (tgt32 + 0.8 * rng.standard_normal((B, T, V))).astype(np.float32)
    if dtype == "bf16":
        tgt_t, drf_t = W.bf16(tgt32), W.bf16(drf32)
        tgt_np, drf_np = W.bits(tgt_t), W.bits(drf_t)
        tok = _draft_tokens(rng, drf_t.float().numpy(), par, tl, tau)
    else:
        tgt_t, drf_t = torch.from_numpy(tgt32), torch.from_numpy(drf32)
        tgt_np, drf_np = tgt32, drf32
        tok = _draft_tokens(rng, drf32, par, tl, tau)
    u_acc, u_res, ref = _oracle_clean(tgt_np, drf_np, par, tok, tl, kl, max_path, tau, rng, bf16=dtype == "bf16")
    assert ref["status"] == 0
    # the case mixes accepted drafts, rejections and cut walks
    assert (ref["accept_len"] == 1).any() and (ref["accept_len"] >= 3).any()
    k = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    v = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    kg, vg = k.cuda(), v.cuda()
    r, st = _run(dreams, tgt_t.cuda(), drf_t.cuda(), par, tok, tl, kl, kg, vg, max_path, tau, u_acc, u_res)
    assert st == 0
    _compare(r, ref)
    ko, vo, ost = oracle.kv_compact(W.bits(k), W.bits(v), oracle.KVLayout(cap, Hkv, D), kl, ref["accept_len"],
                                    ref["path"])
    assert ost == 0
    assert np.array_equal(W.bits(kg.cpu()), ko) and np.array_equal(W.bits(vg.cpu()), vo)


def test_speculative_batched_workload(dreams):
    """The batched serving workload (16 sequences, paged cache, trees of
    32-64 nodes, bf16 logits over a 128256-entry vocabulary) with draft logits
    = target + N(0, 0.5) noise, at temperature 1."""
    w = W.make("batched")
    g = to_gpu(w)
    rng = np.random.default_rng(41)
    noise = torch.from_numpy((0.5 * rng.standard_normal((w.B, w.T_max, w.V), dtype=np.float32)))
    drf = (w.logits.float() + noise).to(torch.bfloat16)
    del noise
    par, tok, tl, kl = (x.numpy() for x in (w.parent, w.tokens, w.tree_len, w.kv_len))
    u_acc, u_res, ref = _oracle_clean(W.bits(w.logits), W.bits(drf), par, tok, tl, kl, w.max_path, 1.0, rng,
                                      bf16=True)
    assert ref["status"] == 0
    r, st = _run(dreams, g["logits"], drf.cuda(), par, tok, tl, kl, g["k"], g["v"], w.max_path, 1.0, u_acc, u_res,
                 g["page_table"])
    assert st == 0
    _compare(r, ref)
    assert (ref["accept_len"] >= 2).any()
    ko, vo, ost = oracle.kv_compact(W.bits(w.k), W.bits(w.v), layout(w), kl, ref["accept_len"], ref["path"])
    assert ost == 0
    assert np.array_equal(W.bits(g["k"].cpu()), ko) and np.array_equal(W.bits(g["v"].cpu()), vo)


def test_speculative_low_temperature_is_greedy(dreams):
    """At a tiny temperature both distributions are one-hot at their argmax:
    a draft is accepted exactly when it is the target's argmax and the bonus
    is the argmax, whatever the draft rows, so the step reproduces the greedy
    step (verify_step) on the LLaVA-7B-shaped workload."""
    w = W.make("llava7b")
    g1, g2 = to_gpu(w), to_gpu(w)
    rng = np.random.default_rng(5)
    drf = torch.from_numpy((2.0 * rng.standard_normal((w.B, w.T_max, w.V))).astype(np.float32)).cuda()
    u_acc = torch.from_numpy(rng.random((w.B, w.T_max), dtype=np.float32)).cuda()
    u_res = torch.from_numpy(rng.random((w.B, w.T_max), dtype=np.float32)).cuda()
    r_s = dreams.verify_step_speculative(g1["logits"], drf, g1["tree"], g1["kv"], w.max_path, 1e-30, u_acc, u_res)
    r_g = dreams.verify_step(g2["logits"], g2["tree"], g2["kv"], w.max_path)
    torch.cuda.synchronize()
    for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
        assert torch.equal(r_s[key], r_g[key]), key
    assert torch.equal(g1["k"], g2["k"]) and torch.equal(g1["v"], g2["v"])


@pytest.mark.parametrize("k", [1, 3])
def test_first_token_is_distributed_as_the_target(dreams, k):
    """200 000 one-node trees with k children drawn i.i.d. from q: the kernel's
    first emitted token has the target's distribution p (4.5 standard errors),
    although q puts most of its mass elsewhere; and the kernel's outputs equal
    the oracle's on every sequence with no decision within MARGIN."""
    rng = np.random.default_rng(60 + k)
    n, V, T = 200_000, 5, k + 1
    p_logits = np.array([2.0, 0.5, -1.0, 1.0, -0.3], np.float32)
    q_logits = np.array([-0.5, 1.8, 0.2, -1.0, 1.1], np.float32)
    p = _softmax(p_logits, 1.0)
    q = _softmax(q_logits, 1.0)
    par = np.zeros((n, T), np.int32)
    par[:, 0] = -1
    tok = np.zeros((n, T), np.int32)
    tok[:, 1:] = rng.choice(V, size=(n, k), p=q)
    tgt = np.broadcast_to(p_logits, (n, T, V)).copy()
    drf = np.broadcast_to(q_logits, (n, T, V)).copy()
    tl = np.full(n, T, np.int32)
    kl = np.zeros(n, np.int32)
    u_acc = rng.random((n, T), dtype=np.float32)
    u_res = rng.random((n, T), dtype=np.float32)
    kc = torch.zeros((n, T, 1, 8), dtype=torch.bfloat16, device="cuda")
    r, st = _run(dreams, torch.from_numpy(tgt).cuda(), torch.from_numpy(drf).cuda(), par, tok, tl, kl, kc,
                 kc.clone(), 3, 1.0, u_acc, u_res)
    assert st == 0
    first = r["out_tokens"][:, 0].cpu().numpy()
    freq = np.bincount(first, minlength=V) / n
    assert (np.abs(freq - p) <= 4.5 * np.sqrt(p * (1 - p) / n)).all(), (freq, p)
    ref = oracle.spec_path(tgt, drf, par, tok, tl, kl, 3, 1.0, u_acc, u_res)
    ok = ref["margin"] >= MARGIN
    assert ok.mean() > 0.99
    for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
        np.testing.assert_array_equal(r[key].cpu().numpy()[ok], ref[key][ok], err_msg=key)


def test_leaf_root_cut_and_zero_residual(dreams):
    """Sequences whose root is a leaf, a walk cut at max_path = 1, draft
    tokens outside the vocabulary (always rejected), and rejections whose
    residual sum is exactly zero (target == draft, drafts of zero probability
    under both: the residual stays the target)."""
    rng = np.random.default_rng(77)
    B, T, V, cap = 24, 8, 2100, 64
    par = np.full((B, T), -1, np.int32)
    tl = np.full(B, T, np.int32)
    tl[:6] = 1
    for b in range(6, B):
        par[b] = W.random_tree(rng, T)
    tgt = (1.5 * rng.standard_normal((B, T, V))).astype(np.float32)
    drf = (tgt + 0.6 * rng.standard_normal((B, T, V))).astype(np.float32)
    tok = _draft_tokens(rng, drf, par, tl, 1.0)
    tok[6:9, 1] = V + 3
    tok[9, 1] = -2
    # zero residual: rows 12..17 have target == draft with a support of 40
    # entries, every other logit so low that exp underflows in fp64 as well
    for b in range(12, 18):
        row = np.full(V, -1e4, np.float32)
        sup = rng.choice(V, 40, replace=False)
        row[sup] = rng.standard_normal(40).astype(np.float32)
        tgt[b] = row
        drf[b] = row
        off = np.setdiff1d(np.arange(V), sup)
        for c in range(1, T):
            tok[b, c] = rng.choice(off) if c % 3 else rng.choice(sup)
    kl = rng.integers(0, cap - T + 1, B).astype(np.int32)
    for max_path in (1, 5):
        u_acc, u_res, ref = _oracle_clean(tgt, drf, par, tok, tl, kl, max_path, 1.0, rng)
        k = W.bf16(rng.standard_normal((B, cap, 1, 16), dtype=np.float32))
        v = W.bf16(rng.standard_normal((B, cap, 1, 16), dtype=np.float32))
        kg, vg = k.cuda(), v.cuda()
        r, st = _run(dreams, torch.from_numpy(tgt).cuda(), torch.from_numpy(drf).cuda(), par, tok, tl, kl, kg, vg,
                     max_path, 1.0, u_acc, u_res)
        assert st == 0
        _compare(r, ref)
        if max_path == 1:
            assert (ref["accept_len"] == 1).all()
        ko, vo, _ = oracle.kv_compact(W.bits(k), W.bits(v), oracle.KVLayout(cap, 1, 16), kl, ref["accept_len"],
                                      ref["path"])
        assert np.array_equal(W.bits(kg.cpu()), ko) and np.array_equal(W.bits(vg.cpu()), vo)
    # the bonus at a leaf root is one draw from the target itself
    leaf = slice(0, 6)
    samp = oracle.sample(tgt[leaf, 0], 1.0, u_res[leaf, 0])
    np.testing.assert_array_equal(r["out_tokens"][leaf, 0].cpu().numpy(), samp)


def test_malformed_tree_is_flagged(dreams):
    """A parent after its child: the sequence is flagged, gets accept_len 0,
    rows of -1 and its old kv_len, and its cache is left alone; the other
    sequences are verified as usual."""
    rng = np.random.default_rng(88)
    B, T, V, cap = 3, 10, 500, 32
    par = np.stack([W.random_tree(rng, T) for _ in range(B)]).astype(np.int32)
    par[1, 4] = 6
    tl = np.full(B, T, np.int32)
    tgt = rng.standard_normal((B, T, V)).astype(np.float32)
    drf = (tgt + 0.3 * rng.standard_normal((B, T, V))).astype(np.float32)
    tok = rng.integers(0, V, (B, T)).astype(np.int32)
    kl = np.array([5, 9, 12], np.int32)
    good = par.copy()
    good[1] = W.chain_parent(T)
    u_acc, u_res, ref = _oracle_clean(tgt, drf, good, tok, tl, kl, 4, 1.0, rng)
    k = W.bf16(rng.standard_normal((B, cap, 1, 8), dtype=np.float32))
    kg, vg = k.cuda(), k.clone().cuda()
    r, st = _run(dreams, torch.from_numpy(tgt).cuda(), torch.from_numpy(drf).cuda(), par, tok, tl, kl, kg, vg, 4,
                 1.0, u_acc, u_res)
    assert st & dreams.DATA_BAD_PARENT
    acc = r["accept_len"].cpu().numpy()
    assert acc[1] == 0 and int(r["new_kv_len"][1]) == 9
    assert (r["path"][1] == -1).all() and (r["out_tokens"][1] == -1).all()
    assert torch.equal(kg[1], k[1].cuda())
    for b in (0, 2):
        for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
            np.testing.assert_array_equal(r[key][b].cpu().numpy(), ref[key][b], err_msg=key)


def test_speculative_repeatable(dreams):
    """Two calls on the same inputs give identical outputs (the sums are
    combined in a fixed order, whichever SM ran each CTA)."""
    w = W.make("qwen2vl7b", with_attn=False)
    rng = np.random.default_rng(3)
    drf = (w.logits.float() + torch.from_numpy(0.4 * rng.standard_normal(w.logits.shape).astype(np.float32))).to(
        torch.bfloat16).cuda()
    tgt = w.logits.cuda()
    cap = int(w.kv_len.max()) + w.T_max
    k = torch.zeros((w.B, cap, 1, 8), dtype=torch.bfloat16, device="cuda")
    kv = dreams.KVCache(k, k.clone())
    tree = dreams.Tree(w.parent.cuda(), w.tokens.cuda(), w.tree_len.cuda(), w.kv_len.cuda())
    u_acc = torch.from_numpy(rng.random((w.B, w.T_max), dtype=np.float32)).cuda()
    u_res = torch.from_numpy(rng.random((w.B, w.T_max), dtype=np.float32)).cuda()
    a = dreams.verify_step_speculative(tgt, drf, tree, kv, w.max_path, 1.0, u_acc, u_res)
    a = {key: t.clone() for key, t in a.items()}
    b = dreams.verify_step_speculative(tgt, drf, tree, kv, w.max_path, 1.0, u_acc, u_res)
    torch.cuda.synchronize()
    for key in a:
        assert torch.equal(a[key], b[key]), key


def test_speculative_multi_layer_paged_cache(dreams):
    """Three layer caches in 64-slot pages (a permuted page table), random bit
    patterns in every slot (NaN bf16 included): each cluster moves the accepted
    nodes' K/V of every layer and head; all other bytes are unchanged. One
    sequence's page table points outside the pool: it is flagged, its cache is
    left alone, and the walk outputs are still written."""
    rng = np.random.default_rng(66)
    B, T, V, Hkv, D, n_layers, page, pps = 6, 20, 1500, 2, 64, 3, 64, 3
    cap = pps * page
    par = np.stack([W.random_tree(rng, T) for _ in range(B)]).astype(np.int32)
    tl = np.full(B, T, np.int32)
    tgt = (2.0 * rng.standard_normal((B, T, V))).astype(np.float32)
    drf = (tgt + 0.5 * rng.standard_normal((B, T, V))).astype(np.float32)
    tok = _draft_tokens(rng, drf, par, tl, 1.0)
    kl = rng.integers(0, cap - T + 1, B).astype(np.int32)
    table = rng.permutation(B * pps).astype(np.int32).reshape(B, pps)
    kin = rng.integers(0, 65536, (n_layers, B * pps, page, Hkv, D), dtype=np.uint16)
    vin = rng.integers(0, 65536, (n_layers, B * pps, page, Hkv, D), dtype=np.uint16)
    u_acc, u_res, ref = _oracle_clean(tgt, drf, par, tok, tl, kl, 6, 1.0, rng)
    lay = oracle.KVLayout(cap, Hkv, D, page_table=table, page_size=page, num_pages=B * pps)
    ko, vo, ost = oracle.kv_compact(kin, vin, lay, kl, ref["accept_len"], ref["path"], n_layers=n_layers,
                                    layer_stride=kin[0].size)
    assert ost == 0
    tk = torch.from_numpy(kin.view(np.int16)).view(torch.bfloat16).cuda()
    tv = torch.from_numpy(vin.view(np.int16)).view(torch.bfloat16).cuda()
    r, st = _run(dreams, torch.from_numpy(tgt).cuda(), torch.from_numpy(drf).cuda(), par, tok, tl, kl, tk, tv, 6,
                 1.0, u_acc, u_res, torch.from_numpy(table).cuda())
    assert st == 0
    _compare(r, ref)
    assert np.array_equal(tk.view(torch.int16).cpu().numpy().view(np.uint16), ko)
    assert np.array_equal(tv.view(torch.int16).cpu().numpy().view(np.uint16), vo)
    # a page id outside the pool in a sequence whose walk moves rows
    moved = int(np.argmax(ref["accept_len"]))
    assert ref["accept_len"][moved] >= 2
    bad = table.copy()
    bad[moved, :] = B * pps + 5
    tk2 = torch.from_numpy(kin.view(np.int16)).view(torch.bfloat16).cuda()
    tv2 = torch.from_numpy(vin.view(np.int16)).view(torch.bfloat16).cuda()
    r2, st2 = _run(dreams, torch.from_numpy(tgt).cuda(), torch.from_numpy(drf).cuda(), par, tok, tl, kl, tk2, tv2, 6,
                   1.0, u_acc, u_res, torch.from_numpy(bad).cuda())
    assert st2 & dreams.DATA_BAD_PAGE
    _compare(r2, ref)
    acc_ok = ref["accept_len"].copy()
    acc_ok[moved] = 1  # nothing moves for the flagged sequence
    ko2, vo2, _ = oracle.kv_compact(kin, vin, lay, kl, acc_ok, ref["path"], n_layers=n_layers,
                                    layer_stride=kin[0].size)
    assert np.array_equal(tk2.view(torch.int16).cpu().numpy().view(np.uint16), ko2)
    assert np.array_equal(tv2.view(torch.int16).cpu().numpy().view(np.uint16), vo2)


@pytest.mark.parametrize("B, V, sigma", [(2, 128256, 2.0), (3, 256000, 4.0)])
def test_speculative_clusters_of_16(dreams, B, V, sigma):
    """Clusters of 16 CTAs: a batch of at most 4 over a 128256-entry
    vocabulary (16 CTAs per sequence to spread the passes), and a 256000-entry
    vocabulary, whose rows need 16 slices of shared memory (the non-portable
    cluster size). A draw's margin is at most half the width of the entry it
    lands in, so the larger vocabulary takes more peaked rows (sigma 4), whose
    draws land in entries of percent-level width."""
    rng = np.random.default_rng(B * 7 + V % 97)
    T, cap = 24, 64
    par = np.stack([W.random_tree(rng, T) for _ in range(B)]).astype(np.int32)
    tl = np.full(B, T, np.int32)
    tgt32 = (sigma * rng.standard_normal((B, T, V))).astype(np.float32)
    drf32 = (tgt32 + 0.5 * rng.standard_normal((B, T, V))).astype(np.float32)
    tgt_t, drf_t = W.bf16(tgt32), W.bf16(drf32)
    del tgt32, drf32
    tok = _draft_tokens(rng, drf_t.float().numpy(), par, tl, 1.0)
    kl = rng.integers(0, cap - T + 1, B).astype(np.int32)
    u_acc, u_res, ref = _oracle_clean(W.bits(tgt_t), W.bits(drf_t), par, tok, tl, kl, 6, 1.0, rng, bf16=True)
    k = W.bf16(rng.standard_normal((B, cap, 1, 64), dtype=np.float32))
    kg, vg = k.cuda(), k.clone().cuda()
    r, st = _run(dreams, tgt_t.cuda(), drf_t.cuda(), par, tok, tl, kl, kg, vg, 6, 1.0, u_acc, u_res)
    assert st == 0
    _compare(r, ref)
    assert (ref["accept_len"] >= 2).any()
    ko, _, ost = oracle.kv_compact(W.bits(k), W.bits(k), oracle.KVLayout(cap, 1, 64), kl, ref["accept_len"],
                                   ref["path"])
    assert ost == 0 and np.array_equal(W.bits(kg.cpu()), ko)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_speculative_llava_f32_temperature_1(dreams, seed):
    """The LLaVA-7B-shaped workload (f32 logits over 32000 entries, one
    sequence, a cluster of 8 CTAs) at temperature 1, drafts = target + N(0, 0.5)
    noise, against the oracle."""
    w = W.make("llava7b", with_attn=False)
    rng = np.random.default_rng(500 + seed)
    tgt = w.logits.numpy()
    drf = (tgt + 0.5 * rng.standard_normal(tgt.shape, dtype=np.float32)).astype(np.float32)
    par, tok, tl, kl = (x.numpy() for x in (w.parent, w.tokens, w.tree_len, w.kv_len))
    u_acc, u_res, ref = _oracle_clean(tgt, drf, par, tok, tl, kl, w.max_path, 1.0, rng)
    assert ref["status"] == 0
    cap = int(kl.max()) + w.T_max
    k = torch.zeros((w.B, cap, 1, 8), dtype=torch.bfloat16, device="cuda")
    r, st = _run(dreams, torch.from_numpy(tgt).cuda(), torch.from_numpy(drf).cuda(), par, tok, tl, kl, k, k.clone(),
                 w.max_path, 1.0, u_acc, u_res)
    assert st == 0
    _compare(r, ref)
