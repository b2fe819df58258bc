"""Pins for the oracle's speculative sampling over a draft tree (Leviathan et
al.'s rule, cited in Sec. 1 of the paper; verification at T = 1, Table 2): a
draft is accepted with probability min(1, p/q), a rejection moves the target
to the renormalised residual max(0, p - q), and the bonus token is drawn from
what is left. The defining property of the rule is that the first emitted
token is distributed as the target p, whatever the draft distribution q; the
tests check that by sampling, the greedy limit against the (independently
pinned) greedy walk, and the closed-form acceptance rate."""
import numpy as np
import pytest

import oracle
import workloads as W

V_SMALL = 5


def _node_case(rng, n, k, p_logits, q_logits, tau=1.0):
    """n sequences of one node with k children whose drafts are drawn i.i.d.
    from q = softmax(q_logits / tau); returns the oracle's output."""
    T = k + 1
    q = np.exp((q_logits - q_logits.max()) / tau)
    q /= q.sum()
    parent = np.full((n, T), 0, np.int32)
    parent[:, 0] = -1
    tokens = np.zeros((n, T), np.int32)
    tokens[:, 1:] = rng.choice(len(q), size=(n, k), p=q)
    target = np.zeros((n, T, len(q)), np.float32)
    target[:, :] = p_logits
    draft = np.zeros((n, T, len(q)), np.float32)
    draft[:, :] = q_logits
    u_acc = rng.random((n, T), dtype=np.float32)
    u_res = rng.random((n, T), dtype=np.float32)
    res = oracle.spec_path(target, draft, parent, tokens, np.full(n, T, np.int32), np.zeros(n, np.int32), 3, tau,
                           u_acc, u_res)
    return res, tokens


def _first_token_freq(res, n, V):
    first = np.where(res["accept_len"] >= 2, res["out_tokens"][:, 0], res["out_tokens"][:, 0])
    return np.bincount(first, minlength=V) / n


@pytest.mark.parametrize("k", [1, 2, 3])
def test_first_token_is_distributed_as_the_target(k):
    """The output token of a node with k children drawn i.i.d. from q has the
    target's distribution p (4.5 standard errors over 200 000 draws). p and q
    differ a lot, so an unnormalised residual, a later child tested against p
    instead of the residual, a bonus drawn from p, or an inverted ratio all
    move some probability by far more than the tolerance."""
    rng = np.random.default_rng(100 + k)
    p_logits = np.array([2.0, 0.5, -1.0, 1.0, -0.3])
    q_logits = np.array([-0.5, 1.8, 0.2, -1.0, 1.1])
    p = np.exp(p_logits - p_logits.max())
    p /= p.sum()
    n = 200_000
    res, _ = _node_case(rng, n, k, p_logits, q_logits)
    freq = _first_token_freq(res, n, V_SMALL)
    se = np.sqrt(p * (1 - p) / n)
    assert (np.abs(freq - p) <= 4.5 * se).all(), (freq, p)


def test_acceptance_rate_closed_form():
    """One child drawn from q: P(accept) = sum_x q(x) min(1, p(x)/q(x)) =
    sum_x min(p(x), q(x)) (one minus the total-variation distance)."""
    rng = np.random.default_rng(7)
    p_logits = np.array([1.0, -0.5, 0.3, 2.0, 0.0])
    q_logits = np.array([0.0, 1.5, 0.3, 0.5, -1.0])
    p = np.exp(p_logits - p_logits.max())
    p /= p.sum()
    q = np.exp(q_logits - q_logits.max())
    q /= q.sum()
    n = 200_000
    res, _ = _node_case(rng, n, 1, p_logits, q_logits)
    rate = float((res["accept_len"] == 2).mean())
    exact = float(np.minimum(p, q).sum())
    assert abs(rate - exact) <= 4.5 * np.sqrt(exact * (1 - exact) / n), (rate, exact)


def test_second_token_after_acceptance_follows_the_child_target():
    """A chain root -> c1 -> c2: given that c1 was accepted, the next emitted
    token is distributed as the target at c1 (the same guarantee one level
    down)."""
    rng = np.random.default_rng(9)
    n, V = 200_000, 4
    q0 = np.array([0.2, 0.1, 0.6, 0.1])
    p0_logits = np.log(np.array([0.3, 0.2, 0.4, 0.1]))
    p1 = np.array([0.1, 0.5, 0.15, 0.25])
    q1 = np.array([0.4, 0.2, 0.2, 0.2])
    parent = np.tile(np.array([-1, 0, 1], np.int32), (n, 1))
    tokens = np.zeros((n, 3), np.int32)
    tokens[:, 1] = rng.choice(V, size=n, p=q0)
    tokens[:, 2] = rng.choice(V, size=n, p=q1)
    target = np.zeros((n, 3, V), np.float32)
    target[:, 0] = p0_logits
    target[:, 1] = np.log(p1)
    target[:, 2] = 0.0
    draft = np.zeros((n, 3, V), np.float32)
    draft[:, 0] = np.log(q0)
    draft[:, 1] = np.log(q1)
    res = oracle.spec_path(target, draft, parent, tokens, np.full(n, 3, np.int32), np.zeros(n, np.int32), 4, 1.0,
                           rng.random((n, 3), dtype=np.float32), rng.random((n, 3), dtype=np.float32))
    took = res["accept_len"] >= 2
    second = res["out_tokens"][took, 1]
    m = int(took.sum())
    freq = np.bincount(second, minlength=V) / m
    se = np.sqrt(p1 * (1 - p1) / m)
    assert (np.abs(freq - p1) <= 4.5 * se).all(), (freq, p1)
    first = res["out_tokens"][:, 0]
    p0 = np.exp(p0_logits)
    f0 = np.bincount(first, minlength=V) / n
    assert (np.abs(f0 - p0) <= 4.5 * np.sqrt(p0 * (1 - p0) / n)).all(), (f0, p0)


def _distinct_sibling_tree(rng, T, V):
    parent = W.random_tree(rng, T).astype(np.int32)
    tokens = np.zeros(T, np.int32)
    for i in range(T):
        kids = [c for c in range(i + 1, T) if parent[c] == i]
        toks = rng.choice(V, size=len(kids), replace=False)
        for c, t in zip(kids, toks):
            tokens[c] = t
    return parent, tokens


def test_greedy_limit_matches_the_greedy_walk():
    """At a temperature of 1e-4 both distributions are one-hot at their argmax
    (the other weights underflow to exactly 0 in fp64 for the planted margins),
    so a draft is accepted exactly when it is the target's argmax and the bonus
    is the argmax: with distinct sibling tokens the walk is the greedy walk of
    oracle.accept_path, whatever the draft rows and the uniforms."""
    rng = np.random.default_rng(11)
    B, T, V = 40, 24, 50
    par = np.zeros((B, T), np.int32)
    tok = np.zeros((B, T), np.int32)
    for b in range(B):
        par[b], tok[b] = _distinct_sibling_tree(rng, T, V)
    target = rng.standard_normal((B, T, V)).astype(np.float32)
    draft = rng.standard_normal((B, T, V)).astype(np.float32)
    for b in range(B):
        for i in range(T):
            kids = [c for c in range(i + 1, T) if par[b, c] == i]
            if kids and rng.random() < 0.7:
                target[b, i, tok[b, rng.choice(kids)]] = 10.0  # planted argmax: margin >= 5
            else:
                target[b, i, rng.integers(V)] = 10.0
            draft[b, i, rng.integers(V)] = 10.0
    am = target.argmax(axis=2).astype(np.int32)
    ref = oracle.accept_path(am, par, tok, np.full(B, T, np.int32), np.zeros(B, np.int32), 8)
    res = oracle.spec_path(target, draft, par, tok, np.full(B, T, np.int32), np.zeros(B, np.int32), 8, 1e-4,
                           rng.random((B, T), dtype=np.float32), rng.random((B, T), dtype=np.float32))
    for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
        np.testing.assert_array_equal(res[key], ref[key], err_msg=key)
    assert (res["accept_len"] >= 2).any() and (res["accept_len"] == 1).any()


def test_equal_distributions_accept_the_first_child():
    """q == p: the ratio is 1 and every first child is accepted (u < 1)."""
    rng = np.random.default_rng(13)
    B, T, V = 30, 20, 16
    par = np.stack([W.random_tree(rng, T) for _ in range(B)]).astype(np.int32)
    tok = rng.integers(0, V, (B, T)).astype(np.int32)
    target = rng.standard_normal((B, T, V)).astype(np.float32)
    res = oracle.spec_path(target, target, par, tok, np.full(B, T, np.int32), np.zeros(B, np.int32), 64, 0.8,
                           rng.random((B, T), dtype=np.float32) * 0.999, rng.random((B, T), dtype=np.float32))
    for b in range(B):
        cur, path = 0, [0]
        while True:
            kids = [c for c in range(cur + 1, T) if par[b, c] == cur]
            if not kids:
                break
            cur = kids[0]
            path.append(cur)
        assert res["accept_len"][b] == len(path)
        np.testing.assert_array_equal(res["path"][b, :len(path)], path)


def test_leaf_root_and_cut_draw_from_the_target():
    """At a leaf, and at the max_path cut, the bonus is one draw from the
    target itself: the same inverse-transform draw as oracle.sample."""
    rng = np.random.default_rng(17)
    B, V = 64, 37
    tgt = (rng.standard_normal((B, 1, V)) * 2).astype(np.float32)
    u = rng.random((B, 1), dtype=np.float32)
    res = oracle.spec_path(tgt, tgt, np.full((B, 1), -1, np.int32), np.zeros((B, 1), np.int32),
                           np.ones(B, np.int32), np.zeros(B, np.int32), 4, 0.7, u, u)
    ref = oracle.sample(tgt[:, 0], 0.7, u[:, 0])
    ok = res["margin"] > 1e-9
    np.testing.assert_array_equal(res["out_tokens"][ok, 0], ref[ok])
    assert (res["accept_len"] == 1).all() and ok.mean() > 0.9
    # max_path 1: no draft is tried, the bonus is the root's own draw
    T = 6
    par = np.tile(np.array([-1, 0, 0, 1, 1, 2], np.int32), (B, 1))
    tgt2 = (rng.standard_normal((B, T, V)) * 2).astype(np.float32)
    u2 = rng.random((B, T), dtype=np.float32)
    res2 = oracle.spec_path(tgt2, tgt2, par, rng.integers(0, V, (B, T)).astype(np.int32), np.full(B, T, np.int32),
                            np.zeros(B, np.int32), 1, 0.7, u2, u2)
    assert (res2["accept_len"] == 1).all()
    ref2 = oracle.sample(tgt2[:, 0], 0.7, u2[:, 0])
    ok2 = res2["margin"] > 1e-9
    np.testing.assert_array_equal(res2["out_tokens"][ok2, 0], ref2[ok2])


def test_malformed_tree_is_flagged():
    par = np.array([[-1, 0, 5]], np.int32)
    res = oracle.spec_path(np.zeros((1, 3, 4), np.float32), np.zeros((1, 3, 4), np.float32), par,
                           np.zeros((1, 3), np.int32), np.array([3], np.int32), np.array([10], np.int32), 4, 1.0,
                           np.zeros((1, 3), np.float32), np.zeros((1, 3), np.float32))
    assert res["status"] & 1 and res["accept_len"][0] == 0 and res["new_kv_len"][0] == 10
    assert (res["path"] == -1).all()
