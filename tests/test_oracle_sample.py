"""Pins for the oracle's temperature-tau sample (inverse transform of
softmax(x / tau) with a caller-supplied uniform), CPU only.

Each pin fixes the answer by a route that does not retype the oracle's loop:
the logistic closed form for two tokens, exact integer arithmetic for weights
that are integers, the uniform limit of a huge temperature, the argmax limit of
a tiny one (numpy's argmax), scipy's softmax for the frequencies over a grid of
uniforms, and invariants (shift invariance, monotonicity in u)."""
import numpy as np
import pytest
import scipy.special

import oracle
import workloads as W


def _draw(x, tau, u, bf16=False):
    x = np.asarray(x, np.float32)
    if x.ndim == 1:
        x = x[None]
    u = np.broadcast_to(np.asarray(u, np.float32), (x.shape[0],))
    if bf16:
        return oracle.sample(W.bits(W.bf16(x)), tau, u, bf16_bits=True)
    return oracle.sample(x, tau, u)


@pytest.mark.parametrize("a,b,tau", [(0.0, 1.0, 1.0), (2.5, -1.0, 0.7), (3.0, 3.5, 2.0), (-4.0, 1.0, 5.0)])
def test_two_tokens_logistic_threshold(a, b, tau):
    # P(draw = 0) = 1 / (1 + exp((b - a) / tau)): u just below draws 0, just above draws 1
    p0 = 1.0 / (1.0 + np.exp((b - a) / tau))
    for u, expect in ((p0 * (1 - 1e-4), 0), (p0 + (1 - p0) * 1e-4, 1), (0.0, 0), (np.nextafter(np.float32(1), 0), 1)):
        assert _draw([a, b], tau, [u])[0] == expect, (u, p0)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_integer_weights_exact_buckets(seed):
    # logits tau * log(k_v) give weights proportional to the integers k_v; the
    # draw for u = (j + 0.5) / N, N = sum k, is the v with K_{v-1} <= j < K_v
    # (prefix sums K), an exact integer answer
    rng = np.random.default_rng(seed)
    V = int(rng.integers(2, 40))
    k = rng.integers(0, 9, V)
    k[rng.integers(0, V)] += 1  # at least one positive weight
    tau = float(rng.uniform(0.3, 3.0))
    with np.errstate(divide="ignore"):
        x = (tau * np.log(k.astype(np.float64))).astype(np.float32)
    N = int(k.sum())
    K = np.cumsum(k)
    j = np.arange(N)
    u = ((j + 0.5) / N).astype(np.float32)
    got = oracle.sample(np.repeat(x[None], N, 0), tau, u)
    expect = np.searchsorted(K, j, side="right")
    np.testing.assert_array_equal(got, expect)
    assert (k[got] > 0).all()


def test_huge_temperature_is_uniform():
    rng = np.random.default_rng(4)
    V = 37
    x = rng.standard_normal(V).astype(np.float32)
    j = np.arange(V)
    u = ((j + 0.5) / V).astype(np.float32)
    got = oracle.sample(np.repeat(x[None], V, 0), 1e30, u)
    np.testing.assert_array_equal(got, j)  # floor(u * V)


@pytest.mark.parametrize("bf16", [False, True])
def test_tiny_temperature_is_argmax(bf16):
    rng = np.random.default_rng(5)
    x = rng.standard_normal((50, 300)).astype(np.float32)
    if bf16:
        x = W.bf16(x).float().numpy()
    # distinct maxima with probability one; any u in [0, 1) then draws the argmax
    u = rng.uniform(0, 1, 50).astype(np.float32)
    np.testing.assert_array_equal(_draw(x, 1e-30, u, bf16=bf16), np.argmax(x, axis=1))


def test_tiny_temperature_splits_ties_by_u():
    x = np.array([1.0, 4.0, 2.0, 4.0, 4.0], np.float32)
    # three tied maxima share the mass equally
    assert _draw(x, 1e-30, [0.1])[0] == 1
    assert _draw(x, 1e-30, [0.5])[0] == 3
    assert _draw(x, 1e-30, [0.9])[0] == 4


def test_grid_frequencies_match_softmax():
    rng = np.random.default_rng(6)
    V, N = 12, 4000
    x = (2.0 * rng.standard_normal(V)).astype(np.float32)
    tau = 1.3
    u = ((np.arange(N) + 0.5) / N).astype(np.float32)
    got = oracle.sample(np.repeat(x[None], N, 0), tau, u)
    freq = np.bincount(got, minlength=V) / N
    p = scipy.special.softmax(x.astype(np.float64) / tau)
    assert np.abs(freq - p).max() <= 1.0 / N + 1e-9


def test_shift_invariance_and_monotone_in_u():
    rng = np.random.default_rng(7)
    x = rng.standard_normal(500).astype(np.float32)
    u = np.sort(rng.uniform(0, 1, 200)).astype(np.float32)
    a = oracle.sample(np.repeat(x[None], 200, 0), 0.8, u)
    b = oracle.sample(np.repeat((x + 17.0)[None].astype(np.float32), 200, 0), 0.8, u)
    # +17 is exact in float32 for these magnitudes only up to rounding of x + 17;
    # compare where no boundary is within that rounding
    assert (a == b).mean() > 0.98
    assert (np.diff(a) >= 0).all()


def test_clamped_and_degenerate_rows():
    nan, inf = np.nan, np.inf
    x = np.array([0.0, 1.0, 2.0], np.float32)
    assert _draw(x, 1.0, [-0.5])[0] == _draw(x, 1.0, [0.0])[0] == 0
    assert _draw(x, 1.0, [nan])[0] == 0
    assert _draw(x, 1.0, [1.0])[0] == 2 and _draw(x, 1.0, [7.0])[0] == 2
    # the last token with positive weight, when u = 1 and the tail has zero weight
    assert _draw([0.0, 1.0, -inf, -inf], 1.0, [1.0])[0] == 1
    rows = np.array([
        [1, nan, 9, nan],          # a NaN: the first NaN (the argmax order)
        [-inf, inf, inf, 3],       # +inf maximum: the first +inf
        [-inf, -inf, -inf, -inf],  # no finite value: index 0
        [-inf, 2, -inf, 2],        # -inf entries have weight 0
    ], np.float32)
    u = np.array([0.5, 0.5, 0.5, 0.75], np.float32)
    np.testing.assert_array_equal(oracle.sample(rows, 1.0, u), [1, 1, 0, 3])
    np.testing.assert_array_equal(np.argmax(rows[:3], axis=1), [1, 1, 0])


def test_row_stride_and_bf16_widening():
    rng = np.random.default_rng(8)
    x = rng.standard_normal((16, 64)).astype(np.float32)
    x[:, 40:] = 1e4  # beyond V: ignored
    u = rng.uniform(0, 1, 16).astype(np.float32)
    np.testing.assert_array_equal(oracle.sample(x, 1.0, u, V=40), oracle.sample(x[:, :40].copy(), 1.0, u))
    b = W.bf16(x[:, :40])
    np.testing.assert_array_equal(oracle.sample(W.bits(b), 1.0, u, bf16_bits=True),
                                  oracle.sample(b.float().numpy(), 1.0, u))


def test_sampled_walk_first_token_is_root_draw():
    # The paper's acceptance compares each draft with the target's own output
    # at its parent; with draws in place of argmaxes, the first emitted token
    # is always the root's draw (an accepted child carries the same token, and
    # otherwise the draw is the bonus token).
    rng = np.random.default_rng(9)
    w = W.make("tiny")
    x = w.logits.reshape(-1, w.V).numpy()
    u = rng.uniform(0, 1, x.shape[0]).astype(np.float32)
    draws = oracle.sample(x, 1.0, u).reshape(w.B, w.T_max)
    r = oracle.accept_path(draws, w.parent.numpy(), w.tokens.numpy(), w.tree_len.numpy(), w.kv_len.numpy(), 8)
    assert r["status"] == 0
    assert r["out_tokens"][0, 0] == draws[0, 0]
