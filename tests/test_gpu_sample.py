"""GPU parity of the temperature-tau draws (dreams_vocab_sample) and of the
sampled verification tail (dreams_verify_step_sampled) against the fp64 oracle.

A draw is an integer decided by floating point: the kernel sums f32 weights in
its own fixed order, the oracle sums exact-ish doubles. Where the two differ,
the kernel's draw must still be a valid inverse-transform draw within rounding:
positive weight, and u inside [F(v-1), F(v)] up to DRAW_TOL (F = the exact
cumulative distribution). Such differences must also be rare. Everything
downstream of the draws (walk, outputs, compaction) is compared bit-exactly
against the oracle run on the kernel's own draws."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import layout, to_gpu

pytestmark = pytest.mark.gpu

DRAW_TOL = 2e-5       # in units of probability
MISMATCH_SHARE = 0.01  # at most this share of rows may differ from the oracle


@pytest.fixture(scope="module")
def dreams():
    import paper_2606_00535_gb300 as d
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    d._lib()
    return d


def _status():
    return torch.zeros(1, dtype=torch.int32, device="cuda")


def _cdf_ok(x, tau, u, v):
    """v is a valid draw of softmax(x / tau) for uniform u, within DRAW_TOL."""
    x = np.asarray(x, np.float64)
    if np.isnan(x).any() or np.max(x) == np.inf or np.max(x) == -np.inf:
        return v == int(np.argmax(x))
    u = 0.0 if not (u > 0) else min(float(u), 1.0)
    w = np.exp((x - x.max()) / tau)
    F = np.cumsum(w) / w.sum()
    lo = F[v - 1] if v > 0 else 0.0
    return w[v] > 0 and lo - DRAW_TOL <= u <= F[v] + DRAW_TOL


def _check_draws(x64, tau, u, got, ref):
    """got (kernel) and ref (oracle) over rows of x64; returns the mismatch count."""
    bad = np.nonzero(got != ref)[0]
    for r in bad:
        assert _cdf_ok(x64[r], tau, u[r], int(got[r])), (r, int(got[r]), int(ref[r]), float(u[r]))
    assert len(bad) <= max(2, MISMATCH_SHARE * len(got)), f"{len(bad)} of {len(got)} draws differ"
    return len(bad)


def _run(dreams, x_t, tau, u_np):
    u = torch.from_numpy(np.ascontiguousarray(u_np, np.float32)).cuda()
    out = dreams.vocab_sample(x_t, tau, u)
    torch.cuda.synchronize()
    return out.cpu().numpy()


@pytest.mark.parametrize("V", [1, 7, 255, 256, 257, 1000, 32000, 128256])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_sample_matches_oracle(dreams, V, dtype):
    rng = np.random.default_rng(V + (0 if dtype == "f32" else 1))
    rows = 40 if V > 10000 else 200
    x = (2.0 * rng.standard_normal((rows, V))).astype(np.float32)
    x[rng.integers(0, rows, rows // 4), rng.integers(0, V, rows // 4)] += 6.0  # peaked rows
    u = rng.uniform(0, 1, rows).astype(np.float32)
    for tau in (0.5, 1.0, 2.0):
        if dtype == "bf16":
            t = W.bf16(x)
            got = _run(dreams, t.cuda(), tau, u)
            ref = oracle.sample(W.bits(t), tau, u, bf16_bits=True)
            x64 = t.float().numpy()
        else:
            got = _run(dreams, torch.from_numpy(x).cuda(), tau, u)
            ref = oracle.sample(x, tau, u)
            x64 = x
        _check_draws(x64, tau, u, got, ref)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_sample_unaligned_rows_and_stride(dreams, dtype):
    """Rows that do not start on 16 bytes take scalar loads; padding past V is ignored."""
    rng = np.random.default_rng(21)
    rows, V, stride = 33, 5001, 5003
    x = rng.standard_normal((rows, stride)).astype(np.float32)
    x[:, V:] = 50.0
    u = rng.uniform(0, 1, rows).astype(np.float32)
    t = torch.from_numpy(x) if dtype == "f32" else W.bf16(x)
    got = _run(dreams, t.cuda()[:, :V], 1.0, u)  # a strided view
    ref = oracle.sample(W.bits(t) if dtype == "bf16" else x, 1.0, u, V=V, bf16_bits=dtype == "bf16")
    _check_draws(t.float().numpy()[:, :V], 1.0, u, got, ref)


def test_sample_degenerate_rows_and_uniform_edges(dreams):
    nan, inf = np.nan, np.inf
    V = 600
    rows = np.zeros((8, V), np.float32)
    rows[0, [3, 400]] = nan                   # first NaN
    rows[1, [10, 299, 599]] = inf             # first +inf
    rows[2, :] = -inf                         # no finite value: 0
    rows[3, :] = -inf
    rows[3, [257, 511]] = 1.0                 # two equal survivors
    rows[4, :] = np.linspace(-3, 3, V)
    rows[5, :] = np.linspace(-3, 3, V)
    rows[6, :] = np.linspace(-3, 3, V)
    rows[7, :] = np.linspace(-3, 3, V)
    u = np.array([0.5, 0.5, 0.5, 0.75, 0.0, 1.0, nan, -3.0], np.float32)
    got = _run(dreams, torch.from_numpy(rows).cuda(), 0.7, u)
    ref = oracle.sample(rows, 0.7, u)
    np.testing.assert_array_equal(ref[:4], [3, 10, 0, 511])
    np.testing.assert_array_equal(got, ref)
    assert got[5] == V - 1 and got[4] == 0 and got[6] == 0 and got[7] == 0


def test_sample_grid_frequencies_match_softmax(dreams):
    """One row, a grid of uniforms: the draw frequencies are the softmax probabilities."""
    import scipy.special
    rng = np.random.default_rng(22)
    V, N = 50, 20000
    x = (1.5 * rng.standard_normal(V)).astype(np.float32)
    u = ((np.arange(N) + 0.5) / N).astype(np.float32)
    got = _run(dreams, torch.from_numpy(np.repeat(x[None], N, 0)).cuda(), 0.9, u)
    freq = np.bincount(got, minlength=V) / N
    p = scipy.special.softmax(x.astype(np.float64) / 0.9)
    assert np.abs(freq - p).max() <= 2.0 / N
    assert (np.diff(got) >= 0).all()  # monotone in u


def test_sample_rejects_bad_arguments(dreams):
    x = torch.zeros((4, 100), device="cuda")
    u = torch.zeros(4, device="cuda")
    for tau in (0.0, -1.0, float("inf"), float("nan"), 1e-39):
        with pytest.raises(RuntimeError):
            dreams.vocab_sample(x, tau, u)


CONFIGS = ["tiny", "llava7b", "qwen2vl7b", "long13b", "batched"]


@pytest.mark.parametrize("name", CONFIGS)
def test_verify_step_sampled_matches_oracle(dreams, name):
    w = W.make(name)
    g = to_gpu(w)
    rng = np.random.default_rng(31)
    tau = 1.0
    u_np = rng.uniform(0, 1, (w.B, w.T_max)).astype(np.float32)
    u = torch.from_numpy(u_np).cuda()
    draws = torch.full((w.B, w.T_max), -7, dtype=torch.int32, device="cuda")
    st = _status()
    r = dreams.verify_step_sampled(g["logits"], g["tree"], g["kv"], w.max_path, tau, u, sample_out=draws, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    d_gpu = draws.cpu().numpy()
    x = w.logits.reshape(-1, w.V)
    bf16 = w.logits_dtype == "bf16"
    ref_all = oracle.sample(W.bits(x) if bf16 else x.numpy(), tau, u_np.reshape(-1), bf16_bits=bf16)
    ref_all = ref_all.reshape(w.B, w.T_max)
    x64 = x.float().numpy().reshape(w.B, w.T_max, w.V)
    got_rows, ref_rows, xs, us = [], [], [], []
    for b in range(w.B):
        t = int(w.tree_len[b])
        assert (d_gpu[b, t:] == -7).all()
        got_rows.append(d_gpu[b, :t])
        ref_rows.append(ref_all[b, :t])
        xs.append(x64[b, :t])
        us.append(u_np[b, :t])
    _check_draws(np.concatenate(xs), tau, np.concatenate(us), np.concatenate(got_rows), np.concatenate(ref_rows))
    # the walk and the compaction, from the kernel's own draws
    ref = oracle.accept_path(d_gpu, w.parent.numpy(), w.tokens.numpy(), w.tree_len.numpy(), w.kv_len.numpy(),
                             w.max_path)
    for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
        np.testing.assert_array_equal(r[key].cpu().numpy(), ref[key], err_msg=key)
    # the first emitted token is always the root's draw
    np.testing.assert_array_equal(r["out_tokens"][:, 0].cpu().numpy(), d_gpu[:, 0])
    ko, vo, ost = oracle.kv_compact(W.bits(w.k), W.bits(w.v), layout(w), w.kv_len.numpy(), ref["accept_len"],
                                    ref["path"])
    assert ost == 0
    assert np.array_equal(W.bits(g["k"].cpu()), ko)
    assert np.array_equal(W.bits(g["v"].cpu()), vo)


def test_verify_step_sampled_low_temperature_is_greedy(dreams):
    """At a tiny temperature the draws are the argmaxes (distinct maxima), so
    the sampled step reproduces the greedy step."""
    w = W.make("llava7b")
    g1, g2 = to_gpu(w), to_gpu(w)
    u = torch.rand((w.B, w.T_max), generator=torch.Generator().manual_seed(3)).cuda()
    r_s = dreams.verify_step_sampled(g1["logits"], g1["tree"], g1["kv"], w.max_path, 1e-30, u)
    r_g = dreams.verify_step(g2["logits"], g2["tree"], g2["kv"], w.max_path)
    torch.cuda.synchronize()
    for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
        assert torch.equal(r_s[key], r_g[key]), key
    assert torch.equal(g1["k"], g2["k"]) and torch.equal(g1["v"], g2["v"])


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_sample_split_rows_repeat(dreams, dtype):
    """Few long rows, each split between CTAs; two calls on one workspace agree."""
    rng = np.random.default_rng(23)
    rows, V = 5, 300_001
    x = (2.0 * rng.standard_normal((rows, V))).astype(np.float32)
    u = rng.uniform(0, 1, rows).astype(np.float32)
    t = torch.from_numpy(x) if dtype == "f32" else W.bf16(x)
    need = dreams._lib().dreams_vocab_sample_workspace_size(rows, V)
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    ut = torch.from_numpy(u).cuda()
    a = dreams.vocab_sample(t.cuda(), 1.0, ut, workspace=ws).cpu().numpy()
    ws.fill_(0xA5)  # the workspace holds no state: garbage in it changes nothing
    b = dreams.vocab_sample(t.cuda(), 1.0, ut, workspace=ws).cpu().numpy()
    np.testing.assert_array_equal(a, b)
    ref = oracle.sample(W.bits(t) if dtype == "bf16" else x, 1.0, u, bf16_bits=dtype == "bf16")
    _check_draws(t.float().numpy(), 1.0, u, a, ref)


def test_sample_workspace_reused_across_shapes(dreams):
    """One workspace for calls of different shapes (the binding caches one per stream)."""
    rng = np.random.default_rng(24)
    need = max(dreams._lib().dreams_vocab_sample_workspace_size(r, V) for r, V in ((3, 200_000), (40, 32000)))
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    for rows, V in ((3, 200_000), (40, 32000), (3, 200_000), (7, 1000)):
        x = rng.standard_normal((rows, V)).astype(np.float32)
        u = rng.uniform(0, 1, rows).astype(np.float32)
        got = dreams.vocab_sample(torch.from_numpy(x).cuda(), 1.0, torch.from_numpy(u).cuda(), workspace=ws)
        _check_draws(x, 1.0, u, got.cpu().numpy(), oracle.sample(x, 1.0, u))
