"""GPU parity: every kernel, through the C ABI, against the fp64 oracle on the
same seeded inputs (bit-exact for indices, paths, tokens and the compacted
cache; attention within max-abs 1e-2 / mean-abs 1e-3 and lse within 1e-3
relative)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import compare_attention, layout, logits_rows_oracle, oracle_attention, to_gpu

pytestmark = pytest.mark.gpu

CONFIGS = ["tiny", "llava7b", "qwen2vl7b", "long13b", "batched"]


@pytest.fixture(scope="module")
def dreams():
    import paper_2606_00535_gb300 as d
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    d._lib()  # fails loudly when the library is missing
    return d


def _status():
    return torch.zeros(1, dtype=torch.int32, device="cuda")


# ------------------------------------------------------------------ attention
@pytest.mark.parametrize("name", CONFIGS)
def test_attention_matches_oracle(dreams, name):
    w = W.make(name, with_logits=False)
    g = to_gpu(w)
    st = _status()
    out, lse = dreams.tree_verify_attn(g["q"], g["kv"], g["tree"], w.scale, want_lse=True, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    rng = np.random.default_rng(5)
    if name == "batched":  # all heads of sampled nodes, plus every node of one sequence
        sel = []
        for b in range(w.B):
            for t in rng.choice(int(w.tree_len[b]), 6, replace=False):
                sel += [(b, int(t), h) for h in range(w.Hq)]
        sel += [(3, t, h) for t in range(int(w.tree_len[3])) for h in (0, 13, 31)]
        sel = np.array(sel, np.int32)
    else:
        sel = None
    ref, ref_lse, sel, ost = oracle_attention(w, sel)
    assert ost == 0
    compare_attention(out, lse, ref, ref_lse, sel)


@pytest.mark.parametrize("name,L,key_scale", [("tiny", 0, 1.0), ("tiny", 16, 8.0), ("llava7b", 16, 8.0),
                                              ("qwen2vl7b", 0, 8.0), ("tiny", 300, 8.0), ("batched", 16, 8.0),
                                              ("batched", 0, 8.0)])
def test_attention_mask_sensitive(dreams, name, L, key_scale):
    """Short prefixes and tree keys scaled x8: the tree columns dominate, so a
    wrong ancestor mask moves the output far outside the tolerance (the
    batched cases run it on the paged, many-sequence layout).

    The tolerance is the task's (max-abs 1e-2, mean-abs 1e-3) on outputs of
    magnitude <= 1, relative above that. A dominated softmax makes |out| ~ |V|
    (up to ~4), where no bf16 result can meet a fixed absolute 1e-2: bf16 keeps
    8 significant bits (unit roundoff u = 2^-8, 0.0156 at 4), and the
    probabilities enter the PV product rounded to bf16 too. With a = the
    attention weights, the error is at most u |out| (output rounding) +
    u sum_j a_j |V_j| (probability rounding) + f32 accumulation; where one key
    dominates the second term is ~u |out|, so each element must satisfy
    |err| <= max(1e-2, 2u |ref|), and the mean of |err| / max(1, |ref|) must
    stay within 1e-3."""
    w = W.make(name, with_logits=False, kv_len_override=L, tree_key_scale=key_scale)
    g = to_gpu(w)
    st = _status()
    out, lse = dreams.tree_verify_attn(g["q"], g["kv"], g["tree"], w.scale, want_lse=True, status=st)
    sel = None
    if name == "batched":  # every head of 8 nodes of each sequence, and one whole sequence
        rng = np.random.default_rng(9)
        sel = [(b, int(t), h) for b in range(w.B) for t in rng.choice(int(w.tree_len[b]), 8, replace=False)
               for h in range(w.Hq)]
        sel += [(5, t, h) for t in range(int(w.tree_len[5])) for h in range(w.Hq)]
        sel = np.array(sorted(set(sel)), np.int32)
    ref, ref_lse, sel, _ = oracle_attention(w, sel)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    # the lse and the finiteness checks of the plain comparison, output bound below
    compare_attention(out, lse, ref, ref_lse, sel, max_abs=np.inf, mean_abs=np.inf)
    o = out.float().cpu().numpy()[sel[:, 0], sel[:, 1], sel[:, 2]].astype(np.float64)
    err = np.abs(o - ref)
    lim = np.maximum(1e-2, 2.0 ** -7 * np.abs(ref))
    worst = np.unravel_index(np.argmax(err / lim), err.shape)
    assert (err <= lim).all(), f"err {err[worst]:.3e} at |ref| {abs(ref[worst]):.3f} (limit {lim[worst]:.3e})"
    rel_mean = float((err / np.maximum(1.0, np.abs(ref))).mean())
    assert rel_mean <= 1e-3, f"mean relative error {rel_mean:.3e}"
    # the tree keys do dominate here: outputs reach well past the prefix-average scale
    if key_scale > 1:
        assert np.abs(ref).max() > 1.0


@pytest.mark.parametrize("B,Hq,Hkv,D,T,L,cap", [
    (1, 1, 1, 64, 1, 0, 1),        # root only, empty prefix
    (1, 2, 1, 128, 1, 5, 8),       # root only
    (2, 8, 2, 128, 17, 63, 200),   # ragged tile boundary
    (3, 4, 4, 64, 64, 129, 400),   # maximum tree
    (2, 16, 2, 128, 64, 1000, 1100),  # 512 query rows per KV head: several row blocks
    (2, 14, 2, 128, 40, 300, 400),    # group of 7 heads: 18 nodes (126 rows) per row block
    (1, 100, 1, 64, 5, 100, 200),     # group of 100 heads: one node per row block
    (2, 128, 1, 64, 3, 50, 100),      # the largest group (128 heads)
    (1, 3, 1, 128, 64, 2000, 2304),   # 2 row blocks, KV range split
    (1, 5, 1, 128, 64, 2000, 2304),   # 3 row blocks, KV range split
    (1, 6, 1, 128, 64, 2000, 2304),   # 4 row blocks, KV range split
    (2, 10, 2, 64, 61, 1500, 1600),   # head dim 64, ragged split tail
])
def test_attention_edge_shapes(dreams, B, Hq, Hkv, D, T, L, cap):
    rng = np.random.default_rng(B * 1000 + T)
    par = np.full((B, T), -1, np.int32)
    for b in range(B):
        par[b] = W.random_tree(rng, T)
    tl = np.full(B, T, np.int32)
    tl[-1] = max(1, T - 3)
    par[-1, tl[-1]:] = -1
    kl = rng.integers(max(0, L - 5), L + 1, B).astype(np.int32)
    kl = np.minimum(kl, cap - tl)
    q = W.bf16(rng.standard_normal((B, T, Hq, D), dtype=np.float32))
    k = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    v = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    scale = 1.0 / np.sqrt(D)
    kv = dreams.KVCache(k.cuda(), v.cuda())
    tree = dreams.Tree(torch.from_numpy(par).cuda(), torch.zeros((B, T), dtype=torch.int32, device="cuda"),
                       torch.from_numpy(tl).cuda(), torch.from_numpy(kl).cuda())
    out = torch.full((B, T, Hq, D), 7.0, dtype=torch.bfloat16, device="cuda")
    out, lse = dreams.tree_verify_attn(q.cuda(), kv, tree, scale, out=out, want_lse=True)
    ref, ref_lse, sel, st = oracle.tree_attention(W.bits(q), W.bits(k), W.bits(v), oracle.KVLayout(cap, Hkv, D),
                                                  par, tl, kl, Hq, scale)
    assert st == 0
    compare_attention(out, lse, ref, ref_lse, sel)
    # rows past tree_len are untouched
    assert (out[-1, tl[-1]:].float() == 7.0).all()


def test_attention_uneven_lengths(dreams):
    """Sequences of very different lengths in one call: the long ones are
    split over several CTAs and merged, the short ones are not, and the
    items run longest first."""
    rng = np.random.default_rng(77)
    B, Hq, Hkv, D, T, cap = 5, 8, 2, 128, 24, 4096
    par = np.stack([W.random_tree(rng, T) for _ in range(B)]).astype(np.int32)
    tl = np.array([24, 1, 17, 24, 9], np.int32)
    for b in range(B):
        par[b, tl[b]:] = -1
    kl = np.array([4000, 0, 1500, 63, 3333], np.int32)
    kl = np.minimum(kl, cap - tl)
    q = W.bf16(rng.standard_normal((B, T, Hq, D), dtype=np.float32))
    k = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    v = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    scale = 1.0 / np.sqrt(D)
    kv = dreams.KVCache(k.cuda(), v.cuda())
    tree = dreams.Tree(torch.from_numpy(par).cuda(), torch.zeros((B, T), dtype=torch.int32, device="cuda"),
                       torch.from_numpy(tl).cuda(), torch.from_numpy(kl).cuda())
    st = _status()
    out, lse = dreams.tree_verify_attn(q.cuda(), kv, tree, scale, want_lse=True, status=st)
    ref, ref_lse, sel, ost = oracle.tree_attention(W.bits(q), W.bits(k), W.bits(v), oracle.KVLayout(cap, Hkv, D),
                                                   par, tl, kl, Hq, scale)
    assert ost == 0 and int(st.item()) == 0
    compare_attention(out, lse, ref, ref_lse, sel)


@pytest.mark.parametrize("B", [64, 80])
def test_attention_many_sequences(dreams, B):
    """64 (sequence, split) pairs are the most each CTA ranks itself; 80 take
    the separate ordering pass. Lengths repeat, so equal work sizes tie."""
    rng = np.random.default_rng(B)
    Hq, Hkv, D, T, cap = 4, 2, 64, 8, 320
    par = np.stack([W.random_tree(rng, T) for _ in range(B)]).astype(np.int32)
    tl = rng.integers(1, T + 1, B).astype(np.int32)
    for b in range(B):
        par[b, tl[b]:] = -1
    kl = rng.choice([0, 5, 127, 128, 200, 311], B).astype(np.int32)
    kl = np.minimum(kl, cap - tl)
    q = W.bf16(rng.standard_normal((B, T, Hq, D), dtype=np.float32))
    k = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    v = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    scale = 1.0 / np.sqrt(D)
    kv = dreams.KVCache(k.cuda(), v.cuda())
    tree = dreams.Tree(torch.from_numpy(par).cuda(), torch.zeros((B, T), dtype=torch.int32, device="cuda"),
                       torch.from_numpy(tl).cuda(), torch.from_numpy(kl).cuda())
    assert dreams.tree_verify_attn_launches(kv, tree, Hq) == (1 if B <= 64 else 2)
    st = _status()
    out, lse = dreams.tree_verify_attn(q.cuda(), kv, tree, scale, want_lse=True, status=st)
    ref, ref_lse, sel, ost = oracle.tree_attention(W.bits(q), W.bits(k), W.bits(v), oracle.KVLayout(cap, Hkv, D),
                                                   par, tl, kl, Hq, scale)
    assert ost == 0 and int(st.item()) == 0
    compare_attention(out, lse, ref, ref_lse, sel)


@pytest.mark.parametrize("B", [1, 3])
def test_attention_malformed_tree(dreams, B):
    """A sequence whose parent array is malformed (a parent after its child)
    is flagged and its output rows are left untouched, while the MMAs and
    copies of its CTAs stop through the abort flag; the other sequences are
    computed as usual. B = 1 splits the KV range, B = 3 ranks the pairs."""
    rng = np.random.default_rng(90 + B)
    Hq, Hkv, D, T, cap = 8, 2, 128, 40, 1536
    par = np.stack([W.random_tree(rng, T) for _ in range(B)]).astype(np.int32)
    bad = B // 2
    good_par = par.copy()
    par[bad, 7] = 9
    tl = np.full(B, T, np.int32)
    kl = np.array([1000, 700, 1200][:B], np.int32)
    q = W.bf16(rng.standard_normal((B, T, Hq, D), dtype=np.float32))
    k = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    v = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    scale = 1.0 / np.sqrt(D)
    kv = dreams.KVCache(k.cuda(), v.cuda())
    tree = dreams.Tree(torch.from_numpy(par).cuda(), torch.zeros((B, T), dtype=torch.int32, device="cuda"),
                       torch.from_numpy(tl).cuda(), torch.from_numpy(kl).cuda())
    out = torch.full((B, T, Hq, D), 7.0, dtype=torch.bfloat16, device="cuda")
    st = _status()
    out, lse = dreams.tree_verify_attn(q.cuda(), kv, tree, scale, out=out, want_lse=True, status=st)
    s = int(st.item())
    assert s & dreams.DATA_BAD_PARENT and not s & dreams.DATA_TIMEOUT, hex(s)
    assert (out[bad].float() == 7.0).all()
    others = [b for b in range(B) if b != bad]
    if others:
        sel = np.array([(b, t, h) for b in others for t in range(T) for h in range(Hq)], np.int32)
        ref, ref_lse, sel, ost = oracle.tree_attention(W.bits(q), W.bits(k), W.bits(v),
                                                       oracle.KVLayout(cap, Hkv, D), good_par, tl, kl, Hq, scale,
                                                       sel=sel)
        assert ost == 0
        compare_attention(out, lse, ref, ref_lse, sel)


def test_attention_paged_equals_contiguous(dreams):
    """The batched workload copied into a contiguous cache gives bit-identical
    results to its paged form."""
    w = W.make("batched", with_logits=False)
    g = to_gpu(w)
    out_p, lse_p = dreams.tree_verify_attn(g["q"], g["kv"], g["tree"], w.scale, want_lse=True)
    pt = w.page_table.numpy()
    cap = w.capacity
    kc = torch.zeros((w.B, cap, w.Hkv, w.D), dtype=torch.bfloat16)
    vc = torch.zeros_like(kc)
    for b in range(w.B):
        for j in range(w.pages_per_seq):
            if pt[b, j] >= 0:
                kc[b, j * 64:(j + 1) * 64] = w.k[pt[b, j]]
                vc[b, j * 64:(j + 1) * 64] = w.v[pt[b, j]]
    kv_c = dreams.KVCache(kc.cuda(), vc.cuda())
    out_c, lse_c = dreams.tree_verify_attn(g["q"], kv_c, g["tree"], w.scale, want_lse=True)
    for b in range(w.B):
        t = int(w.tree_len[b])
        assert torch.equal(out_p[b, :t], out_c[b, :t])
        assert torch.equal(lse_p[b, :t], lse_c[b, :t])


def test_attention_repeatable(dreams):
    """Two calls on the same inputs give identical bits (the split merge has a
    fixed order, whichever SM computed each split)."""
    w = W.make("long13b", with_logits=False)
    g = to_gpu(w)
    a, la = dreams.tree_verify_attn(g["q"], g["kv"], g["tree"], w.scale, want_lse=True)
    a = a.clone()
    la = la.clone()
    b, lb = dreams.tree_verify_attn(g["q"], g["kv"], g["tree"], w.scale, want_lse=True)
    assert torch.equal(a, b) and torch.equal(la, lb)


# ------------------------------------------------------------------ argmax
@pytest.mark.parametrize("name", CONFIGS)
def test_argmax_matches_oracle(dreams, name):
    w = W.make(name, with_attn=False)
    x = w.logits.cuda()
    am = dreams.vocab_argmax(x)
    ref = logits_rows_oracle(w)
    np.testing.assert_array_equal(am.cpu().numpy(), ref)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_argmax_edge_rows(dreams, dtype):
    nan, inf = float("nan"), float("inf")
    V = 4099  # not a multiple of the vector width
    rng = np.random.default_rng(9)
    x = rng.standard_normal((12, V)).astype(np.float32)
    x[0, :] = 1.0                   # all equal -> 0
    x[1, [5, 4000]] = 50.0          # tie across chunks -> 5
    x[2, :] = -0.0
    x[2, 3000] = 0.0                # +0 == -0 -> 0
    x[3, :] = -inf                  # -> 0
    x[4, [17, 2000]] = nan          # first NaN -> 17
    x[5, 4098] = 99.0               # tail element
    x[6, 0] = inf
    x[6, 1] = inf                   # -> 0
    x[7, :] = -1.0
    x[7, 4097] = -0.5               # tail
    x[8, 3] = nan
    x[8, 2] = inf                   # NaN beats inf -> 3
    x[9, 4096:] = 1e30              # tail maxima, first wins
    t = torch.from_numpy(x).to(dtype)
    ref = (oracle.argmax(W.bits(t), bf16_bits=True) if dtype == torch.bfloat16 else oracle.argmax(x))
    np.testing.assert_array_equal(dreams.vocab_argmax(t.cuda()).cpu().numpy(), ref)
    np.testing.assert_array_equal(ref[:10], [0, 5, 0, 0, 17, 4098, 0, 4097, 3, 4096])
    # padded rows (row_stride > V) and a base that is not 16-byte aligned
    pad = torch.full((12, V + 5), 1e30, dtype=dtype)
    pad[:, 1:V + 1] = t
    got = dreams.vocab_argmax(pad.cuda()[:, 1:V + 1])
    np.testing.assert_array_equal(got.cpu().numpy(), ref)


@pytest.mark.parametrize("rows,V", [(1, 1), (3, 7), (1, 152064), (700, 9), (2, 1_000_003)])
def test_argmax_shapes(dreams, rows, V):
    rng = np.random.default_rng(rows + V)
    x = (rng.standard_normal((rows, V)) * 3).astype(np.float32)
    t = torch.from_numpy(x).to(torch.bfloat16)
    np.testing.assert_array_equal(dreams.vocab_argmax(t.cuda()).cpu().numpy(),
                                  oracle.argmax(W.bits(t), bf16_bits=True))
    np.testing.assert_array_equal(dreams.vocab_argmax(torch.from_numpy(x).cuda()).cpu().numpy(),
                                  oracle.argmax(x))


# ------------------------------------------------------------------ acceptance
def _tree_gpu(dreams, parent, tokens, tree_len, kv_len):
    f = lambda a: torch.as_tensor(np.asarray(a, np.int32)).cuda()
    return dreams.Tree(f(parent), f(tokens), f(tree_len), f(kv_len))


@pytest.mark.parametrize("seed", range(6))
def test_accept_path_random_trees(dreams, seed):
    rng = np.random.default_rng(seed)
    B, T_max = 40, 64
    par = np.full((B, T_max), -1, np.int32)
    tl = rng.integers(1, T_max + 1, B).astype(np.int32)
    for b in range(B):
        par[b, :tl[b]] = W.random_tree(rng, int(tl[b]))
    vocab = [2, 3, 5, 50][seed % 4]
    tok = rng.integers(0, vocab, (B, T_max)).astype(np.int32)
    am = rng.integers(0, vocab, (B, T_max)).astype(np.int32)
    kl = rng.integers(0, 5000, B).astype(np.int32)
    max_path = [65, 8, 3, 1, 30, 65][seed]
    tree = _tree_gpu(dreams, par, tok, tl, kl)
    r = dreams.accept_path(torch.from_numpy(am).cuda(), tree, max_path)
    ref = oracle.accept_path(am, par, tok, tl, kl, max_path)
    for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
        np.testing.assert_array_equal(r[key].cpu().numpy(), ref[key], err_msg=key)


def test_accept_path_bad_data(dreams):
    par = np.array([[-1, 0, 0, 1], [-1, 0, 2, 1], [0, 0, 1, 2], [-1, 0, 0, 0]], np.int32)
    tl = np.array([4, 4, 4, 9], np.int32)
    kl = np.array([3, 3, 3, 3], np.int32)
    kl2 = np.array([-1, 3, 3, 3], np.int32)
    tok = np.zeros((4, 4), np.int32)
    am = np.zeros((4, 4), np.int32)
    st = _status()
    r = dreams.accept_path(torch.from_numpy(am).cuda(), _tree_gpu(dreams, par, tok, tl, kl2), 5, status=st)
    s = int(st.item())
    assert s & dreams.DATA_BAD_PARENT and s & dreams.DATA_BAD_TREE_LEN and s & dreams.DATA_BAD_KV_LEN
    np.testing.assert_array_equal(r["accept_len"].cpu().numpy(), [0, 0, 0, 0])
    np.testing.assert_array_equal(r["new_kv_len"].cpu().numpy(), kl2)
    assert (r["path"].cpu().numpy() == -1).all()


# ------------------------------------------------------------------ compaction
@pytest.mark.parametrize("paged", [False, True])
def test_kv_compact_matches_oracle(dreams, paged):
    rng = np.random.default_rng(31 + paged)
    B, cap, Hkv, D, n_layers, page = 5, 256, 4, 128, 3, 64
    k = rng.integers(0, 65536, (n_layers, B, cap, Hkv, D), dtype=np.uint16)
    v = rng.integers(0, 65536, (n_layers, B, cap, Hkv, D), dtype=np.uint16)
    L = np.array([10, 0, 60, 100, 180], np.int32)
    max_path = 9
    acc = np.array([3, 1, 8, 0, 9], np.int32)
    path = np.full((B, max_path), -1, np.int32)
    path[0, :3] = [0, 2, 3]
    path[1, :1] = [0]
    path[2, :8] = [0, 1, 5, 7, 9, 10, 30, 63]
    path[4, :9] = [0, 3, 4, 6, 8, 20, 40, 70, 75]
    if paged:
        pps = cap // page
        table = rng.permutation(B * pps).astype(np.int32).reshape(B, pps)
        kin = np.empty((n_layers, B * pps, page, Hkv, D), np.uint16)
        vin = np.empty_like(kin)
        for b in range(B):
            for j in range(pps):
                kin[:, table[b, j]] = k[:, b, j * page:(j + 1) * page]
                vin[:, table[b, j]] = v[:, b, j * page:(j + 1) * page]
        lay = oracle.KVLayout(cap, Hkv, D, page_table=table, page_size=page, num_pages=B * pps)
        pt = torch.from_numpy(table).cuda()
    else:
        kin, vin, pt = k, v, None
        lay = oracle.KVLayout(cap, Hkv, D)
    ko, vo, ost = oracle.kv_compact(kin, vin, lay, L, acc, path, n_layers=n_layers,
                                    layer_stride=kin[0].size)
    assert ost == 0
    tk = torch.from_numpy(kin.view(np.int16)).view(torch.bfloat16).cuda()
    tv = torch.from_numpy(vin.view(np.int16)).view(torch.bfloat16).cuda()
    kv = dreams.KVCache(tk, tv, pt)
    st = _status()
    f = lambda a: torch.from_numpy(a).cuda()
    dreams.kv_compact(kv, f(L), f(acc), f(path), status=st)
    assert int(st.item()) == 0
    assert np.array_equal(tk.view(torch.int16).cpu().numpy().view(np.uint16), ko)
    assert np.array_equal(tv.view(torch.int16).cpu().numpy().view(np.uint16), vo)


def test_kv_compact_bad_path_untouched(dreams):
    B, cap, Hkv, D = 3, 64, 1, 64
    k = torch.randn((B, cap, Hkv, D)).to(torch.bfloat16).cuda()
    k0 = k.clone()
    kv = dreams.KVCache(k, k.clone())
    path = torch.tensor([[1, 2, 3], [0, 2, 2], [0, 1, 60]], dtype=torch.int32, device="cuda")
    st = _status()
    dreams.kv_compact(kv, torch.tensor([0, 0, 10], dtype=torch.int32, device="cuda"),
                      torch.tensor([3, 3, 3], dtype=torch.int32, device="cuda"), path, status=st)
    s = int(st.item())
    assert s & dreams.DATA_BAD_PATH and s & dreams.DATA_BAD_KV_LEN
    assert torch.equal(k, k0)


# ------------------------------------------------------------------ fused step
@pytest.mark.parametrize("name", CONFIGS)
def test_verify_step_matches_oracle(dreams, name):
    w = W.make(name)
    g = to_gpu(w)
    max_path = w.max_path
    am_out = torch.full((w.B, w.T_max), -7, dtype=torch.int32, device="cuda")
    st = _status()
    r = dreams.verify_step(g["logits"], g["tree"], g["kv"], max_path, argmax_out=am_out, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    am_ref = logits_rows_oracle(w)
    am_gpu = am_out.cpu().numpy()
    for b in range(w.B):
        t = int(w.tree_len[b])
        np.testing.assert_array_equal(am_gpu[b, :t], am_ref[b, :t])
        assert (am_gpu[b, t:] == -7).all()
    ref = oracle.accept_path(am_ref, w.parent.numpy(), w.tokens.numpy(), w.tree_len.numpy(),
                             w.kv_len.numpy(), max_path)
    for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
        np.testing.assert_array_equal(r[key].cpu().numpy(), ref[key], err_msg=key)
    # planted structure: mean acceptance is well above 1
    assert ref["accept_len"].mean() > 1.5
    ko, vo, ost = oracle.kv_compact(W.bits(w.k), W.bits(w.v), layout(w), w.kv_len.numpy(), ref["accept_len"],
                                    ref["path"])
    assert ost == 0
    assert np.array_equal(W.bits(g["k"].cpu()), ko)
    assert np.array_equal(W.bits(g["v"].cpu()), vo)


@pytest.mark.parametrize("name", ["batched", "llava7b"])
def test_verify_step_per_sequence_views(dreams, name):
    """verify_step called once per sequence, on views of that sequence's row
    of every input and output (a KV cache view: its page-table row, or its
    slice of a contiguous cache), gives what one batched call gives: the same
    predictions, walk outputs and compacted cache, bit for bit. The bench's
    end-to-end step verifies each sequence as its logits land this way."""
    w = W.make(name)
    a, b_ = to_gpu(w), to_gpu(w)
    st = _status()
    am_a = torch.full((w.B, w.T_max), -7, dtype=torch.int32, device="cuda")
    r_a = dreams.verify_step(a["logits"], a["tree"], a["kv"], w.max_path, argmax_out=am_a, status=st)
    am_b = torch.full((w.B, w.T_max), -7, dtype=torch.int32, device="cuda")
    outs = (torch.full((w.B,), -9, dtype=torch.int32, device="cuda"),
            torch.full((w.B, w.max_path), -9, dtype=torch.int32, device="cuda"),
            torch.full((w.B, w.max_path), -9, dtype=torch.int32, device="cuda"),
            torch.full((w.B,), -9, dtype=torch.int32, device="cuda"))
    tr = b_["tree"]
    for s in range(w.B):
        one = slice(s, s + 1)
        kv_s = (dreams.KVCache(b_["k"], b_["v"], b_["page_table"][one]) if b_["page_table"] is not None
                else dreams.KVCache(b_["k"][one], b_["v"][one]))
        tree_s = dreams.Tree(tr.parent[one], tr.tokens[one], tr.tree_len[one], tr.kv_len[one])
        dreams.verify_step(b_["logits"][one], tree_s, kv_s, w.max_path, argmax_out=am_b[one],
                           outputs=tuple(o[one] for o in outs), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert torch.equal(am_a, am_b)
    for key, o in zip(("accept_len", "path", "out_tokens", "new_kv_len"), outs):
        assert torch.equal(r_a[key], o), key
    assert torch.equal(a["k"], b_["k"]) and torch.equal(a["v"], b_["v"])


def test_verify_step_bad_sequences(dreams):
    """Bad data in one sequence is reported and leaves the others intact."""
    w = W.make("batched", with_attn=True)
    am_ref = logits_rows_oracle(w)
    ref = oracle.accept_path(am_ref, w.parent.numpy(), w.tokens.numpy(), w.tree_len.numpy(), w.kv_len.numpy(),
                             w.max_path)
    pb = [b for b in range(9, w.B) if ref["accept_len"][b] >= 2][0]  # has moves to make
    par = w.parent.clone()
    par[2, 5] = 7            # parent not below the node
    tl = w.tree_len.clone()
    tl[4] = 0                # empty tree
    kl = w.kv_len.clone()
    kl[6] = w.capacity       # no room for the tree
    pt = w.page_table.clone()
    lo, hi = int(w.kv_len[pb]) // 64, (int(w.kv_len[pb]) + int(w.tree_len[pb]) - 1) // 64
    pt[pb, lo:hi + 1] = w.num_pages + 3  # bad pages under the tree slots
    w2 = W.Workload(**{**w.__dict__, "parent": par, "tree_len": tl, "kv_len": kl, "page_table": pt})
    g = to_gpu(w2)
    st = _status()
    r = dreams.verify_step(g["logits"], g["tree"], g["kv"], w.max_path, status=st)
    s = int(st.item())
    assert s & dreams.DATA_BAD_PARENT and s & dreams.DATA_BAD_TREE_LEN and s & dreams.DATA_BAD_KV_LEN
    assert s & dreams.DATA_BAD_PAGE
    acc = r["accept_len"].cpu().numpy()
    assert acc[2] == 0 and acc[4] == 0 and acc[6] == 0
    good = [b for b in range(w.B) if b not in (2, 4, 6, pb)]
    np.testing.assert_array_equal(acc[good], ref["accept_len"][good])


def test_status_word_clean_on_valid_input(dreams):
    w = W.make("tiny")
    g = to_gpu(w)
    st = _status()
    dreams.tree_verify_attn(g["q"], g["kv"], g["tree"], w.scale, status=st)
    dreams.verify_step(g["logits"], g["tree"], g["kv"], w.max_path, status=st)
    assert int(st.item()) == 0


# ------------------------------------------------------------------ scan partition
def test_argmax_many_short_rows(dreams):
    """More rows than eight per CTA: every CTA takes whole rows (no workspace)."""
    rows, V = 5003, 37
    rng = np.random.default_rng(11)
    x = (rng.standard_normal((rows, V)) * 2).astype(np.float32)
    x[::7, 5] = x[::7, 30] = 99.0  # ties inside a row
    assert dreams._lib().dreams_vocab_argmax_workspace_size(rows, V) == 0
    for t in (torch.from_numpy(x), torch.from_numpy(x).to(torch.bfloat16)):
        ref = (oracle.argmax(W.bits(t), bf16_bits=True) if t.dtype == torch.bfloat16 else oracle.argmax(x))
        np.testing.assert_array_equal(dreams.vocab_argmax(t.cuda()).cpu().numpy(), ref)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_argmax_split_rows_repeat(dreams, dtype):
    """Rows split between many CTAs, aligned and unaligned bases, two calls on
    one explicit workspace: same answers, workspace zero-filled afterwards."""
    rows, V = 5, 300_001
    rng = np.random.default_rng(12)
    x = rng.standard_normal((rows, V)).astype(np.float32)
    x[0, [17, 250_000]] = 40.0   # equal maxima far apart: lowest index wins
    x[1, V - 1] = 40.0           # the maximum in the partial last vector
    x[2, 123_457] = float("nan")
    t = torch.from_numpy(x).to(dtype)
    ref = (oracle.argmax(W.bits(t), bf16_bits=True) if dtype == torch.bfloat16 else oracle.argmax(x))
    need = dreams._lib().dreams_vocab_argmax_workspace_size(rows, V)
    assert need > 0
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    pad = torch.zeros((rows, V + 3), dtype=dtype)
    pad[:, 1:V + 1] = t
    for src in (t.cuda(), pad.cuda()[:, 1:V + 1]):
        for _ in range(2):
            got = dreams.vocab_argmax(src, workspace=ws)
            np.testing.assert_array_equal(got.cpu().numpy(), ref)
            assert int(ws.count_nonzero().item()) == 0


@pytest.mark.parametrize("dtype,aligned", [(torch.bfloat16, True), (torch.float32, False)])
def test_verify_step_ragged_repeat(dreams, dtype, aligned):
    """Ragged and invalid trees, a vocabulary that is not a multiple of the
    vector width, rows split between CTAs; two calls on one workspace."""
    rng = np.random.default_rng(13)
    B, T_max, V, Hkv, D, cap = 7, 9, 100_003, 2, 16, 64
    tl = np.array([1, 9, 0, 5, 9, 2, 3], np.int32)  # sequence 2 is invalid
    par = np.full((B, T_max), -1, np.int32)
    for b in range(B):
        if tl[b] > 0:
            par[b, :tl[b]] = W.random_tree(rng, int(tl[b]))
    tok = rng.integers(0, V, (B, T_max)).astype(np.int32)
    x = rng.standard_normal((B, T_max, V)).astype(np.float32)
    for b in range(B):  # plant matches along the first child of each node
        for i in range(1, int(tl[b])):
            x[b, par[b, i], tok[b, i]] = 50.0 + i
    kl = np.array([0, 10, 5, 40, 55, 3, 20], np.int32)
    k = torch.from_numpy(rng.standard_normal((B, cap, Hkv, D)).astype(np.float32)).to(torch.bfloat16)
    v = torch.from_numpy(rng.standard_normal((B, cap, Hkv, D)).astype(np.float32)).to(torch.bfloat16)
    t = torch.from_numpy(x).to(dtype)
    rows_ref = (oracle.argmax(W.bits(t.reshape(-1, V)), bf16_bits=True) if dtype == torch.bfloat16
                else oracle.argmax(x.reshape(-1, V))).reshape(B, T_max)
    ref = oracle.accept_path(rows_ref, par, tok, tl, kl, T_max + 1)
    if aligned:
        lg = t.cuda()
    else:
        pad = torch.zeros((B, T_max, V + 1), dtype=dtype)
        pad[:, :, 1:] = t
        lg = pad.cuda()[:, :, 1:]
    f = lambda a: torch.as_tensor(a).cuda()
    tree = dreams.Tree(f(par), f(tok), f(tl), f(kl))
    kv = dreams.KVCache(k.cuda(), v.cuda())
    ws = torch.zeros(dreams.verify_step_workspace_size(tree, V), dtype=torch.uint8, device="cuda")
    lay = oracle.KVLayout(cap, Hkv, D)
    ko, vo = W.bits(k), W.bits(v)
    for call in range(2):
        st = _status()
        am = torch.full((B, T_max), -7, dtype=torch.int32, device="cuda")
        r = dreams.verify_step(lg, tree, kv, T_max + 1, argmax_out=am, workspace=ws, status=st)
        torch.cuda.synchronize()
        assert int(st.item()) == dreams.DATA_BAD_TREE_LEN
        assert int(ws.count_nonzero().item()) == 0
        amc = am.cpu().numpy()
        for b in range(B):
            np.testing.assert_array_equal(amc[b, :tl[b]], rows_ref[b, :tl[b]])
            assert (amc[b, tl[b]:] == -7).all()
        for key in ("accept_len", "path", "out_tokens", "new_kv_len"):
            np.testing.assert_array_equal(r[key].cpu().numpy(), ref[key], err_msg=key)
        ko, vo, ost = oracle.kv_compact(ko, vo, lay, kl, ref["accept_len"], ref["path"])
        assert ost == 0
        assert np.array_equal(W.bits(kv.k.cpu()), ko) and np.array_equal(W.bits(kv.v.cpu()), vo)


@pytest.mark.parametrize("tail", [1, 63, 64, 65, 127])
def test_attention_paged_ragged_tails(dreams, tail):
    """A paged cache (pages in a seeded random order) whose sequences end `tail`
    keys into their last 128-key tile: before, at and after the 64-key halves
    in which P goes to the MMA thread, for a long sequence split over several
    CTAs, a medium one and a one-tile one. The paged run equals the contiguous
    run bit for bit, and both match the oracle."""
    rng = np.random.default_rng(1000 + tail)
    B, Hq, Hkv, D, T, cap = 3, 8, 2, 128, 24, 1024
    tl = np.array([24, 9, 1], np.int32)
    tiles = np.array([7, 2, 0])
    kl = (128 * tiles + tail - tl).astype(np.int32)
    kl[2] = max(0, tail - 1)
    assert (kl >= 0).all() and (kl + tl <= cap).all()
    par = np.stack([W.random_tree(rng, T) for _ in range(B)]).astype(np.int32)
    for b in range(B):
        par[b, tl[b]:] = -1
    q = W.bf16(rng.standard_normal((B, T, Hq, D), dtype=np.float32))
    k = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    v = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    pps = cap // 64
    perm = torch.randperm(B * pps, generator=torch.Generator().manual_seed(tail))
    table = perm.view(B, pps).to(torch.int32)
    kp = torch.empty((B * pps, 64, Hkv, D), dtype=torch.bfloat16)
    vp = torch.empty_like(kp)
    for b in range(B):
        for pg in range(pps):
            kp[table[b, pg]] = k[b, 64 * pg:64 * (pg + 1)]
            vp[table[b, pg]] = v[b, 64 * pg:64 * (pg + 1)]
    tree = dreams.Tree(torch.from_numpy(par).cuda(), torch.zeros((B, T), dtype=torch.int32, device="cuda"),
                       torch.from_numpy(tl).cuda(), torch.from_numpy(kl).cuda())
    scale = 1.0 / np.sqrt(D)
    st = _status()
    res = []
    for kv in (dreams.KVCache(k.cuda(), v.cuda()), dreams.KVCache(kp.cuda(), vp.cuda(), table.cuda())):
        res.append(dreams.tree_verify_attn(q.cuda(), kv, tree, scale, want_lse=True, status=st))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    for b in range(B):
        for x, y in zip(res[0], res[1]):
            assert torch.equal(x[b, :tl[b]], y[b, :tl[b]])
    ref, ref_lse, sel, ost = oracle.tree_attention(W.bits(q), W.bits(k), W.bits(v), oracle.KVLayout(cap, Hkv, D),
                                                   par, tl, kl, Hq, scale)
    assert ost == 0
    compare_attention(res[1][0], res[1][1], ref, ref_lse, sel)
