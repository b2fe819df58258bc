"""The bounded pipeline waits of the tcgen05 kernels, made to run out on
purpose without any fault: the test hook dreams_test_set_stall withholds the
TMA copies of each CTA from a given tile on (the consumers then wait on
barriers that nothing completes) and shortens every wait to 20 ms. The kernels
must flag DREAMS_DATA_TIMEOUT, leave the output rows they did not finish
untouched, wait for the copies and MMAs they did issue and free their tensor
memory: the next normal call on the same device must then be bit-identical to
a call made before the stall (a CTA that kept its tensor memory would leave the
next kernel unable to allocate)."""
import numpy as np
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu

SENTINEL = 0x7F7F  # bf16 bit pattern no attention output takes here (3.4e38)


@pytest.fixture(scope="module")
def dreams():
    import paper_2606_00535_gb300 as d
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    d._lib()
    yield d
    d.test_set_stall(0, -1)


def _uneven_case(dreams, Hq):
    """Five sequences: two fit in one 128-key tile (they finish before any
    stall at the second tile), three span 12 to 32 tiles. With 4 query heads
    per KV head the 24 nodes fill one row block per KV head; with 8, two."""
    rng = np.random.default_rng(77)
    B, Hkv, D, T, cap = 5, 2, 128, 24, 4096
    par = np.stack([W.random_tree(rng, T) for _ in range(B)]).astype(np.int32)
    tl = np.array([24, 1, 17, 24, 9], np.int32)
    for b in range(B):
        par[b, tl[b]:] = -1
    kl = np.array([4000, 0, 1500, 63, 3333], np.int32)
    kl = np.minimum(kl, cap - tl)
    q = W.bf16(rng.standard_normal((B, T, Hq, D), dtype=np.float32)).cuda()
    k = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32)).cuda()
    v = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32)).cuda()
    kv = dreams.KVCache(k, v)
    tree = dreams.Tree(torch.from_numpy(par).cuda(), torch.zeros((B, T), dtype=torch.int32, device="cuda"),
                       torch.from_numpy(tl).cuda(), torch.from_numpy(kl).cuda())
    return q, kv, tree, tl, D ** -0.5


def _attend(dreams, q, kv, tree, scale):
    out = torch.full(q.shape, 0, dtype=torch.int16, device="cuda").fill_(SENTINEL).view(torch.bfloat16)
    lse = torch.full(q.shape[:3], -7.0, dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    dreams.tree_verify_attn(q, kv, tree, scale, out=out, lse=lse, status=st)
    torch.cuda.synchronize()
    return out.view(torch.int16).clone(), lse.clone(), int(st.item())


@pytest.mark.parametrize("Hq", [8, 16])
def test_attention_wait_runs_out_then_recovers(dreams, Hq):
    q, kv, tree, tl, scale = _uneven_case(dreams, Hq)
    ref_out, ref_lse, st = _attend(dreams, q, kv, tree, scale)
    assert st == 0
    try:
        # no K tile is ever issued: every CTA's first wait runs out
        dreams.test_set_stall(dreams.TEST_ATTENTION, 0, 20_000_000)
        out, lse, st = _attend(dreams, q, kv, tree, scale)
    finally:
        dreams.test_set_stall(0, -1)
    assert st == dreams.DATA_TIMEOUT
    assert (out == SENTINEL).all() and (lse == -7.0).all()
    # tensor memory and workspace are clean: the next call matches the first
    out2, lse2, st2 = _attend(dreams, q, kv, tree, scale)
    assert st2 == 0
    assert torch.equal(out2, ref_out) and torch.equal(lse2, ref_lse)


@pytest.mark.parametrize("Hq", [8, 16])
def test_attention_partial_stall_leaves_unfinished_rows_untouched(dreams, Hq):
    """Copies withheld from the second K tile on: the one-tile sequences (1 and
    3) finish and match the normal call bit for bit; every row of the long
    ones, whether written directly or through the merge of the KV splits (a
    KV split spans at least two tiles, so the first split of every row block
    gives up and tells the merge to skip the row), is untouched."""
    q, kv, tree, tl, scale = _uneven_case(dreams, Hq)
    ref_out, ref_lse, _ = _attend(dreams, q, kv, tree, scale)
    try:
        dreams.test_set_stall(dreams.TEST_ATTENTION, 1, 20_000_000)
        out, lse, st = _attend(dreams, q, kv, tree, scale)
    finally:
        dreams.test_set_stall(0, -1)
    assert st == dreams.DATA_TIMEOUT
    for b in range(len(tl)):
        n = int(tl[b])
        if b in (1, 3):
            assert torch.equal(out[b, :n], ref_out[b, :n]) and torch.equal(lse[b, :n], ref_lse[b, :n])
        else:
            assert (out[b] == SENTINEL).all() and (lse[b] == -7.0).all(), b
    out2, lse2, st2 = _attend(dreams, q, kv, tree, scale)
    assert st2 == 0 and torch.equal(out2, ref_out) and torch.equal(lse2, ref_lse)


def test_lm_head_wait_runs_out_then_recovers(dreams):
    g = torch.Generator().manual_seed(8)
    rows, K, V = 300, 1024, 40000
    h = torch.randn((rows, K), generator=g).to(torch.bfloat16).cuda()
    w = (torch.randn((V, K), generator=g) / 32).to(torch.bfloat16).cuda()
    ws = torch.zeros(dreams._lib().dreams_lm_head_argmax_workspace_size(rows), dtype=torch.uint8, device="cuda")

    def run():
        idx = torch.full((rows,), -5, dtype=torch.int32, device="cuda")
        mx = torch.full((rows,), -5.0, dtype=torch.float32, device="cuda")
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        dreams.lm_head_argmax(h, w, out=idx, out_max=mx, workspace=ws, status=st)
        torch.cuda.synchronize()
        return idx.clone(), mx.clone(), int(st.item())

    ref_idx, ref_mx, st = run()
    assert st == 0
    try:
        dreams.test_set_stall(dreams.TEST_LM_HEAD, 0, 20_000_000)
        idx, mx, st = run()
        assert st == dreams.DATA_TIMEOUT
        assert (idx == -5).all() and (mx == -5.0).all()   # no tile reached any row
        assert int(ws.count_nonzero().item()) == 0
        # a stall mid-way: indices unreliable, but the flag is set and the
        # workspace is left zero-filled
        dreams.test_set_stall(dreams.TEST_LM_HEAD, 40, 20_000_000)
        _, _, st = run()
        assert st == dreams.DATA_TIMEOUT
        assert int(ws.count_nonzero().item()) == 0
    finally:
        dreams.test_set_stall(0, -1)
    idx2, mx2, st2 = run()
    assert st2 == 0 and torch.equal(idx2, ref_idx) and torch.equal(mx2, ref_mx)
