"""GPU parity of the fused LM-head argmax (tcgen05 GEMM + epilogue argmax)
against the fp64 oracle. The GEMM sums f32 products in the tensor cores' order,
so two logits within rounding of each other may swap: where an index differs
from the oracle's, its exact logit must lie within the accumulation error
bound of the exact maximum (and such rows must be rare)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dreams():
    import paper_2606_00535_gb300 as d
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    d._lib()
    return d


def _case(rng, rows, K, V, scale=1.0):
    h = W.bf16((rng.standard_normal((rows, K)) * scale).astype(np.float32))
    w = W.bf16((rng.standard_normal((V, K)) / np.sqrt(K)).astype(np.float32))
    return h, w


def _check(h, w, idx, mx):
    ref_idx, ref_max, logits = oracle.lm_head_argmax(W.bits(h), W.bits(w))
    hf = h.double().numpy()
    wf = w.double().numpy()
    bad = np.nonzero(idx != ref_idx)[0]
    for r in bad:
        # f32 accumulation of K exact products: |error| <= K * 2^-24 * sum |h_k w_vk|
        bound = 2.0 * hf.shape[1] * 2.0 ** -24 * np.abs(hf[r]) @ np.abs(wf[int(idx[r])])
        assert ref_max[r] - logits[r, int(idx[r])] <= bound, (r, int(idx[r]), int(ref_idx[r]))
    assert len(bad) <= max(1, 0.01 * len(idx)), f"{len(bad)} of {len(idx)} rows differ"
    rel = np.abs(mx - ref_max) / np.maximum(np.abs(ref_max), 1e-3)
    assert rel.max() < 1e-3, rel.max()


@pytest.mark.parametrize("rows,K,V", [(1, 64, 1), (5, 256, 1000), (60, 4096, 32000), (130, 128, 5003),
                                      (300, 512, 257), (128, 1024, 65536)])
def test_lm_head_argmax_matches_oracle(dreams, rows, K, V):
    rng = np.random.default_rng(rows * 7 + K + V)
    h, w = _case(rng, rows, K, V)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    idx, mx = dreams.lm_head_argmax(h.cuda(), w.cuda(), want_max=True, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    _check(h, w, idx.cpu().numpy(), mx.cpu().numpy())


def test_lm_head_planted_and_strided(dreams):
    """Planted winners (one aligned weight row per hidden row), row strides
    larger than K, and a second call on the same workspace."""
    rng = np.random.default_rng(5)
    rows, K, V, ld = 70, 512, 20000, 520
    h32 = rng.standard_normal((rows, ld)).astype(np.float32)
    w32 = (rng.standard_normal((V, ld)) * 0.02).astype(np.float32)
    plant = rng.choice(V, rows, replace=False)
    w32[plant] = h32 * 0.5
    h, w = W.bf16(h32), W.bf16(w32)
    need = dreams._lib().dreams_lm_head_argmax_workspace_size(rows)
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    hd, wd = h.cuda()[:, :K], w.cuda()[:, :K]
    for _ in range(2):
        idx = dreams.lm_head_argmax(hd, wd, workspace=ws)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(idx.cpu().numpy(), plant)
    assert int(ws.count_nonzero().item()) == 0


def test_lm_head_rejects_bad_shapes(dreams):
    h = torch.zeros((4, 96), dtype=torch.bfloat16, device="cuda")  # K not a multiple of 64
    w = torch.zeros((10, 96), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(RuntimeError):
        dreams.lm_head_argmax(h, w)


def _oracle_over_vocab_chunks(h_sel, w, chunk=8192):
    """Oracle argmax over the whole vocabulary for the rows h_sel, taken chunk
    by chunk of the vocabulary through oracle.lm_head_argmax (fp64 products);
    the first chunk holding the greatest value wins, as the lowest index does."""
    best_idx = np.zeros(h_sel.shape[0], np.int64)
    best_val = np.full(h_sel.shape[0], -np.inf)
    hb = W.bits(h_sel)
    for v0 in range(0, w.shape[0], chunk):
        idx, mx, _ = oracle.lm_head_argmax(hb, W.bits(w[v0:v0 + chunk]))
        take = mx > best_val
        best_val = np.where(take, mx, best_val)
        best_idx = np.where(take, idx + v0, best_idx)
    return best_idx, best_val


@pytest.mark.parametrize("rows,K,V,nsample", [(854, 4096, 128256, 128), (48, 3584, 152064, 48)])
def test_lm_head_argmax_at_benched_shapes(dreams, rows, K, V, nsample):
    """The shapes the LM-head line of the benchmark times: the 854 tree-node
    rows of the batched-serving workload at hidden 4096 and vocabulary 128256,
    and the Qwen2-VL-shaped 48 rows x 3584 x 152064. Sampled rows cover every
    128-row tile (its first and last row included); each is compared with the
    fp64 oracle over the full vocabulary and hidden size, with the same
    accumulation bound as the smaller cases."""
    g = torch.Generator().manual_seed(rows + K)
    h = torch.randn((rows, K), generator=g).to(torch.bfloat16)
    w = torch.empty((V, K), dtype=torch.bfloat16)
    for v0 in range(0, V, 16384):  # in slices, to bound the f32 temporaries
        n = min(16384, V - v0)
        w[v0:v0 + n] = (torch.randn((n, K), generator=g) * K ** -0.5).to(torch.bfloat16)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    idx, mx = dreams.lm_head_argmax(h.cuda(), w.cuda(), want_max=True, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    idx, mx = idx.cpu().numpy(), mx.cpu().numpy()
    rng = np.random.default_rng(rows)
    sel = set()
    tiles = (rows + 127) // 128
    for m in range(tiles):
        lo, hi = 128 * m, min(rows, 128 * m + 128)
        sel |= {lo, hi - 1}
        sel |= set(int(x) for x in rng.choice(np.arange(lo, hi), min(hi - lo, nsample // tiles), replace=False))
    sel = np.array(sorted(sel))
    assert len(sel) >= min(rows, 128)
    ref_idx, ref_max = _oracle_over_vocab_chunks(h[sel], w)
    hf = h[sel].double().numpy()
    bad = np.nonzero(idx[sel] != ref_idx)[0]
    for i in bad:
        r = int(sel[i])
        wv = w[int(idx[r])].double().numpy()
        exact = float(hf[i] @ wv)
        bound = 2.0 * K * 2.0 ** -24 * float(np.abs(hf[i]) @ np.abs(wv))
        assert ref_max[i] - exact <= bound, (r, int(idx[r]), int(ref_idx[i]))
    assert len(bad) <= max(1, 0.01 * len(sel)), f"{len(bad)} of {len(sel)} rows differ"
    rel = np.abs(mx[sel] - ref_max) / np.maximum(np.abs(ref_max), 1e-3)
    assert rel.max() < 1e-3, rel.max()
