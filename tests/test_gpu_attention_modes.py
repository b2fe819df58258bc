"""GPU parity of attention without a tree (dreams_attention): the draft's
cross-attention to target features (ATTN_FULL) and a layer's causal prefill
(ATTN_CAUSAL), with each row's entropy, against the fp64 oracle on bf16-rounded
inputs. Output within max-abs 1e-2 / mean-abs 1e-3, lse within 1e-3 relative,
entropy within 2e-3 absolute (P is f32 in the entropy sum)."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dreams():
    import paper_2606_00535_gb300 as d
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    d._lib()
    return d


def _case(seed, B, T_max, Hq, Hkv, D, cap):
    g = torch.Generator().manual_seed(seed)
    q = torch.randn((B, T_max, Hq, D), generator=g).to(torch.bfloat16)
    k = torch.randn((B, cap, Hkv, D), generator=g).to(torch.bfloat16)
    v = torch.randn((B, cap, Hkv, D), generator=g).to(torch.bfloat16)
    return q, k, v


def _run(dreams, q, k, v, q_len, kv_len, scale, mode):
    kvc = dreams.KVCache(k.cuda(), v.cuda(), None)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out, lse, ent = dreams.attention(q.cuda(), kvc, torch.tensor(q_len, dtype=torch.int32, device="cuda"),
                                     torch.tensor(kv_len, dtype=torch.int32, device="cuda"), scale, mode,
                                     want_lse=True, want_entropy=True, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return out.float().cpu().numpy(), lse.cpu().numpy(), ent.cpu().numpy()


def _compare(q, k, v, q_len, kv_len, scale, causal, got, rng, nsel=400):
    B, T_max, Hq = q.shape[:3]
    sel = [(b, t, h) for b in range(B) for t in range(q_len[b]) for h in range(Hq)]
    if len(sel) > nsel:
        sel = [sel[i] for i in rng.choice(len(sel), nsel, replace=False)]
    out, lse, ent = oracle.attention_rows(q.float().numpy(), k.float().numpy(), v.float().numpy(), q_len, kv_len,
                                          scale, causal, sel)
    go, gl, ge = got
    idx = tuple(np.array(sel).T)
    err = np.abs(go[idx] - out)
    assert np.isfinite(go[idx]).all()
    assert err.max() <= 1e-2 and err.mean() <= 1e-3, (err.max(), err.mean())
    assert (np.abs(gl[idx] - lse) / np.maximum(np.abs(lse), 1.0)).max() <= 1e-3
    assert np.abs(ge[idx] - ent).max() <= 2e-3, np.abs(ge[idx] - ent).max()


@pytest.mark.parametrize("Hq,Hkv,D", [(32, 32, 128), (28, 4, 128), (8, 8, 64)])
def test_cross_attention_matches_oracle(dreams, Hq, Hkv, D):
    """Draft queries (a few positions each) against the target features of the whole prompt."""
    B, T_max, cap = 2, 7, 3392
    q, k, v = _case(Hq + D, B, T_max, Hq, Hkv, D, cap)
    q_len, kv_len = [7, 3], [3392, 1500]
    got = _run(dreams, q, k, v, q_len, kv_len, D ** -0.5, dreams.ATTN_FULL)
    _compare(q, k, v, q_len, kv_len, D ** -0.5, False, got, np.random.default_rng(1))


@pytest.mark.parametrize("T,L,Hq,Hkv", [(512, 0, 8, 8), (300, 100, 8, 2), (1100, 0, 4, 4)])
def test_causal_prefill_matches_oracle(dreams, T, L, Hq, Hkv):
    B, D = 1, 128
    q, k, v = _case(T + L, B, T, Hq, Hkv, D, L + T)
    got = _run(dreams, q, k, v, [T], [L], D ** -0.5, dreams.ATTN_CAUSAL)
    _compare(q, k, v, [T], [L], D ** -0.5, True, got, np.random.default_rng(2))


def test_entropy_closed_forms(dreams):
    """Equal scores (q = 0): entropy ln n for cross-attention, ln(t + 1) for causal rows."""
    B, T, H, D, cap = 1, 64, 4, 64, 640
    q = torch.zeros((B, T, H, D), dtype=torch.bfloat16)
    g = torch.Generator().manual_seed(5)
    k = torch.randn((B, cap, H, D), generator=g).to(torch.bfloat16)
    v = torch.randn((B, cap, H, D), generator=g).to(torch.bfloat16)
    _, _, e_full = _run(dreams, q, k, v, [T], [cap], 0.125, dreams.ATTN_FULL)
    np.testing.assert_allclose(e_full[0], np.log(cap), atol=1e-4)
    _, _, e_causal = _run(dreams, q, k[:, :T].contiguous(), v[:, :T].contiguous(), [T], [0], 0.125,
                          dreams.ATTN_CAUSAL)
    np.testing.assert_allclose(e_causal[0], np.log(np.arange(1, T + 1))[:, None].repeat(H, 1), atol=1e-4)


def _paged(k, v, seed):
    """The same cache as a pool of 64-slot pages in a seeded random order,
    with its page table."""
    B, cap, Hkv, D = k.shape
    pps = cap // 64
    perm = torch.randperm(B * pps, generator=torch.Generator().manual_seed(seed))
    kp = torch.empty((B * pps, 64, Hkv, D), dtype=k.dtype)
    vp = torch.empty_like(kp)
    table = perm.view(B, pps).to(torch.int32)
    for b in range(B):
        for p in range(pps):
            kp[table[b, p]] = k[b, 64 * p:64 * (p + 1)]
            vp[table[b, p]] = v[b, 64 * p:64 * (p + 1)]
    return kp, vp, table


@pytest.mark.parametrize("mode", ["full", "causal"])
def test_attention_modes_paged_equal_contiguous(dreams, mode):
    """Cross-attention and causal prefill on a paged cache (pages in a random
    order, several sequences of different lengths, a split KV range): the same
    output, lse and entropy bits as on the contiguous cache, and the oracle's
    values."""
    B, Hq, Hkv, D, cap = 3, 8, 2, 128, 2048
    causal = mode == "causal"
    T_max = 300 if causal else 24
    q, k, v = _case(77 if causal else 78, B, T_max, Hq, Hkv, D, cap)
    q_len = [300, 129, 1] if causal else [24, 5, 1]
    kv_len = [1500, 0, 1747] if causal else [2048, 700, 1]
    m = dreams.ATTN_CAUSAL if causal else dreams.ATTN_FULL
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ql = torch.tensor(q_len, dtype=torch.int32, device="cuda")
    kl = torch.tensor(kv_len, dtype=torch.int32, device="cuda")
    kp, vp, table = _paged(k, v, 5)
    res = []
    for kvc in (dreams.KVCache(k.cuda(), v.cuda(), None), dreams.KVCache(kp.cuda(), vp.cuda(), table.cuda())):
        res.append(dreams.attention(q.cuda(), kvc, ql, kl, D ** -0.5, m, want_lse=True, want_entropy=True, status=st))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    for b in range(B):
        t = q_len[b]
        for x, y in zip(res[0], res[1]):
            assert torch.equal(x[b, :t], y[b, :t])
    got = tuple(x.float().cpu().numpy() for x in res[1])
    _compare(q, k, v, q_len, kv_len, D ** -0.5, causal, got, np.random.default_rng(3))
