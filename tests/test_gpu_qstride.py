"""Queries as a strided view: Q taken straight out of a fused QKV projection
output [B, T, 3, Hq, D] (each token's head rows dense, tokens 3 Hq D elements
apart), through the C ABI's q_stride_b / q_stride_t. The kernels read Q
through a tensor map built from those strides, so the result must be
bit-identical to the same call on a dense copy of Q, and within the attention
tolerance of the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import compare_attention, oracle_attention, to_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dreams():
    import paper_2606_00535_gb300 as d
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    d._lib()
    return d


def _fused(q: torch.Tensor, seed: int) -> torch.Tensor:
    """A [B, T, 3, Hq, D] buffer whose slice [:, :, 0] equals q, with random
    K and V projections around it."""
    B, T, Hq, D = q.shape
    g = torch.Generator().manual_seed(seed)
    qkv = torch.randn((B, T, 3, Hq, D), generator=g).to(torch.bfloat16)
    qkv[:, :, 0] = q
    return qkv


@pytest.mark.parametrize("name", ["tiny", "qwen2vl7b", "batched"])
def test_tree_attention_fused_qkv_view(dreams, name):
    w = W.make(name, with_logits=False)
    g = to_gpu(w)
    qkv = _fused(w.q, 11).cuda()
    qv = qkv[:, :, 0]
    assert not qv.is_contiguous() and qv.stride(1) == 3 * w.Hq * w.D
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out_v, lse_v = dreams.tree_verify_attn(qv, g["kv"], g["tree"], w.scale, want_lse=True, status=st)
    out_d, lse_d = dreams.tree_verify_attn(g["q"], g["kv"], g["tree"], w.scale, want_lse=True)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    rows = [(b, t) for b in range(w.B) for t in range(int(w.tree_len[b]))]
    bi = torch.tensor([r[0] for r in rows])
    ti = torch.tensor([r[1] for r in rows])
    assert torch.equal(out_v[bi, ti].view(torch.int16), out_d[bi, ti].view(torch.int16))
    assert torch.equal(lse_v[bi, ti], lse_d[bi, ti])
    rng = np.random.default_rng(3)
    sel = np.array([(b, t, h) for b, t in rows if rng.random() < 0.1 for h in range(w.Hq)] or
                   [(0, 0, 0)], np.int32)
    ref, ref_lse, sel, ost = oracle_attention(w, sel)
    assert ost == 0
    compare_attention(out_v, lse_v, ref, ref_lse, sel)


def test_causal_attention_fused_qkv_view(dreams):
    """The same through dreams_attention (causal prefill after a prefix)."""
    rng = np.random.default_rng(21)
    B, T, Hq, Hkv, D, L = 2, 200, 8, 2, 128, 150
    cap = L + T
    q = W.bf16(rng.standard_normal((B, T, Hq, D), dtype=np.float32))
    k = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    v = W.bf16(rng.standard_normal((B, cap, Hkv, D), dtype=np.float32))
    kv = dreams.KVCache(k.cuda(), v.cuda())
    q_len = torch.full((B,), T, dtype=torch.int32, device="cuda")
    kv_len = torch.full((B,), L, dtype=torch.int32, device="cuda")
    qkv = _fused(q, 12).cuda()
    scale = D ** -0.5
    out_v, lse_v, ent_v = dreams.attention(qkv[:, :, 0], kv, q_len, kv_len, scale, dreams.ATTN_CAUSAL,
                                           want_lse=True, want_entropy=True)
    out_d, lse_d, ent_d = dreams.attention(q.cuda(), kv, q_len, kv_len, scale, dreams.ATTN_CAUSAL,
                                           want_lse=True, want_entropy=True)
    torch.cuda.synchronize()
    assert torch.equal(out_v.view(torch.int16), out_d.view(torch.int16))
    assert torch.equal(lse_v, lse_d) and torch.equal(ent_v, ent_d)
    sel = [(b, t, h) for b in range(B) for t in (0, 1, 63, 64, 127, 199) for h in (0, 5)]
    ref, ref_lse, _ = oracle.attention_rows(q.float().numpy(), k.float().numpy(), v.float().numpy(), [T] * B,
                                            [L] * B, scale, True, sel)
    compare_attention(out_v, lse_v, ref, ref_lse, np.array(sel, np.int32))
