"""Shared test helpers: move a seeded workload to the GPU and run the oracle on
the same inputs. Only tests import this module."""
from __future__ import annotations

import numpy as np
import torch

import oracle
import workloads as W

# Attention tolerance for bf16 inputs with fp32 accumulation and one bf16
# rounding of the output (max-abs, mean-abs over all compared elements).
ATTN_MAX_ABS = 1e-2
ATTN_MEAN_ABS = 1e-3
LSE_REL = 1e-3


def layout(w: W.Workload) -> oracle.KVLayout:
    if w.paged:
        return oracle.KVLayout(w.capacity, w.Hkv, w.D, page_table=w.page_table.numpy(),
                               page_size=w.page_size, num_pages=w.num_pages)
    return oracle.KVLayout(w.capacity, w.Hkv, w.D)


def to_gpu(w: W.Workload, dev="cuda"):
    import paper_2606_00535_gb300 as dreams
    g = {}
    g["q"] = w.q.to(dev)
    g["k"] = w.k.to(dev)
    g["v"] = w.v.to(dev)
    g["page_table"] = None if w.page_table is None else w.page_table.to(dev)
    g["kv"] = dreams.KVCache(g["k"], g["v"], g["page_table"])
    g["tree"] = dreams.Tree(w.parent.to(dev), w.tokens.to(dev), w.tree_len.to(dev), w.kv_len.to(dev))
    g["logits"] = w.logits.to(dev) if w.logits.numel() else None
    return g


def oracle_attention(w: W.Workload, sel=None):
    return oracle.tree_attention(W.bits(w.q), W.bits(w.k), W.bits(w.v), layout(w), w.parent.numpy(),
                                 w.tree_len.numpy(), w.kv_len.numpy(), w.Hq, w.scale, sel=sel)


def compare_attention(out_gpu: torch.Tensor, lse_gpu, ref_out, ref_lse, sel, max_abs=ATTN_MAX_ABS,
                      mean_abs=ATTN_MEAN_ABS, lse_rel=LSE_REL):
    sel = np.asarray(sel)
    o = out_gpu.float().cpu().numpy()[sel[:, 0], sel[:, 1], sel[:, 2]].astype(np.float64)
    err = np.abs(o - ref_out)
    assert np.isfinite(o).all(), "non-finite attention output"
    assert err.max() <= max_abs, f"max-abs {err.max():.3e} > {max_abs}"
    assert err.mean() <= mean_abs, f"mean-abs {err.mean():.3e} > {mean_abs}"
    if lse_gpu is not None:
        lg = lse_gpu.cpu().numpy()[sel[:, 0], sel[:, 1], sel[:, 2]].astype(np.float64)
        rel = np.abs(lg - ref_lse) / np.maximum(np.abs(ref_lse), 1.0)
        assert rel.max() <= lse_rel, f"lse rel {rel.max():.3e} > {lse_rel}"
    return float(err.max()), float(err.mean())


def logits_rows_oracle(w: W.Workload) -> np.ndarray:
    """Oracle argmax of every row of w.logits, shape [B, T_max]."""
    x = w.logits.reshape(-1, w.V)
    if w.logits_dtype == "bf16":
        am = oracle.argmax(W.bits(x), bf16_bits=True)
    else:
        am = oracle.argmax(x.numpy())
    return am.reshape(w.B, w.T_max)
