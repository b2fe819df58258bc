"""Plain fp64 CPU oracle for the DREAM-S tree verification step.

TEST INFRASTRUCTURE. Only the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package. The CUDA library in
``paper_2606_00535_gb300`` never imports it, and this package imports nothing
from there: the two share no code.

The arithmetic lives in ``oracle.c`` (straight double-precision loops, one
thread); this module only marshals numpy arrays into it. Each wrapper names the
paper passage its C routine follows:

* :func:`tree_attention` -- softmax(scale * q K^T) V of each draft-tree query
  over the prefix cache plus its own ancestors (paper Sec. 2 "Speculative
  decoding": one parallel target pass over the drafts; Sec. 2 "Vision-Language
  Models": cached visual and text tokens take part in every decoding step;
  Sec. 3.2: attention = softmax(Q K^T / sqrt(z))).
* :func:`argmax` -- the target's greedy (temperature 0) prediction per node
  (Sec. 2 "Speculative decoding"; Table 2, Temperature = 0).
* :func:`sample` -- the target's own sample per node at temperature tau > 0,
  by inverse transform of softmax(x / tau) with a caller-supplied uniform
  (Sec. 2 "Speculative decoding": drafts are checked against the target's own
  sampling; Table 2, Temperature = 1).
* :func:`lm_head_argmax` -- the target's greedy prediction from its final
  hidden states: argmax over the vocabulary of H W^T, in fp64 (numpy's matmul
  as the product step), the same total order as :func:`argmax`.
* :func:`visual_importance` -- the importance of each visual token, the mean of
  its column of the final-layer attention over heads and queries, and the r
  most important tokens kept (Sec. 3.2 "Visual Token Compression", Eq. 2);
  :func:`top_r` is the selection alone.
* :func:`attention_rows` -- attention without a tree: the draft's cross-attention
  to the target's features (every query sees slots 0 .. L-1; Sec. 3.2, "Adaptive
  Target Feature Injection") or a layer's causal prefill (query t sees slots
  0 .. L+t), with each row's attention entropy -sum_j a_j ln a_j, whose mean
  over rows and heads is AE(l) (Sec. 3.3).
* :func:`spec_path` -- speculative sampling over the tree (Leviathan et al.,
  cited in Sec. 1; T = 1 in Table 2): drafts accepted with probability
  min(1, p/q), the bonus drawn from the renormalised residual max(0, p - q).
* :func:`accept_path` -- sequential acceptance with the target's token
  replacing the first mismatch (Sec. 2 "Speculative decoding"), over a tree.
* :func:`kv_compact` -- the accepted nodes' K/V moved into contiguous slots
  (Sec. 2 "Vision-Language Models": the cache persists across steps).
* :func:`ancestor_mask` -- the tree mask the attention uses, for inspection.

Parity of this oracle against the paper's own numbers is unpinned for every
routine: the paper prints no worked example of this step. Each routine is
pinned instead by closed forms, special cases that reduce to library
routines, brute force on tiny inputs and invariants (see ``tests/``).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

BAD_PARENT = 0x1
BAD_TREE_LEN = 0x2
BAD_KV_LEN = 0x4
BAD_PAGE = 0x8
BAD_PATH = 0x10


def build(force: bool = False) -> str:
    """Compile ``oracle.c`` into ``liboracle.so`` with gcc (no fast-math)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
             "-ffp-contract=off", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib: Optional[ctypes.CDLL] = None


def _load() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        i64, i32, f64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
        p = ctypes.c_void_p
        _lib.oracle_ancestor_mask.argtypes = [p, i32, p]
        _lib.oracle_ancestor_mask.restype = ctypes.c_int
        _lib.oracle_tree_attention.argtypes = [
            p, p, p, i64, p, i64, i64, i64, p, p, p, i64, i64, i64, i64, i64, f64, p, i64, p, p]
        _lib.oracle_tree_attention.restype = ctypes.c_int
        _lib.oracle_argmax_f32.argtypes = [p, i64, i64, i64, p]
        _lib.oracle_argmax_f32.restype = None
        _lib.oracle_argmax_bf16.argtypes = [p, i64, i64, i64, p]
        _lib.oracle_argmax_bf16.restype = None
        _lib.oracle_sample_f32.argtypes = [p, i64, i64, i64, f64, p, p]
        _lib.oracle_sample_f32.restype = None
        _lib.oracle_sample_bf16.argtypes = [p, i64, i64, i64, f64, p, p]
        _lib.oracle_sample_bf16.restype = None
        _lib.oracle_accept_path.argtypes = [p, p, p, p, p, i64, i64, i64, p, p, p, p]
        _lib.oracle_accept_path.restype = ctypes.c_int
        for nm in ("oracle_spec_path_f32", "oracle_spec_path_bf16"):
            fn = getattr(_lib, nm)
            fn.argtypes = [p, p, i64, i64, p, p, p, p, i64, i64, i64, f64, p, p, p, p, p, p, p]
            fn.restype = ctypes.c_int
        _lib.oracle_kv_compact.argtypes = [
            p, p, i64, i64, i64, p, i64, i64, i64, i64, i64, i64, p, p, p, i64]
        _lib.oracle_kv_compact.restype = ctypes.c_int
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


def ancestor_mask(parent) -> np.ndarray:
    """[T, T] uint8: mask[i, a] = 1 iff a is i or an ancestor of i."""
    par = _c(parent, np.int32)
    T = par.shape[0]
    out = np.zeros((T, T), dtype=np.uint8)
    st = _load().oracle_ancestor_mask(_ptr(par), T, _ptr(out))
    if st:
        raise ValueError(f"malformed tree (status {st:#x})")
    return out


class KVLayout:
    """How one layer's K/V cache is laid out (see ``oracle.c``).

    ``page_table is None``: contiguous ``[B, capacity, Hkv, D]``.
    Otherwise paged ``[num_pages, page_size, Hkv, D]`` with
    ``page_table[B, pages_per_seq]`` physical page ids.
    """

    def __init__(self, capacity, Hkv, D, page_table=None, page_size=64, num_pages=0):
        self.capacity = int(capacity)
        self.Hkv = int(Hkv)
        self.D = int(D)
        self.page_table = None if page_table is None else _c(page_table, np.int32)
        self.page_size = int(page_size)
        self.pages_per_seq = 0 if page_table is None else int(self.page_table.shape[1])
        self.num_pages = int(num_pages)


def tree_attention(q_bits, k_bits, v_bits, layout: KVLayout, parent, tree_len, kv_len,
                   Hq: int, scale: float, sel=None):
    """fp64 tree-masked attention for the selected (b, t, h) triples.

    q_bits: uint16 bf16 patterns [B, T_max, Hq, D]; k_bits / v_bits: uint16
    patterns of one layer cache. ``sel`` is an [n, 3] int array of (b, t, h);
    None selects every valid row (t < tree_len[b]). Returns (out [n, D],
    lse [n], sel, status).
    """
    q = _c(q_bits, np.uint16)
    k = _c(k_bits, np.uint16)
    v = _c(v_bits, np.uint16)
    par = _c(parent, np.int32)
    tl = _c(tree_len, np.int32)
    kl = _c(kv_len, np.int32)
    B, T_max, _, D = q.shape
    if sel is None:
        sel = np.array([(b, t, h) for b in range(B) for t in range(int(tl[b]))
                        for h in range(Hq)], dtype=np.int32).reshape(-1, 3)
    sel = _c(sel, np.int32).reshape(-1, 3)
    n = sel.shape[0]
    out = np.empty((n, D), dtype=np.float64)
    lse = np.empty((n,), dtype=np.float64)
    st = _load().oracle_tree_attention(
        _ptr(q), _ptr(k), _ptr(v), layout.capacity, _ptr(layout.page_table), layout.page_size,
        layout.pages_per_seq, layout.num_pages, _ptr(par), _ptr(tl), _ptr(kl), B, T_max, Hq,
        layout.Hkv, D, float(scale), _ptr(sel), n, _ptr(out), _ptr(lse))
    return out, lse, sel, st


def argmax(logits, V: Optional[int] = None, bf16_bits: bool = False) -> np.ndarray:
    """Row-wise argmax of a 2-D array (float32, or uint16 bf16 patterns)."""
    x = np.asarray(logits)
    rows = x.shape[0]
    V = x.shape[1] if V is None else int(V)
    out = np.empty((rows,), dtype=np.int32)
    if bf16_bits:
        x = _c(x, np.uint16)
        _load().oracle_argmax_bf16(_ptr(x), rows, V, x.shape[1], _ptr(out))
    else:
        x = _c(x, np.float32)
        _load().oracle_argmax_f32(_ptr(x), rows, V, x.shape[1], _ptr(out))
    return out


def sample(logits, temperature: float, u, V: Optional[int] = None, bf16_bits: bool = False) -> np.ndarray:
    """One draw per row of a 2-D array (float32, or uint16 bf16 patterns) from
    softmax(row / temperature), by inverse transform with the row's uniform
    ``u[r]`` (float32); degenerate rows take their argmax."""
    x = np.asarray(logits)
    rows = x.shape[0]
    V = x.shape[1] if V is None else int(V)
    uu = _c(np.asarray(u, dtype=np.float32).reshape(rows), np.float32)
    out = np.empty((rows,), dtype=np.int32)
    if bf16_bits:
        x = _c(x, np.uint16)
        _load().oracle_sample_bf16(_ptr(x), rows, V, x.shape[1], float(temperature), _ptr(uu), _ptr(out))
    else:
        x = _c(x, np.float32)
        _load().oracle_sample_f32(_ptr(x), rows, V, x.shape[1], float(temperature), _ptr(uu), _ptr(out))
    return out


def lm_head_argmax(hidden_bits, weight_bits):
    """(indices, maxima, logits) of the LM head: logits = H W^T in float64 from
    bf16 bit patterns (uint16 [rows, K] and [V, K]); argmax with the lowest
    index among equal values (numpy's argmax; NaN first, as torch)."""
    h = _bf16_to_f64(hidden_bits)
    w = _bf16_to_f64(weight_bits)
    logits = np.matmul(h, w.T)
    idx = np.argmax(logits, axis=1).astype(np.int32)
    return idx, logits[np.arange(logits.shape[0]), idx], logits


def _bf16_to_f64(bits):
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def top_r(values, r: int, v0: int = 0) -> np.ndarray:
    """Positions v0 + j of the r largest values per row (equal values: the
    lower position first; NaN above every number), in increasing order."""
    x = np.asarray(values)
    B, n = x.shape
    out = np.empty((B, r), np.int32)
    for b in range(B):
        row = x[b]
        nan = np.isnan(row)
        key = np.where(nan, np.inf, row)
        order = np.lexsort((np.arange(n), -key, ~nan))  # NaN first, then larger, then lower position
        out[b] = np.sort(order[:r]) + v0
    return out


def visual_importance(attn, v0: int, n_vis: int, r: int, bf16_bits: bool = False):
    """(importance [B, n_vis] float64, keep [B, r]) from attention weights
    [B, H, Q, K] (float32, or uint16 bf16 patterns): I_j = the sum over heads
    and queries of A[:, :, :, v0 + j] divided by H Q (Eq. 2), summed head by
    head in float64; keep = the r largest, positions in increasing order."""
    a = np.asarray(attn)
    B, H, Q, K = a.shape
    imp = np.zeros((B, n_vis), np.float64)
    for b in range(B):
        for h in range(H):
            blk = a[b, h, :, v0:v0 + n_vis]
            blk = _bf16_to_f64(blk) if bf16_bits else blk.astype(np.float64)
            imp[b] += blk.sum(axis=0)
    imp /= float(H * Q)
    return imp, top_r(imp, r, v0)


def attention_rows(q, k, v, q_len, kv_len, scale: float, causal: bool, sel):
    """(out [n, D], lse [n], entropy [n]) in float64 for the selected (b, t, h)
    triples. q: float [B, T_max, Hq, D]; k, v: float [B, capacity, Hkv, D]
    (contiguous caches). Row (b, t, h) attends slots 0 .. kv_len[b] - 1
    (causal=False) or 0 .. kv_len[b] + t (causal=True) of KV head h // G:
        s_j = scale <q, K_j>, m = max s, w_j = exp(s_j - m), Z = sum w,
        out = sum w_j V_j / Z, lse = m + ln Z, entropy = -sum (w/Z) ln(w/Z)."""
    q = np.asarray(q, np.float64)
    k = np.asarray(k, np.float64)
    v = np.asarray(v, np.float64)
    Hq, Hkv = q.shape[2], k.shape[2]
    G = Hq // Hkv
    outs, lses, ents = [], [], []
    for b, t, h in sel:
        n = int(kv_len[b]) + (int(t) + 1 if causal else 0)
        g = h // G
        s = scale * (k[b, :n, g, :] @ q[b, t, h, :])
        m = s.max()
        w = np.exp(s - m)
        Z = w.sum()
        a = w / Z
        outs.append((a[:, None] * v[b, :n, g, :]).sum(axis=0))
        lses.append(m + np.log(Z))
        nz = a > 0
        ents.append(-(a[nz] * np.log(a[nz])).sum())
    return np.array(outs), np.array(lses), np.array(ents)


def accept_path(am, parent, tokens, tree_len, kv_len, max_path: int):
    """Greedy tree acceptance. Returns dict of accept_len, path, out_tokens,
    new_kv_len and the OR of data-error bits."""
    am = _c(am, np.int32)
    par = _c(parent, np.int32)
    tok = _c(tokens, np.int32)
    tl = _c(tree_len, np.int32)
    kl = _c(kv_len, np.int32)
    B, T_max = par.shape
    acc = np.empty((B,), np.int32)
    path = np.empty((B, max_path), np.int32)
    outt = np.empty((B, max_path), np.int32)
    nkl = np.empty((B,), np.int32)
    st = _load().oracle_accept_path(_ptr(am), _ptr(par), _ptr(tok), _ptr(tl), _ptr(kl), B, T_max,
                                    max_path, _ptr(acc), _ptr(path), _ptr(outt), _ptr(nkl))
    return {"accept_len": acc, "path": path, "out_tokens": outt, "new_kv_len": nkl, "status": st}


def spec_path(target, draft, parent, tokens, tree_len, kv_len, max_path: int, temperature: float, u_accept,
              u_resample, bf16_bits: bool = False):
    """Speculative sampling over the draft trees (Leviathan et al., cited in
    Sec. 1; verification at T = 1, Table 2) -- see ``oracle_spec_path`` in
    oracle.c. target, draft: [B, T_max, V] logits (float32, or uint16 bf16
    patterns); u_accept, u_resample: float32 [B, T_max]. Returns dict of
    accept_len, path, out_tokens, new_kv_len, the OR of data-error bits and
    margin [B] (the smallest distance of a uniform from its threshold)."""
    par = _c(parent, np.int32)
    B, T_max = par.shape
    dt = np.uint16 if bf16_bits else np.float32
    t = _c(target, dt)
    d = _c(draft, dt)
    V = t.shape[-1]
    t = t.reshape(B * T_max, V)
    d = d.reshape(B * T_max, V)
    acc = np.empty((B,), np.int32)
    path = np.empty((B, max_path), np.int32)
    outt = np.empty((B, max_path), np.int32)
    nkl = np.empty((B,), np.int32)
    mg = np.empty((B,), np.float64)
    fn = _load().oracle_spec_path_bf16 if bf16_bits else _load().oracle_spec_path_f32
    st = fn(_ptr(t), _ptr(d), V, V, _ptr(par), _ptr(_c(tokens, np.int32)), _ptr(_c(tree_len, np.int32)),
            _ptr(_c(kv_len, np.int32)), B, T_max, max_path, float(temperature),
            _ptr(_c(np.asarray(u_accept, np.float32).reshape(B, T_max), np.float32)),
            _ptr(_c(np.asarray(u_resample, np.float32).reshape(B, T_max), np.float32)),
            _ptr(acc), _ptr(path), _ptr(outt), _ptr(nkl), _ptr(mg))
    return {"accept_len": acc, "path": path, "out_tokens": outt, "new_kv_len": nkl, "status": st, "margin": mg}


def kv_compact(k_bits, v_bits, layout: KVLayout, kv_len, accept_len, path, n_layers: int = 1,
               layer_stride: int = 0):
    """In-place compaction on copies of the caches. Returns (k, v, status)."""
    k = np.array(k_bits, dtype=np.uint16, copy=True, order="C")
    v = np.array(v_bits, dtype=np.uint16, copy=True, order="C")
    kl = _c(kv_len, np.int32)
    acc = _c(accept_len, np.int32)
    pth = _c(path, np.int32)
    B, max_path = pth.shape
    st = _load().oracle_kv_compact(
        _ptr(k), _ptr(v), n_layers, layer_stride, layout.capacity, _ptr(layout.page_table),
        layout.page_size, layout.pages_per_seq, layout.num_pages, layout.Hkv, layout.D, B,
        _ptr(kl), _ptr(acc), _ptr(pth), max_path)
    return k, v, st
