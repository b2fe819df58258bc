"""Seeded synthetic inputs for the tree verification step.

This module only draws inputs. It computes no attention, argmax, acceptance
or compaction, so both the CPU oracle (``oracle/``) and the CUDA library can be
fed from it without sharing any of the method's arithmetic.

The five workloads follow the shapes of the VLM decoding the paper measures:
LLaVA-v1.6-7B/13B-shaped and Qwen2-VL-7B-shaped target models, whose KV cache
holds the visual tokens followed by the text tokens (paper Sec. 2,
"Vision-Language Models"), verified against a draft tree. The paper's own
datasets and weights are not used; random values of the stated distributions
stand in for them.

Recipe (seed = 20260 + workload index, numpy PCG64):

* Q, K, V ~ N(0, 1), rounded to bf16. Every cache slot is filled, including
  the tree slots [L, L + T) that the verify pass has just written.
* Draft tree: nodes are numbered level by level, so parent[i] < i. Level
  widths are filled greedily up to a cap (10 = "top-10 expansion per level"),
  and each node's parent is drawn uniformly from the previous level. The tiny
  tree is a depth-4 chain plus nodes hung under uniformly drawn parents with
  fewer than 3 children and depth < 4.
* Draft tokens uniform in [0, V).
* Logits sigma * N(0, 1) clipped to +-7 sigma. For every node with at least one
  child, with probability p one child c is drawn and logits[node, tokens[c]] is
  set to 8 sigma, which is strictly above every other value in the row (in
  fp32 and after bf16 rounding), so the target's prediction equals that
  child's token.
* Batched workload: L_b ~ U{1500..6000}, T_b ~ U{32..64}, depth 6, p_b ~ U[0.5,
  0.9]; the cache is paged (64-token pages) with physical pages in a seeded
  random order.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import numpy as np
import torch

PAGE = 64


@dataclasses.dataclass(frozen=True)
class Spec:
    name: str
    index: int
    B: int
    Hq: int
    Hkv: int
    D: int
    visual: Optional[int]  # fixed prefix split (visual + text); None -> drawn per sequence
    text: Optional[int]
    T: Optional[int]  # tree nodes incl. the root; None -> drawn per sequence
    depth: int
    level_cap: Optional[int]  # None -> even split over depth levels
    V: int
    logits_dtype: str  # "f32" | "bf16"
    sigma: float
    p_match: Optional[float]  # None -> drawn per sequence in [0.5, 0.9]
    paged: bool
    description: str


SPECS: List[Spec] = [
    Spec("tiny", 0, 1, 4, 4, 64, 144, 112, 16, 4, None, 1024, "f32", 1.0, 0.7, False,
         "batch 1, 4 heads MHA, head_dim 64, KV 256 (144 visual + 112 text), tree 16 nodes depth 4, "
         "fp32 logits vocab 1024"),
    Spec("llava7b", 1, 1, 32, 32, 128, 2880, 512, 60, 6, 10, 32000, "f32", 2.0, 0.75, False,
         "LLaVA-v1.6-7B-shaped: batch 1, 32 heads MHA, head_dim 128, KV 2880 visual + 512 text, "
         "tree 60 nodes depth 6, fp32 logits vocab 32000"),
    Spec("qwen2vl7b", 2, 1, 28, 4, 128, 1200, 800, 48, 5, 10, 152064, "bf16", 2.0, 0.7, False,
         "Qwen2-VL-7B-shaped GQA: batch 1, 28 q / 4 KV heads, head_dim 128, KV 1200 visual + 800 text, "
         "tree 48 nodes depth 5, bf16 logits vocab 152064"),
    Spec("long13b", 3, 1, 40, 40, 128, 5760, 2048, 64, 7, 10, 32000, "f32", 2.0, 0.8, False,
         "long-prefix 13B-shaped: batch 1, 40 heads MHA, head_dim 128, KV 5760 visual + 2048 text, "
         "tree 64 nodes depth 7, fp32 logits vocab 32000"),
    Spec("batched", 4, 16, 32, 8, 128, None, None, None, 6, None, 128256, "bf16", 2.0, None, True,
         "batched serving: batch 16, 32 q / 8 KV heads, head_dim 128, KV length U[1500,6000] paged "
         "(64-token pages), trees of 32-64 nodes depth 6, bf16 logits vocab 128256"),
]
SPEC_BY_NAME: Dict[str, Spec] = {s.name: s for s in SPECS}


@dataclasses.dataclass
class Workload:
    spec: Spec
    B: int
    Hq: int
    Hkv: int
    D: int
    T_max: int
    V: int
    logits_dtype: str
    capacity: int
    paged: bool
    page_size: int
    pages_per_seq: int
    num_pages: int
    scale: float
    q: torch.Tensor  # bf16 [B, T_max, Hq, D]
    k: torch.Tensor  # bf16 [B, capacity, Hkv, D] or [num_pages, 64, Hkv, D]
    v: torch.Tensor
    page_table: Optional[torch.Tensor]  # int32 [B, pages_per_seq] (-1 = unused) or None
    parent: torch.Tensor  # int32 [B, T_max] (-1 past tree_len)
    tokens: torch.Tensor  # int32 [B, T_max]
    tree_len: torch.Tensor  # int32 [B]
    kv_len: torch.Tensor  # int32 [B]
    logits: torch.Tensor  # f32 or bf16 [B, T_max, V]
    depth: List[int]
    p_match: List[float]

    @property
    def max_path(self) -> int:
        return max(self.depth) + 1


def bf16(x: np.ndarray) -> torch.Tensor:
    """float32 numpy -> bf16 torch (round to nearest even)."""
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)


def bits(t: torch.Tensor) -> np.ndarray:
    """bf16 torch tensor -> its uint16 bit patterns as numpy (no copy when contiguous)."""
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def level_sizes(n_nodes: int, depth: int, cap: Optional[int]) -> List[int]:
    """Widths of levels 1..depth holding n_nodes non-root nodes, filled greedily
    up to ``cap`` per level (cap None: as even as possible), each level >= 1."""
    if depth < 1 or n_nodes < depth:
        raise ValueError("need at least one node per level")
    if cap is None:
        cap = math.ceil(n_nodes / depth)
    sizes = []
    left = n_nodes
    for lvl in range(depth):
        levels_after = depth - lvl - 1
        w = min(cap, left - levels_after)
        sizes.append(w)
        left -= w
    if left != 0:
        raise ValueError(f"{n_nodes} nodes do not fit {depth} levels of width <= {cap}")
    return sizes


def level_tree(rng: np.random.Generator, T: int, depth: int, cap: Optional[int]) -> np.ndarray:
    """Parent array of a T-node tree (root included) numbered level by level."""
    parent = np.full((T,), -1, dtype=np.int32)
    prev = [0]
    nxt = 1
    for w in level_sizes(T - 1, depth, cap):
        cur = list(range(nxt, nxt + w))
        for i in cur:
            parent[i] = prev[int(rng.integers(len(prev)))]
        prev = cur
        nxt += w
    return parent


def tiny_tree(rng: np.random.Generator, T: int, depth: int, max_children: int = 3) -> np.ndarray:
    """Depth-``depth`` chain, then nodes under random parents with < max_children
    children and depth < ``depth``."""
    parent = np.full((T,), -1, dtype=np.int32)
    node_depth = [0]
    children = [0]
    for i in range(1, depth + 1):
        parent[i] = i - 1
        node_depth.append(i)
        children.append(0)
        children[i - 1] += 1
    for i in range(depth + 1, T):
        ok = [a for a in range(i) if children[a] < max_children and node_depth[a] < depth]
        a = ok[int(rng.integers(len(ok)))]
        parent[i] = a
        node_depth.append(node_depth[a] + 1)
        children.append(0)
        children[a] += 1
    return parent


def tree_depth(parent: np.ndarray, T: int) -> int:
    d = [0] * T
    for i in range(1, T):
        d[i] = d[parent[i]] + 1
    return max(d)


def make(name: str, seed: Optional[int] = None, kv_len_override: Optional[int] = None,
         tree_key_scale: float = 1.0, with_logits: bool = True, with_attn: bool = True) -> Workload:
    """Build workload ``name`` with its seeded recipe.

    kv_len_override: force every L_b (mask-sensitive variants: 0 or 16).
    tree_key_scale: multiply the K rows in the tree slots by this power of two
    (exact in bf16) so that the tree columns dominate the softmax.
    """
    s = SPEC_BY_NAME[name]
    rng = np.random.Generator(np.random.PCG64(20260 + s.index if seed is None else seed))
    B = s.B
    # -- per-sequence lengths, trees, tokens
    if s.T is None:
        T_b = rng.integers(32, 65, size=B).astype(np.int32)
        L_b = rng.integers(1500, 6001, size=B).astype(np.int32)
        p_b = rng.uniform(0.5, 0.9, size=B)
    else:
        T_b = np.full((B,), s.T, np.int32)
        L_b = np.full((B,), s.visual + s.text, np.int32)
        p_b = np.full((B,), s.p_match)
    if kv_len_override is not None:
        L_b = np.full((B,), kv_len_override, np.int32)
    T_max = int(T_b.max()) if s.T is None else s.T
    if s.T is None:
        T_max = 64
    parent = np.full((B, T_max), -1, np.int32)
    depth = []
    for b in range(B):
        if s.level_cap is None and s.name == "tiny":
            par = tiny_tree(rng, int(T_b[b]), s.depth)
        else:
            par = level_tree(rng, int(T_b[b]), s.depth, s.level_cap)
        parent[b, :T_b[b]] = par
        depth.append(tree_depth(par, int(T_b[b])))
    tokens = rng.integers(0, s.V, size=(B, T_max)).astype(np.int32)

    # -- KV cache
    if s.paged:
        max_len = 6000 + 64
        pages_per_seq = -(-max_len // PAGE)
        capacity = pages_per_seq * PAGE
        need = [-(-int(L_b[b] + T_b[b]) // PAGE) for b in range(B)]
        num_pages = int(sum(need))
        perm = rng.permutation(num_pages).astype(np.int32)
        page_table = np.full((B, pages_per_seq), -1, np.int32)
        off = 0
        for b in range(B):
            page_table[b, :need[b]] = perm[off:off + need[b]]
            off += need[b]
        kv_shape = (num_pages, PAGE, s.Hkv, s.D)
    else:
        capacity = int(L_b.max()) + T_max
        pages_per_seq = 0
        num_pages = 0
        page_table = None
        kv_shape = (B, capacity, s.Hkv, s.D)

    q = k = v = torch.empty(0, dtype=torch.bfloat16)
    if with_attn:
        q = bf16(rng.standard_normal((B, T_max, s.Hq, s.D), dtype=np.float32))
        kf = rng.standard_normal(kv_shape, dtype=np.float32)
        vf = rng.standard_normal(kv_shape, dtype=np.float32)
        if tree_key_scale != 1.0:
            for b in range(B):
                for i in range(int(T_b[b])):
                    slot = int(L_b[b]) + i
                    if s.paged:
                        kf[page_table[b, slot // PAGE], slot % PAGE] *= tree_key_scale
                    else:
                        kf[b, slot] *= tree_key_scale
        k = bf16(kf)
        v = bf16(vf)
        del kf, vf

    # -- logits with planted matches
    if with_logits:
        lf = rng.standard_normal((B, T_max, s.V), dtype=np.float32)
        lf *= np.float32(s.sigma)
        np.clip(lf, -7.0 * s.sigma, 7.0 * s.sigma, out=lf)
        for b in range(B):
            Tb = int(T_b[b])
            kids: List[List[int]] = [[] for _ in range(Tb)]
            for i in range(1, Tb):
                kids[parent[b, i]].append(i)
            for i in range(Tb):
                if kids[i] and rng.random() < p_b[b]:
                    c = kids[i][int(rng.integers(len(kids[i])))]
                    lf[b, i, tokens[b, c]] = np.float32(8.0 * s.sigma)
        if s.logits_dtype == "bf16":
            logits = bf16(lf)
        else:
            logits = torch.from_numpy(lf)
        del lf
    else:
        logits = torch.empty(0, dtype=torch.float32)

    return Workload(
        spec=s, B=B, Hq=s.Hq, Hkv=s.Hkv, D=s.D, T_max=T_max, V=s.V, logits_dtype=s.logits_dtype,
        capacity=capacity, paged=s.paged, page_size=PAGE, pages_per_seq=pages_per_seq,
        num_pages=num_pages, scale=1.0 / math.sqrt(s.D), q=q, k=k, v=v,
        page_table=None if page_table is None else torch.from_numpy(page_table),
        parent=torch.from_numpy(parent), tokens=torch.from_numpy(tokens),
        tree_len=torch.from_numpy(T_b.copy()), kv_len=torch.from_numpy(L_b.copy()),
        logits=logits, depth=depth, p_match=[float(x) for x in p_b])


def chain_parent(T: int) -> np.ndarray:
    """Parent array of a chain root -> 1 -> 2 -> ... -> T-1."""
    return np.arange(-1, T - 1, dtype=np.int32)


def random_tree(rng: np.random.Generator, T: int) -> np.ndarray:
    """Uniform random recursive tree: parent[i] uniform in [0, i)."""
    parent = np.full((T,), -1, np.int32)
    for i in range(1, T):
        parent[i] = int(rng.integers(i))
    return parent
