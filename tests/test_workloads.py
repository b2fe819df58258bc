"""The seeded input recipe: tree shapes, planted predictions, page tables."""
import numpy as np
import pytest

import workloads as W


@pytest.mark.parametrize("name", ["tiny", "llava7b", "qwen2vl7b", "long13b", "batched"])
def test_tree_shapes(name):
    w = W.make(name, with_logits=False, with_attn=False)
    s = w.spec
    for b in range(w.B):
        T = int(w.tree_len[b])
        par = w.parent[b].numpy()
        assert par[0] == -1 and all(0 <= par[i] < i for i in range(1, T))
        assert (par[T:] == -1).all()
        assert W.tree_depth(par, T) == s.depth
        if s.T is not None:
            assert T == s.T and int(w.kv_len[b]) == s.visual + s.text
        else:
            assert 32 <= T <= 64 and 1500 <= int(w.kv_len[b]) <= 6000
        if name == "tiny":
            kids = np.bincount(par[1:T], minlength=T)
            assert kids.max() <= 3
        if s.level_cap:
            assert max(W.level_sizes(T - 1, s.depth, s.level_cap)) <= s.level_cap
    if w.paged:
        pt = w.page_table.numpy()
        used = pt[pt >= 0]
        assert len(np.unique(used)) == len(used) == w.num_pages
        for b in range(w.B):
            need = -(-(int(w.kv_len[b]) + int(w.tree_len[b])) // 64)
            assert (pt[b, :need] >= 0).all() and (pt[b, need:] == -1).all()


@pytest.mark.parametrize("name", ["tiny", "llava7b"])
def test_planted_predictions(name):
    """Planted rows have the child's token as their unique maximum."""
    w = W.make(name, with_attn=False)
    lg = w.logits.float().numpy()
    planted = 0
    for b in range(w.B):
        T = int(w.tree_len[b])
        par = w.parent[b].numpy()
        for i in range(T):
            kids = [c for c in range(1, T) if par[c] == i]
            row = lg[b, i]
            top = np.argmax(row)
            if row[top] == 8.0 * w.spec.sigma:
                assert (row == row[top]).sum() == 1
                assert any(w.tokens[b, c] == top for c in kids)
                planted += 1
            else:
                assert row.max() <= 7.0 * w.spec.sigma
    n_parents = sum(1 for i in range(int(w.tree_len[0])) if (w.parent[0].numpy() == i).any())
    assert 0.4 * n_parents <= planted <= n_parents


def test_level_sizes():
    assert W.level_sizes(59, 6, 10) == [10, 10, 10, 10, 10, 9]
    assert W.level_sizes(47, 5, 10) == [10, 10, 10, 10, 7]
    assert W.level_sizes(63, 7, 10) == [10, 10, 10, 10, 10, 10, 3]
    assert W.level_sizes(31, 6, None) == [6, 6, 6, 6, 6, 1]
