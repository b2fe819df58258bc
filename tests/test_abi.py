"""The C ABI on the CPU: the library builds for sm_103a, loads, exports every
function include/dreams.h declares, and rejects bad arguments on the host
before any launch. No compute runs here."""
import ctypes
import os
import subprocess
import sys

import pytest
import torch

import paper_2606_00535_gb300 as dreams
from paper_2606_00535_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return dreams._lib()


def test_exports_every_declared_function(lib):
    names = dreams.declared_functions()
    assert len(names) >= 11
    for n in names:
        assert hasattr(lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", dreams.LIB_PATH], capture_output=True, text=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    assert set(names) <= exported


def test_version_and_strings(lib):
    assert dreams.version() == 10000
    for code, text in [(0, b"ok"), (1, b"invalid argument"), (3, b"workspace missing or too small"),
                       (99, b"unknown status")]:
        assert lib.dreams_status_string(code) == text


def test_binding_fails_loudly_without_library(tmp_path):
    code = ("import paper_2606_00535_gb300 as d; d.LIB_PATH='/nonexistent/libdreams.so'\n"
            "try:\n    d._lib()\nexcept ImportError as e:\n    print('raised', e)\n")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, capture_output=True, text=True)
    assert "raised" in r.stdout


def test_workspace_sizes(lib):
    k = torch.empty(0, dtype=torch.bfloat16)
    kvc = dreams._KVCache(16, 16, 1, 0, 8, 128, 6080, None, 0, 0, 0)
    one = dreams._Tree(16, 16, 16, 16, 1, 64)     # one sequence: the KV range is split over CTAs
    n = lib.dreams_tree_verify_attn_workspace_size(ctypes.byref(kvc), ctypes.byref(one), 32)
    assert n > 0 and n % 256 == 0
    tr = dreams._Tree(16, 16, 16, 16, 16, 64)
    # 16 sequences, one split each: the CTAs rank the 16 pairs themselves, no workspace
    assert lib.dreams_tree_verify_attn_workspace_size(ctypes.byref(kvc), ctypes.byref(tr), 32) == 0
    # 128 sequences: the longest-first order of the work items needs room
    tr = dreams._Tree(16, 16, 16, 16, 128, 64)
    assert lib.dreams_tree_verify_attn_workspace_size(ctypes.byref(kvc), ctypes.byref(tr), 32) >= 128 * 4
    bad = dreams._KVCache(16, 16, 1, 0, 8, 128, 6080, None, 0, 0, 0)
    assert lib.dreams_tree_verify_attn_workspace_size(ctypes.byref(bad), ctypes.byref(tr), 30) == 0
    assert lib.dreams_vocab_argmax_workspace_size(768, 128256) >= 0
    assert lib.dreams_verify_step_workspace_size(ctypes.byref(tr), 128256) >= 16 * 64 * 16


def test_attention_workspace_covers_every_row_block(lib):
    """The split partials are kept per row block: with 5 query heads per KV
    head and 64 nodes there are 3 row blocks (25 nodes each), so one split
    needs 3 x 128 rows of (O, m, l)."""
    kvc = dreams._KVCache(16, 16, 1, 0, 1, 128, 2304, None, 0, 0, 0)
    one = dreams._Tree(16, 16, 16, 16, 1, 64)
    ws = lib.dreams_tree_verify_attn_workspace_size(ctypes.byref(kvc), ctypes.byref(one), 5)
    per_split = 3 * 128 * (128 * 4 + 8)
    assert ws > 0 and ws % per_split == 0, ws


def test_attention_launch_count(lib):
    """One sequence: the attention, plus a merge when the KV range is split
    (the workspace then holds the partials). Several sequences are taken
    longest first: up to 64 (sequence, split) pairs each CTA ranks them
    itself, beyond that a separate ordering pass runs first (its order lives
    in the workspace). Rejected shapes make no launch."""
    kvc = dreams._KVCache(16, 16, 1, 0, 8, 128, 6080, None, 0, 0, 0)
    one = dreams._Tree(16, 16, 16, 16, 1, 64)
    split = lib.dreams_tree_verify_attn_workspace_size(ctypes.byref(kvc), ctypes.byref(one), 32) > 0
    assert lib.dreams_tree_verify_attn_launches(ctypes.byref(kvc), ctypes.byref(one), 32) == 1 + int(split)
    many = dreams._Tree(16, 16, 16, 16, 16, 64)  # 16 sequences x 8 KV heads x 2 row blocks: one split
    assert lib.dreams_tree_verify_attn_workspace_size(ctypes.byref(kvc), ctypes.byref(many), 32) == 0
    assert lib.dreams_tree_verify_attn_launches(ctypes.byref(kvc), ctypes.byref(many), 32) == 1
    lots = dreams._Tree(16, 16, 16, 16, 128, 64)  # 128 pairs: the ordering pass
    assert lib.dreams_tree_verify_attn_workspace_size(ctypes.byref(kvc), ctypes.byref(lots), 32) >= 128 * 4
    assert lib.dreams_tree_verify_attn_launches(ctypes.byref(kvc), ctypes.byref(lots), 32) == 2
    assert lib.dreams_tree_verify_attn_launches(ctypes.byref(kvc), ctypes.byref(many), 30) == 0
    d96 = dreams._KVCache(16, 16, 1, 0, 8, 96, 6080, None, 0, 0, 0)
    assert lib.dreams_tree_verify_attn_launches(ctypes.byref(d96), ctypes.byref(many), 32) == 0


@pytest.mark.skipif(torch.cuda.is_available(), reason="host-validation cases use placeholder pointers")
def test_invalid_arguments_rejected_before_launch(lib):
    """Each case breaks exactly one rule and must be refused on the host."""
    P = 0x1000  # placeholder, never dereferenced: every call below fails validation
    null = None
    tr = dreams._Tree(P, P, P, P, 2, 8)
    kvc = dreams._KVCache(P, P, 1, 0, 2, 128, 256, None, 0, 0, 0)
    st = ctypes.c_void_p(P)
    s = ctypes.c_void_p(0)

    def attn(q=P, kv=kvc, layer=0, tree=tr, Hq=4, scale=0.1, out=P, ws=None, wsb=0, sb=8 * 4 * 128,
             stt=4 * 128):
        return lib.dreams_tree_verify_attn(q, sb, stt, ctypes.byref(kv), layer, ctypes.byref(tree), Hq, scale, out,
                                           null, ws, wsb, st, s)

    assert attn(q=null) == dreams.ERR_INVALID_ARG
    assert attn(out=null) == dreams.ERR_INVALID_ARG
    assert attn(q=P + 2) == dreams.ERR_INVALID_ARG           # misaligned
    # Q strides (elements): a fused-QKV view [B, T, 3, Hq, D] is accepted by
    # the host checks; a token stride that is not a 16-byte multiple, one
    # below the token's Hq * D head rows, or a short sequence stride is not
    assert attn(stt=3 * 4 * 128 + 4) == dreams.ERR_INVALID_ARG
    assert attn(stt=4 * 128 - 8) == dreams.ERR_INVALID_ARG
    assert attn(sb=8 * 4 * 128 + 12) == dreams.ERR_INVALID_ARG
    assert attn(sb=0) == dreams.ERR_INVALID_ARG
    assert attn(stt=1 << 38) == dreams.ERR_INVALID_ARG
    assert attn(stt=3 * 4 * 128, sb=8 * 3 * 4 * 128, q=null) == dreams.ERR_INVALID_ARG  # strides fine, q null
    assert attn(Hq=3) == dreams.ERR_INVALID_ARG              # Hq % Hkv
    assert attn(Hq=258) == dreams.ERR_INVALID_ARG            # more than 128 query heads per KV head
    assert attn(layer=1) == dreams.ERR_INVALID_ARG
    assert attn(scale=float("inf")) == dreams.ERR_INVALID_ARG
    assert attn(tree=dreams._Tree(P, P, P, P, 2, 65)) == dreams.ERR_INVALID_ARG   # T_max > 64
    assert attn(tree=dreams._Tree(P, P, P, P, 0, 8)) == dreams.ERR_INVALID_ARG
    assert attn(kv=dreams._KVCache(P, P, 1, 0, 2, 96, 256, None, 0, 0, 0)) == dreams.ERR_UNSUPPORTED
    assert attn(kv=dreams._KVCache(P, P, 1, 0, 2, 128, 256, P, 32, 8, 4)) == dreams.ERR_UNSUPPORTED
    assert attn(kv=dreams._KVCache(P, P, 1, 0, 2, 128, 256, P, 64, 5, 4)) == dreams.ERR_INVALID_ARG
    big = dreams._KVCache(P, P, 1, 0, 1, 128, 100000, None, 0, 0, 0)
    need = lib.dreams_tree_verify_attn_workspace_size(ctypes.byref(big), ctypes.byref(tr), 1)
    assert need > 0
    assert attn(kv=big, Hq=1, ws=None, wsb=0) == dreams.ERR_WORKSPACE
    assert attn(kv=big, Hq=1, ws=P, wsb=need - 1) == dreams.ERR_WORKSPACE

    am = lib.dreams_vocab_argmax
    assert am(null, 0, 4, 100, 100, P, null, 0, s) == dreams.ERR_INVALID_ARG
    assert am(P, 0, 4, 100, 99, P, null, 0, s) == dreams.ERR_INVALID_ARG     # stride < V
    assert am(P, 7, 4, 100, 100, P, null, 0, s) == dreams.ERR_UNSUPPORTED
    assert am(P + 1, 1, 4, 100, 100, P, null, 0, s) == dreams.ERR_INVALID_ARG  # misaligned bf16
    assert am(P, 0, 1, 10_000_000, 10_000_000, P, null, 0, s) == dreams.ERR_WORKSPACE

    ap = lib.dreams_accept_path
    assert ap(P, ctypes.byref(tr), 0, P, P, P, P, st, s) == dreams.ERR_INVALID_ARG
    assert ap(P, ctypes.byref(dreams._Tree(P, null, P, P, 2, 8)), 4, P, P, P, P, st, s) == dreams.ERR_INVALID_ARG
    assert ap(null, ctypes.byref(tr), 4, P, P, P, P, st, s) == dreams.ERR_INVALID_ARG

    kc = lib.dreams_kv_compact
    assert kc(ctypes.byref(kvc), 0, P, P, P, 4, st, s) == dreams.ERR_INVALID_ARG
    assert kc(ctypes.byref(kvc), 2, P, P, P, 66, st, s) == dreams.ERR_INVALID_ARG
    assert kc(ctypes.byref(dreams._KVCache(P + 8, P, 1, 0, 2, 128, 256, None, 0, 0, 0)), 2, P, P, P, 4, st,
              s) == dreams.ERR_INVALID_ARG

    vs = lib.dreams_verify_step
    wsb = lib.dreams_verify_step_workspace_size(ctypes.byref(tr), 1000)
    assert vs(P, 0, 1000, 1000, ctypes.byref(tr), ctypes.byref(kvc), 5, null, P, P, P, P, P, wsb - 1, st,
              s) == dreams.ERR_WORKSPACE
    assert vs(P, 0, 1000, 999, ctypes.byref(tr), ctypes.byref(kvc), 5, null, P, P, P, P, P, wsb, st,
              s) == dreams.ERR_INVALID_ARG
    assert vs(P, 3, 1000, 1000, ctypes.byref(tr), ctypes.byref(kvc), 5, null, P, P, P, P, P, wsb, st,
              s) == dreams.ERR_UNSUPPORTED

    def spec(tgt=P, drf=P, dt=1, V=1000, rs=1000, tree=tr, mp=5, tau=1.0, ua=P, ur=P):
        return lib.dreams_verify_step_speculative(tgt, drf, dt, V, rs, ctypes.byref(tree), ctypes.byref(kvc), mp,
                                                  tau, ua, ur, P, P, P, P, st, s)

    assert spec(tgt=null) == dreams.ERR_INVALID_ARG
    assert spec(drf=null) == dreams.ERR_INVALID_ARG
    assert spec(ua=null) == dreams.ERR_INVALID_ARG
    assert spec(ur=P + 2) == dreams.ERR_INVALID_ARG          # misaligned uniforms
    assert spec(drf=P + 1) == dreams.ERR_INVALID_ARG         # misaligned bf16 rows
    assert spec(rs=999) == dreams.ERR_INVALID_ARG            # stride < V
    assert spec(mp=0) == dreams.ERR_INVALID_ARG
    assert spec(mp=66) == dreams.ERR_INVALID_ARG
    assert spec(tree=dreams._Tree(P, null, P, P, 2, 8)) == dreams.ERR_INVALID_ARG  # the drafts are needed
    assert spec(dt=7) == dreams.ERR_UNSUPPORTED
    assert spec(V=393217, rs=393217) == dreams.ERR_UNSUPPORTED  # more than 16 CTAs' shared memory
    assert spec(tau=0.0) == dreams.ERR_INVALID_ARG
    assert spec(tau=float("nan")) == dreams.ERR_INVALID_ARG
    assert spec(tau=1e-45) == dreams.ERR_INVALID_ARG         # log2(e) / tau overflows


def test_stall_hook_argument_checks(lib):
    """The test hook of the bounded waits: only the two kernel families, a
    wait limit of 1 us .. 2 s; a negative stall restores normal operation
    whatever the other arguments."""
    assert lib.dreams_test_set_stall(0, 0, 10_000_000) == dreams.ERR_INVALID_ARG
    assert lib.dreams_test_set_stall(4, 0, 10_000_000) == dreams.ERR_INVALID_ARG
    assert lib.dreams_test_set_stall(dreams.TEST_ATTENTION, 0, 999) == dreams.ERR_INVALID_ARG
    assert lib.dreams_test_set_stall(dreams.TEST_LM_HEAD, 0, 2_000_000_001) == dreams.ERR_INVALID_ARG
    assert lib.dreams_test_set_stall(dreams.TEST_ATTENTION | dreams.TEST_LM_HEAD, 3, 10_000_000) == dreams.OK
    assert lib.dreams_test_set_stall(7, -1, 0) == dreams.OK


def test_binding_checks_before_any_call():
    """The wrappers refuse on the host, before any library call: a no-allocation
    argmax over more rows than its fixed scratch, an output shorter than the
    rows written, leading dimensions that flatten only by copying (which would
    allocate), and a query tensor whose head rows are not dense."""
    x = torch.zeros((dreams.NOALLOC_ARGMAX_MAX_ROWS + 1, 8), dtype=torch.float32)
    out = torch.zeros(dreams.NOALLOC_ARGMAX_MAX_ROWS + 1, dtype=torch.int32)
    with pytest.raises(ValueError, match="fixed scratch"):
        dreams.vocab_argmax_noalloc(x, out)
    x = torch.zeros((6, 8), dtype=torch.float32)
    with pytest.raises(ValueError, match="holds 5 elements"):
        dreams.vocab_argmax_noalloc(x, torch.zeros(5, dtype=torch.int32))
    with pytest.raises(ValueError, match="holds 5 elements"):
        dreams.vocab_argmax(x, out=torch.zeros(5, dtype=torch.int32))
    y = torch.zeros((4, 3, 8), dtype=torch.float32).transpose(0, 1)  # [3, 4, 8], not viewable as [12, 8]
    with pytest.raises(ValueError, match="without a copy"):
        dreams.vocab_argmax_noalloc(y, torch.zeros(12, dtype=torch.int32))
    q = torch.zeros((2, 5, 4, 64), dtype=torch.bfloat16).transpose(2, 1)  # heads strided
    with pytest.raises(ValueError, match="head rows must be dense"):
        dreams._q_strides(q)
    fused = torch.zeros((2, 5, 3, 4, 64), dtype=torch.bfloat16)
    assert dreams._q_strides(fused[:, :, 0]) == (5 * 3 * 4 * 64, 3 * 4 * 64)


def test_speculative_binding_checks_before_any_call():
    """verify_step_speculative refuses on the host, before any library call:
    target and draft logits of different dtypes or shapes, rows that are not
    [B, T_max, V] with contiguous rows, logits of another dtype, and uniforms
    of the wrong shape or dtype."""
    B, T, V = 2, 4, 16
    tree = dreams.Tree(torch.full((B, T), -1, dtype=torch.int32), torch.zeros((B, T), dtype=torch.int32),
                       torch.ones(B, dtype=torch.int32), torch.zeros(B, dtype=torch.int32))
    k = torch.zeros((B, 8, 1, 64), dtype=torch.bfloat16)
    kv = dreams.KVCache(k, k.clone())
    tgt = torch.zeros((B, T, V), dtype=torch.float32)
    u = torch.zeros((B, T), dtype=torch.float32)
    with pytest.raises(ValueError, match="share dtype, shape and strides"):
        dreams.verify_step_speculative(tgt, tgt.to(torch.bfloat16).float()[:, :, :8], tree, kv, 3, 1.0, u, u)
    with pytest.raises(ValueError, match="share dtype, shape and strides"):
        dreams.verify_step_speculative(tgt, tgt.to(torch.bfloat16), tree, kv, 3, 1.0, u, u)
    with pytest.raises(ValueError, match="uniformly strided contiguous rows"):
        dreams.verify_step_speculative(tgt.transpose(1, 2), tgt.transpose(1, 2), tree, kv, 3, 1.0, u, u)
    with pytest.raises(TypeError, match="float32/bfloat16"):
        dreams.verify_step_speculative(tgt.double(), tgt.double(), tree, kv, 3, 1.0, u, u)
    with pytest.raises(ValueError, match=r"u_accept must be \[B, T_max\]"):
        dreams.verify_step_speculative(tgt, tgt, tree, kv, 3, 1.0, torch.zeros((B, 2), dtype=torch.float32), u)
    with pytest.raises((TypeError, ValueError)):
        dreams.verify_step_speculative(tgt, tgt, tree, kv, 3, 1.0, u, u.double())


def test_binding_checks_outputs_status_and_workspace():
    """The verify-step wrappers check caller-provided outputs (dtype, and at
    least the elements the kernels write), the status word (int32, one
    element) and the workspace (a contiguous tensor on the tensors' device)
    before any library call."""
    B, T, V, P = 2, 4, 16, 3
    tree = dreams.Tree(torch.full((B, T), -1, dtype=torch.int32), torch.zeros((B, T), dtype=torch.int32),
                       torch.ones(B, dtype=torch.int32), torch.zeros(B, dtype=torch.int32))
    k = torch.zeros((B, 8, 1, 64), dtype=torch.bfloat16)
    kv = dreams.KVCache(k, k.clone())
    lg = torch.zeros((B, T, V), dtype=torch.float32)
    u = torch.zeros((B, T), dtype=torch.float32)
    good = (torch.zeros(B, dtype=torch.int32), torch.zeros((B, P), dtype=torch.int32),
            torch.zeros((B, P), dtype=torch.int32), torch.zeros(B, dtype=torch.int32))
    short_path = (good[0], torch.zeros((B, P - 1), dtype=torch.int32), good[2], good[3])
    wrong_dtype = (good[0].long(), good[1], good[2], good[3])
    calls = [
        lambda **kw: dreams.verify_step(lg, tree, kv, P, **kw),
        lambda **kw: dreams.verify_step_sampled(lg, tree, kv, P, 1.0, u, **kw),
        lambda **kw: dreams.verify_step_speculative(lg, lg, tree, kv, P, 1.0, u, u, **kw),
    ]
    for call in calls:
        with pytest.raises(ValueError, match="path holds"):
            call(outputs=short_path)
        with pytest.raises(TypeError, match="accept_len must be"):
            call(outputs=wrong_dtype)
        with pytest.raises(ValueError, match="outputs must be"):
            call(outputs=good[:3])
        with pytest.raises(TypeError, match="status must be"):
            call(outputs=good, status=torch.zeros(1, dtype=torch.int64))
        with pytest.raises(ValueError, match="status holds"):
            call(outputs=good, status=torch.zeros(0, dtype=torch.int32))
    with pytest.raises(ValueError, match="argmax_out holds"):
        dreams.verify_step(lg, tree, kv, P, argmax_out=torch.zeros(B * T - 1, dtype=torch.int32), outputs=good)
    with pytest.raises(ValueError, match="sample_out holds"):
        dreams.verify_step_sampled(lg, tree, kv, P, 1.0, u, sample_out=torch.zeros(B * T - 1, dtype=torch.int32),
                                   outputs=good)
    with pytest.raises(ValueError, match="workspace must be a contiguous tensor"):
        dreams.verify_step(lg, tree, kv, P, outputs=good, workspace=torch.zeros((64, 4), dtype=torch.uint8).t())


def test_binding_checks_batch_and_head_dims():
    """Queries that do not match the tree's (B, T_max), a head dim other than
    the cache's, a cache with fewer sequences than the call addresses, and
    length arrays shorter than the batch are refused before any call."""
    B, T, H, D = 3, 4, 2, 64
    tree = dreams.Tree(torch.full((B, T), -1, dtype=torch.int32), torch.zeros((B, T), dtype=torch.int32),
                       torch.ones(B, dtype=torch.int32), torch.zeros(B, dtype=torch.int32))
    k = torch.zeros((B, 16, H, D), dtype=torch.bfloat16)
    kv = dreams.KVCache(k, k.clone())
    small = dreams.KVCache(k[:2].contiguous(), k[:2].contiguous())
    q = torch.zeros((B, T, H, D), dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="the tree's B"):
        dreams.tree_verify_attn(q[:2], kv, tree, 0.1)
    with pytest.raises(ValueError, match="the tree's B"):
        dreams.tree_verify_attn(torch.zeros((B, T + 1, H, D), dtype=torch.bfloat16), kv, tree, 0.1)
    with pytest.raises(ValueError, match="head dim"):
        dreams.tree_verify_attn(torch.zeros((B, T, H, 2 * D), dtype=torch.bfloat16), kv, tree, 0.1)
    with pytest.raises(ValueError, match="holds 2 sequences"):
        dreams.tree_verify_attn(q, small, tree, 0.1)
    lens = torch.ones(B, dtype=torch.int32)
    with pytest.raises(ValueError, match="q_len holds 2 entries"):
        dreams.attention(q, kv, lens[:2], lens, 0.1, dreams.ATTN_FULL)
    with pytest.raises(ValueError, match="holds 2 sequences"):
        dreams.attention(q, small, lens, lens, 0.1, dreams.ATTN_FULL)
    lg = torch.zeros((B, T, 8), dtype=torch.float32)
    with pytest.raises(ValueError, match="holds 2 sequences"):
        dreams.verify_step(lg, tree, small, 3)
    path = torch.zeros((B, 3), dtype=torch.int32)
    with pytest.raises(ValueError, match="kv_len holds 2 entries"):
        dreams.kv_compact(kv, lens[:2], lens, path)
    with pytest.raises(ValueError, match="holds 2 sequences"):
        dreams.kv_compact(small, lens, lens, path)
    with pytest.raises(ValueError, match="argmax holds"):
        dreams.accept_path(torch.zeros(B * T - 1, dtype=torch.int32), tree, 3)
