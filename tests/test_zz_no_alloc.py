"""The no-allocation argmax entry point, through the C ABI and its wrapper.

dreams_vocab_argmax_noalloc serves callers that must not allocate device
memory while the argmax runs (an engine plugin whose host owns every device
allocation, a server that reserves its whole memory budget at start-up). It
must give the same indices as dreams_vocab_argmax, which uses a
caller-provided workspace, call after call. Its fixed scratch is shared by
all calls; each call clears the part it uses before the kernel runs (and the
kernel resets what it used at the end), so a call with fewer rows after one
with more must not see the earlier call's slots.

This file is collected last so that a run stopping at the first failure has
already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _logits(rows, V, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn((rows, V), generator=g) * 2
    x[0, :] = 1.0                   # all equal: index 0
    x[1, [7, V - 3]] = 50.0         # a tie across vocabulary chunks: the first
    x[2, V // 2] = float("nan")     # NaN wins
    return x.to(dtype).cuda()


def test_noalloc_argmax_matches_workspace_entry_point():
    import paper_2606_00535_gb300 as dreams
    lib = dreams._lib()
    fn = lib.dreams_vocab_argmax_noalloc
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    # two calls in a row through the C symbol, each splitting its rows over
    # several CTAs (so the shared scratch slots are used), the second with
    # fewer rows than the first
    for seed, (rows, V, dtype) in enumerate([(60, 152064, torch.bfloat16), (48, 32000, torch.float32)]):
        x = _logits(rows, V, dtype, seed)
        ref = dreams.vocab_argmax(x)          # the workspace entry point
        out = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
        st = fn(ctypes.c_void_p(x.data_ptr()), dreams.BF16 if dtype == torch.bfloat16 else dreams.F32, rows, V, V,
                ctypes.c_void_p(out.data_ptr()), stream)
        assert st == dreams.OK, lib.dreams_status_string(st)
        torch.cuda.synchronize()
        assert torch.equal(out, ref)
        assert out[0].item() == 0 and out[1].item() == 7 and out[2].item() == V // 2
        np.testing.assert_array_equal(out.cpu().numpy(), torch.argmax(x.float(), dim=1).int().cpu().numpy())


def test_noalloc_wrapper_more_rows_then_fewer():
    """Through the Python wrapper: a split-row call over many rows, then one
    over fewer rows on the same scratch; both equal torch.argmax and the
    workspace entry point."""
    import paper_2606_00535_gb300 as dreams
    for seed, (rows, V) in enumerate([(100, 128256), (9, 128256), (3, 20000)]):
        x = _logits(rows, V, torch.bfloat16, 10 + seed)
        out = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
        dreams.vocab_argmax_noalloc(x, out)
        torch.cuda.synchronize()
        assert torch.equal(out, dreams.vocab_argmax(x))
        np.testing.assert_array_equal(out.cpu().numpy(), torch.argmax(x.float(), dim=1).int().cpu().numpy())


def test_noalloc_wrapper_at_the_row_limit():
    """Exactly DREAMS_NOALLOC_ARGMAX_MAX_ROWS rows, as a [.., .., V] tensor
    that flattens without a copy."""
    import paper_2606_00535_gb300 as dreams
    rows, V = dreams.NOALLOC_ARGMAX_MAX_ROWS, 1000
    x = _logits(rows, V, torch.float32, 30).view(128, rows // 128, V)
    out = torch.full((128, rows // 128), -1, dtype=torch.int32, device="cuda")
    dreams.vocab_argmax_noalloc(x, out)
    torch.cuda.synchronize()
    assert torch.equal(out, torch.argmax(x, dim=-1).int())


def test_noalloc_wrapper_rejects_before_launch():
    """A short output, more rows than the scratch, and leading dimensions that
    only flatten by copying are refused on the host; the output stays as it was."""
    import paper_2606_00535_gb300 as dreams
    x = _logits(8, 512, torch.float32, 40)
    short = torch.full((7,), -3, dtype=torch.int32, device="cuda")
    with pytest.raises(ValueError):
        dreams.vocab_argmax_noalloc(x, short)
    assert (short == -3).all()
    big = torch.zeros((dreams.NOALLOC_ARGMAX_MAX_ROWS + 1, 16), dtype=torch.float32, device="cuda")
    with pytest.raises(ValueError):
        dreams.vocab_argmax_noalloc(big, torch.zeros(big.shape[0], dtype=torch.int32, device="cuda"))
    y = torch.zeros((4, 3, 16), dtype=torch.float32, device="cuda").transpose(0, 1)
    with pytest.raises(ValueError):
        dreams.vocab_argmax_noalloc(y, torch.zeros(12, dtype=torch.int32, device="cuda"))


def test_noalloc_argmax_rejects_rows_beyond_its_scratch():
    import paper_2606_00535_gb300 as dreams
    lib = dreams._lib()
    x = torch.zeros((4, 64), dtype=torch.float32, device="cuda")
    out = torch.zeros((4,), dtype=torch.int32, device="cuda")
    st = lib.dreams_vocab_argmax_noalloc(ctypes.c_void_p(x.data_ptr()), dreams.F32, dreams.NOALLOC_ARGMAX_MAX_ROWS + 1,
                                         64, 64, ctypes.c_void_p(out.data_ptr()), None)
    assert st == dreams.ERR_SCRATCH_LIMIT
    assert b"fixed scratch" in lib.dreams_status_string(st)
