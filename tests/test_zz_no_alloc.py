"""The no-allocation argmax entry point, through the C ABI.

dreams_vocab_argmax_noalloc serves callers that must not allocate device
memory while the argmax runs (an engine plugin whose host owns every device
allocation, a server that reserves its whole memory budget at start-up). It
must give the same indices as dreams_vocab_argmax, which uses a
caller-provided workspace, call after call, because the fixed scratch it uses
instead is shared by all calls and keeps each call's leftovers.

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
    # two calls in a row, with shapes that split rows over several CTAs, so
    # the second call runs on the scratch the first one left behind
    for seed, (rows, V, dtype) in enumerate([(48, 152064, torch.bfloat16), (60, 32000, torch.float32)]):
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


def test_noalloc_argmax_rejects_rows_beyond_its_scratch():
    import paper_2606_00535_gb300 as dreams
    lib = dreams._lib()
    x = torch.zeros((4, 64), dtype=torch.float32, device="cuda")
    out = torch.zeros((4,), dtype=torch.int32, device="cuda")
    st = lib.dreams_vocab_argmax_noalloc(ctypes.c_void_p(x.data_ptr()), dreams.F32, dreams.NOALLOC_ARGMAX_MAX_ROWS + 1,
                                         64, 64, ctypes.c_void_p(out.data_ptr()), None)
    assert st == dreams.ERR_SCRATCH_LIMIT
    assert b"fixed scratch" in lib.dreams_status_string(st)
