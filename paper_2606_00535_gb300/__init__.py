"""GB300 (sm_103a) tree verification for DREAM-S speculative decoding.

A thin binding over the C ABI of ``libdreams.so`` (declared in
``include/dreams.h``): each function checks the dtype, device and layout of
its torch tensors, passes their ``data_ptr()`` and the current CUDA stream to
the C entry point of the same name, and raises on a non-OK status. Every
step of the computation runs in the library's CUDA kernels; there is no CPU
or PyTorch fallback, and importing this package on a machine without the
built library raises.

The step it implements (paper Sec. 2, "Speculative decoding"): the target
model scores all draft tokens in one pass, then accepts drafts while they
equal its own greedy prediction; here the drafts form a tree.

    out, lse = tree_verify_attn(q, kv, tree, scale)          # per layer
    res = verify_step(logits, tree, kv, max_path)            # argmax + walk + compaction
"""
from __future__ import annotations

import ctypes
import os
import re
import threading
from dataclasses import dataclass
from typing import Dict, Optional, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdreams.so")
HEADER = os.path.join(os.path.dirname(_HERE), "include", "dreams.h")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_WORKSPACE, ERR_CUDA, ERR_SCRATCH_LIMIT = 0, 1, 2, 3, 4, 5
NOALLOC_ARGMAX_MAX_ROWS = 16384
F32, BF16 = 0, 1
DATA_BAD_PARENT, DATA_BAD_TREE_LEN, DATA_BAD_KV_LEN, DATA_BAD_PAGE, DATA_BAD_PATH = 1, 2, 4, 8, 16
DATA_TIMEOUT = 0x20  # a kernel gave up waiting on its own pipeline
TEST_ATTENTION, TEST_LM_HEAD = 1, 2  # kernel families of test_set_stall


class DreamsError(RuntimeError):
    def __init__(self, fn: str, status: int):
        msg = _lib().dreams_status_string(status).decode()
        if status == ERR_CUDA:
            msg += f" (cudaError {_lib().dreams_last_cuda_error()})"
        super().__init__(f"{fn}: {msg}")
        self.status = status


class _KVCache(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("n_layers", ctypes.c_int32),
                ("layer_stride", ctypes.c_int64), ("Hkv", ctypes.c_int32), ("D", ctypes.c_int32),
                ("capacity", ctypes.c_int32), ("page_table", ctypes.c_void_p),
                ("page_size", ctypes.c_int32), ("pages_per_seq", ctypes.c_int32),
                ("num_pages", ctypes.c_int32)]


class _Tree(ctypes.Structure):
    _fields_ = [("parent", ctypes.c_void_p), ("tokens", ctypes.c_void_p), ("tree_len", ctypes.c_void_p),
                ("kv_len", ctypes.c_void_p), ("B", ctypes.c_int32), ("T_max", ctypes.c_int32)]


_LIB: Optional[ctypes.CDLL] = None
_LOCK = threading.Lock()


def _lib() -> ctypes.CDLL:
    global _LIB
    if _LIB is None:
        with _LOCK:
            if _LIB is None:
                if not os.path.exists(LIB_PATH):
                    raise ImportError(f"libdreams.so is not built ({LIB_PATH}); run "
                                      "`python -c 'import __graft_entry__ as g; g.build()'`")
                lib = ctypes.CDLL(LIB_PATH)
                p, i32, i64, sz, f32 = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t,
                                        ctypes.c_float)
                pkv, ptr = ctypes.POINTER(_KVCache), ctypes.POINTER(_Tree)
                sig = {
                    "dreams_tree_verify_attn_workspace_size": (sz, [pkv, ptr, i32]),
                    "dreams_tree_verify_attn_launches": (i32, [pkv, ptr, i32]),
                    "dreams_tree_verify_attn": (ctypes.c_int, [p, i64, i64, pkv, i32, ptr, i32, f32, p, p, p, sz, p,
                                                               p]),
                    "dreams_vocab_argmax_workspace_size": (sz, [i64, i64]),
                    "dreams_vocab_argmax": (ctypes.c_int, [p, ctypes.c_int, i64, i64, i64, p, p, sz, p]),
                    "dreams_accept_path": (ctypes.c_int, [p, ptr, i32, p, p, p, p, p, p]),
                    "dreams_kv_compact": (ctypes.c_int, [pkv, i32, p, p, p, i32, p, p]),
                    "dreams_verify_step_workspace_size": (sz, [ptr, i64]),
                    "dreams_verify_step": (ctypes.c_int, [p, ctypes.c_int, i64, i64, ptr, pkv, i32, p, p, p, p,
                                                          p, p, sz, p, p]),
                    "dreams_vocab_argmax_noalloc": (ctypes.c_int, [p, ctypes.c_int, i64, i64, i64, p, p]),
                    "dreams_attention_workspace_size": (sz, [pkv, i32, i32, i32, i32, i32]),
                    "dreams_attention": (ctypes.c_int, [p, i64, i64, pkv, i32, p, p, i32, i32, i32, f32, i32, p, p,
                                                        p, p, sz, p, p]),
                    "dreams_lm_head_argmax_workspace_size": (sz, [i64]),
                    "dreams_lm_head_argmax": (ctypes.c_int, [p, i64, i64, i64, p, i64, i64, p, p, p, sz, p, p]),
                    "dreams_visual_importance_workspace_size": (sz, [i64, i64, i64, i64]),
                    "dreams_visual_importance": (ctypes.c_int, [p, ctypes.c_int, i64, i64, i64, i64, i64, i64, i32,
                                                                p, p, p, sz, p]),
                    "dreams_vocab_sample_workspace_size": (sz, [i64, i64]),
                    "dreams_vocab_sample": (ctypes.c_int, [p, ctypes.c_int, i64, i64, i64, f32, p, p, p, sz, p]),
                    "dreams_verify_step_sampled_workspace_size": (sz, [ptr, i64]),
                    "dreams_verify_step_sampled": (ctypes.c_int, [p, ctypes.c_int, i64, i64, ptr, pkv, i32, f32, p,
                                                                  p, p, p, p, p, p, sz, p, p]),
                    "dreams_verify_step_speculative": (ctypes.c_int, [p, p, ctypes.c_int, i64, i64, ptr, pkv, i32,
                                                                      f32, p, p, p, p, p, p, p, p]),
                    "dreams_test_set_stall": (ctypes.c_int, [i32, i32, i64]),
                    "dreams_status_string": (ctypes.c_char_p, [ctypes.c_int]),
                    "dreams_version": (i32, []),
                    "dreams_last_cuda_error": (i32, []),
                }
                for name, (res, args) in sig.items():
                    fn = getattr(lib, name)
                    fn.restype = res
                    fn.argtypes = args
                _LIB = lib
    return _LIB


def declared_functions() -> list:
    """Names of the functions ``include/dreams.h`` declares."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\s\*]*?\b(dreams_\w+)\s*\(", text, re.M)))


def version() -> int:
    return int(_lib().dreams_version())


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream, dev: torch.device) -> ctypes.c_void_p:
    """The given stream, or the current stream of the tensors' device ``dev``."""
    s = torch.cuda.current_stream(dev) if stream is None else stream
    if s.device != dev:
        raise ValueError(f"stream is on {s.device}, the tensors on {dev}")
    return ctypes.c_void_p(s.cuda_stream)


def _check(name: str, st: int):
    if st != OK:
        raise DreamsError(name, st)


def _call(name: str, dev: torch.device, *args) -> None:
    """Calls the C entry point with the tensors' device current (the library
    runs on the current CUDA device) and raises on a non-OK status."""
    if dev.type != "cuda":
        raise ValueError(f"{name}: tensors must be on a CUDA device, got {dev}")
    with torch.cuda.device(dev):
        st = getattr(_lib(), name)(*args)
    _check(name, st)


def _rows_view(logits: torch.Tensor) -> torch.Tensor:
    """[rows, V] view of ``logits`` (no copy) with contiguous rows."""
    if logits.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError("logits must be float32 or bfloat16")
    V = int(logits.shape[-1])
    try:
        x = logits if logits.dim() == 2 else logits.view(-1, V)
    except RuntimeError as e:
        raise ValueError("logits' leading dimensions must flatten without a copy") from e
    if x.stride(-1) != 1:
        raise ValueError("logits rows must be contiguous")
    return x


def _need_out(out: torch.Tensor, name: str, dtype, dev, numel: int) -> torch.Tensor:
    _need(out, name, dtype, dev)
    if out.numel() < numel:
        raise ValueError(f"{name} holds {out.numel()} elements, the call uses {numel}")
    return out


def _ws(workspace: Optional[torch.Tensor], dev):
    """Pointer and byte size of a caller's workspace (contiguous, on dev), or
    (None, 0)."""
    if workspace is None:
        return None, 0
    if not isinstance(workspace, torch.Tensor) or workspace.device != dev or not workspace.is_contiguous():
        raise ValueError(f"workspace must be a contiguous tensor on {dev}")
    return _ptr(workspace), workspace.numel() * workspace.element_size()


def _status(status: Optional[torch.Tensor], dev):
    """Pointer to the caller's device status word (int32, on dev), or None."""
    return None if status is None else _ptr(_need_out(status, "status", torch.int32, dev, 1))


def _outputs(outputs: Optional[tuple], B: int, max_path: int, dev) -> tuple:
    """(accept_len [B], path [B, max_path], out_tokens [B, max_path],
    new_kv_len [B]): the caller's, checked, or new."""
    if outputs is None:
        return _walk_outputs(B, max_path, dev)
    if len(outputs) != 4:
        raise ValueError("outputs must be (accept_len, path, out_tokens, new_kv_len)")
    acc, path, toks, nkl = outputs
    return (_need_out(acc, "accept_len", torch.int32, dev, B),
            _need_out(path, "path", torch.int32, dev, B * max_path),
            _need_out(toks, "out_tokens", torch.int32, dev, B * max_path),
            _need_out(nkl, "new_kv_len", torch.int32, dev, B))


def _need(t: torch.Tensor, name: str, dtype, dev) -> torch.Tensor:
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if t.device != dev:
        raise ValueError(f"{name} must be on {dev}, got {t.device}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


@dataclass
class KVCache:
    """K/V cache of one or more layers (bf16).

    Contiguous: ``k, v`` of shape ``[B, capacity, Hkv, D]`` (one layer) or
    ``[n_layers, B, capacity, Hkv, D]``. Paged: ``[num_pages, 64, Hkv, D]``
    (or with a leading layer dim) plus ``page_table`` int32 ``[B, pages_per_seq]``.
    """
    k: torch.Tensor
    v: torch.Tensor
    page_table: Optional[torch.Tensor] = None

    def __post_init__(self):
        if self.k.shape != self.v.shape:
            raise ValueError("k and v shapes differ")
        dev = self.k.device
        _need(self.k, "k", torch.bfloat16, dev)
        _need(self.v, "v", torch.bfloat16, dev)
        nd = self.k.dim()
        if nd not in (4, 5):
            raise ValueError("k must be 4-D or 5-D")
        self.n_layers = self.k.shape[0] if nd == 5 else 1
        shp = self.k.shape[1:] if nd == 5 else self.k.shape
        self.layer_stride = int(shp.numel()) if nd == 5 else 0
        self.Hkv, self.D = int(shp[2]), int(shp[3])
        if self.page_table is None:
            self.B = int(shp[0])
            self.capacity = int(shp[1])
            self.page_size = self.pages_per_seq = self.num_pages = 0
        else:
            _need(self.page_table, "page_table", torch.int32, dev)
            self.B = int(self.page_table.shape[0])
            self.page_size = int(shp[1])
            self.pages_per_seq = int(self.page_table.shape[1])
            self.num_pages = int(shp[0])
            self.capacity = self.pages_per_seq * self.page_size
        self._c = _KVCache(self.k.data_ptr(), self.v.data_ptr(), self.n_layers, self.layer_stride, self.Hkv,
                           self.D, self.capacity,
                           None if self.page_table is None else self.page_table.data_ptr(),
                           self.page_size, self.pages_per_seq, self.num_pages)


@dataclass
class Tree:
    """Draft trees of a batch: int32 ``parent``, ``tokens`` [B, T_max];
    ``tree_len``, ``kv_len`` [B] (all on the same CUDA device)."""
    parent: torch.Tensor
    tokens: torch.Tensor
    tree_len: torch.Tensor
    kv_len: torch.Tensor

    def __post_init__(self):
        dev = self.parent.device
        for n in ("parent", "tokens", "tree_len", "kv_len"):
            _need(getattr(self, n), n, torch.int32, dev)
        self.B, self.T_max = (int(x) for x in self.parent.shape)
        if tuple(self.tokens.shape) != (self.B, self.T_max) or self.tree_len.numel() != self.B or \
                self.kv_len.numel() != self.B:
            raise ValueError("tree tensor shapes disagree")
        self._c = _Tree(self.parent.data_ptr(), self.tokens.data_ptr(), self.tree_len.data_ptr(),
                        self.kv_len.data_ptr(), self.B, self.T_max)


# Zero-filled workspaces, one per (function, device, stream); the kernels
# leave them zero-filled after each call.
_WS: Dict[Tuple[str, int, int], torch.Tensor] = {}


def _workspace(kind: str, nbytes: int, device: torch.device, stream) -> Optional[torch.Tensor]:
    if nbytes == 0:
        return None
    key = (kind, device.index if device.index is not None else torch.cuda.current_device(),
           (torch.cuda.current_stream(device) if stream is None else stream).cuda_stream)
    ws = _WS.get(key)
    if ws is None or ws.numel() < nbytes:
        ws = torch.zeros(nbytes, dtype=torch.uint8, device=device)
        _WS[key] = ws
    return ws


def tree_verify_attn_workspace_size(kv: KVCache, tree: Tree, Hq: int) -> int:
    return int(_lib().dreams_tree_verify_attn_workspace_size(ctypes.byref(kv._c), ctypes.byref(tree._c), Hq))


def tree_verify_attn_launches(kv: KVCache, tree: Tree, Hq: int) -> int:
    """Kernel launches one tree_verify_attn call with these shapes makes."""
    return int(_lib().dreams_tree_verify_attn_launches(ctypes.byref(kv._c), ctypes.byref(tree._c), Hq))


VERIFY_STEP_LAUNCHES = 2  # dreams_verify_step: the argmax, then the walk and compaction
VERIFY_STEP_SAMPLED_LAUNCHES = 3  # draw statistics, draw selection, walk + compaction


def _cache_covers(kv: "KVCache", B: int, D: Optional[int] = None) -> None:
    """The cache holds (at least) the B sequences a call reads or writes, with
    head dim D when given."""
    if kv.B < B:
        raise ValueError(f"the KV cache holds {kv.B} sequences, the call addresses {B}")
    if D is not None and kv.D != D:
        raise ValueError(f"q's head dim {D} differs from the cache's {kv.D}")


def _q_strides(q: torch.Tensor) -> Tuple[int, int]:
    """(sequence stride, token stride) in elements of a bf16 [B, T, Hq, D]
    query tensor whose head rows are dense (a view into a fused QKV output
    qualifies)."""
    if not isinstance(q, torch.Tensor) or q.dtype != torch.bfloat16 or q.dim() != 4:
        raise TypeError("q must be a 4-D bfloat16 tensor [B, T, Hq, D]")
    if q.stride(3) != 1 or q.stride(2) != q.shape[3]:
        raise ValueError("q's head rows must be dense (strides [.., .., D, 1])")
    return int(q.stride(0)), int(q.stride(1))


def tree_verify_attn(q: torch.Tensor, kv: KVCache, tree: Tree, scale: float, layer: int = 0,
                     out: Optional[torch.Tensor] = None, lse: Optional[torch.Tensor] = None,
                     want_lse: bool = False, workspace: Optional[torch.Tensor] = None,
                     status: Optional[torch.Tensor] = None, stream=None):
    """Tree-masked attention of the tree tokens' queries ``q`` (bf16
    [B, T_max, Hq, D], head rows dense, tokens and sequences may be strided)
    over the cache. Returns (out, lse or None); out is dense."""
    dev = q.device
    sb, stt = _q_strides(q)
    Hq = int(q.shape[2])
    if tuple(q.shape[:2]) != (tree.B, tree.T_max):
        raise ValueError(f"q must be [B, T_max, Hq, D] with the tree's B = {tree.B}, T_max = {tree.T_max}")
    _cache_covers(kv, tree.B, int(q.shape[3]))
    if out is None:
        out = torch.empty(tuple(q.shape), dtype=torch.bfloat16, device=dev)
    _need(out, "out", torch.bfloat16, dev)
    if tuple(out.shape) != tuple(q.shape):
        raise ValueError("out must have q's shape")
    if lse is None and want_lse:
        lse = torch.empty(q.shape[:3], dtype=torch.float32, device=dev)
    if lse is not None:
        _need(lse, "lse", torch.float32, dev)
        if tuple(lse.shape) != tuple(q.shape[:3]):
            raise ValueError("lse must be [B, T_max, Hq]")
    need = tree_verify_attn_workspace_size(kv, tree, Hq)
    if workspace is None:
        workspace = _workspace("attn", need, dev, stream)
    _call("dreams_tree_verify_attn", dev,
          _ptr(q), sb, stt, ctypes.byref(kv._c), layer, ctypes.byref(tree._c), Hq, float(scale), _ptr(out),
          _ptr(lse), *_ws(workspace, dev),
          _status(status, dev), _stream(stream, dev))
    return out, lse


def vocab_argmax(logits: torch.Tensor, out: Optional[torch.Tensor] = None,
                 workspace: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Row-wise argmax of a 2-D (or flattened leading dims) f32 / bf16 tensor."""
    x = _rows_view(logits)
    rows, V = int(x.shape[0]), int(x.shape[1])
    dev = logits.device
    if out is None:
        out = torch.empty(logits.shape[:-1], dtype=torch.int32, device=dev)
    _need_out(out, "out", torch.int32, dev, rows)
    need = int(_lib().dreams_vocab_argmax_workspace_size(rows, V))
    if workspace is None:
        workspace = _workspace("argmax", need, dev, stream)
    _call("dreams_vocab_argmax", dev,
          _ptr(x), F32 if x.dtype == torch.float32 else BF16, rows, V, int(x.stride(0)), _ptr(out),
          *_ws(workspace, dev), _stream(stream, dev))
    return out


def vocab_argmax_noalloc(logits: torch.Tensor, out: torch.Tensor, stream=None) -> torch.Tensor:
    """Row-wise argmax into a caller-provided ``out`` without any device
    allocation, for callers that must not allocate while it runs (see
    ``dreams_vocab_argmax_noalloc`` in include/dreams.h): the library's fixed
    scratch serves at most NOALLOC_ARGMAX_MAX_ROWS rows, and calls that overlap
    on the GPU race. Nothing here allocates: ``logits`` must flatten to
    [rows, V] as a view, and ``out`` must hold at least ``rows`` int32."""
    x = _rows_view(logits)
    rows, V = int(x.shape[0]), int(x.shape[1])
    if rows > NOALLOC_ARGMAX_MAX_ROWS:
        raise ValueError(f"{rows} rows exceed the fixed scratch of {NOALLOC_ARGMAX_MAX_ROWS} rows")
    dev = logits.device
    _need_out(out, "out", torch.int32, dev, rows)
    _call("dreams_vocab_argmax_noalloc", dev, _ptr(x), F32 if x.dtype == torch.float32 else BF16, rows, V,
          int(x.stride(0)), _ptr(out), _stream(stream, dev))
    return out


def vocab_sample(logits: torch.Tensor, temperature: float, uniforms: torch.Tensor,
                 out: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                 stream=None) -> torch.Tensor:
    """One draw per row of a 2-D (or flattened leading dims) f32 / bf16 tensor
    from softmax(row / temperature), by inverse transform with the row's
    uniform (``uniforms``: f32, one per row, on the same device)."""
    x = _rows_view(logits)
    rows, V = int(x.shape[0]), int(x.shape[1])
    dev = logits.device
    _need(uniforms, "uniforms", torch.float32, dev)
    if uniforms.numel() != rows:
        raise ValueError("uniforms must hold one value per row")
    if out is None:
        out = torch.empty(logits.shape[:-1], dtype=torch.int32, device=dev)
    _need_out(out, "out", torch.int32, dev, rows)
    need = int(_lib().dreams_vocab_sample_workspace_size(rows, V))
    if workspace is None:
        workspace = _workspace("sample", need, dev, stream)
    _call("dreams_vocab_sample", dev,
          _ptr(x), F32 if x.dtype == torch.float32 else BF16, rows, V, int(x.stride(0)), float(temperature),
          _ptr(uniforms), _ptr(out), *_ws(workspace, dev),
          _stream(stream, dev))
    return out


ATTN_FULL = 1    # query t attends slots 0 .. kv_len - 1 (cross-attention)
ATTN_CAUSAL = 2  # query t attends slots 0 .. kv_len + t (prefill self-attention)


def attention(q: torch.Tensor, kv: KVCache, q_len: torch.Tensor, kv_len: torch.Tensor, scale: float, mode: int,
              layer: int = 0, out: Optional[torch.Tensor] = None, want_lse: bool = False,
              want_entropy: bool = False, workspace: Optional[torch.Tensor] = None,
              status: Optional[torch.Tensor] = None, stream=None):
    """Attention without a tree (ATTN_FULL: the draft's cross-attention to
    target features; ATTN_CAUSAL: a layer's prefill). q: bf16 [B, T_max, Hq,
    D], head rows dense, tokens and sequences may be strided. Returns (out,
    lse, entropy); out is dense; lse and entropy are None unless asked."""
    dev = q.device
    sb, stt = _q_strides(q)
    B, T_max, Hq = int(q.shape[0]), int(q.shape[1]), int(q.shape[2])
    for n, t in (("q_len", q_len), ("kv_len", kv_len)):
        _need(t, n, torch.int32, dev)
        if t.numel() < B:
            raise ValueError(f"{n} holds {t.numel()} entries, q has {B} sequences")
    _cache_covers(kv, B, int(q.shape[3]))
    if out is None:
        out = torch.empty(tuple(q.shape), dtype=torch.bfloat16, device=dev)
    _need(out, "out", torch.bfloat16, dev)
    if tuple(out.shape) != tuple(q.shape):
        raise ValueError("out must have q's shape")
    lse = torch.empty((B, T_max, Hq), dtype=torch.float32, device=dev) if want_lse else None
    ent = torch.empty((B, T_max, Hq), dtype=torch.float32, device=dev) if want_entropy else None
    need = int(_lib().dreams_attention_workspace_size(ctypes.byref(kv._c), B, T_max, Hq, mode, int(want_entropy)))
    if workspace is None:
        workspace = _workspace("attention", need, dev, stream)
    _call("dreams_attention", dev, _ptr(q), sb, stt, ctypes.byref(kv._c), layer, _ptr(q_len), _ptr(kv_len), B,
          T_max, Hq, float(scale), mode, _ptr(out), _ptr(lse), _ptr(ent), *_ws(workspace, dev),
          _status(status, dev), _stream(stream, dev))
    return out, lse, ent


def lm_head_argmax(hidden: torch.Tensor, weight: torch.Tensor, out: Optional[torch.Tensor] = None,
                   out_max: Optional[torch.Tensor] = None, want_max: bool = False,
                   workspace: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
                   stream=None):
    """argmax over the vocabulary of hidden @ weight.T (bf16 [rows, K] and
    [V, K], f32 accumulation) without writing the logits. Returns the indices
    (int32 [rows]) and, with ``want_max``, the maximum logits (f32 [rows])."""
    for n, t in (("hidden", hidden), ("weight", weight)):
        if t.dtype != torch.bfloat16 or t.dim() != 2 or t.stride(1) != 1:
            raise TypeError(f"{n} must be a 2-D bf16 tensor with contiguous rows")
    if weight.device != hidden.device or weight.shape[1] != hidden.shape[1]:
        raise ValueError("hidden and weight must share the device and the hidden size")
    rows, K = int(hidden.shape[0]), int(hidden.shape[1])
    V = int(weight.shape[0])
    dev = hidden.device
    if out is None:
        out = torch.empty(rows, dtype=torch.int32, device=dev)
    _need_out(out, "out", torch.int32, dev, rows)
    if out_max is None and want_max:
        out_max = torch.empty(rows, dtype=torch.float32, device=dev)
    if out_max is not None:
        _need_out(out_max, "out_max", torch.float32, dev, rows)
    need = int(_lib().dreams_lm_head_argmax_workspace_size(rows))
    if workspace is None:
        workspace = _workspace("lm_head", need, dev, stream)
    _call("dreams_lm_head_argmax", dev, _ptr(hidden), rows, K, int(hidden.stride(0)), _ptr(weight), V,
          int(weight.stride(0)), _ptr(out), _ptr(out_max), *_ws(workspace, dev), _status(status, dev),
          _stream(stream, dev))
    return (out, out_max) if want_max or out_max is not None else out


def visual_importance(attn: torch.Tensor, v0: int, n_vis: int, r: int, workspace: Optional[torch.Tensor] = None,
                      stream=None):
    """Eq. 2 importance of the visual tokens (key positions v0 .. v0+n_vis-1)
    from attention weights [B, H, Q, K] (f32 / bf16, contiguous), and the r
    kept positions in increasing order. Returns (importance f32 [B, n_vis],
    keep int32 [B, r])."""
    if attn.dtype not in (torch.float32, torch.bfloat16) or attn.dim() != 4 or not attn.is_contiguous():
        raise TypeError("attn must be a contiguous [B, H, Q, K] float32/bfloat16 tensor")
    B, H, Q, K = (int(x) for x in attn.shape)
    dev = attn.device
    imp = torch.empty((B, n_vis), dtype=torch.float32, device=dev)
    keep = torch.empty((B, r), dtype=torch.int32, device=dev)
    need = int(_lib().dreams_visual_importance_workspace_size(B, H, Q, n_vis))
    if workspace is None:
        workspace = _workspace("importance", need, dev, stream)
    _call("dreams_visual_importance", dev, _ptr(attn), F32 if attn.dtype == torch.float32 else BF16, B, H, Q, K, v0,
          n_vis, r, _ptr(imp), _ptr(keep), *_ws(workspace, dev),
          _stream(stream, dev))
    return imp, keep


def _walk_outputs(B: int, max_path: int, dev):
    return (torch.empty(B, dtype=torch.int32, device=dev),
            torch.empty((B, max_path), dtype=torch.int32, device=dev),
            torch.empty((B, max_path), dtype=torch.int32, device=dev),
            torch.empty(B, dtype=torch.int32, device=dev))


def accept_path(argmax: torch.Tensor, tree: Tree, max_path: int, status: Optional[torch.Tensor] = None,
                stream=None) -> dict:
    """Greedy acceptance over the trees. Returns a dict of device tensors."""
    dev = tree.parent.device
    _need_out(argmax, "argmax", torch.int32, dev, tree.B * tree.T_max)
    acc, path, toks, nkl = _walk_outputs(tree.B, max_path, dev)
    _call("dreams_accept_path", dev, _ptr(argmax), ctypes.byref(tree._c), max_path, _ptr(acc), _ptr(path),
          _ptr(toks), _ptr(nkl), _status(status, dev), _stream(stream, dev))
    return {"accept_len": acc, "path": path, "out_tokens": toks, "new_kv_len": nkl}


def kv_compact(kv: KVCache, kv_len: torch.Tensor, accept_len: torch.Tensor, path: torch.Tensor,
               status: Optional[torch.Tensor] = None, stream=None) -> None:
    """Moves the accepted slots into place, in all layers of ``kv``."""
    dev = kv.k.device
    for n, t in (("kv_len", kv_len), ("accept_len", accept_len), ("path", path)):
        _need(t, n, torch.int32, dev)
    if path.dim() != 2:
        raise ValueError("path must be [B, max_path]")
    B, max_path = (int(x) for x in path.shape)
    for n, t in (("kv_len", kv_len), ("accept_len", accept_len)):
        if t.numel() < B:
            raise ValueError(f"{n} holds {t.numel()} entries, path has {B} rows")
    _cache_covers(kv, B)
    _call("dreams_kv_compact", dev, ctypes.byref(kv._c), B, _ptr(kv_len), _ptr(accept_len), _ptr(path), max_path,
          _status(status, dev), _stream(stream, dev))


def verify_step_sampled_workspace_size(tree: Tree, V: int) -> int:
    return int(_lib().dreams_verify_step_sampled_workspace_size(ctypes.byref(tree._c), V))


def verify_step_workspace_size(tree: Tree, V: int) -> int:
    return int(_lib().dreams_verify_step_workspace_size(ctypes.byref(tree._c), V))


def verify_step(logits: torch.Tensor, tree: Tree, kv: KVCache, max_path: int,
                argmax_out: Optional[torch.Tensor] = None, outputs: Optional[tuple] = None,
                workspace: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
                stream=None) -> dict:
    """Argmax of the tree rows of ``logits`` ([B, T_max, V] f32/bf16), greedy
    acceptance and KV compaction, in one call (two kernel launches)."""
    dev = tree.parent.device
    if logits.dtype not in (torch.float32, torch.bfloat16) or logits.device != dev:
        raise TypeError("logits must be float32/bfloat16 on the tree's device")
    if logits.dim() != 3 or tuple(logits.shape[:2]) != (tree.B, tree.T_max) or logits.stride(-1) != 1 or \
            logits.stride(0) != logits.shape[1] * logits.stride(1):
        raise ValueError("logits must be [B, T_max, V] with uniformly strided contiguous rows")
    V = int(logits.shape[2])
    if argmax_out is not None:
        _need_out(argmax_out, "argmax_out", torch.int32, dev, tree.B * tree.T_max)
    acc, path, toks, nkl = _outputs(outputs, tree.B, max_path, dev)
    st = _status(status, dev)
    _cache_covers(kv, tree.B)
    need = verify_step_workspace_size(tree, V)
    if workspace is None:
        workspace = _workspace("step", need, dev, stream)
    _call("dreams_verify_step", dev,
          _ptr(logits), F32 if logits.dtype == torch.float32 else BF16, V, int(logits.stride(1)),
          ctypes.byref(tree._c), ctypes.byref(kv._c), max_path, _ptr(argmax_out), _ptr(acc), _ptr(path),
          _ptr(toks), _ptr(nkl), *_ws(workspace, dev), st,
          _stream(stream, dev))
    return {"accept_len": acc, "path": path, "out_tokens": toks, "new_kv_len": nkl}


def verify_step_sampled(logits: torch.Tensor, tree: Tree, kv: KVCache, max_path: int, temperature: float,
                        uniforms: torch.Tensor, sample_out: Optional[torch.Tensor] = None,
                        outputs: Optional[tuple] = None, workspace: Optional[torch.Tensor] = None,
                        status: Optional[torch.Tensor] = None, stream=None) -> dict:
    """The verification tail at temperature > 0: the target's draw per tree
    node (``uniforms``: f32 [B, T_max]) takes the place of the argmax, then
    acceptance and KV compaction, in one call (three kernel launches)."""
    dev = tree.parent.device
    if logits.dtype not in (torch.float32, torch.bfloat16) or logits.device != dev:
        raise TypeError("logits must be float32/bfloat16 on the tree's device")
    if logits.dim() != 3 or tuple(logits.shape[:2]) != (tree.B, tree.T_max) or logits.stride(-1) != 1 or \
            logits.stride(0) != logits.shape[1] * logits.stride(1):
        raise ValueError("logits must be [B, T_max, V] with uniformly strided contiguous rows")
    _need(uniforms, "uniforms", torch.float32, dev)
    if tuple(uniforms.shape) != (tree.B, tree.T_max):
        raise ValueError("uniforms must be [B, T_max]")
    V = int(logits.shape[2])
    if sample_out is not None:
        _need_out(sample_out, "sample_out", torch.int32, dev, tree.B * tree.T_max)
    acc, path, toks, nkl = _outputs(outputs, tree.B, max_path, dev)
    st = _status(status, dev)
    _cache_covers(kv, tree.B)
    need = verify_step_sampled_workspace_size(tree, V)
    if workspace is None:
        workspace = _workspace("step_sampled", need, dev, stream)
    _call("dreams_verify_step_sampled", dev,
          _ptr(logits), F32 if logits.dtype == torch.float32 else BF16, V, int(logits.stride(1)),
          ctypes.byref(tree._c), ctypes.byref(kv._c), max_path, float(temperature), _ptr(uniforms),
          _ptr(sample_out), _ptr(acc), _ptr(path), _ptr(toks), _ptr(nkl), *_ws(workspace, dev),
          st, _stream(stream, dev))
    return {"accept_len": acc, "path": path, "out_tokens": toks, "new_kv_len": nkl}


def verify_step_speculative(target_logits: torch.Tensor, draft_logits: torch.Tensor, tree: Tree, kv: KVCache,
                            max_path: int, temperature: float, u_accept: torch.Tensor, u_resample: torch.Tensor,
                            outputs: Optional[tuple] = None, status: Optional[torch.Tensor] = None,
                            stream=None) -> dict:
    """The verification tail at temperature > 0 by speculative sampling over
    the tree: a draft is accepted with probability min(1, r/q) against the
    current residual r, a rejection renormalises max(0, r - q), and the bonus is
    drawn from what is left (``dreams_verify_step_speculative``). target_logits
    and draft_logits: [B, T_max, V] f32/bf16 with the same strides; u_accept,
    u_resample: f32 [B, T_max]. Then acceptance outputs and KV compaction."""
    dev = tree.parent.device
    for n, t in (("target_logits", target_logits), ("draft_logits", draft_logits)):
        if t.dtype not in (torch.float32, torch.bfloat16) or t.device != dev:
            raise TypeError(f"{n} must be float32/bfloat16 on the tree's device")
        if t.dim() != 3 or tuple(t.shape[:2]) != (tree.B, tree.T_max) or t.stride(-1) != 1 or \
                t.stride(0) != t.shape[1] * t.stride(1):
            raise ValueError(f"{n} must be [B, T_max, V] with uniformly strided contiguous rows")
    if draft_logits.dtype != target_logits.dtype or draft_logits.shape != target_logits.shape or \
            draft_logits.stride() != target_logits.stride():
        raise ValueError("target and draft logits must share dtype, shape and strides")
    for n, t in (("u_accept", u_accept), ("u_resample", u_resample)):
        _need(t, n, torch.float32, dev)
        if tuple(t.shape) != (tree.B, tree.T_max):
            raise ValueError(f"{n} must be [B, T_max]")
    V = int(target_logits.shape[2])
    acc, path, toks, nkl = _outputs(outputs, tree.B, max_path, dev)
    st = _status(status, dev)
    _cache_covers(kv, tree.B)
    _call("dreams_verify_step_speculative", dev,
          _ptr(target_logits), _ptr(draft_logits), F32 if target_logits.dtype == torch.float32 else BF16, V,
          int(target_logits.stride(1)), ctypes.byref(tree._c), ctypes.byref(kv._c), max_path, float(temperature),
          _ptr(u_accept), _ptr(u_resample), _ptr(acc), _ptr(path), _ptr(toks), _ptr(nkl), st,
          _stream(stream, dev))
    return {"accept_len": acc, "path": path, "out_tokens": toks, "new_kv_len": nkl}


VERIFY_STEP_SPECULATIVE_LAUNCHES = 1  # one cluster per sequence: walk, residual sums, bonus, compaction


def test_set_stall(kernels: int, stall_at: int, wait_limit_ns: int = 20_000_000) -> None:
    """Test hook for the bounded pipeline waits (``dreams_test_set_stall``):
    later launches of the selected kernel families withhold their copies from
    the ``stall_at``-th tile on and give up waiting after ``wait_limit_ns``.
    ``stall_at < 0`` restores normal operation."""
    _check("dreams_test_set_stall", _lib().dreams_test_set_stall(int(kernels), int(stall_at), int(wait_limit_ns)))
