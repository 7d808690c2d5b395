"""ctypes binding of ``libtk.so`` (include/tk.h), one Python function per entry point.

Argument marshalling only: each function checks that the torch tensors it
is given have the dtype, device and contiguity the C ABI expects, passes
their ``data_ptr()`` and the current CUDA stream, and raises ``TkError`` on
a non-OK status.  Every step of the computation runs in the library's
kernels; there is no CPU or PyTorch fallback, and a missing library raises.
"""

from __future__ import annotations

import ctypes
import math
import os
from dataclasses import dataclass

import torch

TK_OK, TK_ERR_INVALID_ARG, TK_ERR_UNSUPPORTED, TK_ERR_WORKSPACE, TK_ERR_CUDA, TK_ERR_DEVICE = range(6)
TK_BF16, TK_F32, TK_I8, TK_I4 = 0, 1, 2, 3

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libtk.so")

EXPORTED = ("tk_kv_append", "tk_attn_prefill", "tk_decode_workspace_size", "tk_attn_decode",
            "tk_attn_decode_append", "tk_attn_decode_noalloc", "tk_attn_prefill_cached",
            "tk_prefill_cached_workspace_size",
            "tk_attn_forward", "tk_backward_workspace_size", "tk_attn_backward", "tk_copy_async",
            "tk_check_wait_timeout", "tk_get_device_error", "tk_status_string", "tk_last_error",
            "tk_abi_version", "tk_graph_begin", "tk_graph_end", "tk_graph_launch",
            "tk_graph_destroy")


class TkError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        super().__init__(f"{where}: {_status_name(status)}: {detail}")
        self.status = status


class tk_cache_desc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "batch", "h_q", "h_kv", "r", "d_v", "capacity", "page_size", "num_pages",
        "max_pages_per_seq", "k_dtype")]


_lib = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libtk.so once and declare the C signatures; raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is not built; run `python -m paper_2603_04427_gb300.build` "
                           "(or __graft_entry__.build()) first")
    L = ctypes.CDLL(path)
    vp, i32, f32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_float, ctypes.c_size_t
    dp = ctypes.POINTER(tk_cache_desc)
    sig = {
        "tk_kv_append": (i32, [dp, vp, vp, vp, vp, vp, vp, vp, i32, vp]),
        "tk_attn_prefill": (i32, [vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, i32, f32, i32, vp]),
        "tk_decode_workspace_size": (sz, [dp, i32]),
        "tk_attn_forward": (i32, [vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, i32, f32, i32,
                                  vp]),
        "tk_backward_workspace_size": (sz, [i32, i32, i32]),
        "tk_attn_backward": (i32, [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, i32, i32, i32, i32,
                                   i32, i32, f32, i32, vp]),
        "tk_attn_prefill_cached": (i32, [dp, vp, vp, vp, vp, vp, vp, vp, vp, i32, i32, vp, i32,
                                         f32, i32, vp, sz, vp]),
        "tk_prefill_cached_workspace_size": (sz, [dp, i32]),
        "tk_attn_decode": (i32, [dp, vp, vp, vp, vp, vp, vp, i32, vp, i32, f32, vp, sz, vp]),
        "tk_attn_decode_append": (i32, [dp, vp, vp, vp, vp, vp, vp, vp, vp, i32, vp, i32, f32, vp,
                                        sz, vp]),
        "tk_attn_decode_noalloc": (i32, [dp, vp, vp, vp, vp, vp, vp, i32, vp, i32, f32, vp]),
        "tk_get_device_error": (i32, [ctypes.POINTER(i32), vp]),
        "tk_check_wait_timeout": (i32, [i32, vp]),
        "tk_copy_async": (i32, [vp, vp, sz, vp]),
        "tk_graph_begin": (i32, [vp]),
        "tk_graph_end": (i32, [vp, ctypes.POINTER(vp)]),
        "tk_graph_launch": (i32, [vp, vp]),
        "tk_graph_destroy": (i32, [vp]),
        "tk_status_string": (ctypes.c_char_p, [i32]),
        "tk_last_error": (ctypes.c_char_p, []),
        "tk_abi_version": (i32, []),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype, fn.argtypes = res, args
    _lib = L
    return L


def _status_name(s: int) -> str:
    names = {0: "TK_OK", 1: "TK_ERR_INVALID_ARG", 2: "TK_ERR_UNSUPPORTED", 3: "TK_ERR_WORKSPACE",
             4: "TK_ERR_CUDA", 5: "TK_ERR_DEVICE"}
    return names.get(s, f"status {s}")


def _check(status: int, where: str):
    if status != TK_OK:
        raise TkError(status, where, load_library().tk_last_error().decode())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need_out(t, name, device):
    """An output: float32 or bfloat16, contiguous, on `device` or in page-locked host memory
    (the kernel then writes it zero-copy)."""
    if t.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError(f"{name} must be float32 or bfloat16")
    if t.is_cuda:
        _need(t, t.dtype, name, device)
    elif not t.is_pinned() or not t.is_contiguous():
        raise ValueError(f"{name} must be a CUDA tensor or a contiguous page-locked host tensor")


def _need(t, dtype, name, device=None):
    if t is None:
        return
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


# ------------------------------------------------------------------ cache helper

@dataclass
class ThinKeyCache:
    """Caller-owned thin-key / full-value cache tensors plus their descriptor.

    Contiguous: k [B, H_kv, cap, r] (bf16 or int8; uint8 [B, H_kv, cap, r/2] of
    packed int4 codes), k_scale [B, H_kv, cap] fp32, v [B, H_kv, cap, d_v] bf16.
    Paged: pools [P, H_kv, page_size, ...] and a page table [B, max_pages] int32.
    """
    desc: tk_cache_desc
    k: torch.Tensor
    v: torch.Tensor
    k_scale: torch.Tensor | None = None
    page_table: torch.Tensor | None = None

    @staticmethod
    def allocate(batch, h_q, h_kv, r, d_v, capacity=0, page_size=0, num_pages=0,
                 page_table=None, k_int8=False, device="cuda", fill=0, k_int4=False):
        if page_size:
            if page_table is None:
                raise ValueError("a paged cache needs a page table")
            page_table = page_table.to(device=device, dtype=torch.int32).contiguous()
            lead = (num_pages, h_kv, page_size)
            max_pages = page_table.shape[1]
        else:
            lead = (batch, h_kv, capacity)
            max_pages = 0
        if k_int8 and k_int4:
            raise ValueError("k_int8 and k_int4 are exclusive")
        kd = torch.int8 if k_int8 else (torch.uint8 if k_int4 else torch.bfloat16)
        k = torch.full(lead + (r // 2 if k_int4 else r,), fill, dtype=kd, device=device)
        v = torch.full(lead + (d_v,), fill, dtype=torch.bfloat16, device=device)
        ks = torch.zeros(lead, dtype=torch.float32, device=device) if (k_int8 or k_int4) else None
        desc = tk_cache_desc(batch, h_q, h_kv, r, d_v, 0 if page_size else capacity, page_size,
                             num_pages if page_size else 0, max_pages,
                             TK_I8 if k_int8 else (TK_I4 if k_int4 else TK_BF16))
        return ThinKeyCache(desc, k, v, ks, page_table)


# ------------------------------------------------------------------ entry points

def tk_abi_version() -> int:
    return int(load_library().tk_abi_version())


def tk_status_string(status: int) -> str:
    return load_library().tk_status_string(status).decode()


def tk_last_error() -> str:
    return load_library().tk_last_error().decode()


def tk_kv_append(cache: ThinKeyCache, k_new, v_new, seq_lens, stream=None):
    """Append k_new [B, H_kv, T, r] / v_new [B, H_kv, T, d_v] (bf16) at seq_lens[b]."""
    d = cache.desc
    dev = cache.k.device
    _need(k_new, torch.bfloat16, "k_new", dev)
    _need(v_new, torch.bfloat16, "v_new", dev)
    _need(seq_lens, torch.int32, "seq_lens", dev)
    T = k_new.shape[2]
    if tuple(k_new.shape) != (d.batch, d.h_kv, T, d.r) or tuple(v_new.shape) != (d.batch, d.h_kv, T, d.d_v):
        raise ValueError(f"k_new {tuple(k_new.shape)} / v_new {tuple(v_new.shape)} do not match the cache")
    L = load_library()
    _check(L.tk_kv_append(ctypes.byref(d), _ptr(cache.k), _ptr(cache.v), _ptr(cache.k_scale),
                          _ptr(cache.page_table), _ptr(seq_lens), _ptr(k_new), _ptr(v_new), T,
                          _stream(stream)), "tk_kv_append")


def tk_decode_workspace_size(desc: tk_cache_desc, max_seq_len: int) -> int:
    n = int(load_library().tk_decode_workspace_size(ctypes.byref(desc), int(max_seq_len)))
    if n == 0:
        raise TkError(TK_ERR_INVALID_ARG, "tk_decode_workspace_size", tk_last_error())
    return n


def decode_workspace(desc: tk_cache_desc, max_seq_len: int, device="cuda") -> torch.Tensor:
    """A zero-filled workspace of the size tk_attn_decode needs (torch owns the memory)."""
    return torch.zeros(tk_decode_workspace_size(desc, max_seq_len), dtype=torch.uint8, device=device)


def tk_attn_decode(cache: ThinKeyCache, q, seq_lens, max_seq_len: int, out, workspace,
                   scale: float | None = None, stream=None):
    """One decode step: q [B, H_q, r] bf16 -> out [B, H_q, d_v] (fp32 or bf16, on the GPU or
    in page-locked host memory, which the kernel then writes directly)."""
    d = cache.desc
    dev = cache.k.device
    _need(q, torch.bfloat16, "q", dev)
    _need(seq_lens, torch.int32, "seq_lens", dev)
    _need(workspace, torch.uint8, "workspace", dev)
    _need_out(out, "out", dev)
    if tuple(q.shape) != (d.batch, d.h_q, d.r) or tuple(out.shape) != (d.batch, d.h_q, d.d_v):
        raise ValueError(f"q {tuple(q.shape)} / out {tuple(out.shape)} do not match the cache")
    scale = 1.0 / math.sqrt(d.r) if scale is None else float(scale)
    L = load_library()
    _check(L.tk_attn_decode(ctypes.byref(d), _ptr(q), _ptr(cache.k), _ptr(cache.v),
                            _ptr(cache.k_scale), _ptr(cache.page_table), _ptr(seq_lens),
                            int(max_seq_len), _ptr(out),
                            TK_F32 if out.dtype == torch.float32 else TK_BF16, scale,
                            _ptr(workspace), workspace.numel(), _stream(stream)), "tk_attn_decode")
    return out


def tk_attn_decode_append(cache: ThinKeyCache, q, k_new, v_new, seq_lens, max_seq_len: int, out,
                          workspace, scale: float | None = None, stream=None):
    """Append one token per sequence (k_new [B, H_kv, r], v_new [B, H_kv, d_v] bf16) at
    seq_lens[b] and decode q [B, H_q, r] over the seq_lens[b] + 1 tokens, in one launch."""
    d = cache.desc
    dev = cache.k.device
    _need(q, torch.bfloat16, "q", dev)
    _need(k_new, torch.bfloat16, "k_new", dev)
    _need(v_new, torch.bfloat16, "v_new", dev)
    _need(seq_lens, torch.int32, "seq_lens", dev)
    _need(workspace, torch.uint8, "workspace", dev)
    _need_out(out, "out", dev)
    if tuple(q.shape) != (d.batch, d.h_q, d.r) or tuple(out.shape) != (d.batch, d.h_q, d.d_v):
        raise ValueError(f"q {tuple(q.shape)} / out {tuple(out.shape)} do not match the cache")
    if tuple(k_new.shape) != (d.batch, d.h_kv, d.r) or tuple(v_new.shape) != (d.batch, d.h_kv, d.d_v):
        raise ValueError(f"k_new {tuple(k_new.shape)} / v_new {tuple(v_new.shape)} do not match the cache")
    scale = 1.0 / math.sqrt(d.r) if scale is None else float(scale)
    L = load_library()
    _check(L.tk_attn_decode_append(ctypes.byref(d), _ptr(q), _ptr(cache.k), _ptr(cache.v),
                                   _ptr(cache.k_scale), _ptr(cache.page_table), _ptr(seq_lens),
                                   _ptr(k_new), _ptr(v_new), int(max_seq_len), _ptr(out),
                                   TK_F32 if out.dtype == torch.float32 else TK_BF16, scale,
                                   _ptr(workspace), workspace.numel(), _stream(stream)),
           "tk_attn_decode_append")
    return out


def tk_attn_forward(q, k, v, out, lse, scale: float | None = None, causal: bool = True, stream=None):
    """tk_attn_prefill that also writes lse [B, H_q, S] (fp32), each row's logsumexp."""
    dev = q.device
    for t, n in ((q, "q"), (k, "k"), (v, "v")):
        _need(t, torch.bfloat16, n, dev)
    _need(lse, torch.float32, "lse", dev)
    if out.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError("out must be float32 or bfloat16")
    _need(out, out.dtype, "out", dev)
    B, hq, S, r = q.shape
    hkv, dv = k.shape[1], v.shape[3]
    if tuple(k.shape) != (B, hkv, S, r) or tuple(v.shape) != (B, hkv, S, dv) or \
            tuple(out.shape) != (B, hq, S, dv) or tuple(lse.shape) != (B, hq, S):
        raise ValueError("q / k / v / out / lse shapes are inconsistent")
    scale = 1.0 / math.sqrt(r) if scale is None else float(scale)
    L = load_library()
    _check(L.tk_attn_forward(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(lse),
                             TK_F32 if out.dtype == torch.float32 else TK_BF16,
                             B, hq, hkv, S, r, dv, scale, 1 if causal else 0, _stream(stream)),
           "tk_attn_forward")
    return out, lse


def tk_attn_backward(q, k, v, out, d_out, lse, dq, dk, dv, workspace=None,
                     scale: float | None = None, causal: bool = True, stream=None):
    """Gradients dq [B, H_q, S, r], dk [B, H_kv, S, r], dv [B, H_kv, S, d_v] (fp32)
    of prefill attention for dL/d(out) = d_out (bf16), from the forward's lse."""
    dev = q.device
    for t, n in ((q, "q"), (k, "k"), (v, "v"), (out, "out"), (d_out, "d_out")):
        _need(t, torch.bfloat16, n, dev)
    for t, n in ((lse, "lse"), (dq, "dq"), (dk, "dk"), (dv, "dv")):
        _need(t, torch.float32, n, dev)
    B, hq, S, r = q.shape
    hkv, d_v = k.shape[1], v.shape[3]
    if tuple(k.shape) != (B, hkv, S, r) or tuple(v.shape) != (B, hkv, S, d_v) or \
            tuple(out.shape) != (B, hq, S, d_v) or tuple(d_out.shape) != (B, hq, S, d_v) or \
            tuple(lse.shape) != (B, hq, S) or tuple(dq.shape) != tuple(q.shape) or \
            tuple(dk.shape) != tuple(k.shape) or tuple(dv.shape) != tuple(v.shape):
        raise ValueError("backward tensor shapes are inconsistent")
    L = load_library()
    if workspace is None:
        workspace = torch.empty(int(L.tk_backward_workspace_size(B, hq, S)), dtype=torch.uint8,
                                device=dev)
    _need(workspace, torch.uint8, "workspace", dev)
    scale = 1.0 / math.sqrt(r) if scale is None else float(scale)
    _check(L.tk_attn_backward(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(d_out), _ptr(lse),
                              _ptr(dq), _ptr(dk), _ptr(dv), _ptr(workspace), workspace.numel(),
                              B, hq, hkv, S, r, d_v, scale, 1 if causal else 0, _stream(stream)),
           "tk_attn_backward")
    return dq, dk, dv


def prefill_cached_workspace(cache: ThinKeyCache, max_seq_len: int):
    """The device workspace tk_attn_prefill_cached needs for this cache and this
    bound of seq_lens[b] + S (int8 / int4 keys), or None (bf16 keys)."""
    n = int(load_library().tk_prefill_cached_workspace_size(ctypes.byref(cache.desc), int(max_seq_len)))
    return torch.empty(n, dtype=torch.uint8, device=cache.k.device) if n else None


def tk_attn_prefill_cached(cache: ThinKeyCache, q, k_new, v_new, seq_lens, max_seq_len: int, out,
                           scale: float | None = None, causal: bool = True, workspace=None,
                           stream=None):
    """Append a chunk (k_new [B, H_kv, S, r], v_new [B, H_kv, S, d_v] bf16) at seq_lens[b]
    and prefill its queries q [B, H_q, S, r] over the cache (query i at position
    seq_lens[b] + i) -> out [B, H_q, S, d_v] (fp32 or bf16).  bf16, int8 or int4 keys;
    quantised keys need a workspace (prefill_cached_workspace; allocated here if None)."""
    d = cache.desc
    dev = cache.k.device
    for t, n in ((q, "q"), (k_new, "k_new"), (v_new, "v_new")):
        _need(t, torch.bfloat16, n, dev)
    _need(seq_lens, torch.int32, "seq_lens", dev)
    if out.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError("out must be float32 or bfloat16")
    _need(out, out.dtype, "out", dev)
    S = q.shape[2]
    if tuple(q.shape) != (d.batch, d.h_q, S, d.r) or tuple(out.shape) != (d.batch, d.h_q, S, d.d_v) \
            or tuple(k_new.shape) != (d.batch, d.h_kv, S, d.r) \
            or tuple(v_new.shape) != (d.batch, d.h_kv, S, d.d_v):
        raise ValueError("q / k_new / v_new / out shapes do not match the cache")
    scale = 1.0 / math.sqrt(d.r) if scale is None else float(scale)
    L = load_library()
    if workspace is None and d.k_dtype != TK_BF16:
        workspace = prefill_cached_workspace(cache, max_seq_len)
    if workspace is not None:
        _need(workspace, torch.uint8, "workspace", dev)
    _check(L.tk_attn_prefill_cached(ctypes.byref(d), _ptr(q), _ptr(cache.k), _ptr(cache.v),
                                    _ptr(cache.k_scale), _ptr(cache.page_table), _ptr(seq_lens),
                                    _ptr(k_new), _ptr(v_new),
                                    S, int(max_seq_len), _ptr(out),
                                    TK_F32 if out.dtype == torch.float32 else TK_BF16, scale,
                                    1 if causal else 0, _ptr(workspace),
                                    0 if workspace is None else workspace.numel(),
                                    _stream(stream)), "tk_attn_prefill_cached")
    return out


class PreparedCall:
    """Entry-point calls with their arguments checked and marshalled once.

    For serving loops whose buffers stay fixed between steps: calling the
    object re-issues the same C calls in order (same pointers, same stream)
    without the per-call Python checks, and raises TkError on a non-OK status.
    With graph=True (a non-default stream required) the calls are run once,
    then recorded once into a CUDA graph (tk_graph_begin / tk_graph_end), and
    each call of the object is one tk_graph_launch of that graph."""

    def __init__(self, name: str, args: tuple, keep: tuple, before: tuple = (), graph: bool = False,
                 stream=None):
        L = load_library()
        self._calls = tuple((getattr(L, n), n, a) for n, a in (*before, (name, args)))
        self._keep = keep  # the tensors whose pointers are in args stay alive
        self._graph = None
        if graph:
            if stream is None:
                raise ValueError("graph=True needs a non-default stream")
            self._stream = _stream(stream)
            self._run_calls()                     # first run: checks and set-up outside capture
            _check(L.tk_graph_begin(self._stream), "tk_graph_begin")
            try:
                self._run_calls()
            finally:
                g = ctypes.c_void_p()
                st = L.tk_graph_end(self._stream, ctypes.byref(g))
            _check(st, "tk_graph_end")
            self._graph = g
            self._launch = L.tk_graph_launch
            self._destroy = L.tk_graph_destroy

    def _run_calls(self):
        for fn, name, args in self._calls:
            st = fn(*args)
            if st != TK_OK:
                _check(st, name)

    def __call__(self):
        if self._graph is not None:
            st = self._launch(self._graph, self._stream)
            if st != TK_OK:
                _check(st, "tk_graph_launch")
            return
        self._run_calls()

    def __del__(self):
        g = getattr(self, "_graph", None)
        if g is not None and g.value:
            self._destroy(g)
            self._graph = None


def tk_copy_async(dst, src, stream=None):
    """Stream-ordered copy between device memory and page-locked host memory (same byte size)."""
    for t, n in ((dst, "dst"), (src, "src")):
        if not t.is_contiguous() or not (t.is_cuda or t.is_pinned()):
            raise ValueError(f"{n} must be contiguous, on a GPU or page-locked")
    nb = dst.numel() * dst.element_size()
    if src.numel() * src.element_size() != nb:
        raise ValueError("dst and src differ in size")
    _check(load_library().tk_copy_async(_ptr(dst), _ptr(src), nb, _stream(stream)), "tk_copy_async")
    return dst


def prepare_decode_append(cache: ThinKeyCache, q, k_new, v_new, seq_lens, max_seq_len: int, out,
                          workspace, scale: float | None = None, stream=None,
                          copy_in=None, graph: bool = False) -> PreparedCall:
    """tk_attn_decode_append with every argument checked once (see that function).

    copy_in = (dst, src): a device tensor and a page-locked host tensor of the
    same byte size, copied (tk_copy_async) before each decode -- e.g. the
    step's q, k_new and v_new packed in one host buffer.  `out` may be a
    page-locked host tensor: the kernel then writes the result there directly.
    graph=True records the step (copy and decode) as one CUDA graph launched
    per call; preparing it runs the step twice (once eagerly, once recorded:
    the recorded run does not execute), so the cache gets the new token once."""
    d = cache.desc
    dev = cache.k.device
    for t, n in ((q, "q"), (k_new, "k_new"), (v_new, "v_new")):
        _need(t, torch.bfloat16, n, dev)
    _need(seq_lens, torch.int32, "seq_lens", dev)
    _need(workspace, torch.uint8, "workspace", dev)
    _need_out(out, "out", dev)
    before = ()
    keep_in = ()
    if copy_in is not None:
        dst, src = copy_in
        if not dst.is_cuda or dst.device != dev or not dst.is_contiguous():
            raise ValueError("copy_in: dst must be a contiguous tensor on the cache's device")
        if src.is_cuda or not src.is_pinned() or not src.is_contiguous():
            raise ValueError("copy_in: src must be a contiguous page-locked host tensor")
        nb = dst.numel() * dst.element_size()
        if src.numel() * src.element_size() != nb:
            raise ValueError("copy_in: dst and src differ in size")
        before = (("tk_copy_async", (_ptr(dst), _ptr(src), ctypes.c_size_t(nb), _stream(stream))),)
        keep_in = (dst, src)
    if tuple(q.shape) != (d.batch, d.h_q, d.r) or tuple(out.shape) != (d.batch, d.h_q, d.d_v):
        raise ValueError(f"q {tuple(q.shape)} / out {tuple(out.shape)} do not match the cache")
    if tuple(k_new.shape) != (d.batch, d.h_kv, d.r) or tuple(v_new.shape) != (d.batch, d.h_kv, d.d_v):
        raise ValueError(f"k_new {tuple(k_new.shape)} / v_new {tuple(v_new.shape)} do not match the cache")
    scale = 1.0 / math.sqrt(d.r) if scale is None else float(scale)
    args = (ctypes.byref(d), _ptr(q), _ptr(cache.k), _ptr(cache.v), _ptr(cache.k_scale),
            _ptr(cache.page_table), _ptr(seq_lens), _ptr(k_new), _ptr(v_new), int(max_seq_len),
            _ptr(out), TK_F32 if out.dtype == torch.float32 else TK_BF16, ctypes.c_float(scale),
            _ptr(workspace), ctypes.c_size_t(workspace.numel()), _stream(stream))
    return PreparedCall("tk_attn_decode_append", args,
                        (cache, q, k_new, v_new, seq_lens, out, workspace) + keep_in, before,
                        graph=graph, stream=stream)


def tk_attn_prefill(q, k, v, out, scale: float | None = None, causal: bool = True, stream=None):
    """Prefill: q [B, H_q, S, r], k [B, H_kv, S, r], v [B, H_kv, S, d_v] bf16 -> out [B, H_q, S, d_v]."""
    dev = q.device
    for t, n in ((q, "q"), (k, "k"), (v, "v")):
        _need(t, torch.bfloat16, n, dev)
    if out.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError("out must be float32 or bfloat16")
    _need(out, out.dtype, "out", dev)
    B, hq, S, r = q.shape
    hkv, dv = k.shape[1], v.shape[3]
    if tuple(k.shape) != (B, hkv, S, r) or tuple(v.shape) != (B, hkv, S, dv) or \
            tuple(out.shape) != (B, hq, S, dv):
        raise ValueError("q / k / v / out shapes are inconsistent")
    scale = 1.0 / math.sqrt(r) if scale is None else float(scale)
    L = load_library()
    _check(L.tk_attn_prefill(_ptr(q), _ptr(k), _ptr(v), _ptr(out),
                             TK_F32 if out.dtype == torch.float32 else TK_BF16,
                             B, hq, hkv, S, r, dv, scale, 1 if causal else 0, _stream(stream)),
           "tk_attn_prefill")
    return out


def tk_attn_decode_noalloc(cache: ThinKeyCache, q, seq_lens, max_seq_len: int, out,
                           scale: float | None = None, stream=None):
    """tk_attn_decode without a workspace: uses the library's fixed device scratch.

    For callers that cannot allocate device memory.  Calls that may overlap on
    the GPU share the scratch and race; see include/tk.h.
    """
    d = cache.desc
    dev = cache.k.device
    _need(q, torch.bfloat16, "q", dev)
    _need(seq_lens, torch.int32, "seq_lens", dev)
    _need_out(out, "out", dev)
    if tuple(q.shape) != (d.batch, d.h_q, d.r) or tuple(out.shape) != (d.batch, d.h_q, d.d_v):
        raise ValueError(f"q {tuple(q.shape)} / out {tuple(out.shape)} do not match the cache")
    scale = 1.0 / math.sqrt(d.r) if scale is None else float(scale)
    L = load_library()
    _check(L.tk_attn_decode_noalloc(ctypes.byref(d), _ptr(q), _ptr(cache.k), _ptr(cache.v),
                                    _ptr(cache.k_scale), _ptr(cache.page_table), _ptr(seq_lens),
                                    int(max_seq_len), _ptr(out),
                                    TK_F32 if out.dtype == torch.float32 else TK_BF16, scale,
                                    _stream(stream)), "tk_attn_decode_noalloc")
    return out


def tk_check_wait_timeout(limit_us: int, stream=None):
    """Run the failure-detection diagnostic: a bounded wait that must run out
    after limit_us microseconds and record code 2 (see include/tk.h)."""
    _check(load_library().tk_check_wait_timeout(int(limit_us), _stream(stream)),
           "tk_check_wait_timeout")


def tk_get_device_error(stream=None) -> int:
    """Synchronise the stream and return (and clear) the device error word (0 = none)."""
    code = ctypes.c_int32(0)
    st = load_library().tk_get_device_error(ctypes.byref(code), _stream(stream))
    if st not in (TK_OK, TK_ERR_DEVICE):
        _check(st, "tk_get_device_error")
    return int(code.value)
