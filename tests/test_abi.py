"""The C-ABI library builds, loads and exports every symbol include/tk.h declares.

Also checks the host-side argument validation, which returns before any
CUDA call and therefore runs without a GPU.
"""

import ctypes
import os
import re

import pytest

from paper_2603_04427_gb300 import binding as tb
from paper_2603_04427_gb300 import build as tbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    tbuild.build()
    return tb.load_library()


def _declared():
    src = open(os.path.join(ROOT, "include", "tk.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tk_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("tk_kv_append", "tk_attn_prefill", "tk_attn_decode", "tk_decode_workspace_size"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for name in _declared():
        assert hasattr(lib, name), name
    assert set(_declared()) == set(tb.EXPORTED)


def test_abi_version_and_status_strings(lib):
    assert tb.tk_abi_version() == 4
    assert tb.tk_status_string(tb.TK_OK) == "TK_OK"
    assert tb.tk_status_string(tb.TK_ERR_WORKSPACE) == "TK_ERR_WORKSPACE"
    assert tb.tk_status_string(99) == "TK_ERR_UNKNOWN"


def _desc(**kw):
    d = dict(batch=2, h_q=8, h_kv=2, r=32, d_v=128, capacity=256, page_size=0, num_pages=0,
             max_pages_per_seq=0, k_dtype=tb.TK_BF16)
    d.update(kw)
    return tb.tk_cache_desc(**d)


FAKE = ctypes.c_void_p(0x10000)  # never dereferenced: validation fails first


@pytest.mark.parametrize("kw,status,msg", [
    (dict(h_q=6, h_kv=4), tb.TK_ERR_INVALID_ARG, "multiple"),
    (dict(h_q=32, h_kv=2), tb.TK_ERR_UNSUPPORTED, "h_q/h_kv"),
    (dict(r=48), tb.TK_ERR_UNSUPPORTED, "r=48"),
    (dict(d_v=96), tb.TK_ERR_UNSUPPORTED, "d_v=96"),
    (dict(capacity=100), tb.TK_ERR_INVALID_ARG, "capacity"),
    (dict(page_size=48, num_pages=4, max_pages_per_seq=2), tb.TK_ERR_UNSUPPORTED, "page_size"),
    (dict(page_size=64, num_pages=0, max_pages_per_seq=2), tb.TK_ERR_INVALID_ARG, "num_pages"),
    (dict(k_dtype=7), tb.TK_ERR_UNSUPPORTED, "k_dtype"),
    (dict(k_dtype=tb.TK_I4, r=16), tb.TK_ERR_UNSUPPORTED, "TK_I4"),
])
def test_descriptor_validation(lib, kw, status, msg):
    d = _desc(**kw)
    st = lib.tk_kv_append(ctypes.byref(d), FAKE, FAKE, None, None, FAKE, FAKE, FAKE, 1, None)
    assert st == status
    assert msg in tb.tk_last_error()
    st = lib.tk_attn_decode(ctypes.byref(d), FAKE, FAKE, FAKE, None, None, FAKE, 16, FAKE,
                            tb.TK_F32, 0.1, FAKE, 1 << 20, None)
    assert st == status
    st = lib.tk_attn_decode_append(ctypes.byref(d), FAKE, FAKE, FAKE, None, None, FAKE, FAKE,
                                   FAKE, 16, FAKE, tb.TK_F32, 0.1, FAKE, 1 << 20, None)
    assert st == status
    assert lib.tk_decode_workspace_size(ctypes.byref(d), 16) == 0


def test_pointer_and_option_validation(lib):
    d = _desc()
    mis = ctypes.c_void_p(0x10008)
    assert lib.tk_kv_append(ctypes.byref(d), mis, FAKE, None, None, FAKE, FAKE, FAKE, 1,
                            None) == tb.TK_ERR_INVALID_ARG
    assert "aligned" in tb.tk_last_error()
    d8 = _desc(k_dtype=tb.TK_I8)
    assert lib.tk_kv_append(ctypes.byref(d8), FAKE, FAKE, None, None, FAKE, FAKE, FAKE, 1,
                            None) == tb.TK_ERR_INVALID_ARG
    assert "k_scale" in tb.tk_last_error()
    dp = _desc(page_size=64, num_pages=8, max_pages_per_seq=4, capacity=0)
    assert lib.tk_kv_append(ctypes.byref(dp), FAKE, FAKE, None, None, FAKE, FAKE, FAKE, 1,
                            None) == tb.TK_ERR_INVALID_ARG
    assert "page_table" in tb.tk_last_error()
    assert lib.tk_kv_append(ctypes.byref(d), FAKE, FAKE, None, None, FAKE, FAKE, FAKE, -1,
                            None) == tb.TK_ERR_INVALID_ARG
    # zero new tokens and an empty batch are no-ops (no CUDA call is made)
    assert lib.tk_kv_append(ctypes.byref(d), None, None, None, None, None, None, None, 0,
                            None) == tb.TK_OK
    assert lib.tk_attn_decode(ctypes.byref(d), FAKE, FAKE, FAKE, None, None, FAKE, 16, FAKE,
                              5, 0.1, FAKE, 1 << 20, None) == tb.TK_ERR_UNSUPPORTED
    assert lib.tk_attn_decode(ctypes.byref(d), FAKE, FAKE, FAKE, None, None, FAKE, -1, FAKE,
                              tb.TK_F32, 0.1, FAKE, 1 << 20, None) == tb.TK_ERR_INVALID_ARG
    assert lib.tk_attn_decode(ctypes.byref(d), FAKE, FAKE, FAKE, None, None, FAKE, 16, FAKE,
                              tb.TK_F32, float("nan"), FAKE, 1 << 20, None) == tb.TK_ERR_INVALID_ARG


def test_decode_append_validation(lib):
    d = _desc()
    mis = ctypes.c_void_p(0x10008)
    A = lib.tk_attn_decode_append
    assert A(ctypes.byref(d), FAKE, FAKE, FAKE, None, None, FAKE, None, FAKE, 16, FAKE,
             tb.TK_F32, 0.1, FAKE, 1 << 20, None) == tb.TK_ERR_INVALID_ARG
    assert "k_new" in tb.tk_last_error()
    assert A(ctypes.byref(d), FAKE, FAKE, FAKE, None, None, FAKE, FAKE, mis, 16, FAKE,
             tb.TK_F32, 0.1, FAKE, 1 << 20, None) == tb.TK_ERR_INVALID_ARG
    assert "aligned" in tb.tk_last_error()
    d8 = _desc(k_dtype=tb.TK_I8)
    assert A(ctypes.byref(d8), FAKE, FAKE, FAKE, None, None, FAKE, FAKE, FAKE, 16, FAKE,
             tb.TK_F32, 0.1, FAKE, 1 << 20, None) == tb.TK_ERR_INVALID_ARG
    assert "k_scale" in tb.tk_last_error()


def test_prefill_cached_validation(lib):
    P = lib.tk_attn_prefill_cached
    d = _desc()
    d8 = _desc(k_dtype=tb.TK_I8)
    # int8 keys need their scales
    assert P(ctypes.byref(d8), FAKE, FAKE, FAKE, None, None, FAKE, FAKE, FAKE, 64, 256, FAKE,
             tb.TK_BF16, 0.1, 1, None, 0, None) == tb.TK_ERR_INVALID_ARG
    assert "k_scale" in tb.tk_last_error()
    assert P(ctypes.byref(d), FAKE, FAKE, FAKE, None, None, FAKE, FAKE, FAKE, 64, 32, FAKE,
             tb.TK_BF16, 0.1, 1, None, 0, None) == tb.TK_ERR_INVALID_ARG      # max_seq_len < seq
    assert P(ctypes.byref(d), None, FAKE, FAKE, None, None, FAKE, FAKE, FAKE, 64, 256, FAKE,
             tb.TK_BF16, 0.1, 1, None, 0, None) == tb.TK_ERR_INVALID_ARG      # q is NULL
    assert P(ctypes.byref(d), FAKE, FAKE, FAKE, None, None, FAKE, FAKE, FAKE, 64, 256, FAKE,
             tb.TK_BF16, -1.0, 1, None, 0, None) == tb.TK_ERR_INVALID_ARG     # scale <= 0
    assert P(ctypes.byref(d), None, None, None, None, None, None, None, None, 0, 0, None,
             tb.TK_BF16, 0.1, 1, None, 0, None) == tb.TK_OK                    # empty chunk: no-op
    # int8 keys need a workspace: NULL, misaligned or too small is rejected
    # before anything is launched
    need = lib.tk_prefill_cached_workspace_size(ctypes.byref(d8), 256)
    assert need > 0
    args = (ctypes.byref(d8), FAKE, FAKE, FAKE, FAKE, None, FAKE, FAKE, FAKE, 64, 256, FAKE,
            tb.TK_BF16, 0.1, 1)
    assert P(*args, None, need, None) == tb.TK_ERR_WORKSPACE
    assert P(*args, ctypes.c_void_p(0x10010), need, None) == tb.TK_ERR_WORKSPACE
    assert P(*args, FAKE, need - 1, None) == tb.TK_ERR_WORKSPACE
    assert "needed" in tb.tk_last_error()


@pytest.mark.parametrize("r,k_dtype,two_planes", [
    (32, tb.TK_I8, True), (32, tb.TK_I4, True), (64, tb.TK_I8, True), (128, tb.TK_I8, False),
    (128, tb.TK_I4, False), (16, tb.TK_I8, True)])
def test_prefill_cached_workspace_size(lib, r, k_dtype, two_planes):
    """Widened keys: hi and lo bf16 planes of r per token and kv head (r <= 64), or one
    bf16 plane and an fp32 scale (r = 128), over min(max_seq_len, cache tokens) rows
    rounded up to 4; nothing for bf16 keys, int4 keys with r < 32 or a bad descriptor."""
    size = lib.tk_prefill_cached_workspace_size
    d = _desc(r=r, k_dtype=k_dtype)                 # batch 2, h_kv 2, capacity 256
    for max_len, rows in ((100, 100), (101, 104), (1000, 256)):
        per_row = 4 * r if two_planes else 2 * r + 4
        assert size(ctypes.byref(d), max_len) == 2 * 2 * rows * per_row
    assert size(ctypes.byref(_desc(r=r)), 100) == 0                       # bf16 keys
    assert size(ctypes.byref(_desc(r=16, k_dtype=tb.TK_I4)), 100) == 0    # int4 needs r >= 32
    assert size(ctypes.byref(_desc(r=24, k_dtype=tb.TK_I8)), 100) == 0    # invalid descriptor
    assert size(ctypes.byref(d), 0) == 0
    paged = _desc(r=r, k_dtype=k_dtype, capacity=0, page_size=16, num_pages=64, max_pages_per_seq=8)
    per_row = 4 * r if two_planes else 2 * r + 4
    assert size(ctypes.byref(paged), 1000) == 2 * 2 * 128 * per_row      # 8 pages of 16 tokens


def test_forward_and_backward_validation(lib):
    F = lib.tk_attn_forward
    assert F(FAKE, FAKE, FAKE, FAKE, None, tb.TK_BF16, 2, 4, 4, 128, 32, 128, 0.1, 1,
             None) == tb.TK_ERR_INVALID_ARG                 # lse is NULL
    assert lib.tk_backward_workspace_size(2, 4, 100) >= 2 * 4 * 100 * 4
    assert lib.tk_backward_workspace_size(-1, 4, 100) == 0
    Bw = lib.tk_attn_backward
    base = [FAKE] * 10
    assert Bw(*base, 1 << 20, 2, 4, 4, 128, 24, 128, 0.1, 1, None) == tb.TK_ERR_UNSUPPORTED
    assert Bw(*base, 1 << 20, 2, 6, 4, 128, 32, 128, 0.1, 1, None) == tb.TK_ERR_INVALID_ARG
    assert Bw(*base, 1 << 20, 2, 4, 4, 128, 32, 128, 0.0, 1, None) == tb.TK_ERR_INVALID_ARG
    ws_small = [FAKE] * 9 + [ctypes.c_void_p(0x10000)]
    assert Bw(*ws_small, 16, 2, 4, 4, 128, 32, 128, 0.1, 1, None) == tb.TK_ERR_WORKSPACE
    nulls = [FAKE] * 5 + [None] + [FAKE] * 4
    assert Bw(*nulls, 1 << 20, 2, 4, 4, 128, 32, 128, 0.1, 1, None) == tb.TK_ERR_INVALID_ARG


def test_prefill_validation(lib):
    P = lib.tk_attn_prefill
    assert P(FAKE, FAKE, FAKE, FAKE, tb.TK_BF16, 2, 6, 4, 128, 32, 128, 0.1, 1, None) == tb.TK_ERR_INVALID_ARG
    assert P(FAKE, FAKE, FAKE, FAKE, tb.TK_BF16, 2, 4, 4, 128, 24, 128, 0.1, 1, None) == tb.TK_ERR_UNSUPPORTED
    assert P(FAKE, FAKE, FAKE, FAKE, tb.TK_BF16, 2, 4, 4, 128, 32, 80, 0.1, 1, None) == tb.TK_ERR_UNSUPPORTED
    assert P(FAKE, FAKE, FAKE, FAKE, tb.TK_I8, 2, 4, 4, 128, 32, 128, 0.1, 1, None) == tb.TK_ERR_UNSUPPORTED
    assert P(FAKE, FAKE, FAKE, FAKE, tb.TK_BF16, 2, 4, 4, -1, 32, 128, 0.1, 1, None) == tb.TK_ERR_INVALID_ARG
    assert P(None, None, None, None, tb.TK_BF16, 2, 4, 4, 0, 32, 128, 0.1, 1, None) == tb.TK_OK
    assert P(None, FAKE, FAKE, FAKE, tb.TK_BF16, 2, 4, 4, 64, 32, 128, 0.1, 1, None) == tb.TK_ERR_INVALID_ARG


def test_copy_async_validation(lib):
    """tk_copy_async: an empty copy is a no-op and NULL pointers are rejected, before any CUDA call."""
    assert lib.tk_copy_async(None, None, 0, None) == tb.TK_OK
    assert lib.tk_copy_async(None, FAKE, 16, None) == tb.TK_ERR_INVALID_ARG
    assert lib.tk_copy_async(FAKE, None, 16, None) == tb.TK_ERR_INVALID_ARG


def test_host_output_needs_page_locked_memory():
    """The binding accepts a host output only when it is page-locked (the kernel writes it zero-copy)."""
    import torch
    with pytest.raises(ValueError):
        tb._need_out(torch.empty(4, 8), "out", None)          # pageable host memory
    with pytest.raises(TypeError):
        tb._need_out(torch.empty(4, 8, dtype=torch.float16), "out", None)


def test_wait_timeout_check_validation(lib):
    """tk_check_wait_timeout rejects a limit outside 1 us .. 1 s before any CUDA call."""
    assert lib.tk_check_wait_timeout(0, None) == tb.TK_ERR_INVALID_ARG
    assert "limit_us" in tb.tk_last_error()
    assert lib.tk_check_wait_timeout(1000001, None) == tb.TK_ERR_INVALID_ARG


def test_graph_entry_points_validate_before_cuda(lib):
    """tk_graph_*: NULL streams / graphs are rejected before any CUDA call."""
    g = ctypes.c_void_p()
    assert lib.tk_graph_begin(None) == tb.TK_ERR_INVALID_ARG
    assert lib.tk_graph_end(None, ctypes.byref(g)) == tb.TK_ERR_INVALID_ARG
    assert lib.tk_graph_end(FAKE, None) == tb.TK_ERR_INVALID_ARG
    assert lib.tk_graph_launch(None, None) == tb.TK_ERR_INVALID_ARG
    assert lib.tk_graph_destroy(None) == tb.TK_ERR_INVALID_ARG

