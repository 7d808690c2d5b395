"""tk_attn_decode_noalloc: the decode entry point for callers that cannot allocate.

Such callers (a runtime whose device memory is all held by its own pool, a
plugin host that only hands over inputs and outputs, a real-time loop that
must not call the allocator between steps) get the split partials and
counters from a fixed scratch array inside the library instead of a
workspace argument.  These tests call it through the C ABI and compare its
output with the regular workspace entry point's, within the parity bar the
other decode tests use, on two calls in a row (the second call finds the
scratch as the first one left it).  This file sorts last so that a run
stopping at the first failure has already run every other test.
"""

import ctypes
import math

import pytest
import torch

from _helpers import f64, parity, require_gpu
from paper_2603_04427_gb300 import binding as tb
from paper_2603_04427_gb300 import inputs

pytestmark = pytest.mark.gpu


def _cache(B, hq, hkv, r, dv, lens, k_int8, seed):
    cap = (max(lens) + 15) // 16 * 16
    cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=cap, k_int8=k_int8)
    kn = inputs.normal_bf16((B, hkv, cap, r), seed, device="cuda")
    vn = inputs.normal_bf16((B, hkv, cap, dv), seed + 1, device="cuda")
    tb.tk_kv_append(cache, kn, vn, torch.zeros(B, dtype=torch.int32, device="cuda"))
    return cache


SHAPES = {
    # Mistral-7B-shaped GQA decode, every context 4096
    "mistral": dict(B=16, hq=32, hkv=8, r=32, dv=128, lens=[4096] * 16, k_int8=False),
    # ragged contexts, int8 keys, including an empty and a one-token context
    "ragged_int8": dict(B=4, hq=16, hkv=4, r=64, dv=64, lens=[3000, 0, 1, 1234], k_int8=True),
}


def _case(name, seed):
    s = SHAPES[name]
    cache = _cache(s["B"], s["hq"], s["hkv"], s["r"], s["dv"], s["lens"], s["k_int8"], seed=seed)
    q = inputs.normal_bf16((s["B"], s["hq"], s["r"]), seed + 1, device="cuda")
    sl = torch.tensor(s["lens"], dtype=torch.int32, device="cuda")
    L = max(s["lens"])
    assert tb.tk_decode_workspace_size(cache.desc, L) <= 8 << 20
    # the regular entry point, with a workspace of its own, zero-filled
    ref = torch.empty(s["B"], s["hq"], s["dv"], device="cuda")
    tb.tk_attn_decode(cache, q, sl, L, ref, tb.decode_workspace(cache.desc, L))
    return cache, q, sl, L, ref


@pytest.mark.parametrize("name", sorted(SHAPES))
def test_noalloc_matches_workspace_decode_twice(name):
    require_gpu()
    cache, q, sl, L, ref = _case(name, seed=77)
    for _ in range(2):
        out = torch.full_like(ref, float("nan"))
        tb.tk_attn_decode_noalloc(cache, q, sl, L, out)
        assert tb.tk_get_device_error() == 0
        parity(f64(out), f64(ref), what="noalloc vs workspace decode")
        assert torch.equal(out, ref)  # same kernel and split plan: identical bits


def test_noalloc_alternating_shapes():
    """Calls of different shapes in a row: each finds the scratch as a call of
    the other shape (another batch x h_kv, other partial records) left it."""
    require_gpu()
    cases = {n: _case(n, seed=91 + 10 * i) for i, n in enumerate(("mistral", "ragged_int8"))}
    for name in ("mistral", "ragged_int8", "mistral", "ragged_int8"):
        cache, q, sl, L, ref = cases[name]
        out = torch.full_like(ref, float("nan"))
        tb.tk_attn_decode_noalloc(cache, q, sl, L, out)
        assert tb.tk_get_device_error() == 0
        parity(f64(out), f64(ref), what=f"noalloc {name} after another shape")
        assert torch.equal(out, ref)


def test_noalloc_rejects_shapes_beyond_its_scratch():
    require_gpu()
    # 1024 sequences x 4096 kv heads need 16 MiB of arrival counters alone,
    # more than the 8 MiB scratch.
    d = tb.tk_cache_desc(1024, 4096, 4096, 32, 128, 8192, 0, 0, 0, tb.TK_BF16)
    assert tb.tk_decode_workspace_size(d, 8192) > 8 << 20
    fake = torch.empty(16, dtype=torch.uint8, device="cuda")
    L = tb.load_library()
    p = fake.data_ptr()
    st = L.tk_attn_decode_noalloc(ctypes.byref(d), p, p, p, None, None, p, 8192, p, tb.TK_F32,
                                  1 / math.sqrt(32), None)
    assert st == tb.TK_ERR_WORKSPACE
    assert "needed" in tb.tk_last_error()
