"""Failure detection on the GPU, without a fault.

Every wait in the library's kernels is bounded: when a phase does not
complete in time the wait records code 2 in the device error word and the
kernel returns.  tk_check_wait_timeout makes one such wait run out on a
barrier that nothing arrives at (a limit of a few milliseconds instead of
the kernels' 1 s); the host then reads code 2, and the device keeps
answering: the next decode still matches the oracle.  The bad-index path
(code 1) is covered in test_gpu_decode.py and test_gpu_append.py.
"""

import math
import time

import pytest
import torch

from _helpers import f64, parity, require_gpu
from oracle import attention as oa
from paper_2603_04427_gb300 import binding as tb
from paper_2603_04427_gb300 import inputs

pytestmark = pytest.mark.gpu


def _small_decode_parity():
    B, hq, hkv, r, dv, L = 2, 8, 2, 32, 128, 300
    cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=304)
    kn = inputs.normal_bf16((B, hkv, 304, r), 501, device="cuda")
    vn = inputs.normal_bf16((B, hkv, 304, dv), 502, device="cuda")
    tb.tk_kv_append(cache, kn, vn, torch.zeros(B, dtype=torch.int32, device="cuda"))
    q = inputs.normal_bf16((B, hq, r), 503, device="cuda")
    out = torch.empty(B, hq, dv, device="cuda")
    sl = torch.full((B,), L, dtype=torch.int32, device="cuda")
    tb.tk_attn_decode(cache, q, sl, L, out, tb.decode_workspace(cache.desc, L))
    assert tb.tk_get_device_error() == 0
    parity(f64(out), oa.attention_decode(f64(q), f64(cache.k), f64(cache.v), [L] * B,
                                         1 / math.sqrt(r)), what="decode after a timed-out wait")


@pytest.mark.parametrize("limit_us", [50, 3000])
def test_bounded_wait_runs_out_and_records_code_2(limit_us):
    require_gpu()
    assert tb.tk_get_device_error() == 0
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    tb.tk_check_wait_timeout(limit_us)
    code = tb.tk_get_device_error()        # synchronises the stream
    elapsed = time.perf_counter() - t0
    assert code == 2
    assert elapsed >= limit_us * 1e-6      # the wait did last its limit
    assert elapsed < 5.0                   # and then gave up
    assert tb.tk_get_device_error() == 0   # reading the word cleared it
    _small_decode_parity()                 # the context is still usable
