"""tk_attn_prefill (tcgen05 / TMEM / TMA) on the GPU against the fp64 oracle.

Small cases span several 128-row tiles with ragged tails, every compiled
(r, d_v), GQA and MHA, causal and full attention, fp32 and bf16 output.
A crafted case makes the running max grow by more than the lazy-rescale
threshold from tile to tile so the O / l rescale path runs.  The
GPT-2-small-shaped prefill is checked in full here; the 7B MHA prefill is in
test_gpu_fullsize.py.
"""

import math

import numpy as np
import pytest
import torch

from _helpers import f64, parity, parity_bf16, require_gpu
from oracle import attention as oa
from paper_2603_04427_gb300 import binding as tb
from paper_2603_04427_gb300 import inputs

pytestmark = pytest.mark.gpu


def _qkv(B, hq, hkv, S, r, dv, seed):
    return (inputs.normal_bf16((B, hq, S, r), seed, device="cuda"),
            inputs.normal_bf16((B, hkv, S, r), seed + 1, device="cuda"),
            inputs.normal_bf16((B, hkv, S, dv), seed + 2, device="cuda"))


def _prefill(q, k, v, dtype=torch.float32, causal=True, scale=None):
    B, hq, S, _ = q.shape
    out = torch.full((B, hq, S, v.shape[3]), float("nan"), dtype=dtype, device="cuda")
    tb.tk_attn_prefill(q, k, v, out, scale=scale, causal=causal)
    assert tb.tk_get_device_error() == 0
    return out


@pytest.mark.parametrize("r,dv", [(16, 64), (32, 128), (64, 64), (128, 128), (32, 64), (16, 128)])
@pytest.mark.parametrize("causal", [True, False])
def test_prefill_small_matches_oracle(r, dv, causal):
    require_gpu()
    B, hq, hkv, S = 2, 4, 2, 300
    q, k, v = _qkv(B, hq, hkv, S, r, dv, seed=10 + r + dv)
    out = _prefill(q, k, v, causal=causal)
    ref = oa.attention_prefill(f64(q), f64(k), f64(v), 1 / math.sqrt(r), causal=causal)
    parity(f64(out), ref, what=f"prefill r={r} dv={dv} causal={causal}")


@pytest.mark.parametrize("S", [1, 7, 128, 129, 256, 513])
def test_prefill_lengths_and_bf16_output(S):
    require_gpu()
    B, hq, hkv, r, dv = 1, 8, 8, 32, 128
    q, k, v = _qkv(B, hq, hkv, S, r, dv, seed=S)
    out = _prefill(q, k, v, dtype=torch.bfloat16)
    ref = oa.attention_prefill(f64(q), f64(k), f64(v), 1 / math.sqrt(r))
    parity_bf16(f64(out), ref, what=f"prefill S={S} bf16 out")
    # causal row 0 is v[0] (a single visible key)
    assert torch.equal(out[:, :, 0], v[:, :, 0])


def test_prefill_gqa_groups_of_8():
    require_gpu()
    B, hq, hkv, S, r, dv = 2, 16, 2, 200, 64, 128
    q, k, v = _qkv(B, hq, hkv, S, r, dv, seed=5)
    out = _prefill(q, k, v)
    parity(f64(out), oa.attention_prefill(f64(q), f64(k), f64(v), 1 / math.sqrt(r)), what="gqa8")


def test_prefill_rescale_path():
    """Logits that grow along the sequence force the running max up every tile."""
    require_gpu()
    B, hq, hkv, S, r, dv = 1, 2, 2, 640, 32, 64
    q, k, v = _qkv(B, hq, hkv, S, r, dv, seed=9)
    q = torch.ones_like(q)
    grow = (torch.arange(S, device="cuda", dtype=torch.float32) / 16.0)[None, None, :, None]
    k = (k.float().abs() * 0.1 + grow).to(torch.bfloat16)   # q.k grows by ~2 per 16 keys
    out = _prefill(q, k, v)
    ref = oa.attention_prefill(f64(q), f64(k), f64(v), 1 / math.sqrt(r))
    parity(f64(out), ref, what="rescale path")


def test_prefill_explicit_scale_and_determinism():
    require_gpu()
    B, hq, hkv, S, r, dv = 1, 4, 4, 384, 16, 64
    q, k, v = _qkv(B, hq, hkv, S, r, dv, seed=3)
    a = _prefill(q, k, v, scale=0.11)
    b = _prefill(q, k, v, scale=0.11)
    assert torch.equal(a, b)
    parity(f64(a), oa.attention_prefill(f64(q), f64(k), f64(v), 0.11), what="scale 0.11")


def test_prefill_row_equals_decode_with_prefix():
    """Row i of causal prefill matches decode over the first i+1 keys."""
    require_gpu()
    B, hq, hkv, S, r, dv = 2, 8, 2, 300, 32, 128
    q, k, v = _qkv(B, hq, hkv, S, r, dv, seed=21)
    pre = _prefill(q, k, v)
    cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=304)
    tb.tk_kv_append(cache, k, v, torch.zeros(B, dtype=torch.int32, device="cuda"))
    for i in (0, 127, 128, 299):
        out = torch.empty(B, hq, dv, device="cuda")
        sl = torch.full((B,), i + 1, dtype=torch.int32, device="cuda")
        tb.tk_attn_decode(cache, q[:, :, i].contiguous(), sl, i + 1, out,
                          tb.decode_workspace(cache.desc, i + 1))
        parity(f64(pre[:, :, i]), f64(out), what=f"row {i}")


def test_gpt2_small_prefill_full():
    """B=1, 12 heads, r=16, d_v=64, S=256, fp32 output: all outputs."""
    require_gpu()
    q, k, v = _qkv(1, 12, 12, 256, 16, 64, seed=1000)
    out = _prefill(q, k, v)
    parity(f64(out), oa.attention_prefill(f64(q), f64(k), f64(v), 0.25), what="gpt2 prefill")
