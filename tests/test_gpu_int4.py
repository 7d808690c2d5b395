"""int4 thin keys (two codes per byte, one fp32 scale per token) on the GPU.

The append must store exactly the oracle's packed codes and scales; decode
must match the fp64 oracle on the dequantised keys for every (r >= 32, d_v,
G), give identical bits for paged and contiguous caches, and the fused
append + decode must equal the two calls.  The full-size shape (B=64,
context 32768) at every r is in test_gpu_fullsize.py.
"""

import math

import numpy as np
import pytest
import torch

from _helpers import f64, parity, require_gpu
from oracle import attention as oa
from oracle import cache as oc
from paper_2603_04427_gb300 import binding as tb
from paper_2603_04427_gb300 import inputs

pytestmark = pytest.mark.gpu


def _filled(B, hq, hkv, r, dv, cap, seed, ps=0, lens=None):
    """A cache whose first cap (or lens[b]) tokens were written by tk_kv_append."""
    lens = lens or [cap] * B
    if ps:
        table, n_pages = inputs.paged_layout(lens, ps, seed=seed, extra_pages=2)
        cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, page_size=ps, num_pages=n_pages,
                                         page_table=table, k_int4=True)
    else:
        cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=cap, k_int4=True)
    kn = inputs.normal_bf16((B, hkv, cap, r), seed, device="cuda")
    vn = inputs.normal_bf16((B, hkv, cap, dv), seed + 1, device="cuda")
    if ps:
        for b, n in enumerate(lens):
            one = tb.ThinKeyCache(tb.tk_cache_desc(1, hq, hkv, r, dv, 0, ps, cache.desc.num_pages,
                                                   cache.desc.max_pages_per_seq, tb.TK_I4),
                                  cache.k, cache.v, cache.k_scale, cache.page_table[b:b + 1].contiguous())
            tb.tk_kv_append(one, kn[b:b + 1, :, :n].contiguous(), vn[b:b + 1, :, :n].contiguous(),
                            torch.zeros(1, dtype=torch.int32, device="cuda"))
    else:
        tb.tk_kv_append(cache, kn, vn, torch.zeros(B, dtype=torch.int32, device="cuda"))
    assert tb.tk_get_device_error() == 0
    return cache, kn, vn


@pytest.mark.parametrize("r", [32, 64, 128])
def test_int4_append_exact(r):
    require_gpu()
    B, hq, hkv, dv, cap = 3, 4, 2, 64, 80
    cache, kn, vn = _filled(B, hq, hkv, r, dv, cap, seed=100 + r)
    codes, sc = oc.quantize_int4_per_token(kn.float().cpu().numpy())
    assert np.array_equal(cache.k.cpu().numpy(), oc.pack_int4(codes))
    assert np.array_equal(cache.k_scale.cpu().numpy().view(np.uint32), sc.view(np.uint32))
    assert torch.equal(cache.v, vn)


def _oracle(cache, q, kn, lens, scale):
    codes, sc = oc.quantize_int4_per_token(kn.float().cpu().numpy())
    return oa.attention_decode(f64(q), codes, f64(cache.v), lens, scale, k_scale=sc)


def _run(cache, q, lens, max_len=None, out_dtype=torch.float32):
    B = q.shape[0]
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    max_len = max(lens) if max_len is None else max_len
    out = torch.full((B, cache.desc.h_q, cache.desc.d_v), float("nan"), dtype=out_dtype, device="cuda")
    tb.tk_attn_decode(cache, q, sl, max_len, out, tb.decode_workspace(cache.desc, max_len))
    assert tb.tk_get_device_error() == 0
    return out


@pytest.mark.parametrize("G", [1, 2, 4, 8])
@pytest.mark.parametrize("r,dv", [(32, 128), (64, 64), (128, 128), (32, 64)])
def test_int4_decode_matches_oracle(G, r, dv):
    require_gpu()
    B, hkv = 4, 2
    hq = G * hkv
    lens = [777, 1, 0, 64]
    cache, kn, _ = _filled(B, hq, hkv, r, dv, 784, seed=200 + r + G)
    q = inputs.normal_bf16((B, hq, r), seed=7, device="cuda")
    out = _run(cache, q, lens)
    parity(f64(out), _oracle(cache, q, kn, lens, 1 / math.sqrt(r)), what=f"int4 r={r} dv={dv} G={G}")
    assert torch.all(out[2] == 0)


@pytest.mark.parametrize("ps", [16, 64, 256])
def test_int4_paged_equals_contiguous_bitwise(ps):
    require_gpu()
    B, hq, hkv, r, dv = 3, 8, 2, 32, 128
    lens = [1000, 333, 65]
    cont, kn, vn = _filled(B, hq, hkv, r, dv, 1024, seed=31)
    paged, _, _ = _filled(B, hq, hkv, r, dv, 1024, seed=31, ps=ps, lens=lens)
    q = inputs.normal_bf16((B, hq, r), seed=9, device="cuda")
    a = _run(cont, q, lens)
    p = _run(paged, q, lens)
    assert torch.equal(a, p)
    parity(f64(p), _oracle(cont, q, kn, lens, 1 / math.sqrt(r)), what=f"int4 paged ps={ps}")


def test_int4_fused_append_decode_equals_two_calls():
    require_gpu()
    B, hq, hkv, r, dv = 4, 32, 8, 32, 128
    lens = [0, 63, 64, 700]
    cap = 704
    a, _, _ = _filled(B, hq, hkv, r, dv, cap, seed=41)
    f = tb.ThinKeyCache(a.desc, a.k.clone(), a.v.clone(), a.k_scale.clone(), None)
    q = inputs.normal_bf16((B, hq, r), seed=42, device="cuda")
    k1 = inputs.normal_bf16((B, hkv, r), seed=43, device="cuda")
    v1 = inputs.normal_bf16((B, hkv, dv), seed=44, device="cuda")
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    L = max(lens) + 1
    out_a = torch.empty(B, hq, dv, device="cuda")
    out_f = torch.empty(B, hq, dv, device="cuda")
    tb.tk_kv_append(a, k1[:, :, None].contiguous(), v1[:, :, None].contiguous(), sl)
    tb.tk_attn_decode(a, q, sl + 1, L, out_a, tb.decode_workspace(a.desc, L))
    tb.tk_attn_decode_append(f, q, k1, v1, sl, L, out_f, tb.decode_workspace(f.desc, L))
    assert tb.tk_get_device_error() == 0
    assert torch.equal(out_a, out_f)
    assert torch.equal(a.k, f.k) and torch.equal(a.k_scale, f.k_scale) and torch.equal(a.v, f.v)
