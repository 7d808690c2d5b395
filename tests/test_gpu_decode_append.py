"""tk_attn_decode_append (the append fused into the decode launch) on the GPU.

The fused call must equal tk_kv_append of one token followed by
tk_attn_decode over the grown context, bit for bit: the outputs and every
byte of the cache (keys or int8 codes, key scales, values).  Cases cover
contiguous and paged caches (pages smaller than, equal to and larger than
the 64-token chunk), bf16 and int8 keys, every (r, d_v), G = 1 and 8, and new
positions at 0, at a chunk start, at a chunk end and mid-chunk.  The fused
result is also compared with the fp64 oracle, and a sequence whose new token
does not fit gets no write and flags the device error word.
"""

import dataclasses
import math

import pytest
import torch

from _helpers import f64, parity, require_gpu
from oracle import attention as oa
from oracle import cache as oc
from paper_2603_04427_gb300 import binding as tb
from paper_2603_04427_gb300 import inputs

pytestmark = pytest.mark.gpu


def _clone(cache):
    return dataclasses.replace(
        cache, k=cache.k.clone(), v=cache.v.clone(),
        k_scale=None if cache.k_scale is None else cache.k_scale.clone())


def _make(B, hq, hkv, r, dv, lens, k_int8, ps, seed, cap=None):
    """A cache holding lens[b] random tokens per sequence, written by tk_kv_append."""
    cap = cap or (max(lens) + 1 + 15) // 16 * 16
    if ps:
        table, n_pages = inputs.paged_layout([n + 1 for n in lens], ps, seed=seed, extra_pages=2)
        cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, page_size=ps, num_pages=n_pages,
                                         page_table=table, k_int8=k_int8)
    else:
        cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=cap, k_int8=k_int8)
    T = max(lens)
    kn = inputs.normal_bf16((B, hkv, T, r), seed, device="cuda")
    vn = inputs.normal_bf16((B, hkv, T, dv), seed + 1, device="cuda")
    zero = torch.zeros(B, dtype=torch.int32, device="cuda")
    if T:
        # only the first lens[b] tokens of each sequence are part of its context;
        # the rest of the block is overwritten by the new token or never read
        if ps:
            for b, n in enumerate(lens):
                if n:
                    one = _clone_desc(cache, b)
                    tb.tk_kv_append(one, kn[b:b + 1, :, :n].contiguous(), vn[b:b + 1, :, :n].contiguous(),
                                    zero[:1])
        else:
            tb.tk_kv_append(cache, kn, vn, zero)
    return cache, kn, vn


def _clone_desc(cache, b):
    """A one-sequence view of a paged cache (same pools, page-table row b)."""
    d = cache.desc
    desc = tb.tk_cache_desc(1, d.h_q, d.h_kv, d.r, d.d_v, d.capacity, d.page_size, d.num_pages,
                            d.max_pages_per_seq, d.k_dtype)
    return dataclasses.replace(cache, desc=desc, page_table=cache.page_table[b:b + 1].contiguous())


def _both(cache, q, k1, v1, lens, out_dtype=torch.float32):
    """(two-call result, fused result): outputs and caches."""
    B = q.shape[0]
    d = cache.desc
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    sl1 = sl + 1
    L = max(lens) + 1
    a, f = _clone(cache), _clone(cache)
    out_a = torch.full((B, d.h_q, d.d_v), float("nan"), dtype=out_dtype, device="cuda")
    out_f = out_a.clone()
    tb.tk_kv_append(a, k1[:, :, None].contiguous(), v1[:, :, None].contiguous(), sl)
    tb.tk_attn_decode(a, q, sl1, L, out_a, tb.decode_workspace(d, L))
    ws = tb.decode_workspace(d, L)
    tb.tk_attn_decode_append(f, q, k1, v1, sl, L, out_f, ws)
    assert tb.tk_get_device_error() == 0
    assert int(ws[:4 * B * d.h_kv].view(torch.int32).abs().sum()) == 0
    return (a, out_a), (f, out_f)


def _same_cache(a, f):
    assert torch.equal(a.k, f.k)
    assert torch.equal(a.v, f.v)
    if a.k_scale is not None:
        assert torch.equal(a.k_scale, f.k_scale)


@pytest.mark.parametrize("k_int8", [False, True])
@pytest.mark.parametrize("ps", [0, 16, 64, 128])
def test_fused_equals_append_then_decode(k_int8, ps):
    require_gpu()
    B, hq, hkv, r, dv = 6, 16, 4, 32, 128
    lens = [0, 63, 64, 127, 200, 1000]   # new token at 0, chunk end, chunk start, ...
    cache, _, _ = _make(B, hq, hkv, r, dv, lens, k_int8, ps, seed=11 + ps)
    q = inputs.normal_bf16((B, hq, r), seed=12, device="cuda")
    k1 = inputs.normal_bf16((B, hkv, r), seed=13, device="cuda")
    v1 = inputs.normal_bf16((B, hkv, dv), seed=14, device="cuda")
    (a, oa_), (f, of_) = _both(cache, q, k1, v1, lens)
    assert torch.equal(oa_, of_)
    _same_cache(a, f)


@pytest.mark.parametrize("r,dv,G", [(16, 64, 1), (64, 64, 8), (128, 128, 8), (128, 64, 2)])
@pytest.mark.parametrize("k_int8", [False, True])
def test_fused_every_shape(r, dv, G, k_int8):
    require_gpu()
    B, hkv = 3, 2
    hq = G * hkv
    lens = [5, 300, 64]
    cache, _, _ = _make(B, hq, hkv, r, dv, lens, k_int8, 0, seed=20 + r + G)
    q = inputs.normal_bf16((B, hq, r), seed=21, device="cuda")
    k1 = inputs.normal_bf16((B, hkv, r), seed=22, device="cuda")
    v1 = inputs.normal_bf16((B, hkv, dv), seed=23, device="cuda")
    (a, oa_), (f, of_) = _both(cache, q, k1, v1, lens, out_dtype=torch.bfloat16)
    assert torch.equal(oa_, of_)
    _same_cache(a, f)


@pytest.mark.parametrize("k_int8", [False, True])
def test_fused_matches_oracle(k_int8):
    require_gpu()
    B, hq, hkv, r, dv = 4, 32, 8, 32, 128
    lens = [4095, 17, 0, 2048]
    cache, kn, vn = _make(B, hq, hkv, r, dv, lens, k_int8, 0, seed=31, cap=4096)
    q = inputs.normal_bf16((B, hq, r), seed=32, device="cuda")
    k1 = inputs.normal_bf16((B, hkv, r), seed=33, device="cuda")
    v1 = inputs.normal_bf16((B, hkv, dv), seed=34, device="cuda")
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    out = torch.empty(B, hq, dv, device="cuda")
    tb.tk_attn_decode_append(cache, q, k1, v1, sl, 4096, out, tb.decode_workspace(cache.desc, 4096))
    assert tb.tk_get_device_error() == 0
    # the oracle's cache: the first lens[b] tokens of the block, then the new token
    n1 = [n + 1 for n in lens]
    K = torch.zeros(B, hkv, 4096, r, dtype=torch.bfloat16, device="cuda")
    V = torch.zeros(B, hkv, 4096, dv, dtype=torch.bfloat16, device="cuda")
    for b, n in enumerate(lens):
        K[b, :, :n] = kn[b, :, :n]
        V[b, :, :n] = vn[b, :, :n]
        K[b, :, n] = k1[b]
        V[b, :, n] = v1[b]
    scale = 1 / math.sqrt(r)
    if k_int8:
        codes, sc = oc.quantize_int8_per_token(K.float().cpu().numpy())
        ref = oa.attention_decode(f64(q), codes, f64(V), n1, scale, k_scale=sc)
    else:
        ref = oa.attention_decode(f64(q), f64(K), f64(V), n1, scale)
    parity(f64(out), ref, what=f"fused append+decode int8={k_int8}")


def test_fused_position_beyond_capacity_is_flagged():
    require_gpu()
    B, hq, hkv, r, dv = 2, 8, 2, 32, 128
    lens = [64, 10]
    cache, _, _ = _make(B, hq, hkv, r, dv, lens, False, 0, seed=41, cap=64)  # seq 0 is full
    before = _clone(cache)
    q = inputs.normal_bf16((B, hq, r), seed=42, device="cuda")
    k1 = inputs.normal_bf16((B, hkv, r), seed=43, device="cuda")
    v1 = inputs.normal_bf16((B, hkv, dv), seed=44, device="cuda")
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    out = torch.empty(B, hq, dv, device="cuda")
    tb.tk_attn_decode_append(cache, q, k1, v1, sl, 65, out, tb.decode_workspace(cache.desc, 65))
    assert tb.tk_get_device_error() == 1   # index out of range
    assert torch.equal(cache.k[0], before.k[0]) and torch.equal(cache.v[0], before.v[0])
    assert torch.equal(cache.k[1, :, 10], k1[1]) and torch.equal(cache.v[1, :, 10], v1[1])
    assert torch.isfinite(out).all()


def test_prepared_call_equals_direct_call():
    """binding.prepare_decode_append checks once and re-issues the same call."""
    require_gpu()
    B, hq, hkv, r, dv = 4, 32, 8, 32, 128
    lens = [100, 640, 1, 300]
    cache, _, _ = _make(B, hq, hkv, r, dv, lens, False, 0, seed=51)
    other = _clone(cache)
    q = inputs.normal_bf16((B, hq, r), seed=52, device="cuda")
    k1 = inputs.normal_bf16((B, hkv, r), seed=53, device="cuda")
    v1 = inputs.normal_bf16((B, hkv, dv), seed=54, device="cuda")
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    out_d = torch.empty(B, hq, dv, device="cuda")
    out_p = torch.empty(B, hq, dv, device="cuda")
    tb.tk_attn_decode_append(other, q, k1, v1, sl, 641, out_d, tb.decode_workspace(other.desc, 641))
    call = tb.prepare_decode_append(cache, q, k1, v1, sl, 641, out_p,
                                    tb.decode_workspace(cache.desc, 641))
    call()
    torch.cuda.synchronize()
    assert tb.tk_get_device_error() == 0
    assert torch.equal(out_d, out_p)
    _same_cache(other, cache)
    call()  # again: the same token rewritten at the same positions, same result
    torch.cuda.synchronize()
    assert torch.equal(out_d, out_p)
    with pytest.raises(ValueError):
        tb.prepare_decode_append(cache, q[:, :4], k1, v1, sl, 641, out_p,
                                 tb.decode_workspace(cache.desc, 641))


def test_prepared_call_with_host_input_and_zero_copy_output():
    """copy_in from page-locked host memory and a page-locked host `out` (written by the
    kernel directly) give the same bits as the all-device call."""
    require_gpu()
    B, hq, hkv, r, dv = 4, 32, 8, 32, 128
    lens = [100, 640, 1, 300]
    cache, _, _ = _make(B, hq, hkv, r, dv, lens, False, 0, seed=61)
    other = _clone(cache)
    q = inputs.normal_bf16((B, hq, r), seed=62, device="cuda")
    k1 = inputs.normal_bf16((B, hkv, r), seed=63, device="cuda")
    v1 = inputs.normal_bf16((B, hkv, dv), seed=64, device="cuda")
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    out_d = torch.empty(B, hq, dv, device="cuda")
    tb.tk_attn_decode_append(other, q, k1, v1, sl, 641, out_d, tb.decode_workspace(other.desc, 641))
    # the step's q, k_new, v_new packed in one device buffer, filled from one host buffer
    io = torch.empty(q.numel() + k1.numel() + v1.numel(), dtype=torch.bfloat16, device="cuda")
    hio = torch.cat([q.flatten(), k1.flatten(), v1.flatten()]).cpu().pin_memory()
    nq, nk = q.numel(), k1.numel()
    qv = io[:nq].view(B, hq, r)
    kv = io[nq:nq + nk].view(B, hkv, r)
    vv = io[nq + nk:].view(B, hkv, dv)
    out_h = torch.full((B, hq, dv), float("nan")).pin_memory()
    stream = torch.cuda.Stream()
    call = tb.prepare_decode_append(cache, qv, kv, vv, sl, 641, out_h, tb.decode_workspace(cache.desc, 641),
                                    stream=stream, copy_in=(io, hio))
    call()
    stream.synchronize()
    assert tb.tk_get_device_error() == 0
    assert torch.equal(out_h, out_d.cpu())
    _same_cache(other, cache)
    with pytest.raises(ValueError):
        tb.prepare_decode_append(cache, qv, kv, vv, sl, 641, out_h, tb.decode_workspace(cache.desc, 641),
                                 copy_in=(io, hio[:-1]))


def test_prepared_call_as_cuda_graph():
    """graph=True: the copy-in and the fused decode recorded as one CUDA graph; each
    replay takes the host buffer's current contents and gives the eager call's bits."""
    require_gpu()
    B, hq, hkv, r, dv = 4, 32, 8, 32, 128
    lens = [100, 640, 1, 300]
    cache, _, _ = _make(B, hq, hkv, r, dv, lens, False, 0, seed=71)
    other = _clone(cache)
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    io = torch.empty(B * hq * r + B * hkv * (r + dv), dtype=torch.bfloat16, device="cuda")
    nq, nk = B * hq * r, B * hkv * r
    qv, kv, vv = io[:nq].view(B, hq, r), io[nq:nq + nk].view(B, hkv, r), io[nq + nk:].view(B, hkv, dv)
    hio = torch.empty(io.numel(), dtype=torch.bfloat16).pin_memory()
    out_h = torch.full((B, hq, dv), float("nan")).pin_memory()
    stream = torch.cuda.Stream()
    ws = tb.decode_workspace(cache.desc, 641)
    for step, seed in enumerate((72, 82)):
        q = inputs.normal_bf16((B, hq, r), seed=seed, device="cuda")
        k1 = inputs.normal_bf16((B, hkv, r), seed=seed + 1, device="cuda")
        v1 = inputs.normal_bf16((B, hkv, dv), seed=seed + 2, device="cuda")
        hio.copy_(torch.cat([q.flatten(), k1.flatten(), v1.flatten()]).cpu())
        if step == 0:   # preparing runs the step once eagerly, then records it
            call = tb.prepare_decode_append(cache, qv, kv, vv, sl, 641, out_h, ws, stream=stream,
                                            copy_in=(io, hio), graph=True)
        call()
        stream.synchronize()
        assert tb.tk_get_device_error() == 0
        out_d = torch.empty(B, hq, dv, device="cuda")
        tb.tk_attn_decode_append(other, q, k1, v1, sl, 641, out_d, tb.decode_workspace(other.desc, 641))
        torch.cuda.synchronize()
        assert torch.equal(out_h, out_d.cpu())
        _same_cache(other, cache)
    del call
