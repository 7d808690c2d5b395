"""tk_attn_decode on the GPU against the fp64 oracle (and against itself).

Small cases cover every compiled (r, d_v, G, key dtype) combination with
ragged context lengths that span several 64-token chunks, several splits
(so the in-launch merge runs), a single token, and an empty context.
The Mistral-shaped GQA decode is compared in full here at the benchmark's
size; the long-context paged and quantised-key workloads are in
test_gpu_fullsize.py.  Paged and contiguous caches holding the same
tokens must give bit-identical outputs (same split boundaries).
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


def _contiguous(B, hq, hkv, r, dv, cap, lens, k_int8, seed):
    """Cache filled through tk_kv_append with `cap` random tokens per sequence."""
    cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=cap, k_int8=k_int8)
    kn = inputs.normal_bf16((B, hkv, cap, r), seed, device="cuda")
    vn = inputs.normal_bf16((B, hkv, cap, dv), seed + 1, device="cuda")
    tb.tk_kv_append(cache, kn, vn, torch.zeros(B, dtype=torch.int32, device="cuda"))
    return cache, kn, vn


def _run(cache, q, lens, max_len=None, out_dtype=torch.float32):
    B = q.shape[0]
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    max_len = max(lens) if max_len is None else max_len
    ws = tb.decode_workspace(cache.desc, max_len)
    out = torch.full((B, cache.desc.h_q, cache.desc.d_v), float("nan"), dtype=out_dtype, device="cuda")
    tb.tk_attn_decode(cache, q, sl, max_len, out, ws)
    assert tb.tk_get_device_error() == 0
    # the workspace's arrival counters are back at zero
    assert int(ws[:4 * B * cache.desc.h_kv].view(torch.int32).abs().sum()) == 0
    return out


def _oracle(cache, q, kn, lens, scale):
    if cache.desc.k_dtype == tb.TK_I8:
        codes, sc = oc.quantize_int8_per_token(kn.float().cpu().numpy())
        return oa.attention_decode(f64(q), codes, f64(cache.v), lens, scale, k_scale=sc)
    return oa.attention_decode(f64(q), f64(cache.k), f64(cache.v), lens, scale)


@pytest.mark.parametrize("k_int8", [False, True])
@pytest.mark.parametrize("G", [1, 2, 4, 8])
@pytest.mark.parametrize("r,dv", [(16, 64), (32, 128), (64, 64), (128, 128)])
def test_decode_matches_oracle_small(k_int8, G, r, dv):
    require_gpu()
    B, hkv = 4, 2
    hq = G * hkv
    lens = [777, 1, 0, 64]
    cap = 784
    cache, kn, _ = _contiguous(B, hq, hkv, r, dv, cap, lens, k_int8, seed=100 + r + G)
    q = inputs.normal_bf16((B, hq, r), seed=7, device="cuda")
    out = _run(cache, q, lens)
    ref = _oracle(cache, q, kn, lens, 1 / math.sqrt(r))
    parity(f64(out), ref, what=f"decode r={r} dv={dv} G={G} int8={k_int8}")
    assert torch.all(out[2] == 0)                       # empty context
    np.testing.assert_allclose(f64(out[1]), ref[1], rtol=1e-5, atol=1e-6)  # one token: v[0]


def test_decode_bf16_output_and_determinism():
    require_gpu()
    B, hq, hkv, r, dv = 3, 16, 4, 32, 128
    lens = [2000, 1531, 64]
    cache, kn, _ = _contiguous(B, hq, hkv, r, dv, 2048, lens, False, seed=5)
    q = inputs.normal_bf16((B, hq, r), seed=8, device="cuda")
    o1 = _run(cache, q, lens, out_dtype=torch.bfloat16)
    o2 = _run(cache, q, lens, out_dtype=torch.bfloat16)
    assert torch.equal(o1, o2)
    of = _run(cache, q, lens)
    assert torch.equal(o1, of.to(torch.bfloat16))       # bf16 output = RNE of the fp32 output
    parity(f64(o1), _oracle(cache, q, kn, lens, 1 / math.sqrt(r)), what="bf16 out")


@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_zero_copy_host_output_equals_device_output(out_dtype):
    """`out` in page-locked host memory: the kernel writes it directly, same bits."""
    require_gpu()
    B, hq, hkv, r, dv = 3, 16, 4, 32, 128
    lens = [2000, 1531, 64]
    cache, _, _ = _contiguous(B, hq, hkv, r, dv, 2048, lens, False, seed=15)
    q = inputs.normal_bf16((B, hq, r), seed=18, device="cuda")
    dev = _run(cache, q, lens, out_dtype=out_dtype)
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    host = torch.full((B, hq, dv), float("nan"), dtype=out_dtype).pin_memory()
    tb.tk_attn_decode(cache, q, sl, max(lens), host, tb.decode_workspace(cache.desc, max(lens)))
    torch.cuda.synchronize()
    assert tb.tk_get_device_error() == 0
    assert torch.equal(host, dev.cpu())
    with pytest.raises(ValueError):   # pageable host memory is refused
        tb.tk_attn_decode(cache, q, sl, max(lens), torch.empty(B, hq, dv, dtype=out_dtype),
                          tb.decode_workspace(cache.desc, max(lens)))


def _paged_copy(cache, lens, ps, seed):
    """A paged cache holding the same tokens as the contiguous `cache`."""
    d = cache.desc
    table, n_pages = inputs.paged_layout(lens, ps, seed=seed, extra_pages=3)
    pc = tb.ThinKeyCache.allocate(d.batch, d.h_q, d.h_kv, d.r, d.d_v, page_size=ps,
                                  num_pages=n_pages, page_table=table,
                                  k_int8=d.k_dtype == tb.TK_I8)
    for b, n in enumerate(lens):
        for j in range(-(-n // ps)):
            page = int(table[b, j])
            m = min(ps, n - j * ps)
            pc.k[page, :, :m] = cache.k[b, :, j * ps:j * ps + m]
            pc.v[page, :, :m] = cache.v[b, :, j * ps:j * ps + m]
            if pc.k_scale is not None:
                pc.k_scale[page, :, :m] = cache.k_scale[b, :, j * ps:j * ps + m]
    return pc


@pytest.mark.parametrize("k_int8", [False, True])
@pytest.mark.parametrize("ps", [16, 64, 256])
def test_paged_equals_contiguous_bitwise(k_int8, ps):
    require_gpu()
    B, hq, hkv, r, dv = 3, 8, 2, 32, 128
    lens = [1000, 333, 65]
    cache, kn, _ = _contiguous(B, hq, hkv, r, dv, 1024, lens, k_int8, seed=31)
    q = inputs.normal_bf16((B, hq, r), seed=9, device="cuda")
    a = _run(cache, q, lens)
    pc = _paged_copy(cache, lens, ps, seed=4)
    p = _run(pc, q, lens)
    assert torch.equal(a, p)
    parity(f64(p), _oracle(cache, q, kn, lens, 1 / math.sqrt(r)), what=f"paged ps={ps}")


def test_bad_page_id_is_flagged():
    require_gpu()
    B, hq, hkv, r, dv, ps = 1, 4, 1, 32, 64, 64
    table = torch.tensor([[0, 5, 1]], dtype=torch.int32)     # page 5 does not exist
    pc = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, page_size=ps, num_pages=2, page_table=table)
    q = inputs.normal_bf16((B, hq, r), seed=1, device="cuda")
    sl = torch.tensor([150], dtype=torch.int32, device="cuda")
    ws = tb.decode_workspace(pc.desc, 150)
    out = torch.empty(B, hq, dv, device="cuda")
    tb.tk_attn_decode(pc, q, sl, 150, out, ws)
    assert tb.tk_get_device_error() == 1


def test_seq_len_beyond_bound_is_flagged():
    require_gpu()
    cache, _, _ = _contiguous(1, 2, 1, 32, 64, 64, [64], False, seed=3)
    q = inputs.normal_bf16((1, 2, 32), seed=1, device="cuda")
    ws = tb.decode_workspace(cache.desc, 64)
    out = torch.empty(1, 2, 64, device="cuda")
    tb.tk_attn_decode(cache, q, torch.tensor([65], dtype=torch.int32, device="cuda"), 64, out, ws)
    assert tb.tk_get_device_error() == 1
    assert torch.isfinite(out).all()


def test_workspace_too_small_is_rejected():
    require_gpu()
    cache, _, _ = _contiguous(2, 8, 2, 32, 128, 1024, [1024, 1024], False, seed=3)
    need = tb.tk_decode_workspace_size(cache.desc, 1024)
    ws = torch.zeros(need - 256, dtype=torch.uint8, device="cuda")
    out = torch.empty(2, 8, 128, device="cuda")
    q = torch.zeros(2, 8, 32, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(tb.TkError) as e:
        tb.tk_attn_decode(cache, q, torch.tensor([1024, 1024], dtype=torch.int32, device="cuda"),
                          1024, out, ws)
    assert e.value.status == tb.TK_ERR_WORKSPACE


# ------------------------------------------------------------------ full-size workloads

def test_mistral_gqa_decode_full():
    """B=16, H_q=32, H_kv=8, r=32, d_v=128, every context 4096: all outputs vs the oracle."""
    require_gpu()
    B, hq, hkv, r, dv, L = 16, 32, 8, 32, 128, 4096
    cache, kn, _ = _contiguous(B, hq, hkv, r, dv, L, [L] * B, False, seed=1001)
    q = inputs.normal_bf16((B, hq, r), seed=1002, device="cuda")
    out = _run(cache, q, [L] * B)
    ref = oa.attention_decode(f64(q), f64(cache.k), f64(cache.v), [L] * B, 1 / math.sqrt(r))
    parity(f64(out), ref, what="mistral gqa decode")
