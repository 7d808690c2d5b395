"""tk_kv_append on the GPU against the oracle's cache writes: bit-exact.

bf16 rows are copies; int8 keys must match the oracle quantiser's codes and
fp32 scales bit for bit (same binary32 division and ties-to-even rounding).
"""

import numpy as np
import pytest
import torch

from _helpers import require_gpu
from oracle import cache as oc
from paper_2603_04427_gb300 import binding as tb
from paper_2603_04427_gb300 import inputs

pytestmark = pytest.mark.gpu

SENTINEL = 7  # bf16 bits / int8 fill of untouched slots


def _cache_np(cache):
    k = cache.k.cpu()
    k = k.view(torch.int16).numpy() if k.dtype == torch.bfloat16 else k.numpy()
    v = cache.v.cpu().view(torch.int16).numpy()
    ks = None if cache.k_scale is None else cache.k_scale.cpu().numpy()
    return k.copy(), v.copy(), None if ks is None else ks.copy()


@pytest.mark.parametrize("k_int8", [False, True])
@pytest.mark.parametrize("r,dv", [(16, 64), (32, 128), (64, 128), (128, 64)])
def test_append_contiguous_exact(k_int8, r, dv):
    require_gpu()
    B, hq, hkv, cap, T = 3, 4, 2, 96, 37
    lens = [0, 11, 59]
    cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=cap, k_int8=k_int8)
    cache.k.view(torch.uint8 if k_int8 else torch.int16).fill_(SENTINEL)
    cache.v.view(torch.int16).fill_(SENTINEL)
    k0, v0, s0 = _cache_np(cache)
    kn = inputs.normal_bf16((B, hkv, T, r), seed=11)
    vn = inputs.normal_bf16((B, hkv, T, dv), seed=12)
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    tb.tk_kv_append(cache, kn.cuda(), vn.cuda(), sl)
    assert tb.tk_get_device_error() == 0
    k1, v1, s1 = _cache_np(cache)
    # The oracle writes bf16 bit patterns for copies and float32 values for int8 keys.
    vref = v0.copy()
    oc.append_contiguous(np.zeros((B, hkv, cap, r), np.int16), vref, lens,
                         kn.view(torch.int16).numpy(), vn.view(torch.int16).numpy())
    assert np.array_equal(v1, vref)
    if not k_int8:
        kref = k0.copy()
        oc.append_contiguous(kref, v0.copy(), lens, kn.view(torch.int16).numpy(),
                             vn.view(torch.int16).numpy())
        assert np.array_equal(k1, kref)
    else:
        kref, sref = k0.copy(), s0.copy()
        oc.append_contiguous(kref, v0.copy(), lens, kn.float().numpy(), vn.float().numpy(), sref)
        assert np.array_equal(k1, kref)
        assert np.array_equal(s1.view(np.uint32), sref.view(np.uint32))


@pytest.mark.parametrize("k_int8", [False, True])
@pytest.mark.parametrize("ps", [16, 64, 256])
def test_append_paged_exact(k_int8, ps):
    require_gpu()
    B, hq, hkv, r, dv, T = 2, 8, 2, 32, 128, 70
    lens = [5, 130]
    table, n_pages = inputs.paged_layout([n + T for n in lens], ps, seed=3, extra_pages=2)
    cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, page_size=ps, num_pages=n_pages,
                                     page_table=table, k_int8=k_int8)
    cache.k.view(torch.uint8 if k_int8 else torch.int16).fill_(SENTINEL)
    cache.v.view(torch.int16).fill_(SENTINEL)
    k0, v0, s0 = _cache_np(cache)
    kn = inputs.normal_bf16((B, hkv, T, r), seed=21)
    vn = inputs.normal_bf16((B, hkv, T, dv), seed=22)
    tb.tk_kv_append(cache, kn.cuda(), vn.cuda(), torch.tensor(lens, dtype=torch.int32, device="cuda"))
    assert tb.tk_get_device_error() == 0
    k1, v1, s1 = _cache_np(cache)
    tab = table.numpy()
    if not k_int8:
        kref, vref = k0.copy(), v0.copy()
        oc.append_paged(kref, vref, tab, lens, ps, kn.view(torch.int16).numpy(),
                        vn.view(torch.int16).numpy())
        assert np.array_equal(k1, kref) and np.array_equal(v1, vref)
    else:
        kref, vref, sref = k0.copy(), v0.copy(), s0.copy()
        oc.append_paged(kref, vref, tab, lens, ps, kn.float().numpy(), vn.view(torch.int16).numpy(), sref)
        assert np.array_equal(k1, kref) and np.array_equal(v1, vref)
        assert np.array_equal(s1.view(np.uint32), sref.view(np.uint32))


def test_append_int8_special_rows():
    """Zero rows, exact ties and the amax element, bit-exact against the oracle."""
    require_gpu()
    B, hkv, r, dv, T = 1, 1, 32, 64, 4
    rows = np.zeros((T, r), np.float32)
    rows[1, :4] = [127.0, 2.5, 3.5, -2.5]         # scale 1: ties to even
    rows[2, :3] = [-0.75, 0.375, 0.0]             # negative amax
    rows[3] = np.linspace(-3, 3, r).astype(np.float32)
    kn = torch.from_numpy(rows).to(torch.bfloat16).reshape(B, hkv, T, r)
    vn = inputs.normal_bf16((B, hkv, T, dv), seed=5)
    cache = tb.ThinKeyCache.allocate(B, 1, hkv, r, dv, capacity=16, k_int8=True)
    tb.tk_kv_append(cache, kn.cuda(), vn.cuda(), torch.zeros(1, dtype=torch.int32, device="cuda"))
    codes, scales = oc.quantize_int8_per_token(kn.float().numpy())
    assert np.array_equal(cache.k[:, :, :T].cpu().numpy(), codes)
    assert np.array_equal(cache.k_scale[:, :, :T].cpu().numpy().view(np.uint32), scales.view(np.uint32))
    assert cache.k_scale[0, 0, 0].item() == 0.0 and cache.k[0, 0, 1, :4].tolist() == [127, 2, 4, -2]


def test_append_out_of_capacity_is_flagged_not_written():
    require_gpu()
    cache = tb.ThinKeyCache.allocate(1, 1, 1, 32, 64, capacity=16)
    cache.k.view(torch.int16).fill_(SENTINEL)
    kn = inputs.normal_bf16((1, 1, 4, 32), seed=1).cuda()
    vn = inputs.normal_bf16((1, 1, 4, 64), seed=2).cuda()
    tb.tk_kv_append(cache, kn, vn, torch.tensor([14], dtype=torch.int32, device="cuda"))
    assert tb.tk_get_device_error() == 1
    assert tb.tk_get_device_error() == 0  # cleared by the read
    assert torch.equal(cache.k[0, 0, 14:16], kn[0, 0, :2])
    assert bool((cache.k[0, 0, :14].view(torch.int16) == SENTINEL).all())
