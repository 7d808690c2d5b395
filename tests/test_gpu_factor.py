"""A full-key attention layer turned thin-key by factor.factor_keys, run on the kernels.

Rank-32 key projections (d_head 128): the factored queries and thin keys,
rounded to bf16, go through tk_attn_prefill and the cache + tk_attn_decode at
the original model's scale 1/sqrt(d_head); both match the fp64 oracle on the
same inputs, and the oracle's thin-key result equals its full-key result
(before bf16 rounding) -- the Section 2.3 claim, end to end.
"""

import math

import numpy as np
import pytest
import torch

from _helpers import f64, parity, require_gpu
from oracle import attention as oa
from paper_2603_04427_gb300 import binding as tb
from paper_2603_04427_gb300 import factor

pytestmark = pytest.mark.gpu


def test_factored_layer_on_the_kernels():
    require_gpu()
    B, S, d_model, h_q, h_kv, d_head, r, dv = 1, 300, 256, 8, 2, 128, 32, 128
    g = torch.Generator().manual_seed(77)
    x = torch.randn(B, S, d_model, generator=g, dtype=torch.float64)
    wq = torch.randn(d_model, h_q * d_head, generator=g, dtype=torch.float64) / math.sqrt(d_model)
    wk = torch.cat([torch.randn(d_model, r, generator=g, dtype=torch.float64) / math.sqrt(d_model)
                    @ torch.randn(r, d_head, generator=g, dtype=torch.float64) / math.sqrt(r)
                    for _ in range(h_kv)], dim=1)
    wv = torch.randn(d_model, h_kv * dv, generator=g, dtype=torch.float64) / math.sqrt(d_model)
    f = factor.factor_keys(wq, wk, h_q, h_kv, r)

    def heads(t, h, w):  # [B, S, h*w] -> [B, h, S, w]
        return t.reshape(B, S, h, w).permute(0, 2, 1, 3).contiguous()

    q_full, k_full = heads(x @ wq, h_q, d_head), heads(x @ wk, h_kv, d_head)
    q_thin, k_thin = heads(x @ f.w_q, h_q, r), heads(x @ f.w_k, h_kv, r)
    v = heads(x @ wv, h_kv, dv)
    # the oracle: thin-key attention equals full-key attention (Section 2.3)
    full = oa.attention_prefill(q_full.numpy(), k_full.numpy(), v.numpy(), f.scale)
    thin = oa.attention_prefill(q_thin.numpy(), k_thin.numpy(), v.numpy(), f.scale)
    np.testing.assert_allclose(thin, full, rtol=0, atol=1e-9)

    # the kernels on the bf16-rounded factored inputs
    qb = q_thin.to(torch.bfloat16).cuda()
    kb = k_thin.to(torch.bfloat16).cuda()
    vb = v.to(torch.bfloat16).cuda()
    ref = oa.attention_prefill(f64(qb), f64(kb), f64(vb), f.scale)
    out = torch.empty(B, h_q, S, dv, device="cuda")
    tb.tk_attn_prefill(qb, kb, vb, out, scale=f.scale)
    assert tb.tk_get_device_error() == 0
    parity(f64(out), ref, what="factored layer prefill")

    cache = tb.ThinKeyCache.allocate(B, h_q, h_kv, r, dv, capacity=304)
    tb.tk_kv_append(cache, kb, vb, torch.zeros(B, dtype=torch.int32, device="cuda"))
    dec = torch.empty(B, h_q, dv, device="cuda")
    sl = torch.full((B,), S, dtype=torch.int32, device="cuda")
    tb.tk_attn_decode(cache, qb[:, :, S - 1].contiguous(), sl, S, dec,
                      tb.decode_workspace(cache.desc, S), scale=f.scale)
    assert tb.tk_get_device_error() == 0
    parity(f64(dec), ref[:, :, S - 1], what="factored layer decode")
