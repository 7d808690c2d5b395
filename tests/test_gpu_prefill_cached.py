"""tk_attn_prefill_cached: a chunk of queries over a cached context, on the GPU.

The chunk's keys and values land in the cache (bit-exact); its queries at
positions seq_lens[b] + i attend to the cache's first seq_lens[b] + i + 1
tokens (end-aligned causal) and match the fp64 oracle; paged caches give the
same bits as a contiguous one, and an empty context gives the plain prefill
bit for bit.  int8 and int4 key caches (codes and scales written by the
quantising append) match the oracle on the dequantised keys, again with
paged = contiguous bit for bit; cache slots past a context may hold NaN.
A 7B-shaped chunk (4096 new tokens after 4096 cached) is checked on sampled
rows, with bf16 and with int8 keys.
"""

import math

import numpy as np
import pytest
import torch

from _helpers import f64, parity, parity_bf16, require_gpu
from oracle import attention as oa
from oracle import cache as oc
from paper_2603_04427_gb300 import binding as tb
from paper_2603_04427_gb300 import inputs

pytestmark = pytest.mark.gpu


def _setup(B, hq, hkv, r, dv, L0, S, seed, ps=0, kfmt="bf16", garbage=False):
    """A cache holding each sequence's L0[b] cached tokens (written by tk_kv_append),
    the chunk's q / k_new / v_new, and every sequence's whole context K / V (bf16,
    as appended) for the oracle.  garbage: NaN (bf16) / NaN scales everywhere
    before the context is written, so slots past it hold NaN."""
    cap = (max(L0) + S + 15) // 16 * 16
    n = [l0 + S for l0 in L0]
    q8, q4 = kfmt == "int8", kfmt == "int4"
    if ps:
        table, n_pages = inputs.paged_layout(n, ps, seed=seed, extra_pages=2)
        cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, page_size=ps, num_pages=n_pages,
                                         page_table=table, k_int8=q8, k_int4=q4)
    else:
        cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=cap, k_int8=q8, k_int4=q4)
    if garbage:
        cache.v.fill_(float("nan"))
        if kfmt == "bf16":
            cache.k.fill_(float("nan"))
        else:
            cache.k.fill_(0x77)
            cache.k_scale.fill_(float("nan"))
    T = max(L0)
    kc = inputs.normal_bf16((B, hkv, max(T, 1), r), seed, device="cuda")
    vc = inputs.normal_bf16((B, hkv, max(T, 1), dv), seed + 1, device="cuda")
    zero = torch.zeros(1, dtype=torch.int32, device="cuda")
    for b, l0 in enumerate(L0):   # the cached context of each sequence
        if l0:
            d = cache.desc
            ks = cache.k_scale
            one = tb.ThinKeyCache(tb.tk_cache_desc(1, hq, hkv, r, dv, d.capacity, d.page_size,
                                                   d.num_pages, d.max_pages_per_seq, d.k_dtype),
                                  cache.k if ps else cache.k[b:b + 1], cache.v if ps else cache.v[b:b + 1],
                                  None if ks is None else (ks if ps else ks[b:b + 1]),
                                  cache.page_table[b:b + 1].contiguous() if ps else None)
            tb.tk_kv_append(one, kc[b:b + 1, :, :l0].contiguous(), vc[b:b + 1, :, :l0].contiguous(), zero)
    q = inputs.normal_bf16((B, hq, S, r), seed + 2, device="cuda")
    kn = inputs.normal_bf16((B, hkv, S, r), seed + 3, device="cuda")
    vn = inputs.normal_bf16((B, hkv, S, dv), seed + 4, device="cuda")
    # the whole context per sequence, for the oracle
    K = torch.zeros(B, hkv, max(n), r, dtype=torch.bfloat16, device="cuda")
    V = torch.zeros(B, hkv, max(n), dv, dtype=torch.bfloat16, device="cuda")
    for b, l0 in enumerate(L0):
        K[b, :, :l0], V[b, :, :l0] = kc[b, :, :l0], vc[b, :, :l0]
        K[b, :, l0:l0 + S], V[b, :, l0:l0 + S] = kn[b], vn[b]
    return cache, q, kn, vn, K, V, max(n)


def _keys_for_oracle(K, kfmt):
    """The keys the kernels see: bf16 as they are, or the oracle's quantiser's
    codes times scales (per token and kv head), exact in fp64."""
    if kfmt == "bf16":
        return f64(K)
    quant = oc.quantize_int8_per_token if kfmt == "int8" else oc.quantize_int4_per_token
    codes, sc = quant(K.float().cpu().numpy())
    return oa.dequantize_keys(codes, sc)


def _run(cache, q, kn, vn, L0, max_len, dtype=torch.float32, causal=True):
    B, hq, S, _ = q.shape
    out = torch.full((B, hq, S, cache.desc.d_v), float("nan"), dtype=dtype, device="cuda")
    sl = torch.tensor(L0, dtype=torch.int32, device="cuda")
    tb.tk_attn_prefill_cached(cache, q, kn, vn, sl, max_len, out, causal=causal)
    assert tb.tk_get_device_error() == 0
    return out


@pytest.mark.parametrize("r,dv", [(32, 128), (64, 64), (16, 128), (128, 128)])
def test_cached_prefill_matches_oracle(r, dv):
    require_gpu()
    B, hq, hkv, S = 3, 8, 2, 300
    L0 = [0, 100, 777]
    cache, q, kn, vn, K, V, n = _setup(B, hq, hkv, r, dv, L0, S, seed=10 + r)
    out = _run(cache, q, kn, vn, L0, n)
    ref = oa.attention_prefill_cached(f64(q), f64(K), f64(V), L0, 1 / math.sqrt(r))
    parity(f64(out), ref, what=f"cached prefill r={r} dv={dv}")
    for b, l0 in enumerate(L0):   # the chunk is in the cache
        assert torch.equal(cache.k[b, :, l0:l0 + S], kn[b])
        assert torch.equal(cache.v[b, :, l0:l0 + S], vn[b])


def test_cached_prefill_non_causal_and_bf16_out():
    require_gpu()
    B, hq, hkv, r, dv, S = 2, 4, 4, 32, 128, 200
    L0 = [64, 333]
    cache, q, kn, vn, K, V, n = _setup(B, hq, hkv, r, dv, L0, S, seed=3)
    out = _run(cache, q, kn, vn, L0, n, dtype=torch.bfloat16, causal=False)
    ref = oa.attention_prefill_cached(f64(q), f64(K), f64(V), L0, 1 / math.sqrt(r), causal=False)
    parity_bf16(f64(out), ref, what="cached prefill, full attention, bf16 out")


@pytest.mark.parametrize("ps", [16, 64, 128, 256])
def test_cached_prefill_paged_equals_contiguous_bitwise(ps):
    require_gpu()
    B, hq, hkv, r, dv, S = 3, 8, 2, 32, 128, 257
    L0 = [5, 130, 640]
    a = _setup(B, hq, hkv, r, dv, L0, S, seed=21)
    p = _setup(B, hq, hkv, r, dv, L0, S, seed=21, ps=ps)
    out_a = _run(*a[:4], L0, a[6])
    out_p = _run(*p[:4], L0, p[6])
    assert torch.equal(out_a, out_p)


def test_empty_context_equals_plain_prefill():
    require_gpu()
    B, hq, hkv, r, dv, S = 2, 8, 4, 32, 128, 390
    L0 = [0, 0]
    cache, q, kn, vn, _, _, n = _setup(B, hq, hkv, r, dv, L0, S, seed=31)
    out = _run(cache, q, kn, vn, L0, n)
    plain = torch.empty_like(out)
    tb.tk_attn_prefill(q, kn, vn, plain)
    assert torch.equal(out, plain)


def test_7b_chunk_after_4096_cached_sampled():
    """B=2, H=32, r=32, d_v=128: 4096 new tokens after 4096 cached, bf16 out, sampled rows."""
    require_gpu()
    B, H, r, dv, S = 2, 32, 32, 128, 4096
    L0 = [4096, 4096]
    cache, q, kn, vn, K, V, n = _setup(B, H, H, r, dv, L0, S, seed=1005)
    out = _run(cache, q, kn, vn, L0, n, dtype=torch.bfloat16)
    rng = np.random.default_rng(5)
    got, ref = [], []
    for b, h, i in [(int(rng.integers(B)), int(rng.integers(H)), int(i)) for i in
                    list(rng.integers(0, S, 40)) + [0, 127, 128, 4095]]:
        p = L0[b] + i
        ref.append(oa.attention_head(f64(q[b, h, i])[None], f64(K[b, h, :p + 1]),
                                     f64(V[b, h, :p + 1]), 1 / math.sqrt(r))[0])
        got.append(f64(out[b, h, i]))
    parity_bf16(np.stack(got), np.stack(ref), what="7b cached chunk sampled")


@pytest.mark.parametrize("kfmt,r,dv", [(k, r, dv) for k in ("int8", "int4") for r in (16, 32, 64, 128)
                                       for dv in (64, 128) if not (k == "int4" and r < 32)])
def test_quantised_cached_prefill_matches_oracle(kfmt, r, dv):
    require_gpu()
    B, hq, hkv, S = 3, 8, 2, 300
    L0 = [0, 100, 777]
    cache, q, kn, vn, K, V, n = _setup(B, hq, hkv, r, dv, L0, S, seed=40 + r + dv, kfmt=kfmt)
    out = _run(cache, q, kn, vn, L0, n)
    ref = oa.attention_prefill_cached(f64(q), _keys_for_oracle(K, kfmt), f64(V), L0, 1 / math.sqrt(r))
    parity(f64(out), ref, what=f"cached prefill {kfmt} keys r={r} dv={dv}")
    # the chunk's codes and scales are the oracle quantiser's, bit for bit
    quant = oc.quantize_int8_per_token if kfmt == "int8" else oc.quantize_int4_per_token
    for b, l0 in enumerate(L0):
        codes, sc = quant(kn[b].float().cpu().numpy())
        stored = cache.k[b, :, l0:l0 + S].cpu().numpy()
        assert np.array_equal(stored, codes if kfmt == "int8" else oc.pack_int4(codes))
        assert np.array_equal(cache.k_scale[b, :, l0:l0 + S].cpu().numpy().view(np.uint32),
                              sc.view(np.uint32))
        assert torch.equal(cache.v[b, :, l0:l0 + S], vn[b])


@pytest.mark.parametrize("kfmt", ["int8", "int4"])
@pytest.mark.parametrize("ps", [16, 64, 256])
@pytest.mark.parametrize("r,dv", [(32, 128), (128, 64)])
def test_quantised_cached_prefill_paged_equals_contiguous_bitwise(kfmt, ps, r, dv):
    require_gpu()
    B, hq, hkv, S = 3, 8, 2, 257
    L0 = [5, 130, 640]
    a = _setup(B, hq, hkv, r, dv, L0, S, seed=23, kfmt=kfmt)
    p = _setup(B, hq, hkv, r, dv, L0, S, seed=23, ps=ps, kfmt=kfmt)
    out_a = _run(*a[:4], L0, a[6])
    out_p = _run(*p[:4], L0, p[6])
    assert torch.equal(out_a, out_p)
    ref = oa.attention_prefill_cached(f64(a[1]), _keys_for_oracle(a[4], kfmt), f64(a[5]), L0,
                                      1 / math.sqrt(r))
    parity(f64(out_p), ref, what=f"paged {kfmt} ps={ps}")


@pytest.mark.parametrize("kfmt,r,dv,L0,S,causal,bf16_out", [
    ("int8", 32, 128, [128, 0], 128, True, True),     # contexts end on a tile boundary
    ("int4", 64, 128, [256, 3], 129, False, False),   # full attention over the context
    ("int8", 128, 64, [0, 1], 1, True, False),        # a one-token chunk (scales in the softmax)
    ("int4", 32, 64, [1000, 17], 64, False, True),
])
def test_quantised_cached_prefill_edge_cases(kfmt, r, dv, L0, S, causal, bf16_out):
    require_gpu()
    B, hq, hkv = len(L0), 4, 2
    cache, q, kn, vn, K, V, n = _setup(B, hq, hkv, r, dv, L0, S, seed=71 + S, kfmt=kfmt)
    out = _run(cache, q, kn, vn, L0, n, dtype=torch.bfloat16 if bf16_out else torch.float32,
               causal=causal)
    ref = oa.attention_prefill_cached(f64(q), _keys_for_oracle(K, kfmt), f64(V), L0,
                                      1 / math.sqrt(r), causal=causal)
    check = parity_bf16 if bf16_out else parity
    check(f64(out), ref, what=f"{kfmt} r={r} L0={L0} S={S} causal={causal}")


def _bf16_rne(x):
    """float32 array -> bf16 bit patterns (uint16), rounded to nearest even (finite x)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


@pytest.mark.parametrize("kfmt,r,dv", [("int8", 32, 128), ("int4", 64, 128), ("int8", 16, 64),
                                       ("int8", 128, 64), ("int4", 128, 128)])
def test_widened_keys_in_the_workspace(kfmt, r, dv):
    """The workspace after a call holds every context token's key widened as
    tk_prefill_cached_workspace_size documents: for r <= 64, plane 0 = hi =
    bf16(scale * code) and plane 1 = lo = bf16(scale * code - hi) (the product in
    fp32, both roundings to nearest even), so hi + lo is within 2^-17 of the
    product; for r = 128, the codes as exact bf16 and the fp32 scales.  Computed
    here independently from the cache's codes and scales."""
    require_gpu()
    B, hq, hkv, S = 2, 4, 2, 200
    L0 = [0, 333]
    cache, q, kn, vn, K, V, n = _setup(B, hq, hkv, r, dv, L0, S, seed=61 + r, kfmt=kfmt)
    ws = tb.prefill_cached_workspace(cache, n)
    out = torch.empty(B, hq, S, dv, dtype=torch.float32, device="cuda")
    sl = torch.tensor(L0, dtype=torch.int32, device="cuda")
    tb.tk_attn_prefill_cached(cache, q, kn, vn, sl, n, out, workspace=ws)
    torch.cuda.synchronize()
    assert tb.tk_get_device_error() == 0
    rows = (n + 3) // 4 * 4
    plane = B * hkv * rows * r
    w = ws.cpu().numpy()
    p0 = w[:2 * plane].view(np.uint16).reshape(B, hkv, rows, r)
    codes = cache.k.cpu().numpy()
    codes = codes if kfmt == "int8" else oc.unpack_int4(codes)
    scales = cache.k_scale.cpu().numpy()
    two = r <= 64
    assert ws.numel() == (4 * plane if two else 2 * plane + 4 * B * hkv * rows)
    for b, l0 in enumerate(L0):
        c = codes[b, :, :l0 + S].astype(np.float32)
        s = scales[b, :, :l0 + S]
        if two:
            x = c * s[..., None]                                   # fp32 product
            hi = _bf16_rne(x)
            lo = _bf16_rne(x - (hi.astype(np.uint32) << 16).view(np.float32))
            p1 = w[2 * plane:4 * plane].view(np.uint16).reshape(B, hkv, rows, r)
            assert np.array_equal(p0[b, :, :l0 + S], hi)
            assert np.array_equal(p1[b, :, :l0 + S], lo)
            back = (hi.astype(np.uint32) << 16).view(np.float32).astype(np.float64) + \
                (lo.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
            exact = c.astype(np.float64) * s[..., None].astype(np.float64)
            assert np.all(np.abs(back - exact) <= 2.0 ** -17 * np.abs(exact) + 2.0 ** -24 * np.abs(exact))
        else:
            assert np.array_equal(p0[b, :, :l0 + S], _bf16_rne(c))  # small integers: exact
            sp = w[2 * plane:2 * plane + 4 * B * hkv * rows].view(np.float32).reshape(B, hkv, rows)
            assert np.array_equal(sp[b, :, :l0 + S].view(np.uint32), s.view(np.uint32))


def test_workspace_reused_across_calls_and_shapes():
    """One workspace, large enough for the biggest call, serves calls of other
    shapes and key formats in stream order: every result equals, bit for bit,
    the same call with a fresh workspace of its own."""
    require_gpu()
    cases = [("int8", 64, 128, [500, 20], 300), ("int4", 32, 64, [0, 77], 130),
             ("int8", 128, 64, [128, 1], 64), ("int8", 64, 128, [500, 20], 300)]
    sizes = []
    for kfmt, r, dv, L0, S in cases:
        cache, *_rest, n = _setup(len(L0), 4, 2, r, dv, L0, S, seed=3, kfmt=kfmt)
        sizes.append(tb.prefill_cached_workspace(cache, n).numel())
    shared = torch.full((max(sizes),), 0x7F, dtype=torch.uint8, device="cuda")  # garbage
    for i, (kfmt, r, dv, L0, S) in enumerate(cases):
        a = _setup(len(L0), 4, 2, r, dv, L0, S, seed=90 + i, kfmt=kfmt)
        b = _setup(len(L0), 4, 2, r, dv, L0, S, seed=90 + i, kfmt=kfmt)
        sl = torch.tensor(L0, dtype=torch.int32, device="cuda")
        outs = []
        for (cache, q, kn, vn, K, V, n), ws in ((a, shared), (b, None)):
            out = torch.empty(len(L0), 4, S, dv, dtype=torch.float32, device="cuda")
            tb.tk_attn_prefill_cached(cache, q, kn, vn, sl, n, out, workspace=ws)
            outs.append(out)
        torch.cuda.synchronize()
        assert tb.tk_get_device_error() == 0
        assert torch.equal(outs[0], outs[1]), (kfmt, r, dv)


def test_quantised_prefill_rejects_a_short_workspace():
    require_gpu()
    cache, q, kn, vn, K, V, n = _setup(1, 4, 2, 32, 128, [64], 128, seed=5, kfmt="int8")
    ws = tb.prefill_cached_workspace(cache, n)
    out = torch.empty(1, 4, 128, 128, dtype=torch.float32, device="cuda")
    sl = torch.tensor([64], dtype=torch.int32, device="cuda")
    with pytest.raises(RuntimeError, match="TK_ERR_WORKSPACE"):
        tb.tk_attn_prefill_cached(cache, q, kn, vn, sl, n, out, workspace=ws[:-256])


@pytest.mark.parametrize("kfmt,ps", [("bf16", 0), ("int8", 0), ("bf16", 64), ("int4", 16)])
def test_cached_prefill_ignores_garbage_past_the_context(kfmt, ps):
    """Slots past each context hold NaN (values, bf16 keys, key scales): never weighted."""
    require_gpu()
    B, hq, hkv, r, dv, S = 2, 8, 2, 32, 128, 200
    L0 = [50, 301]
    cache, q, kn, vn, K, V, n = _setup(B, hq, hkv, r, dv, L0, S, seed=61, ps=ps, kfmt=kfmt,
                                       garbage=True)
    out = _run(cache, q, kn, vn, L0, n)
    assert torch.isfinite(out).all()
    ref = oa.attention_prefill_cached(f64(q), _keys_for_oracle(K, kfmt), f64(V), L0, 1 / math.sqrt(r))
    parity(f64(out), ref, what=f"garbage past the context, {kfmt} ps={ps}")


def test_7b_chunk_int8_keys_sampled():
    """The 7B chunk (4096 new after 4096 cached) over an int8 key cache, bf16 out: one row
    of every other 128-row query tile of every (sequence, head) plane."""
    require_gpu()
    B, H, r, dv, S = 2, 32, 32, 128, 4096
    L0 = [4096, 4096]
    cache, q, kn, vn, K, V, n = _setup(B, H, H, r, dv, L0, S, seed=1105, kfmt="int8")
    out = _run(cache, q, kn, vn, L0, n, dtype=torch.bfloat16)
    Kq = _keys_for_oracle(K, "int8")
    Vh, qh, oh = V.cpu(), q.cpu(), out.cpu()
    got, ref = [], []
    for b in range(B):
        for h in range(H):
            rows = [t * 128 + (t * 29 + (b * H + h) * 7) % 128 for t in range(0, S // 128, 2)]
            vv = f64(Vh[b, h])
            for i in rows:
                p = L0[b] + i
                ref.append(oa.attention_head(f64(qh[b, h, i])[None], Kq[b, h, :p + 1], vv[:p + 1],
                                             1 / math.sqrt(r))[0])
                got.append(f64(oh[b, h, i]))
    parity_bf16(np.stack(got), np.stack(ref), what="7b cached chunk, int8 keys")
