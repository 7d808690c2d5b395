"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a
pure-Python brute force, closed forms, invariants of softmax attention,
the factored-key identity of Section 2.3, and torch's CPU fp64
scaled_dot_product_attention (an independent library routine).  A
dropped scale, a flipped sign, a transposed operand, a wrong GQA mapping
or an off-by-one causal mask each fails at least one of them.
"""

import math

import numpy as np
import pytest
import torch

from oracle import attention as oa
from oracle import brute
from oracle import cache as oc

RNG = np.random.default_rng(1234)


torch.manual_seed(1234)  # the torch draws below are then the same on every run


def _rand(*shape, scale=1.0):
    return RNG.standard_normal(shape) * scale


# ---------------------------------------------------------------- bf16 conversion

def test_bf16_bits_exact_values():
    bits = np.array([0x3F80, 0xC000, 0x0000, 0x8000, 0x7F7F, 0x0001, 0x3EAB], dtype=np.uint16)
    got = oa.bf16_bits_to_f64(bits)
    want = [1.0, -2.0, 0.0, -0.0, (2 - 2 ** -7) * 2.0 ** 127, 2.0 ** -133,
            (1 + 0x2B / 128) * 2.0 ** -2]
    assert list(got) == want
    assert math.copysign(1, got[3]) == -1


def test_bf16_bits_match_torch_conversion():
    t = torch.randn(4096, dtype=torch.float32).to(torch.bfloat16)
    got = oa.bf16_bits_to_f64(t.view(torch.int16).numpy())
    assert np.array_equal(got, t.to(torch.float64).numpy())


# ---------------------------------------------------------------- brute force

@pytest.mark.parametrize("causal", [True, False])
@pytest.mark.parametrize("h_q,h_kv,S,r,dv", [(1, 1, 1, 1, 1), (2, 1, 5, 3, 4), (2, 2, 4, 2, 3),
                                             (4, 2, 3, 3, 2)])
def test_prefill_matches_brute_force(causal, h_q, h_kv, S, r, dv):
    q, k, v = _rand(1, h_q, S, r), _rand(1, h_kv, S, r), _rand(1, h_kv, S, dv)
    scale = 1 / math.sqrt(r)
    got = oa.attention_prefill(q, k, v, scale, causal=causal)
    want = np.array(brute.prefill(q.tolist(), k.tolist(), v.tolist(), scale, causal=causal))
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-13)


def test_weights_match_brute_force_and_sum_to_one():
    q, k, v = _rand(4, 3), _rand(6, 3), _rand(6, 5)
    out, w = oa.attention_head(q, k, v, 0.7, causal_offset=2, return_weights=True)
    bo, bw = brute.head(q.tolist(), k.tolist(), v.tolist(), 0.7, causal=False)
    # causal_offset=2: row i sees keys 0..i+2
    for i in range(4):
        n = i + 3
        _, bwi = brute.head(q[i:i + 1].tolist(), k[:n].tolist(), v[:n].tolist(), 0.7)
        np.testing.assert_allclose(w[i, :n], bwi[0], rtol=1e-12)
        assert np.all(w[i, n:] == 0)
    np.testing.assert_allclose(w.sum(axis=1), 1.0, rtol=0, atol=1e-14)
    assert np.all(w >= 0)


# ---------------------------------------------------------------- closed forms

def test_crafted_logits_give_one_to_two_weights():
    # r=1, q=1, scale=1: logits 0 and ln 2, so the weights are exactly 1/3 and 2/3.
    q = np.array([[1.0]])
    k = np.array([[0.0], [math.log(2.0)]])
    v = np.array([[3.0, -6.0], [9.0, 12.0]])
    out, w = oa.attention_head(q, k, v, 1.0, return_weights=True)
    np.testing.assert_allclose(w[0], [1 / 3, 2 / 3], rtol=1e-15)
    np.testing.assert_allclose(out[0], [(3 + 2 * 9) / 3, (-6 + 2 * 12) / 3], rtol=1e-15)


def test_scale_is_one_over_sqrt_r():
    # r=4, scale 1/sqrt(4): q.k = 2 ln 2 gives logit ln 2 (weights 1:2).  A dropped
    # scale would give 1:4, a scale of 1/r would give 1:sqrt(2).
    r = 4
    q = np.array([[1.0, 0.0, 0.0, 0.0]])
    k = np.array([[0.0, 5.0, 0.0, 0.0], [2 * math.log(2.0), 0.0, 0.0, 1.0]])
    v = np.array([[1.0], [4.0]])
    out = oa.attention_decode(q[None], k[None, None], v[None, None], [2], 1 / math.sqrt(r))
    assert abs(out[0, 0, 0] - (1 + 2 * 4) / 3) < 1e-14


def test_sign_of_scores():
    # The larger dot product must get the larger weight.
    q = np.array([[1.0, 1.0]])
    k = np.array([[1.0, 1.0], [-1.0, -1.0]])
    v = np.array([[1.0], [0.0]])
    out = oa.attention_head(q, k, v, 1.0)
    assert abs(out[0, 0] - math.exp(2) / (math.exp(2) + math.exp(-2))) < 1e-15


def test_zero_keys_give_mean_of_values():
    dv = 5
    v = _rand(1, 1, 9, dv)
    k = np.zeros((1, 1, 9, 3))
    q = _rand(1, 1, 9, 3)
    pre = oa.attention_prefill(q, k, v, 0.3, causal=True)
    for i in range(9):
        np.testing.assert_allclose(pre[0, 0, i], v[0, 0, :i + 1].mean(axis=0), rtol=1e-13,
                                   atol=1e-15)
    dec = oa.attention_decode(q[:, :, 0], k, v, [6], 0.3)
    np.testing.assert_allclose(dec[0, 0], v[0, 0, :6].mean(axis=0), rtol=1e-13, atol=1e-15)


def test_causal_row0_is_first_value_exactly():
    q, k, v = _rand(1, 2, 7, 4), _rand(1, 2, 7, 4), _rand(1, 2, 7, 6)
    out = oa.attention_prefill(q, k, v, 0.5, causal=True)
    assert np.array_equal(out[0, :, 0], v[0, :, 0])


def test_empty_context_gives_zero_row():
    q, k, v = _rand(2, 4, 8), _rand(2, 2, 5, 8), _rand(2, 2, 5, 16)
    out = oa.attention_decode(q, k, v, [0, 3], 0.35)
    assert np.all(out[0] == 0)
    assert np.all(out[1] != 0)


# ---------------------------------------------------------------- invariants

def test_prefill_row_equals_decode_with_prefix():
    B, hq, hkv, S, r, dv = 2, 4, 2, 11, 5, 7
    q, k, v = _rand(B, hq, S, r), _rand(B, hkv, S, r), _rand(B, hkv, S, dv)
    pre = oa.attention_prefill(q, k, v, 0.4, causal=True)
    for i in range(S):
        dec = oa.attention_decode(q[:, :, i], k, v, [i + 1] * B, 0.4)
        np.testing.assert_allclose(pre[:, :, i], dec, rtol=1e-13, atol=1e-15)
    rows = [(1, 3, 10), (0, 0, 0), (1, 2, 5)]
    got = oa.attention_prefill_rows(q, k, v, 0.4, rows)
    for n, (b, h, i) in enumerate(rows):
        np.testing.assert_allclose(got[n], pre[b, h, i], rtol=1e-13, atol=1e-15)


def test_gqa_equals_mha_with_repeated_kv_heads():
    B, hq, hkv, S, r, dv = 2, 8, 2, 6, 3, 4
    q, k, v = _rand(B, hq, S, r), _rand(B, hkv, S, r), _rand(B, hkv, S, dv)
    G = hq // hkv
    gqa = oa.attention_prefill(q, k, v, 0.6)
    mha = oa.attention_prefill(q, np.repeat(k, G, axis=1), np.repeat(v, G, axis=1), 0.6)
    assert np.array_equal(gqa, mha)
    # Query head h reads kv head h // G: heads of one group see the same keys.
    k2 = k.copy()
    k2[:, 1] *= 2.0   # (a uniform shift would cancel in the softmax)
    changed = oa.attention_prefill(q, k2, v, 0.6)
    assert np.array_equal(changed[:, :G], gqa[:, :G])
    assert not np.allclose(changed[:, G:], gqa[:, G:])


def test_paged_equals_contiguous():
    B, hq, hkv, r, dv, ps = 3, 4, 2, 4, 6, 4
    lens = [9, 1, 12]
    cap = 12
    q = _rand(B, hq, r)
    k, v = _rand(B, hkv, cap, r), _rand(B, hkv, cap, dv)
    n_pages = sum(-(-n // ps) for n in lens) + 2
    perm = RNG.permutation(n_pages)
    table = np.full((B, 3), -1)
    kp, vp = np.full((n_pages, hkv, ps, r), np.nan), np.full((n_pages, hkv, ps, dv), np.nan)
    pos = 0
    for b, n in enumerate(lens):
        for j in range(-(-n // ps)):
            page = perm[pos]
            pos += 1
            table[b, j] = page
            m = min(ps, n - j * ps)
            kp[page, :, :m] = k[b, :, j * ps:j * ps + m]
            vp[page, :, :m] = v[b, :, j * ps:j * ps + m]
    a = oa.attention_decode(q, k, v, lens, 0.5)
    p = oa.attention_decode_paged(q, kp, vp, table, lens, ps, 0.5)
    assert np.array_equal(a, p)
    for b, n in enumerate(lens):
        assert np.array_equal(oa.gather_pages(kp, table[b], n, ps), k[b, :, :n])


# ---------------------------------------------------------------- factored keys (Section 2.3)

def test_absorption_identity_exact_rank_factorisation():
    # W_K of exact rank r; truncated SVD gives W_K = A B with A = U_r S_r, B = V_r^T.
    d, dh, r, n = 24, 16, 4, 13
    W_K = _rand(d, r) @ _rand(r, dh)
    W_Q = _rand(d, dh)
    W_V = _rand(d, 10)
    U, sv, Vt = np.linalg.svd(W_K, full_matrices=False)
    A = U[:, :r] * sv[:r]
    Bm = Vt[:r]
    np.testing.assert_allclose(A @ Bm, W_K, rtol=0, atol=1e-12 * np.abs(W_K).max())
    x = _rand(n, d)
    q, k, v = x @ W_Q, x @ W_K, x @ W_V
    q_thin, k_thin = x @ (W_Q @ Bm.T), x @ A         # Eqs. thin_key / absorbed_query
    np.testing.assert_allclose(q_thin @ k_thin.T, q @ k.T, rtol=1e-10,
                               atol=1e-12 * np.abs(q @ k.T).max())
    scale = 1 / math.sqrt(dh)    # one explicit scale on both sides
    full = oa.attention_prefill(q[None, None], k[None, None], v[None, None], scale)
    thin = oa.attention_prefill(q_thin[None, None], k_thin[None, None], v[None, None], scale)
    np.testing.assert_allclose(thin, full, rtol=1e-10, atol=1e-12)
    # The full-key side also agrees with torch's library attention.
    t = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q)[None, None], torch.from_numpy(k)[None, None],
        torch.from_numpy(v)[None, None], is_causal=True, scale=scale)
    np.testing.assert_allclose(full, t.numpy(), rtol=1e-10, atol=1e-12)


# ---------------------------------------------------------------- library cross-check

def _sdpa(q, k, v, scale, causal):
    return torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q), torch.from_numpy(k), torch.from_numpy(v),
        is_causal=causal, scale=scale, enable_gqa=True).numpy()


@pytest.mark.parametrize("hq,hkv,S,r,dv", [(4, 4, 40, 128, 128),   # r = d_head: standard MHA
                                           (8, 2, 37, 32, 128),
                                           (12, 12, 33, 16, 64),
                                           (6, 3, 17, 5, 3)])
@pytest.mark.parametrize("causal", [True, False])
def test_prefill_matches_torch_sdpa(hq, hkv, S, r, dv, causal):
    q, k, v = _rand(2, hq, S, r), _rand(2, hkv, S, r), _rand(2, hkv, S, dv)
    scale = 1 / math.sqrt(r)
    np.testing.assert_allclose(oa.attention_prefill(q, k, v, scale, causal=causal),
                               _sdpa(q, k, v, scale, causal), rtol=1e-10, atol=1e-12)


def test_decode_matches_torch_sdpa_ragged():
    B, hq, hkv, cap, r, dv = 3, 8, 2, 50, 32, 128
    q, k, v = _rand(B, hq, r), _rand(B, hkv, cap, r), _rand(B, hkv, cap, dv)
    lens = [50, 7, 1]
    got = oa.attention_decode(q, k, v, lens, 1 / math.sqrt(r))
    for b, n in enumerate(lens):
        want = _sdpa(q[b:b + 1, :, None], k[b:b + 1, :, :n], v[b:b + 1, :, :n],
                     1 / math.sqrt(r), False)[:, :, 0]
        np.testing.assert_allclose(got[b:b + 1], want, rtol=1e-10, atol=1e-12)


# ---------------------------------------------------------------- prefill over a cache

def test_cached_prefill_reduces_to_prefill_and_decode():
    B, hq, hkv, S, r, dv = 2, 4, 2, 9, 8, 5
    L0 = [0, 6]
    n = max(L0) + S
    q = _rand(B, hq, S, r)
    k, v = _rand(B, hkv, n, r), _rand(B, hkv, n, dv)
    got = oa.attention_prefill_cached(q, k, v, L0, 0.3)
    # no cached tokens: the plain causal prefill of the chunk
    np.testing.assert_allclose(got[0], oa.attention_prefill(q[:1], k[:1, :, :S], v[:1, :, :S], 0.3)[0],
                               rtol=1e-13, atol=1e-14)
    # each row: decode over the L0 + i + 1 keys it may see
    for i in range(S):
        want = oa.attention_decode(q[:, :, i], k, v, [l0 + i + 1 for l0 in L0], 0.3)
        np.testing.assert_allclose(got[:, :, i], want, rtol=1e-13, atol=1e-14)
    # non-causal: every row sees all L0 + S keys
    full = oa.attention_prefill_cached(q, k, v, L0, 0.3, causal=False)
    for i in range(S):
        want = oa.attention_decode(q[:, :, i], k, v, [l0 + S for l0 in L0], 0.3)
        np.testing.assert_allclose(full[:, :, i], want, rtol=1e-13, atol=1e-14)


def test_cached_prefill_brute_force():
    q, k, v = _rand(1, 1, 3, 4), _rand(1, 1, 5, 4), _rand(1, 1, 5, 3)
    got = oa.attention_prefill_cached(q, k, v, [2], 0.5)
    for i in range(3):
        want = brute.head([q[0, 0, i].tolist()], k[0, 0, :3 + i].tolist(),
                          v[0, 0, :3 + i].tolist(), 0.5)[0][0]
        np.testing.assert_allclose(got[0, 0, i], want, rtol=1e-12, atol=1e-14)


# ---------------------------------------------------------------- backward

@pytest.mark.parametrize("causal", [True, False])
def test_backward_matches_torch_autograd(causal):
    """Independent route: torch autograd through an fp64 softmax attention."""
    B, hq, hkv, S, r, dv = 2, 4, 2, 11, 6, 5
    q, k, v, do = _rand(B, hq, S, r), _rand(B, hkv, S, r), _rand(B, hkv, S, dv), _rand(B, hq, S, dv)
    dq, dk, dv_ = oa.attention_backward(q, k, v, do, 0.37, causal)
    tq, tk, tv = (torch.tensor(x, requires_grad=True) for x in (q, k, v))
    G = hq // hkv
    kk, vv = tk.repeat_interleave(G, dim=1), tv.repeat_interleave(G, dim=1)
    s = 0.37 * tq @ kk.transpose(-1, -2)
    if causal:
        s = s.masked_fill(torch.triu(torch.ones(S, S, dtype=torch.bool), 1), float("-inf"))
    out = torch.softmax(s, dim=-1) @ vv
    (out * torch.tensor(do)).sum().backward()
    np.testing.assert_allclose(dq, tq.grad.numpy(), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(dk, tk.grad.numpy(), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(dv_, tv.grad.numpy(), rtol=1e-11, atol=1e-12)


def test_backward_finite_differences():
    B, hq, hkv, S, r, dv = 1, 2, 1, 5, 3, 2
    q, k, v, do = _rand(B, hq, S, r), _rand(B, hkv, S, r), _rand(B, hkv, S, dv), _rand(B, hq, S, dv)
    grads = oa.attention_backward(q, k, v, do, 0.8)

    def loss(qq, kk, vv):
        return float(np.sum(oa.attention_prefill(qq, kk, vv, 0.8) * do))
    eps = 1e-6
    for idx, (x, gx) in enumerate(zip((q, k, v), grads)):
        for pos in [(0, 0, 2, 1), (0, hq - 1 if idx == 0 else 0, 4, 0), (0, 0, 0, dv - 1 if idx == 2 else 0)]:
            xp, xm = x.copy(), x.copy()
            xp[pos] += eps
            xm[pos] -= eps
            args_p = [q, k, v]; args_p[idx] = xp
            args_m = [q, k, v]; args_m[idx] = xm
            num = (loss(*args_p) - loss(*args_m)) / (2 * eps)
            assert abs(num - gx[pos]) <= 1e-7 * max(1.0, abs(num))


def test_logsumexp_rows():
    q, k = _rand(1, 2, 7, 4), _rand(1, 1, 7, 4)
    lse = oa.logsumexp_rows(q, k, 0.5)
    for h in range(2):
        for i in range(7):
            s = 0.5 * (q[0, h, i] @ k[0, 0, :i + 1].T)
            assert lse[0, h, i] == pytest.approx(math.log(math.fsum(math.exp(x) for x in s)), rel=1e-13)


# ---------------------------------------------------------------- int8 keys

def test_quantiser_ties_round_to_even():
    # amax 127 gives scale exactly 1, so codes are rint(k): ties go to the even code.
    k = np.array([[127.0, 2.5, 3.5, -2.5, 0.5, 1.5, -0.5, -127.0]], dtype=np.float32)
    codes, sc = oc.quantize_int8_per_token(k)
    assert sc[0] == np.float32(1.0)
    assert codes.tolist() == [[127, 2, 4, -2, 0, 2, 0, -127]]


def test_quantiser_closed_form_and_bounds():
    k = torch.randn(64, 8, 32).to(torch.bfloat16).float().numpy()
    codes, sc = oc.quantize_int8_per_token(k)
    amax = np.abs(k).max(axis=-1)
    assert np.array_equal(sc, (amax / np.float32(127)).astype(np.float32))
    assert codes.dtype == np.int8 and np.abs(codes.astype(int)).max() <= 127
    # the largest |k| of each row maps to +-127 with its sign
    idx = np.abs(k).argmax(axis=-1)
    top = np.take_along_axis(codes, idx[..., None], -1)[..., 0]
    assert np.array_equal(np.abs(top.astype(int)), np.full(top.shape, 127))
    assert np.array_equal(np.sign(top), np.sign(np.take_along_axis(k, idx[..., None], -1)[..., 0]))
    # reconstruction error at most half a step (plus binary32 division rounding)
    err = np.abs(k - codes * sc[..., None].astype(np.float64))
    assert np.all(err <= sc[..., None] * (0.5 + 1e-5))
    # odd symmetry
    c2, s2 = oc.quantize_int8_per_token(-k)
    assert np.array_equal(c2, -codes) and np.array_equal(s2, sc)


def test_quantiser_zero_row():
    codes, sc = oc.quantize_int8_per_token(np.zeros((2, 16), dtype=np.float32))
    assert np.all(codes == 0) and np.all(sc == 0)


def test_int8_attention_uses_dequantised_keys():
    B, hq, hkv, cap, r, dv = 2, 4, 2, 30, 16, 8
    g = torch.Generator().manual_seed(40)
    kf = torch.randn(B, hkv, cap, r, generator=g).to(torch.bfloat16).float().numpy()
    codes, sc = oc.quantize_int8_per_token(kf)
    q, v = _rand(B, hq, r), _rand(B, hkv, cap, dv)
    lens = [30, 13]
    got = oa.attention_decode(q, codes, v, lens, 0.25, k_scale=sc)
    deq = codes.astype(np.float64) * sc[..., None].astype(np.float64)
    assert np.array_equal(got, oa.attention_decode(q, deq, v, lens, 0.25))
    # close to the unquantised-key result (keys move by at most half a step)
    ref = oa.attention_decode(q, kf, v, lens, 0.25)
    assert np.abs(got - ref).max() < 0.05


# ---------------------------------------------------------------- int4 keys

def test_int4_quantiser_ties_round_to_even():
    # amax 7 gives scale exactly 1, so codes are rint(k): ties go to the even code.
    k = np.array([[7.0, 2.5, 3.5, -2.5, 0.5, 1.5, -0.5, -7.0]], dtype=np.float32)
    codes, sc = oc.quantize_int4_per_token(k)
    assert sc[0] == np.float32(1.0)
    assert codes.tolist() == [[7, 2, 4, -2, 0, 2, 0, -7]]


def test_int4_quantiser_closed_form_and_bounds():
    k = torch.randn(64, 8, 32).to(torch.bfloat16).float().numpy()
    codes, sc = oc.quantize_int4_per_token(k)
    amax = np.abs(k).max(axis=-1)
    assert np.array_equal(sc, (amax / np.float32(7)).astype(np.float32))
    assert np.abs(codes.astype(int)).max() <= 7
    idx = np.abs(k).argmax(axis=-1)
    top = np.take_along_axis(codes, idx[..., None], -1)[..., 0]
    assert np.array_equal(np.abs(top.astype(int)), np.full(top.shape, 7))
    err = np.abs(k - codes * sc[..., None].astype(np.float64))
    assert np.all(err <= sc[..., None] * (0.5 + 1e-5))
    c2, s2 = oc.quantize_int4_per_token(-k)
    assert np.array_equal(c2, -codes) and np.array_equal(s2, sc)
    z, zs = oc.quantize_int4_per_token(np.zeros((2, 32), dtype=np.float32))
    assert np.all(z == 0) and np.all(zs == 0)


def test_int4_packing():
    # element 2j in the low nibble, 2j+1 in the high nibble, two's complement
    codes = np.array([[1, -1, 7, -7, 0, -8]], dtype=np.int8)
    packed = oc.pack_int4(codes)
    assert packed.tolist() == [[0xF1, 0x97, 0x80]]
    assert np.array_equal(oc.unpack_int4(packed), codes)
    rnd = np.random.default_rng(3).integers(-8, 8, size=(5, 4, 64)).astype(np.int8)
    assert np.array_equal(oc.unpack_int4(oc.pack_int4(rnd)), rnd)
    assert oc.pack_int4(rnd).shape == (5, 4, 32)


def test_int4_attention_uses_dequantised_keys():
    B, hq, hkv, cap, r, dv = 2, 4, 2, 30, 32, 8
    g = torch.Generator().manual_seed(41)
    kf = torch.randn(B, hkv, cap, r, generator=g).to(torch.bfloat16).float().numpy()
    codes, sc = oc.quantize_int4_per_token(kf)
    q, v = _rand(B, hq, r), _rand(B, hkv, cap, dv)
    lens = [30, 13]
    got = oa.attention_decode(q, oc.unpack_int4(oc.pack_int4(codes)), v, lens, 0.25, k_scale=sc)
    deq = codes.astype(np.float64) * sc[..., None].astype(np.float64)
    assert np.array_equal(got, oa.attention_decode(q, deq, v, lens, 0.25))
    # If every score of a row moves by at most D, every softmax weight ratio
    # moves by at most exp(2D), so sum_j |p'_j - p_j| <= exp(2D) - 1 and the
    # output moves by at most max|v| times that.
    ref = oa.attention_decode(q, kf, v, lens, 0.25)
    G = hq // hkv
    for b in range(B):
        n = lens[b]
        for h in range(hq):
            dk = deq[b, h // G, :n] - kf[b, h // G, :n]
            D = 0.25 * np.abs(dk @ q[b, h]).max()
            bound = np.abs(v[b, h // G, :n]).max() * (np.exp(2 * D) - 1)
            assert np.abs(got[b, h] - ref[b, h]).max() <= bound + 1e-12


def test_append_contiguous_and_paged_agree():
    B, hkv, r, dv, ps, cap = 2, 2, 8, 4, 4, 16
    lens = np.array([3, 9])
    T = 5
    kn = torch.randn(B, hkv, T, r).to(torch.bfloat16).float().numpy()
    vn = torch.randn(B, hkv, T, dv).to(torch.bfloat16).float().numpy()
    for bits in (16, 8, 4):
        int8 = bits < 16
        kw = r // 2 if bits == 4 else r
        kdt = np.float64 if bits == 16 else (np.int8 if bits == 8 else np.uint8)
        kc = np.zeros((B, hkv, cap, kw), dtype=kdt)
        vc = np.zeros((B, hkv, cap, dv))
        ksc = np.zeros((B, hkv, cap), dtype=np.float32) if int8 else None
        oc.append_contiguous(kc, vc, lens, kn, vn, ksc, k_bits=4 if bits == 4 else 8)
        table = np.array([[5, 1, 7, 3], [0, 2, 4, 6]])
        kp = np.zeros((8, hkv, ps, kw), dtype=kc.dtype)
        vp = np.zeros((8, hkv, ps, dv))
        ksp = np.zeros((8, hkv, ps), dtype=np.float32) if int8 else None
        oc.append_paged(kp, vp, table, lens, ps, kn, vn, ksp, k_bits=4 if bits == 4 else 8)
        if bits == 4:
            codes, sc = oc.quantize_int4_per_token(kn)
            assert np.array_equal(oc.unpack_int4(kc[1, :, 9:14]), codes[1])
            assert np.array_equal(ksc[1, :, 9:14], sc[1])
        for b in range(B):
            n = lens[b] + T
            assert np.array_equal(oa.gather_pages(kp, table[b], n, ps)[:, lens[b]:],
                                  kc[b, :, lens[b]:n])
            assert np.array_equal(oa.gather_pages(vp, table[b], n, ps)[:, lens[b]:],
                                  vc[b, :, lens[b]:n])
            if int8:
                assert np.array_equal(oa.gather_pages(ksp[..., None], table[b], n, ps)[:, lens[b]:, 0],
                                      ksc[b, :, lens[b]:n])
        assert np.array_equal(vc[0, :, 3:8], vn[0])
    with pytest.raises(ValueError):
        oc.append_contiguous(np.zeros((1, 1, 4, 2)), np.zeros((1, 1, 4, 2)), [3],
                             np.zeros((1, 1, 2, 2)), np.zeros((1, 1, 2, 2)))


# ---------------------------------------------------------------- int4 scale grouping

def test_int4_per_group_reduces_to_per_token_and_is_groupwise():
    """One group spanning the row is the per-token quantiser; smaller groups
    quantise each group on its own (a group's codes ignore the other groups)."""
    rng = np.random.default_rng(31)
    k = rng.standard_normal((3, 5, 64)).astype(np.float32)
    c_tok, s_tok = oc.quantize_int4_per_token(k)
    c_g, s_g = oc.quantize_int4_per_group(k, 64)
    assert np.array_equal(c_g, c_tok) and np.array_equal(s_g[..., 0], s_tok)
    c32, s32 = oc.quantize_int4_per_group(k, 32)
    assert s32.shape == (3, 5, 2)
    for h in range(2):
        ch, sh = oc.quantize_int4_per_token(k[..., 32 * h:32 * h + 32])
        assert np.array_equal(c32[..., 32 * h:32 * h + 32], ch) and np.array_equal(s32[..., h], sh)
    # dequantised error within half a step of each channel's own group scale
    err = np.abs(oc.dequantize_per_group(c32, s32) - k)
    assert np.all(err <= np.repeat(s32, 32, axis=-1) / 2 + 1e-7)
    with pytest.raises(ValueError):
        oc.quantize_int4_per_group(k, 48)


def int4_grouping_errors(r, group, seed=0, n_q=64, n_k=2048, dv=64):
    """Mean relative error (sum|out - ref| / sum|ref|) of decode attention over int4 keys,
    one scale per token vs one per `group` channels, against the unquantised keys."""
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((n_q, r))
    k = rng.standard_normal((n_k, r)).astype(np.float32)
    v = rng.standard_normal((n_k, dv))
    scale = 1 / math.sqrt(r)
    ref = oa.attention_head(q, k.astype(np.float64), v, scale)
    c_t, s_t = oc.quantize_int4_per_token(k)
    c_g, s_g = oc.quantize_int4_per_group(k, group)
    out_t = oa.attention_head(q, oa.dequantize_keys(c_t, s_t), v, scale)
    out_g = oa.attention_head(q, oc.dequantize_per_group(c_g, s_g), v, scale)
    rel = lambda o: float(np.abs(o - ref).sum() / np.abs(ref).sum())
    return rel(out_t), rel(out_g)


@pytest.mark.parametrize("r", [64, 128])
def test_int4_per_token_scale_costs_little_accuracy(r):
    """The library stores one fp32 scale per token.  Groups of 32 channels would cut
    the attention error (the largest |k| of 32 channels is smaller than of r), at the
    price of r / 32 scales per token; measured here on N(0,1) keys and queries."""
    e_tok, e_grp = int4_grouping_errors(r, 32, seed=r)
    print(f"\n[int4 scale grouping] r={r}: mean rel error per token {e_tok:.4f}, "
          f"per 32 channels {e_grp:.4f} (ratio {e_tok / e_grp:.2f})")
    assert e_grp < e_tok < 2.0 * e_grp
