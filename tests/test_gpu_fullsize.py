"""Full-size parity: the benchmark's launch configurations against the oracle.

Each workload runs at the size and in the launch configuration the benchmark
times, and the fp64 oracle computes the checked outputs one by one:

* 7B MHA causal prefill (B=2, H=32, S=8192, r=32, d_v=128, bf16 output):
  one row of EVERY 128-row query tile of every (sequence, head) plane (4096
  rows, so every CTA of the launch is checked; the row's offset inside its
  tile varies from tile to tile and covers the first and last row of a
  tile), plus one whole plane element by element.  Both numbers are also
  reported against the unrounded oracle (the literal bar).
* long-context paged decode (B=4, contexts U[65536, 131072], 64-token pages):
  all 128 (sequence, query head) pairs.
* quantised-key decode (B=64, H_q=32, H_kv=8, context 32768) at every r of
  the sweep {16, 32, 64, 128}, int8 keys and (r >= 32) int4 keys: the stored
  codes and scales of sampled (sequence, kv head) groups bit for bit against
  the oracle's quantiser, and all G query heads of those groups against the
  oracle on the dequantised keys.

Sampling seeds are fixed in the tests.
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


def _mean_rel(got, ref):
    got, ref = np.asarray(got, np.float64), np.asarray(ref, np.float64)
    return float(np.abs(got - ref).sum() / np.abs(ref).sum()), float(np.abs(got - ref).max())


# ------------------------------------------------------------------ 7B MHA prefill

def test_7b_mha_prefill_every_tile_and_one_plane():
    require_gpu()
    B, H, S, r, dv = 2, 32, 8192, 32, 128
    scale = 1 / math.sqrt(r)
    q = inputs.normal_bf16((B, H, S, r), 1002, device="cuda")
    k = inputs.normal_bf16((B, H, S, r), 1003, device="cuda")
    v = inputs.normal_bf16((B, H, S, dv), 1004, device="cuda")
    out = torch.full((B, H, S, dv), float("nan"), dtype=torch.bfloat16, device="cuda")
    tb.tk_attn_prefill(q, k, v, out)
    assert tb.tk_get_device_error() == 0
    assert torch.isfinite(out.float()).all()
    qh, kh, vh, oh = q.cpu(), k.cpu(), v.cpu(), out.cpu()
    n_tiles = S // 128
    got, ref = [], []
    for b in range(B):
        for h in range(H):
            plane = b * H + h
            # row of tile t: its offset cycles through the tile with the plane and
            # the tile (offsets 0 and 127 both occur in every plane)
            rows = [t * 128 + (t * 37 + plane * 11) % 128 for t in range(n_tiles)]
            rows[0], rows[-1] = 0, S - 1
            rows[1], rows[2] = 128 + 127, 256       # last / first row of a tile boundary
            qq = f64(qh[b, h])[None, None]
            kk = f64(kh[b, h])[None, None]
            vv = f64(vh[b, h])[None, None]
            ref.append(oa.attention_prefill_rows(qq, kk, vv, scale, [(0, 0, i) for i in rows]))
            got.append(f64(oh[b, h, rows]))
    got, ref = np.concatenate(got), np.concatenate(ref)
    err_r = parity_bf16(got, ref, what="7b prefill, one row of every query tile")
    lit = _mean_rel(got, ref)
    # one whole plane, element by element, in chunks of 1024 query rows
    b, h = 1, 17
    qq, kk, vv = f64(qh[b, h]), f64(kh[b, h]), f64(vh[b, h])
    ref_p = np.concatenate([oa.attention_head(qq[c:c + 1024], kk[:c + 1024], vv[:c + 1024], scale,
                                              causal_offset=c) for c in range(0, S, 1024)])
    got_p = f64(oh[b, h])
    err_p = parity_bf16(got_p, ref_p, what=f"7b prefill, whole plane (b={b}, h={h})")
    lit_p = _mean_rel(got_p, ref_p)
    print(f"\n[C3 parity] every-tile rows: vs bf16-rounded oracle max abs {err_r[0]:.3e} "
          f"mean rel {err_r[1]:.3e}; vs unrounded oracle max abs {lit[1]:.3e} mean rel {lit[0]:.3e}"
          f"\n[C3 parity] whole plane: vs bf16-rounded oracle max abs {err_p[0]:.3e} "
          f"mean rel {err_p[1]:.3e}; vs unrounded oracle max abs {lit_p[1]:.3e} "
          f"mean rel {lit_p[0]:.3e}")


# ------------------------------------------------------------------ paged long-context decode

def test_long_context_paged_decode_all_pairs():
    require_gpu()
    B, hq, hkv, r, dv, ps = 4, 32, 8, 32, 128, 64
    G = hq // hkv
    lens = inputs.uniform_lengths(B, 65536, 131072, seed=1003)
    table, n_pages = inputs.paged_layout(lens, ps, seed=1004)
    pc = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, page_size=ps, num_pages=n_pages,
                                  page_table=table)
    pc.k.copy_(inputs.normal_bf16(pc.k.shape, 1005, device="cuda"))
    pc.v.copy_(inputs.normal_bf16(pc.v.shape, 1006, device="cuda"))
    q = inputs.normal_bf16((B, hq, r), seed=1007, device="cuda")
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    ws = tb.decode_workspace(pc.desc, max(lens))
    out = torch.full((B, hq, dv), float("nan"), device="cuda")
    tb.tk_attn_decode(pc, q, sl, max(lens), out, ws)
    assert tb.tk_get_device_error() == 0
    tab = table.numpy()
    got, ref = [], []
    for b in range(B):
        pages = torch.from_numpy(tab[b, :-(-lens[b] // ps)].astype(np.int64)).cuda()
        for g in range(hkv):
            # the oracle's explicit gather: logical token t is slot t % 64 of page t // 64
            kk = f64(pc.k[pages, g].reshape(-1, r)[:lens[b]])
            vv = f64(pc.v[pages, g].reshape(-1, dv)[:lens[b]])
            ref.append(oa.attention_head(f64(q[b, g * G:(g + 1) * G]), kk, vv, 1 / math.sqrt(r)))
            got.append(f64(out[b, g * G:(g + 1) * G]))
    parity(np.concatenate(got), np.concatenate(ref), what="paged long context, all 128 pairs")


# ------------------------------------------------------------------ quantised keys, r sweep

@pytest.mark.parametrize("kfmt,r", [("int8", 16), ("int8", 32), ("int8", 64), ("int8", 128),
                                    ("int4", 32), ("int4", 64), ("int4", 128)])
def test_quantised_key_decode_r_sweep(kfmt, r):
    require_gpu()
    B, hq, hkv, dv, L = 64, 32, 8, 128, 32768
    G = hq // hkv
    seed = 1011 + r + (0 if kfmt == "int8" else 500)
    cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=L, k_int8=kfmt == "int8",
                                     k_int4=kfmt == "int4")
    kn = inputs.normal_bf16((B, hkv, L, r), seed, device="cuda")
    tb.tk_kv_append(cache, kn, inputs.normal_bf16((B, hkv, L, dv), seed + 1, device="cuda"),
                    torch.zeros(B, dtype=torch.int32, device="cuda"))
    q = inputs.normal_bf16((B, hq, r), seed + 2, device="cuda")
    sl = torch.full((B,), L, dtype=torch.int32, device="cuda")
    out = torch.full((B, hq, dv), float("nan"), device="cuda")
    tb.tk_attn_decode(cache, q, sl, L, out, tb.decode_workspace(cache.desc, L))
    assert tb.tk_get_device_error() == 0
    assert torch.isfinite(out).all()
    quant = oc.quantize_int8_per_token if kfmt == "int8" else oc.quantize_int4_per_token
    rng = np.random.default_rng(seed)
    got, ref = [], []
    groups = [(0, 0), (B - 1, hkv - 1)] + [(int(b), int(g)) for b, g in
                                            zip(rng.integers(0, B, 6), rng.integers(0, hkv, 6))]
    for b, g in groups:
        codes, sc = quant(kn[b, g].float().cpu().numpy())
        stored = cache.k[b, g].cpu().numpy()
        assert np.array_equal(stored, codes if kfmt == "int8" else oc.pack_int4(codes))
        assert np.array_equal(cache.k_scale[b, g].cpu().numpy().view(np.uint32), sc.view(np.uint32))
        kk = oa.dequantize_keys(codes, sc)
        ref.append(oa.attention_head(f64(q[b, g * G:(g + 1) * G]), kk, f64(cache.v[b, g]),
                                     1 / math.sqrt(r)))
        got.append(f64(out[b, g * G:(g + 1) * G]))
    parity(np.concatenate(got), np.concatenate(ref), what=f"{kfmt} keys r={r}, full size")


# ------------------------------------------------------------------ GPT-2-small layer

def test_gpt2_small_layer_prefill_then_32_decode_steps():
    """The GPT-2-small-shaped layer as the benchmark runs it: causal prefill of 256
    tokens (fp32 out), the prompt appended, then 32 fused append + decode steps;
    every output element of every step against the oracle."""
    require_gpu()
    B, H, r, dv, S, T = 1, 12, 16, 64, 256, 32
    scale = 1 / math.sqrt(r)
    q = inputs.normal_bf16((B, H, S, r), 2001, device="cuda")
    k = inputs.normal_bf16((B, H, S, r), 2002, device="cuda")
    v = inputs.normal_bf16((B, H, S, dv), 2003, device="cuda")
    pre = torch.empty(B, H, S, dv, device="cuda")
    tb.tk_attn_prefill(q, k, v, pre)
    parity(f64(pre), oa.attention_prefill(f64(q), f64(k), f64(v), scale), what="gpt2 layer prefill")
    cache = tb.ThinKeyCache.allocate(B, H, H, r, dv, capacity=S + T)
    tb.tk_kv_append(cache, k, v, torch.zeros(B, dtype=torch.int32, device="cuda"))
    ws = tb.decode_workspace(cache.desc, S + T)
    kk, vv = f64(k)[0], f64(v)[0]
    for t in range(T):
        qd = inputs.normal_bf16((B, H, r), 2100 + 3 * t, device="cuda")
        k1 = inputs.normal_bf16((B, H, r), 2101 + 3 * t, device="cuda")
        v1 = inputs.normal_bf16((B, H, dv), 2102 + 3 * t, device="cuda")
        out = torch.empty(B, H, dv, device="cuda")
        sl = torch.full((B,), S + t, dtype=torch.int32, device="cuda")
        tb.tk_attn_decode_append(cache, qd, k1, v1, sl, S + T, out, ws)
        kk = np.concatenate([kk, f64(k1)[0][:, None]], axis=1)
        vv = np.concatenate([vv, f64(v1)[0][:, None]], axis=1)
        ref = oa.attention_decode(f64(qd), kk[None], vv[None], [S + t + 1], scale)
        parity(f64(out), ref, what=f"gpt2 layer decode step {t}")
    assert tb.tk_get_device_error() == 0
