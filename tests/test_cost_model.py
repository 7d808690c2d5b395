"""Pins of the byte / FLOP model against the numbers the paper prints.

Expected values come from tests/golden/paper_tables.json (each block cites
its table).  Tolerances are the printed rounding: half a unit of the last
printed digit, unless a note says the paper rounded differently.
"""

import json
import os

import pytest

from paper_2603_04427_gb300 import cost_model as cm

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_tables.json")))


def test_kvcache_per_user_128k():
    t = GOLD["kvcache_per_user"]
    c = t["ctx_128k"]
    n, d, L, b = c["n_tokens"], t["d_model"], t["n_layers"], t["bytes_per"]
    std = cm.kv_cache_bytes(n, d, L, b)
    half = cm.kv_cache_bytes(n, d, L, b, d_select=d // 2)
    quarter = cm.kv_cache_bytes(n, d, L, b, d_select=d // 4)
    for got, want in ((std, c["standard"]), (half, c["d_half"]), (quarter, c["d_quarter"])):
        for key in ("k", "v"):
            assert abs(got[key] / 1e9 - want[key]) <= 0.05, (key, got[key], want)
        # The printed totals are sums of the rounded K and V figures
        # (33.6 + 33.6 = 67.2, while the unrounded total is 67.1 GB).
        assert abs(round(got["k"] / 1e9, 1) + round(got["v"] / 1e9, 1) - want["total"]) < 1e-9
    for got, want in ((half, c["d_half"]), (quarter, c["d_quarter"])):
        saved = std["total"] - got["total"]
        assert abs(saved / 1e9 - want["saved"]) <= 0.05
        assert abs(100 * saved / std["total"] - want["saved_pct"]) <= 1e-9


def test_kvcache_per_user_1m():
    t = GOLD["kvcache_per_user"]
    c = t["ctx_1m"]
    n, d, L, b = c["n_tokens"], t["d_model"], t["n_layers"], t["bytes_per"]
    std = cm.kv_cache_bytes(n, d, L, b)["total"] / 1e9
    half = cm.kv_cache_bytes(n, d, L, b, d_select=d // 2)["total"] / 1e9
    quarter = cm.kv_cache_bytes(n, d, L, b, d_select=d // 4)["total"] / 1e9
    assert abs(std - c["standard"]["total"]) <= 0.5
    assert abs(half - c["d_half"]["total"]) <= 0.5
    assert abs(quarter - c["d_quarter"]["total"]) <= 0.5
    # The printed savings are differences of the rounded totals (524 - 328 = 196,
    # while the unrounded difference is 196.6): compare with those.
    assert round(std) - round(half) == c["d_half"]["saved"]
    assert round(std) - round(quarter) == c["d_quarter"]["saved"]


def test_kv_7b_analytical_table():
    t = GOLD["kv_7b_analytical"]
    n, L, H, dh, b = t["n_tokens"], t["n_layers"], t["n_heads"], t["d_head"], t["bytes_per"]
    gib = 2.0 ** 30

    def kv(k_width, v_width):
        k = n * k_width * L * b / gib
        v = n * v_width * L * b / gib
        return k, v, k + v

    mha = kv(H * dh, H * dh)
    rows = {"mha": mha, "thin_quarter": kv(H * dh // 4, H * dh), "gqa8": kv(8 * dh, 8 * dh),
            "gqa8_thin": kv(8 * dh // 4, 8 * dh)}
    for name, (k, v, tot) in rows.items():
        want = t[name]
        assert abs(k - want["k"]) <= 0.05 and abs(v - want["v"]) <= 0.05
        assert abs(tot - want["total"]) <= 0.05
        if "saved_pct" in want:
            assert abs(100 * (1 - tot / mha[2]) - want["saved_pct"]) <= 0.05
    mla = n * (t["mla"]["d_c"] + t["mla"]["d_rope"]) * L * b / gib
    assert abs(mla - t["mla"]["total"]) <= 0.05
    assert abs(100 * (1 - mla / mha[2]) - t["mla"]["saved_pct"]) <= 0.05


def test_mistral_cache_and_weight_bytes():
    t = GOLD["mistral_decode_model"]
    ckv = cm.c_kv(t["n_layers"], t["n_kv_heads"], t["d_head"], t["n_ctx"], t["beta"])
    assert ckv == 2 * 32 * 8 * 128 * 4096 * 2 == 536_870_912
    assert abs(ckv / 1e6 - t["C_kv_MB"]) <= 0.5
    r256 = 256 // t["n_kv_heads"]
    thin = cm.c_kv_thin(t["n_layers"], t["n_kv_heads"], r256, t["d_head"], t["n_ctx"], t["beta"])
    assert thin == 335_544_320
    assert abs(thin / 1e6 - t["C_kv_thin_r256_MB"]) <= 0.5
    saved = cm.projection_bytes_saved(t["d_model"], t["n_q_heads"], t["n_kv_heads"],
                                      t["d_head"], r256, t["n_layers"], t["beta"])
    assert abs((t["W_GB"] * 1e9 - saved) / 1e9 - t["W_thin_r256_GB"]) <= 0.05
    assert abs(ckv / thin - t["max_speedup_r256"]) <= 0.005


@pytest.mark.parametrize("rank,key", [(256, "predicted_speedup_r256"),
                                      (512, "predicted_speedup_r512")])
def test_mistral_predicted_speedups(rank, key):
    t = GOLD["mistral_decode_model"]
    r = rank // t["n_kv_heads"]
    ckv = cm.c_kv(t["n_layers"], t["n_kv_heads"], t["d_head"], t["n_ctx"], t["beta"])
    thin = cm.c_kv_thin(t["n_layers"], t["n_kv_heads"], r, t["d_head"], t["n_ctx"], t["beta"])
    W = t["W_GB"] * 1e9
    # W' for r256 is printed (13.2 GB); for r512 it is not, and is derived from
    # the projection sizes of Section 2.3 (14.2 GB - 0.67 GB).
    W_thin = (t["W_thin_r256_GB"] * 1e9 if rank == 256 else
              W - cm.projection_bytes_saved(t["d_model"], t["n_q_heads"], t["n_kv_heads"],
                                            t["d_head"], r, t["n_layers"], t["beta"]))
    for b, want in zip(t["batches"], t[key]):
        got = cm.decode_speedup(W, ckv, W_thin, thin, b)
        # The paper prints 1.17 at b=8 for r256 where the model gives 1.164; allow 0.01.
        assert abs(got - want) <= 0.01, (rank, b, got, want)


def test_prefill_flops_appendix_e():
    t = GOLD["prefill_flops"]
    f = cm.prefill_flops(1, t["n_heads"], t["seq"], t["d_head"], t["d_head"], causal=True)
    assert abs(f / 1e9 - t["gflop"]) <= 0.5


def test_decode_bytes_configs():
    # Mistral-shaped GQA decode, B=16, every sequence at 4096 tokens: 167.8 MB.
    assert cm.decode_kv_bytes([4096] * 16, 8, 32, 128) == 16 * 8 * 4096 * (64 + 256)
    # int8 keys with an fp32 scale per token and kv head, B=64, context 32768.
    b = cm.decode_kv_bytes([32768] * 64, 8, 32, 128, k_bytes=1, k_scale_bytes=4)
    assert b == 64 * 8 * 32768 * (32 + 4 + 256)
    # Prefill, B=2, H=32, S=8192, r=32, d_v=128: 6.873e11 FLOPs.
    assert abs(cm.prefill_flops(2, 32, 8192, 32, 128) - 6.873e11) / 6.873e11 < 1e-3


def test_llama125m_parameter_counts():
    # Thinning W_Q and W_K to d_select columns removes 2 d_model (d_model - d_select)
    # weights per layer; W_V and everything else is unchanged (Experiment 6).
    t = GOLD["llama125m_params"]
    d, H, L = t["d_model"], t["n_heads"], t["n_layers"]
    base = t["rows"][0]["params_M"]
    for row in t["rows"]:
        r = row["d_select"] // H
        assert r == row["per_head"]
        saved = cm.projection_bytes_saved(d, H, H, d // H, r, L, beta=1)
        assert saved == 2 * L * d * (d - row["d_select"])
        # both the baseline and the row are printed to 0.1 M
        assert abs(base - saved / 1e6 - row["params_M"]) <= 0.1, (row, saved)
        # "QK saved" = 1 - d_select / d_model; 87.5 % is printed as 87, so allow half a unit
        assert abs(100 * (1 - row["d_select"] / d) - row["qk_saved_pct"]) <= 0.5


def test_kv_methods_budget_per_token_and_layer():
    t = GOLD["kv_methods_budget"]
    d, H, dh, L = t["d_model"], t["n_heads"], t["d_head"], t["n_layers"]
    full = cm.c_kv(1, H, dh, 1, beta=1)
    assert full == t["mha"]["kv_budget"]
    assert cm.kv_cache_bytes(1, d, 1, 1)["total"] == full
    for row in t["thin"]:
        r = row["d_select"] // H
        got = cm.c_kv_thin(1, H, r, dh, 1, beta=1)
        assert got == row["kv_budget"] == cm.kv_cache_bytes(1, d, 1, 1, d_select=row["d_select"])["total"]
        assert abs(100 * (1 - got / full) - row["saved_pct"]) <= 0.05
        saved = cm.projection_bytes_saved(d, H, H, dh, r, L, beta=1)
        assert abs(t["mha"]["params_M"] - saved / 1e6 - row["params_M"]) <= 0.1
    for row in t["gqa"]:
        got = cm.c_kv(1, row["n_kv_heads"], dh, 1, beta=1)
        assert got == row["kv_budget"]
        assert abs(100 * (1 - got / full) - row["saved_pct"]) <= 0.05
