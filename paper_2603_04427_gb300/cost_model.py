"""Byte and FLOP accounting for thin-key attention (pure arithmetic, no GPU).

* KV cache size, paper Section 2.4, Eqs. 8-9:
      standard   = 2 * n * d_model * L * b
      asymmetric = n * (d_select + d_model) * L * b
* Decode bandwidth model, paper Section 4.2, Eq. (roofline):
      bytes/step = W + batch * C_kv,  C_kv = 2 * L * n_kv * d_head * n * beta
      speedup(batch) = (W + batch * C_kv) / (W' + batch * C'_kv)
  with the thin-key cache C'_kv = L * n_kv * (r + d_head) * n * beta.
* Prefill attention FLOPs (paper Appendix E): 2 FLOPs per multiply-add,
  r multiply-adds for a score and d_v for the weighted sum, over the
  unmasked (query, key) pairs only.

The per-launch "algorithmic" figures the benchmark divides by kernel time
come from ``decode_kv_bytes`` and ``prefill_flops``.
"""

from __future__ import annotations


def kv_cache_bytes(n_tokens: int, d_model: int, n_layers: int, bytes_per: float,
                   d_select: int | None = None) -> dict:
    """K, V and total cache bytes per user (Eqs. 8-9); d_select=None means standard."""
    dk = d_model if d_select is None else d_select
    k = n_tokens * dk * n_layers * bytes_per
    v = n_tokens * d_model * n_layers * bytes_per
    return {"k": k, "v": v, "total": k + v}


def c_kv(n_layers: int, n_kv: int, d_head: int, n_ctx: int, beta: float = 2) -> float:
    """Standard per-sequence cache bytes read per decode step (Section 4.2)."""
    return 2 * n_layers * n_kv * d_head * n_ctx * beta


def c_kv_thin(n_layers: int, n_kv: int, r_per_head: int, d_v: int, n_ctx: int,
              beta: float = 2) -> float:
    """Thin-key cache bytes per sequence: r-wide keys, d_v-wide values."""
    return n_layers * n_kv * (r_per_head + d_v) * n_ctx * beta


def decode_speedup(weights: float, ckv: float, weights_thin: float, ckv_thin: float,
                   batch: int) -> float:
    """Predicted decode speedup of Eq. (roofline)."""
    return (weights + batch * ckv) / (weights_thin + batch * ckv_thin)


def projection_bytes_saved(d_model: int, n_q_heads: int, n_kv_heads: int, d_head: int,
                           r_per_kv_head: int, n_layers: int, beta: float = 2) -> float:
    """Weight bytes saved by factored keys at rank r_per_kv_head per kv head.

    W_K (d_model x n_kv*d_head) becomes d_model x n_kv*r and the absorbed
    W_Q (d_model x n_q*d_head) becomes d_model x n_q*r (Section 2.3).
    """
    per_layer = d_model * (n_q_heads + n_kv_heads) * (d_head - r_per_kv_head)
    return per_layer * n_layers * beta


def decode_kv_bytes(seq_lens, h_kv: int, r: int, d_v: int, k_bytes: int = 2,
                    k_scale_bytes: int = 0, v_bytes: int = 2) -> int:
    """Algorithmic cache bytes one decode step reads: every cached K and V row once.

    Per token and kv head: r * k_bytes (thin key) + k_scale_bytes (int8 key
    scale, 4 for fp32) + d_v * v_bytes (value).  Query and output bytes are
    counted separately by ``decode_io_bytes``.
    """
    per_tok = r * k_bytes + k_scale_bytes + d_v * v_bytes
    return int(sum(int(n) for n in seq_lens)) * h_kv * per_tok


def decode_io_bytes(batch: int, h_q: int, r: int, d_v: int, out_bytes: int = 4) -> int:
    """Query read (bf16) plus output write of one decode step."""
    return batch * h_q * (r * 2 + d_v * out_bytes)


def causal_pairs(seq: int) -> int:
    """Unmasked (query, key) pairs of one head under the square causal mask."""
    return seq * (seq + 1) // 2


def prefill_flops(batch: int, h_q: int, seq: int, r: int, d_v: int,
                  causal: bool = True, cached: int = 0) -> int:
    """Attention FLOPs of prefill: 2 * (r + d_v) per unmasked pair.  With `cached`
    tokens before the chunk, query i sees cached + i + 1 keys (causal)."""
    if causal:
        pairs = cached * seq + causal_pairs(seq)
    else:
        pairs = (cached + seq) * seq
    return batch * h_q * pairs * 2 * (r + d_v)
