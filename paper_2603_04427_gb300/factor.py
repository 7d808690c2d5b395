"""Factored keys: turn a full-key attention layer into a thin-key one (Section 2.3).

Each key projection is factorised by truncated SVD, W_K ~ A B with A = U_r S_r
(d_model x r) and B = V_r^T (r x d_head) (Eq. 5); the cache then holds the
thin keys k' = x A, and B^T is absorbed into the query projection,
W_Q' = W_Q B^T (the absorbed-query equation), so q' k'^T = x W_Q B^T A^T x^T
equals q k^T whenever W_K has rank <= r, and otherwise differs only by the
truncation (Eckart-Young: the discarded singular values).

Per head.  Attention scores are per head, so the identity only holds when
every kv head's slice of W_K is factorised on its own; with grouped queries
(G query heads per kv head) the B of kv head g is absorbed into each of its
G query heads.  The paper factorises "each layer's W_K" with a total rank
d_select; this library's reading is the per-head split of that rank
(r = d_select / h_kv per kv head), the only one that keeps per-head scores.

The scores keep the original model's scale: a factorised model is run with
scale 1/sqrt(d_head), not 1/sqrt(r), which is why every entry point takes
the scale as an argument.

Weights use the x @ W convention: W_Q [d_model, h_q * d_head] (query head h
is columns h*d_head .. (h+1)*d_head), W_K [d_model, h_kv * d_head].  This is
offline weight preparation (one SVD per kv head), not part of the attention
hot path.
"""

from __future__ import annotations

from dataclasses import dataclass

import torch


@dataclass
class FactoredKeys:
    w_q: torch.Tensor        # [d_model, h_q * r]   absorbed query projection W_Q'
    w_k: torch.Tensor        # [d_model, h_kv * r]  thin key projection W_K' (= A per kv head)
    b: torch.Tensor          # [h_kv, r, d_head]    B per kv head (k ~ k' B)
    discarded: torch.Tensor  # [h_kv, min(d_model, d_head) - r] singular values left out
    scale: float             # the score scale to keep: 1 / sqrt(d_head)


def factor_keys(w_q: torch.Tensor, w_k: torch.Tensor, h_q: int, h_kv: int, r: int,
                dtype=torch.float64) -> FactoredKeys:
    """Per-kv-head truncated SVD of W_K and absorption of B^T into W_Q (see module doc)."""
    d_model = w_k.shape[0]
    if w_k.shape[1] % h_kv or w_q.shape[1] % h_q or h_q % h_kv:
        raise ValueError("head counts do not divide the projection widths")
    d_head = w_k.shape[1] // h_kv
    if w_q.shape[0] != d_model or w_q.shape[1] != h_q * d_head:
        raise ValueError("W_Q and W_K shapes do not match")
    if not 0 < r <= min(d_model, d_head):
        raise ValueError(f"r={r} must be in [1, min(d_model, d_head)]")
    G = h_q // h_kv
    wq = w_q.to(dtype)
    wk = w_k.to(dtype)
    out_q = torch.empty(d_model, h_q * r, dtype=dtype, device=w_k.device)
    out_k = torch.empty(d_model, h_kv * r, dtype=dtype, device=w_k.device)
    bs = torch.empty(h_kv, r, d_head, dtype=dtype, device=w_k.device)
    disc = []
    for g in range(h_kv):
        u, s, vh = torch.linalg.svd(wk[:, g * d_head:(g + 1) * d_head], full_matrices=False)
        a = u[:, :r] * s[:r]          # A = U_r S_r
        b = vh[:r]                    # B = V_r^T
        out_k[:, g * r:(g + 1) * r] = a
        bs[g] = b
        disc.append(s[r:])
        for h in range(g * G, (g + 1) * G):
            out_q[:, h * r:(h + 1) * r] = wq[:, h * d_head:(h + 1) * d_head] @ b.T
    return FactoredKeys(out_q, out_k, bs, torch.stack(disc), 1.0 / d_head ** 0.5)
