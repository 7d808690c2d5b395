"""Brute-force attention in pure Python, for pinning the fp64 oracle on tiny inputs.

TEST INFRASTRUCTURE ONLY.  Deliberately a different computation from
oracle/attention.py: nested lists, ``math.exp`` of the raw logit with no
max subtraction, and ``math.fsum`` (exactly rounded sums).  It follows the
per-head definition of the paper, Section 2.1, Eq. 4, directly:
weight_ij = exp(s_ij) / sum_j' exp(s_ij'), s_ij = scale * <q_i, k_j>,
out_i = sum_j weight_ij v_j.  Only for logits of modest size (|s| < ~700).
"""

from __future__ import annotations

import math


def head(q, k, v, scale, causal=False):
    """q: list of n_q rows (r floats); k: n_k rows (r); v: n_k rows (d_v).

    Returns (out rows, weight rows).  With causal=True row i sees keys 0..i.
    """
    outs, weights = [], []
    for i, qi in enumerate(q):
        visible = range(i + 1) if causal else range(len(k))
        logits = [scale * math.fsum(a * b for a, b in zip(qi, k[j])) for j in visible]
        ex = [math.exp(s) for s in logits]
        z = math.fsum(ex)
        w = [e / z for e in ex]
        d_v = len(v[0])
        out = [math.fsum(w[t] * v[j][c] for t, j in enumerate(visible)) for c in range(d_v)]
        outs.append(out)
        weights.append(w)
    return outs, weights


def prefill(q, k, v, scale, causal=True):
    """q: [B][H_q][S][r], k: [B][H_kv][S][r], v: [B][H_kv][S][d_v] nested lists."""
    B, h_q, h_kv = len(q), len(q[0]), len(k[0])
    group = h_q // h_kv
    return [[head(q[b][h], k[b][h // group], v[b][h // group], scale, causal)[0]
             for h in range(h_q)] for b in range(B)]
