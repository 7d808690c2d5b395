"""fp64 CPU oracle for thin-key ("asymmetric") softmax attention.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import this
module: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It
shares no code with the CUDA library and imports nothing from it.

What it computes (paper, Section 2.1, Eqs. 1-4): for every head i,

    head_i = softmax( Q_i K_i^T / sqrt(d_head^QK) ) V_i

where the query/key width d_head^QK (called ``r`` here, per head) may be
much smaller than the value width d_head^V (``d_v``).  The attention
weights are scalars, so nothing else changes when r != d_v (Section 2.1,
remark after Eq. 4).  ``scale`` is an explicit argument; the configs use
1/sqrt(r), the factor Eq. 4 prints.

Readings of points the paper leaves open:
  * GQA head mapping (the paper composes thin keys with GQA, Section 3.4,
    Mistral-7B 32 query / 8 kv heads in Section 3.5): query head h reads
    kv head h // G with G = H_q / H_kv (contiguous groups).
  * Causal prefill is top-left aligned: query i sees keys 0..i.
  * Decode over an empty context (seq_len 0) returns a zero row.
  * int8 keys are dequantised as code * scale (per token, per kv head).

Every input here is float64 holding exactly the bf16 (or int8 / fp32)
values the GPU receives; ``bf16_bits_to_f64`` converts raw bf16 bit
patterns without rounding.  Arithmetic is plain float64 numpy: one
matrix product for the scores, the textbook max-subtracted softmax, one
matrix product for the weighted sum.  No blocking, no online softmax, no
reordering beyond that definition.
"""

from __future__ import annotations

import numpy as np


def bf16_bits_to_f64(bits) -> np.ndarray:
    """Exact conversion of raw bf16 bit patterns (uint16 or int16) to float64.

    A bf16 value is the upper half of an IEEE binary32 word, so shifting
    the 16 bits into the high half of a uint32 and reinterpreting gives the
    float32 value exactly; widening to float64 is exact as well.
    """
    b = np.asarray(bits)
    if b.dtype == np.int16:
        b = b.view(np.uint16)
    if b.dtype != np.uint16:
        raise TypeError(f"expected uint16/int16 bf16 bit patterns, got {b.dtype}")
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def attention_head(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float,
                   causal_offset: int | None = None,
                   return_weights: bool = False):
    """One head of Eq. 4: softmax(scale * q k^T) v, in float64.

    q: [n_q, r], k: [n_k, r], v: [n_k, d_v].
    causal_offset: None for no mask; otherwise query row i may attend to
    key j only when j <= i + causal_offset (0 gives the square causal
    mask of prefill).
    Returns out [n_q, d_v] (and the weights [n_q, n_k] on request).
    A query row with no visible key (n_k == 0) gives a zero output row.
    """
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    n_q, n_k = q.shape[0], k.shape[0]
    if n_k == 0:
        out = np.zeros((n_q, v.shape[1]), dtype=np.float64)
        return (out, np.zeros((n_q, 0))) if return_weights else out
    # Scores: the scalar selection weights of Eq. 4 before normalisation.
    s = scale * (q @ k.T)
    if causal_offset is not None:
        i = np.arange(n_q)[:, None]
        j = np.arange(n_k)[None, :]
        s = np.where(j <= i + causal_offset, s, -np.inf)
    # Textbook softmax over the key axis.
    m = np.max(s, axis=1, keepdims=True)
    e = np.exp(s - m)
    w = e / np.sum(e, axis=1, keepdims=True)
    out = w @ v
    return (out, w) if return_weights else out


def _kv_head(h: int, h_q: int, h_kv: int) -> int:
    if h_q % h_kv != 0:
        raise ValueError(f"H_q={h_q} is not a multiple of H_kv={h_kv}")
    return h // (h_q // h_kv)


def attention_prefill(q, k, v, scale: float, causal: bool = True) -> np.ndarray:
    """Prefill attention over a whole prompt (Eqs. 1-4, every head).

    q: [B, H_q, S, r], k: [B, H_kv, S, r], v: [B, H_kv, S, d_v] (float64).
    Returns [B, H_q, S, d_v] float64.
    """
    q, k, v = (np.asarray(x, dtype=np.float64) for x in (q, k, v))
    B, h_q, S, _ = q.shape
    h_kv = k.shape[1]
    out = np.zeros((B, h_q, S, v.shape[3]), dtype=np.float64)
    for b in range(B):
        for h in range(h_q):
            g = _kv_head(h, h_q, h_kv)
            out[b, h] = attention_head(q[b, h], k[b, g], v[b, g], scale,
                                       causal_offset=0 if causal else None)
    return out


def attention_prefill_cached(q, k, v, seq_lens, scale: float, causal: bool = True) -> np.ndarray:
    """Prefill of a chunk that continues a cached context (Eqs. 1-4 over the grown context).

    q: [B, H_q, S, r] the chunk's queries; k: [B, H_kv, n, r], v: [B, H_kv, n, d_v]
    the sequence's keys and values, chunk included (n >= seq_lens[b] + S).
    Query i of sequence b sits at position seq_lens[b] + i and attends to keys
    0 .. seq_lens[b] + i (causal) or to all seq_lens[b] + S of them.
    Returns [B, H_q, S, d_v] float64.
    """
    q, k, v = (np.asarray(x, dtype=np.float64) for x in (q, k, v))
    B, h_q, S, _ = q.shape
    h_kv = k.shape[1]
    out = np.zeros((B, h_q, S, v.shape[3]), dtype=np.float64)
    for b in range(B):
        n = int(seq_lens[b]) + S
        for h in range(h_q):
            g = _kv_head(h, h_q, h_kv)
            out[b, h] = attention_head(q[b, h], k[b, g, :n], v[b, g, :n], scale,
                                       causal_offset=int(seq_lens[b]) if causal else None)
    return out


def attention_backward(q, k, v, d_out, scale: float, causal: bool = True):
    """Gradients of prefill attention (Eqs. 1-4) for a loss with dL/d(out) = d_out.

    q: [B, H_q, S, r], k: [B, H_kv, S, r], v: [B, H_kv, S, d_v], d_out: [B, H_q, S, d_v].
    Per head, with s = scale q k^T (masked), p = softmax(s) row-wise, out = p v:
        dv = p^T d_out,  dp = d_out v^T,  ds = p * (dp - rowsum(dp * p)),
        dq = scale ds k,  dk = scale ds^T q
    (the softmax Jacobian diag(p) - p p^T applied row by row); a kv head's dk and dv
    sum the contributions of its G query heads.  Returns (dq, dk, dv) float64.
    """
    q, k, v, d_out = (np.asarray(x, dtype=np.float64) for x in (q, k, v, d_out))
    B, h_q, S, _ = q.shape
    h_kv = k.shape[1]
    dq, dk, dv = np.zeros_like(q), np.zeros_like(k), np.zeros_like(v)
    for b in range(B):
        for h in range(h_q):
            g = _kv_head(h, h_q, h_kv)
            _, p = attention_head(q[b, h], k[b, g], v[b, g], scale,
                                  causal_offset=0 if causal else None, return_weights=True)
            dv[b, g] += p.T @ d_out[b, h]
            dp = d_out[b, h] @ v[b, g].T
            ds = p * (dp - np.sum(dp * p, axis=1, keepdims=True))
            dq[b, h] = scale * (ds @ k[b, g])
            dk[b, g] += scale * (ds.T @ q[b, h])
    return dq, dk, dv


def logsumexp_rows(q, k, scale: float, causal: bool = True) -> np.ndarray:
    """Natural-log logsumexp of each row's scaled (masked) scores: [B, H_q, S]."""
    q, k = np.asarray(q, dtype=np.float64), np.asarray(k, dtype=np.float64)
    B, h_q, S, _ = q.shape
    h_kv = k.shape[1]
    out = np.zeros((B, h_q, S))
    for b in range(B):
        for h in range(h_q):
            s = scale * (q[b, h] @ k[b, _kv_head(h, h_q, h_kv)].T)
            if causal:
                s = np.where(np.arange(S)[None, :] <= np.arange(S)[:, None], s, -np.inf)
            m = s.max(axis=1)
            out[b, h] = m + np.log(np.exp(s - m[:, None]).sum(axis=1))
    return out


def attention_prefill_rows(q, k, v, scale: float, rows, causal: bool = True) -> np.ndarray:
    """Selected output rows of ``attention_prefill``, each computed on its own.

    rows: iterable of (b, h, i).  For causal prefill row i attends to keys
    0..i, i.e. it is a single-query attention over the first i+1 keys.
    Used to check very large launches on a sample of outputs.
    Returns [len(rows), d_v] float64.
    """
    q, k, v = (np.asarray(x) for x in (q, k, v))
    h_q, h_kv = q.shape[1], k.shape[1]
    res = []
    for (b, h, i) in rows:
        g = _kv_head(h, h_q, h_kv)
        n = i + 1 if causal else k.shape[2]
        res.append(attention_head(np.asarray(q[b, h, i:i + 1], dtype=np.float64),
                                  np.asarray(k[b, g, :n], dtype=np.float64),
                                  np.asarray(v[b, g, :n], dtype=np.float64), scale)[0])
    return np.stack(res) if res else np.zeros((0, v.shape[3]))


def dequantize_keys(codes, scales) -> np.ndarray:
    """int8 or int4 key codes [..., r] times their per-token fp32 scale [...] (exact in fp64)."""
    return np.asarray(codes, dtype=np.float64) * np.asarray(scales, dtype=np.float64)[..., None]


def attention_decode(q, k, v, seq_lens, scale: float, k_scale=None) -> np.ndarray:
    """Single-token decode over a contiguous cache (Eq. 4 with one query row).

    q: [B, H_q, r]; k: [B, H_kv, cap, r] (float64 values, or int8 codes when
    ``k_scale`` [B, H_kv, cap] is given); v: [B, H_kv, cap, d_v];
    seq_lens: [B] context lengths.  Sequence b attends to its first
    seq_lens[b] cached tokens.  Returns [B, H_q, d_v] float64.
    """
    q = np.asarray(q, dtype=np.float64)
    v = np.asarray(v)
    B, h_q, _ = q.shape
    h_kv = v.shape[1]
    out = np.zeros((B, h_q, v.shape[3]), dtype=np.float64)
    for b in range(B):
        n = int(seq_lens[b])
        for h in range(h_q):
            g = _kv_head(h, h_q, h_kv)
            if k_scale is None:
                kk = np.asarray(k[b, g, :n], dtype=np.float64)
            else:
                kk = dequantize_keys(k[b, g, :n], k_scale[b, g, :n])
            out[b, h] = attention_head(q[b, h][None, :], kk,
                                       np.asarray(v[b, g, :n], dtype=np.float64), scale)[0]
    return out


def gather_pages(pool, page_table_row, n_tokens: int, page_size: int) -> np.ndarray:
    """Logical token order of one sequence from a paged pool.

    pool: [num_pages, H_kv, page_size, w]; logical token t of the sequence
    lives in page page_table_row[t // page_size], slot t % page_size.
    Returns [H_kv, n_tokens, w] (same dtype as the pool).
    """
    pool = np.asarray(pool)
    out = np.empty((pool.shape[1], n_tokens) + pool.shape[3:], dtype=pool.dtype)
    for t in range(n_tokens):
        page = int(page_table_row[t // page_size])
        out[:, t] = pool[page, :, t % page_size]
    return out


def attention_decode_paged(q, k_pool, v_pool, page_table, seq_lens, page_size: int,
                           scale: float, k_scale_pool=None) -> np.ndarray:
    """Decode over a paged cache: gather each sequence's pages, then ``attention_decode``.

    k_pool: [P, H_kv, page_size, r], v_pool: [P, H_kv, page_size, d_v],
    k_scale_pool: [P, H_kv, page_size] (int8 keys) or None,
    page_table: [B, max_pages] page ids.  Returns [B, H_q, d_v] float64.
    """
    q = np.asarray(q, dtype=np.float64)
    B, h_q, _ = q.shape
    out = np.zeros((B, h_q, np.asarray(v_pool).shape[3]), dtype=np.float64)
    for b in range(B):
        n = int(seq_lens[b])
        kb = gather_pages(k_pool, page_table[b], n, page_size)[None]
        vb = gather_pages(v_pool, page_table[b], n, page_size)[None]
        sb = None
        if k_scale_pool is not None:
            sb = gather_pages(np.asarray(k_scale_pool)[..., None], page_table[b], n,
                              page_size)[None, ..., 0]
        out[b:b + 1] = attention_decode(q[b:b + 1], kb, vb, [n], scale, k_scale=sb)
    return out
