"""Reference thin-key / full-value KV cache writes and the int8 key quantiser.

TEST INFRASTRUCTURE ONLY (see oracle/attention.py): used by tests, smoke()
and the CPU legs of bench.py, never by the product path.

Cache content (paper, Section 2.4, Eqs. 8-9, and the remark after the
absorbed-query equation in Section 2.3): per token and kv head the cache
holds an r-wide thin key and a d_v-wide value.  Appending T new tokens to
sequence b writes logical positions seq_lens[b] .. seq_lens[b]+T-1.

Contiguous layout: k[B][H_kv][cap][r], v[B][H_kv][cap][d_v].
Paged layout: pools k[P][H_kv][page_size][r], v[P][H_kv][page_size][d_v];
logical position t of sequence b lives in page page_table[b][t // page_size]
at slot t % page_size.

int8 keys (the paper's composition with key quantisation, Section 6,
"Flash Attention and composability"; the paper fixes no scheme).  Reading:
symmetric per-token, per-kv-head absmax quantisation in fp32,
    amax  = max_c |k_c|
    scale = amax / 127            (one IEEE binary32 division, round to nearest)
    code  = clamp(rint(k_c / scale), -127, 127)   (binary32 division, ties to even)
and amax == 0 gives scale 0 and all-zero codes.  Dequantised key: code * scale.

int4 keys (the composition the paper's Section 6 singles out: 4-bit thin keys,
"16x combined" with the 4x of r): the same scheme with 7 in place of 127,
    scale = amax / 7,  code = clamp(rint(k_c / scale), -7, 7)
stored two codes per byte, element 2j in the low nibble and 2j+1 in the high
nibble, each as a 4-bit two's complement number.  One fp32 scale per token
and kv head, as for int8 (the paper fixes neither the grouping nor the
packing; this is the library's reading).
"""

from __future__ import annotations

import numpy as np


def quantize_int8_per_token(k) -> tuple[np.ndarray, np.ndarray]:
    """Quantise keys [..., r] (float32 values) to int8 codes [..., r] and fp32 scales [...].

    All arithmetic is binary32 (numpy float32 division is IEEE round-to-nearest;
    np.rint rounds half to even).
    """
    k32 = np.asarray(k, dtype=np.float32)
    amax = np.max(np.abs(k32), axis=-1)
    scale = (amax / np.float32(127.0)).astype(np.float32)
    safe = np.where(scale == 0, np.float32(1.0), scale).astype(np.float32)
    ratio = (k32 / safe[..., None]).astype(np.float32)
    codes = np.clip(np.rint(ratio), -127, 127).astype(np.int8)
    codes[scale == 0] = 0
    return codes, scale


def quantize_int4_per_token(k) -> tuple[np.ndarray, np.ndarray]:
    """Quantise keys [..., r] to int4 codes in [-7, 7] (returned as int8 [..., r])
    and fp32 scales [...]; binary32 arithmetic as in quantize_int8_per_token."""
    k32 = np.asarray(k, dtype=np.float32)
    amax = np.max(np.abs(k32), axis=-1)
    scale = (amax / np.float32(7.0)).astype(np.float32)
    safe = np.where(scale == 0, np.float32(1.0), scale).astype(np.float32)
    ratio = (k32 / safe[..., None]).astype(np.float32)
    codes = np.clip(np.rint(ratio), -7, 7).astype(np.int8)
    codes[scale == 0] = 0
    return codes, scale


def quantize_int4_per_group(k, group: int) -> tuple[np.ndarray, np.ndarray]:
    """Quantise keys [..., r] to int4 codes with one fp32 scale per `group`
    consecutive channels (r a multiple of group): scales [..., r // group].
    Each group is quantised exactly as quantize_int4_per_token quantises a
    whole row (amax / 7, binary32 division, ties to even); with group == r
    the two coincide.  Used to measure what the coarser one-scale-per-token
    reading costs in accuracy; the kernels store one scale per token."""
    k32 = np.asarray(k, dtype=np.float32)
    r = k32.shape[-1]
    if r % group:
        raise ValueError(f"r={r} is not a multiple of group={group}")
    g = k32.reshape(*k32.shape[:-1], r // group, group)
    codes, scales = quantize_int4_per_token(g)
    return codes.reshape(k32.shape), scales


def dequantize_per_group(codes, scales) -> np.ndarray:
    """codes [..., r] times the scale of each channel's group (scales [..., r // group]), in fp64."""
    c = np.asarray(codes, dtype=np.float64)
    s = np.asarray(scales, dtype=np.float64)
    group = c.shape[-1] // s.shape[-1]
    return c * np.repeat(s, group, axis=-1)


def pack_int4(codes) -> np.ndarray:
    """int4 codes [..., r] (r even, values in [-8, 7]) -> bytes [..., r/2]:
    element 2j in bits 0-3, element 2j+1 in bits 4-7."""
    c = np.asarray(codes).astype(np.int16)
    lo = c[..., 0::2] & 0xF
    hi = c[..., 1::2] & 0xF
    return (lo | (hi << 4)).astype(np.uint8)


def unpack_int4(packed) -> np.ndarray:
    """Inverse of pack_int4: bytes [..., r/2] -> int8 codes [..., r]."""
    b = np.asarray(packed).astype(np.int16)
    nib = np.stack([b & 0xF, (b >> 4) & 0xF], axis=-1).reshape(*b.shape[:-1], -1)
    return np.where(nib >= 8, nib - 16, nib).astype(np.int8)


def _quantize(k, k_bits):
    if k_bits == 8:
        return quantize_int8_per_token(k)
    codes, sc = quantize_int4_per_token(k)
    return pack_int4(codes), sc


def append_contiguous(k_cache, v_cache, seq_lens, k_new, v_new, k_scale=None, k_bits=8):
    """Write new tokens into contiguous caches (in place) and return them.

    k_cache: [B, H_kv, cap, r] (values, or int8 codes when k_scale [B, H_kv, cap]
    is given; [B, H_kv, cap, r/2] packed int4 codes when k_bits is 4);
    v_cache: [B, H_kv, cap, d_v]; k_new: [B, H_kv, T, r] float32 values;
    v_new: [B, H_kv, T, d_v].  Positions beyond cap are an error.
    """
    B, _, T, _ = np.asarray(k_new).shape
    cap = k_cache.shape[2]
    for b in range(B):
        p0 = int(seq_lens[b])
        if p0 + T > cap:
            raise ValueError(f"sequence {b}: {p0}+{T} tokens exceed capacity {cap}")
        if k_scale is None:
            k_cache[b, :, p0:p0 + T] = k_new[b]
        else:
            codes, sc = _quantize(k_new[b], k_bits)
            k_cache[b, :, p0:p0 + T] = codes
            k_scale[b, :, p0:p0 + T] = sc
        v_cache[b, :, p0:p0 + T] = v_new[b]
    return k_cache, v_cache, k_scale


def append_paged(k_pool, v_pool, page_table, seq_lens, page_size, k_new, v_new,
                 k_scale_pool=None, k_bits=8):
    """Write new tokens into paged pools (in place) and return them.

    Pools: [P, H_kv, page_size, r|d_v]; scales [P, H_kv, page_size];
    page_table: [B, max_pages].
    """
    B, _, T, _ = np.asarray(k_new).shape
    for b in range(B):
        p0 = int(seq_lens[b])
        if k_scale_pool is not None:
            codes, sc = _quantize(k_new[b], k_bits)
        for t in range(T):
            pos = p0 + t
            page = int(page_table[b][pos // page_size])
            slot = pos % page_size
            if k_scale_pool is None:
                k_pool[page, :, slot] = k_new[b][:, t]
            else:
                k_pool[page, :, slot] = codes[:, t]
                k_scale_pool[page, :, slot] = sc[:, t]
            v_pool[page, :, slot] = v_new[b][:, t]
    return k_pool, v_pool, k_scale_pool
