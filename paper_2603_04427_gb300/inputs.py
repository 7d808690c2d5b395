"""Seeded synthetic inputs shared by the CUDA path, its tests and the oracle.

This module draws numbers only: it holds none of the attention arithmetic.
The paper's workloads are real models on datasets that are not available
here, so every tensor is i.i.d. N(0, 1) rounded to bf16 (round to nearest
even), with the shapes of the paper's models (GPT-2 small, Mistral-7B,
a 7B MHA model).  Ragged lengths are uniform integers, page tables are
seeded random permutations of the page pool.
"""

from __future__ import annotations

import torch


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def normal_bf16(shape, seed: int, device="cpu") -> torch.Tensor:
    """N(0, 1) samples drawn in fp32 with ``torch.randn`` and rounded to bf16."""
    g = _gen(seed, device)
    return torch.randn(tuple(shape), generator=g, device=device,
                       dtype=torch.float32).to(torch.bfloat16)


def uniform_lengths(batch: int, lo: int, hi: int, seed: int) -> list[int]:
    """``batch`` integers uniform in [lo, hi] (inclusive), drawn on the CPU."""
    g = _gen(seed, "cpu")
    return [int(x) for x in torch.randint(lo, hi + 1, (batch,), generator=g)]


def paged_layout(seq_lens, page_size: int, seed: int, extra_pages: int = 0):
    """A page table that scatters each sequence over a shuffled page pool.

    Sequence b needs ceil(len_b / page_size) pages (at least one).  The pool
    holds the sum of those plus ``extra_pages``; page ids are handed out in
    the order of a seeded random permutation.  Returns
    (page_table int32 [B, max_pages] with -1 in unused slots, num_pages).
    """
    need = [max(1, -(-int(n) // page_size)) for n in seq_lens]
    num_pages = sum(need) + int(extra_pages)
    perm = torch.randperm(num_pages, generator=_gen(seed, "cpu")).to(torch.int32)
    max_pages = max(need)
    table = torch.full((len(need), max_pages), -1, dtype=torch.int32)
    pos = 0
    for b, n in enumerate(need):
        table[b, :n] = perm[pos:pos + n]
        pos += n
    return table, num_pages
