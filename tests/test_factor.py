"""Factored-key weight preparation (Section 2.3): per-kv-head truncated SVD of
W_K and absorption of B^T into W_Q.

Pins: scores are preserved exactly (to fp64 rounding) when every kv head's
W_K slice has rank <= r; otherwise the factor error is the discarded
singular values (Eckart-Young: spectral norm = the first, Frobenius norm =
their root sum of squares); with r = d_head any W_K is exact; GQA absorbs
each kv head's B into its own query heads only.
"""

import numpy as np
import pytest
import torch

from paper_2603_04427_gb300 import factor

D_MODEL, D_HEAD = 96, 32


def _weights(h_q, h_kv, rank=None, seed=0):
    g = torch.Generator().manual_seed(seed)
    wq = torch.randn(D_MODEL, h_q * D_HEAD, generator=g, dtype=torch.float64)
    if rank is None:
        wk = torch.randn(D_MODEL, h_kv * D_HEAD, generator=g, dtype=torch.float64)
    else:  # every kv head's slice of exact rank `rank`
        wk = torch.cat([torch.randn(D_MODEL, rank, generator=g, dtype=torch.float64)
                        @ torch.randn(rank, D_HEAD, generator=g, dtype=torch.float64)
                        for _ in range(h_kv)], dim=1)
    return wq, wk


@pytest.mark.parametrize("h_q,h_kv", [(4, 4), (8, 2)])
def test_scores_preserved_for_exact_rank(h_q, h_kv):
    r = 8
    wq, wk = _weights(h_q, h_kv, rank=r, seed=1)
    f = factor.factor_keys(wq, wk, h_q, h_kv, r)
    x = torch.randn(20, D_MODEL, generator=torch.Generator().manual_seed(2), dtype=torch.float64)
    G = h_q // h_kv
    for h in range(h_q):
        g = h // G
        full = (x @ wq[:, h * D_HEAD:(h + 1) * D_HEAD]) @ (x @ wk[:, g * D_HEAD:(g + 1) * D_HEAD]).T
        thin = (x @ f.w_q[:, h * r:(h + 1) * r]) @ (x @ f.w_k[:, g * r:(g + 1) * r]).T
        assert torch.allclose(thin, full, rtol=1e-10, atol=1e-9 * full.abs().max().item())
    assert float(f.discarded.abs().max()) < 1e-10 * float(wk.abs().max())
    assert f.scale == pytest.approx(1 / np.sqrt(D_HEAD))


def test_truncation_error_is_the_discarded_singular_values():
    h_q, h_kv, r = 4, 2, 6
    wq, wk = _weights(h_q, h_kv, seed=3)
    f = factor.factor_keys(wq, wk, h_q, h_kv, r)
    for g in range(h_kv):
        wkg = wk[:, g * D_HEAD:(g + 1) * D_HEAD]
        err = wkg - f.w_k[:, g * r:(g + 1) * r] @ f.b[g]
        sv = torch.linalg.svdvals(wkg)
        assert torch.linalg.matrix_norm(err, ord=2) == pytest.approx(float(sv[r]), rel=1e-10)
        assert torch.linalg.matrix_norm(err) == pytest.approx(float(sv[r:].square().sum().sqrt()), rel=1e-10)
        assert torch.allclose(f.discarded[g], sv[r:], rtol=1e-12)
        # B has orthonormal rows (right singular vectors)
        assert torch.allclose(f.b[g] @ f.b[g].T, torch.eye(r, dtype=torch.float64), atol=1e-12)


def test_full_rank_is_exact_and_gqa_uses_the_group_factor():
    h_q, h_kv = 6, 2
    wq, wk = _weights(h_q, h_kv, seed=4)
    f = factor.factor_keys(wq, wk, h_q, h_kv, D_HEAD)  # r = d_head: no truncation
    x = torch.randn(7, D_MODEL, generator=torch.Generator().manual_seed(5), dtype=torch.float64)
    for h in range(h_q):
        g = h // 3
        full = (x @ wq[:, h * D_HEAD:(h + 1) * D_HEAD]) @ (x @ wk[:, g * D_HEAD:(g + 1) * D_HEAD]).T
        thin = (x @ f.w_q[:, h * D_HEAD:(h + 1) * D_HEAD]) @ (x @ f.w_k[:, g * D_HEAD:(g + 1) * D_HEAD]).T
        assert torch.allclose(thin, full, rtol=1e-10, atol=1e-9 * full.abs().max().item())
        # the absorbed query of head h uses B of its own kv group
        assert torch.allclose(f.w_q[:, h * D_HEAD:(h + 1) * D_HEAD],
                              wq[:, h * D_HEAD:(h + 1) * D_HEAD] @ f.b[g].T)


def test_shape_checks():
    wq, wk = _weights(4, 2, seed=6)
    with pytest.raises(ValueError):
        factor.factor_keys(wq, wk, 4, 2, 0)
    with pytest.raises(ValueError):
        factor.factor_keys(wq, wk, 4, 2, D_HEAD + 1)
    with pytest.raises(ValueError):
        factor.factor_keys(wq[:, :10], wk, 4, 2, 8)
