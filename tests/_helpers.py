"""Test plumbing: tensor <-> oracle conversion and the parity bar.

The parity bar (fp outputs against the fp64 oracle on identical bf16
inputs): max abs error <= 1e-2 and mean relative error, defined as
sum|gpu - ref| / sum|ref| over all compared elements, <= 2e-3.

For kernels whose output is bf16 (``parity_bf16``), both sides take the
final rounding in the same precision: the oracle's fp64 result is rounded
to bf16 (round to nearest even) before the comparison.  Against the
unrounded oracle the rounding of a correct result alone already costs about
1.4e-3 of the 2e-3 budget.  The two rounded values can still differ by one
bf16 unit when the kernel's fp32 value and the exact value fall on either
side of a rounding boundary; for |out| >= 2 that unit (2^-6 and up) exceeds
1e-2, so the per-element bound is max(1e-2, one bf16 unit at |ref|).
"""

import numpy as np
import pytest
import torch

from oracle.attention import bf16_bits_to_f64

MAX_ABS = 1e-2
MEAN_REL = 2e-3


def has_gpu() -> bool:
    return torch.cuda.is_available()


def require_gpu():
    if not has_gpu():
        pytest.skip("needs a CUDA GPU")
    from paper_2603_04427_gb300 import build
    build.build()


def f64(t: torch.Tensor) -> np.ndarray:
    """Exact float64 copy of a bf16 / fp32 / int8 tensor for the oracle."""
    t = t.detach().cpu()
    if t.dtype == torch.bfloat16:
        return bf16_bits_to_f64(t.contiguous().view(torch.int16).numpy())
    return t.numpy().astype(np.float64)


def round_bf16(x) -> np.ndarray:
    """fp64 values rounded to bf16 (round to nearest even), back as fp64."""
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.to(torch.float64).numpy()


def parity(got, ref, max_abs=MAX_ABS, mean_rel=MEAN_REL, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    err = np.abs(got - ref)
    denom = np.abs(ref).sum()
    rel = err.sum() / denom if denom > 0 else err.sum()
    assert err.max() <= max_abs, f"{what}: max abs error {err.max():.3e} > {max_abs}"
    assert rel <= mean_rel, f"{what}: mean relative error {rel:.3e} > {mean_rel}"
    return float(err.max()), float(rel)


def bf16_ulp(x) -> np.ndarray:
    """Spacing of bf16 values at |x| (8 significant bits)."""
    a = np.maximum(np.abs(np.asarray(x, dtype=np.float64)), 2.0 ** -126)
    return 2.0 ** (np.floor(np.log2(a)) - 7)


def parity_bf16(got, ref, max_abs=MAX_ABS, mean_rel=MEAN_REL, what=""):
    """Parity of a bf16 output with the bf16-rounded oracle (see module docstring)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    r = round_bf16(ref)
    assert got.shape == r.shape, (got.shape, r.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    err = np.abs(got - r)
    bound = np.maximum(max_abs, bf16_ulp(ref))
    worst = np.argmax(err - bound)
    assert np.all(err <= bound), (f"{what}: error {err.flat[worst]:.3e} above its bound "
                                  f"{bound.flat[worst]:.3e} at |ref| = {abs(ref.flat[worst]):.3e}")
    denom = np.abs(r).sum()
    rel = err.sum() / denom if denom > 0 else err.sum()
    assert rel <= mean_rel, f"{what}: mean relative error {rel:.3e} > {mean_rel}"
    return float(err.max()), float(rel)
