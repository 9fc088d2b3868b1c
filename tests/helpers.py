"""Shared helpers for the parity tests (tolerances, conversions)."""
import numpy as np
import torch

# Tolerance for bf16 outputs and gradients against the fp64 oracle; both must
# hold.  (1) Element-wise |got - ref| <= 2e-2 * max(1, |ref|): an absolute
# 2e-2 on the O(1) scale, relative 2e-2 above it (bf16 itself rounds a value
# x to within 2^-9 |x|, so no absolute bound can hold for |x| >~ 10).
# (2) Relative L2 error over the tensor <= 1e-2.
MAX_ABS = 2e-2
REL_L2 = 1e-2


def np32(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy()


def check_close(got, ref, name, max_abs=MAX_ABS, rel_l2=REL_L2):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.isfinite(got).all(), f"{name}: non-finite values"
    if ref.size == 0:
        return 0.0, 0.0
    err = np.abs(got - ref) / np.maximum(1.0, np.abs(ref))
    mx = float(err.max())
    denom = float(np.linalg.norm(ref))
    rl2 = float(np.linalg.norm(got - ref) / denom) if denom > 0 else float(np.linalg.norm(got - ref))
    assert mx <= max_abs and rl2 <= rel_l2, f"{name}: max scaled err {mx:.3e} (<= {max_abs}), rel-L2 {rl2:.3e} (<= {rel_l2})"
    return mx, rl2


def seeded(shape, seed, dtype=torch.float32, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(shape, generator=g, dtype=torch.float32) * scale).to(dtype)
