"""Shared helpers for the parity tests (tolerances, conversions).

Tolerance for bf16 outputs and gradients against the fp64 oracle; both parts
must hold for every tensor:

  (1) element-wise |got - ref| <= 2e-2 + 2^-8 |ref|: the stated absolute
      bound (max-abs 2e-2) plus exactly one bf16 rounding of the output.
      bf16 keeps 8 significant bits, so rounding a value x to bf16 moves it
      by at most half an ulp <= 2^-8 |x|; no kernel that returns bf16 can do
      better than that on large values, and nothing more is allowed.
  (2) relative L2 error over the tensor <= 1e-2.

Outputs kept in fp32 (lse, rstd, gains' gradients, dp) pass their own bound
and set `rel` to the fp32 figure they need.

Every call returns the errors it reached.  With LOGO_PARITY_LOG set to a path,
each call also appends one JSON line (test id, tensor, max |got - ref|, the
largest fraction of the bound used, relative L2) so that the headroom of the
kernels is on record.
"""
import json
import os

import numpy as np
import torch

MAX_ABS = 2e-2
REL_L2 = 1e-2
BF16_ROUNDING = 2.0 ** -8


def np32(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy()


def _log(name, n, max_abs_err, frac, rl2):
    path = os.environ.get("LOGO_PARITY_LOG")
    if not path:
        return
    rec = dict(test=os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0], tensor=name, n=int(n),
               max_abs_err=max_abs_err, bound_used=frac, rel_l2=rl2)
    with open(path, "a") as f:
        f.write(json.dumps(rec) + "\n")


def check_close(got, ref, name, max_abs=MAX_ABS, rel_l2=REL_L2, rel=BF16_ROUNDING, scale_ref=None):
    """Assert |got - ref| <= max_abs + rel * |s| element-wise, where s = ref
    (or `scale_ref`, for a result rounded at more than one magnitude), and
    relative L2 <= rel_l2.  Returns (max |got - ref|, largest fraction of the
    element-wise bound used, relative L2)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.isfinite(got).all(), f"{name}: non-finite values"
    if ref.size == 0:
        return 0.0, 0.0, 0.0
    s = np.abs(ref) if scale_ref is None else np.asarray(scale_ref, dtype=np.float64)
    err = np.abs(got - ref)
    bound = max_abs + rel * s
    mx = float(err.max())
    frac = float((err / bound).max())
    denom = float(np.linalg.norm(ref))
    rl2 = float(np.linalg.norm(got - ref) / denom) if denom > 0 else float(np.linalg.norm(got - ref))
    _log(name, ref.size, mx, frac, rl2)
    i = int(np.argmax(err / bound))
    assert frac <= 1.0 and rl2 <= rel_l2, (
        f"{name}: |got-ref| {mx:.3e}, worst element {err.flat[i]:.3e} at |ref| {abs(ref.flat[i]):.3e} "
        f"uses {frac:.2f} of its bound {max_abs:g} + {rel:g}|ref|; rel-L2 {rl2:.3e} (<= {rel_l2})")
    return mx, frac, rl2


def seeded(shape, seed, dtype=torch.float32, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(shape, generator=g, dtype=torch.float32) * scale).to(dtype)
