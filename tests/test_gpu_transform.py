"""Eq. 5 branch transforms through the C ABI (logo_branch_transform / _bwd)
against the oracle: LP (per-head matrix, tensor cores) and SO (scale and
offset), on every row and on the packed selected rows only (rows not listed
are poisoned and must stay untouched); identity initialisation exact;
gradients within the bf16 / fp32 tolerances, in write and accumulate modes;
parameter gradients deterministic."""
import numpy as np
import pytest
import torch

import oracle
from helpers import check_close, np32

pytestmark = pytest.mark.gpu


def L():
    from paper_2608_29539_gb300 import logo
    return logo


def _setup(B, T, H, D, seed, ratio):
    g = torch.Generator().manual_seed(seed)
    u = torch.randn(B, T, H, D, generator=g).bfloat16()
    a = (torch.randn(H, D, D, generator=g) / D ** 0.5).bfloat16()
    s = (1 + 0.2 * torch.randn(H, D, generator=g)).float()
    b = (0.1 * torch.randn(H, D, generator=g)).float()
    dg = torch.randn(B, T, H, D, generator=g).bfloat16()
    dev = torch.device("cuda")
    rows = rows_np = None
    if ratio is not None:
        p = torch.rand(B, T, generator=g).to(dev)
        z, pos, cu_q, row_of, n_sel = L().logo_select(p, L().LOGO_SELECT_RATIO, 0.0, ratio)
        rows = (pos, cu_q, n_sel)
        n = int(n_sel[0])
        cu = cu_q.cpu().numpy()
        rows_np = (np.repeat(np.arange(B), np.diff(cu)), pos.cpu().numpy()[:n])
    return u, a, s, b, dg, rows, rows_np


CASES = [
    # B, T, H, D, ratio (None: every row)
    (2, 300, 4, 128, None),
    (2, 300, 4, 128, 0.25),
    (1, 1000, 2, 64, None),
    (3, 257, 3, 64, 0.5),
    (2, 2048, 32, 128, 0.125),   # several tiles per block, the 16K workload's head count
    # more row tiles per head than blocks per head: the selected-row LP forward
    # fetches a block's next tile while it multiplies the current one (both
    # buffers in use), with a ragged last tile
    (1, 8100, 32, 128, 0.25),
    (1, 16000, 16, 64, 0.25),
]


@pytest.mark.parametrize("B,T,H,D,ratio", CASES)
@pytest.mark.parametrize("form", ["lp", "so"])
def test_branch_transform_forward_and_backward(B, T, H, D, ratio, form):
    u, a, s, b, dg, rows, rows_np = _setup(B, T, H, D, seed=T + H + D, ratio=ratio)
    dev = torch.device("cuda")
    ud, dgd = u.to(dev), dg.to(dev)
    params = dict(a=a.to(dev)) if form == "lp" else dict(s=s.to(dev), b=b.to(dev))
    ug = torch.full_like(ud, float("nan"))
    L().logo_branch_transform(ud, rows=rows, u_g=ug, **params)
    bw = dict(a=params["a"]) if form == "lp" else dict(s=params["s"])
    du = torch.full_like(ud, float("nan"))
    out = L().logo_branch_transform_bwd(ud, dgd, rows=rows, du_l=du, **bw)
    du_in = torch.randn(B, T, H, D, generator=torch.Generator().manual_seed(1)).bfloat16().to(dev)
    out_acc = L().logo_branch_transform_bwd(ud, dgd, rows=rows, du_l=du_in.clone(), accumulate=True, **bw)
    again = L().logo_branch_transform_bwd(ud, dgd, rows=rows, du_l=torch.empty_like(ud), **bw)
    torch.cuda.synchronize()
    oparams = dict(A=np32(a)) if form == "lp" else dict(s=np32(s), b=np32(b))
    ref = oracle.branch_fwd(np32(u), rows=rows_np, **oparams)
    got = np32(ug)
    if rows_np is None:
        check_close(got.reshape(-1, H, D), ref, "u_g")
    else:
        rb, rt = rows_np
        check_close(got[rb, rt], ref, "u_g (selected rows)")
        mask = np.ones((B, T), bool)
        mask[rb, rt] = False
        assert np.isnan(got[mask]).all()  # rows not listed are untouched
    dg_rows = np32(dg).reshape(-1, H, D) if rows_np is None else np32(dg)[rows_np[0], rows_np[1]]
    if form == "lp":
        rdu, rda = oracle.branch_bwd(np32(u), dg_rows, A=np32(a), rows=rows_np)
        check_close(np32(out[1]), rda, "dA")
        assert torch.equal(out[1], again[1])
    else:
        rdu, rds, rdb = oracle.branch_bwd(np32(u), dg_rows, s=np32(s), rows=rows_np)
        check_close(np32(out[1]), rds, "ds")
        check_close(np32(out[2]), rdb, "db")
        assert torch.equal(out[1], again[1]) and torch.equal(out[2], again[2])
    gdu, gacc, din = np32(du), np32(out_acc[0]), np32(du_in)
    if rows_np is None:
        check_close(gdu.reshape(-1, H, D), rdu, "du_l")
        check_close(gacc.reshape(-1, H, D), din.reshape(-1, H, D) + rdu, "du_l accumulated")
    else:
        rb, rt = rows_np
        check_close(gdu[rb, rt], rdu, "du_l (selected rows)")
        check_close(gacc[rb, rt], din[rb, rt] + rdu, "du_l accumulated")
        mask = np.ones((B, T), bool)
        mask[rb, rt] = False
        assert np.isnan(gdu[mask]).all() and np.array_equal(gacc[mask], din[mask])


@pytest.mark.parametrize("D", [64, 128])
def test_branch_transform_identity_initialisation_is_exact(D):
    """Sec. 3.2: both forms start as the identity, so U^G = U^L bit for bit."""
    B, T, H = 2, 130, 3
    dev = torch.device("cuda")
    u = torch.randn(B, T, H, D).bfloat16().to(dev)
    eye = torch.eye(D).expand(H, D, D).contiguous().bfloat16().to(dev)
    lp = L().logo_branch_transform(u, a=eye)
    so = L().logo_branch_transform(u, s=torch.ones(H, D, device=dev), b=torch.zeros(H, D, device=dev))
    torch.cuda.synchronize()
    assert torch.equal(lp, u) and torch.equal(so, u)
