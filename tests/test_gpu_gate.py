"""The Eq. 7 gate fused ahead of the selection (logo_gate_select) and its
backward (logo_gate_bwd), against the oracle: p within rounding of the fp64
gate; the selection bit-exact given the p the kernel compared (the decision is
taken in the kernel's fp32, as the rules for float-decided integers ask);
dx and dw_g within the bf16 / fp32 tolerances; dw_g deterministic."""
import numpy as np
import pytest
import torch

import oracle
from helpers import check_close, np32

pytestmark = pytest.mark.gpu


def L():
    from paper_2608_29539_gb300 import logo
    return logo


def _inputs(B, T, dm, seed):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(B, T, dm, generator=g).bfloat16()
    w = (torch.randn(dm, generator=g) / dm ** 0.5).float()
    return x, w


CASES = [
    # B, T, d_model, mode, b_th, ratio
    (2, 1000, 4096, 1, 0.0, 0.125),    # ragged T, the 16K workload's d_model
    (1, 777, 8192, 0, 0.55, 0.0),      # the largest d_model, threshold mode
    (3, 129, 2056, 1, 0.0, 0.5),       # 257 vectors: threads of a block idle
    (1, 1, 64, 0, 0.3, 0.0),           # one token
]


@pytest.mark.parametrize("B,T,dm,mode,b_th,ratio", CASES)
def test_gate_select_and_backward(B, T, dm, mode, b_th, ratio):
    x, w = _inputs(B, T, dm, seed=dm + T)
    dev = torch.device("cuda")
    xd, wd = x.to(dev), w.to(dev)
    p, z, pos, cu_q, row_of, n_sel = L().logo_gate_select(xd, wd, mode, b_th, ratio)
    torch.cuda.synchronize()
    pk = np32(p)
    np.testing.assert_allclose(pk, oracle.gate(np32(x), np32(w)), rtol=0, atol=1e-5)
    # the selection of the p the kernel computed, bit for bit
    if mode == 1:
        zr = oracle.select_ratio(pk, oracle.k_from_ratio(ratio, T))
    else:
        zr = oracle.select_threshold(pk, b_th)
    assert np.array_equal(z.cpu().numpy(), zr)
    rpos, rcu, rrow, n = oracle.compact(zr)
    assert int(n_sel[0]) == n
    assert np.array_equal(pos.cpu().numpy()[:n], rpos) and np.array_equal(cu_q.cpu().numpy(), rcu)
    # backward: dp nonzero on the selected tokens only (as combine_bwd gives it)
    g = torch.Generator().manual_seed(T)
    dp = (torch.randn(B, T, generator=g) * torch.from_numpy(zr)).float()
    rdx, rdw = oracle.gate_bwd(np32(x), np32(w), np32(dp))
    dx, dw = L().logo_gate_bwd(xd, wd, p, dp.to(dev))
    dx_in = torch.randn(B, T, dm, generator=g).bfloat16().to(dev)
    dx_acc, dw2 = L().logo_gate_bwd(xd, wd, p, dp.to(dev), dx=dx_in.clone(), accumulate=True)
    torch.cuda.synchronize()
    check_close(np32(dx), rdx, "dx")
    check_close(np32(dw), rdw, "dw_g")
    check_close(np32(dx_acc), np32(dx_in) + rdx, "dx accumulated")
    assert torch.equal(dw, dw2)  # blocks summed in a fixed order


def test_gate_zero_init_puts_every_p_at_one_half():
    """Sec. 3.2's near-zero gate initialisation: w_g = 0 gives p = 0.5 exactly,
    so the strict compare of Eq. 7 at b_th = 0.5 selects nothing, and any
    b_th below it selects everything."""
    x, _ = _inputs(2, 300, 512, seed=1)
    dev = torch.device("cuda")
    w = torch.zeros(512, dtype=torch.float32, device=dev)
    p, z, _, _, _, n_sel = L().logo_gate_select(x.to(dev), w, 0, 0.5)
    p2, z2, _, _, _, n2 = L().logo_gate_select(x.to(dev), w, 0, 0.4999)
    torch.cuda.synchronize()
    assert bool((p == 0.5).all()) and int(n_sel[0]) == 0 and int(z.sum()) == 0
    assert int(n2[0]) == 600 and bool((z2 == 1).all())


def test_gate_bwd_dw_only_and_dx_only():
    x, w = _inputs(2, 500, 1024, seed=9)
    dev = torch.device("cuda")
    xd, wd = x.to(dev), w.to(dev)
    p, *_ = L().logo_gate_select(xd, wd, 1, 0.0, 0.25)
    dp = torch.randn(2, 500).float().to(dev)
    dx_only, none_dw = L().logo_gate_bwd(xd, wd, p, dp, want_dw=False)
    none_dx, dw_only = L().logo_gate_bwd(xd, wd, p, dp, want_dx=False)
    dx, dw = L().logo_gate_bwd(xd, wd, p, dp)
    torch.cuda.synchronize()
    assert none_dw is None and none_dx is None
    assert torch.equal(dx_only, dx) and torch.equal(dw_only, dw)
