"""The fused layer path (LogoAttention.forward_fused / backward_fused): Eq. 7
gate + selection, Eq. 5 LP transforms (Q^G on the selected rows only), both
branches, Eq. 9/10, and every gradient back to x, w_g, Q^L/K^L/V^L, the
transform matrices and the ContextNorm gains, against a chain of oracle
functions computed from the same inputs (the oracle takes its own selection
from its fp64 gate; the test asserts it is the kernel's).

Tolerance.  Each piece is checked element by element on identical inputs in
its own test.  Here errors compound through the chain: a gradient that sums
hundreds of terms over tokens, each carrying the bf16 rounding of an
upstream GPU output, keeps an absolute error of a few 1e-2 where the sum
cancels to near zero.  So every tensor must hold relative L2 <= 1e-2, as
everywhere, and max |got - ref| <= 2e-2 * max(1, max |ref|), the max-abs
bound taken against the tensor's own scale."""
import numpy as np
import pytest
import torch

import oracle
from helpers import check_close as _check_close, np32


def check_close(got, ref, name):
    ref = np.asarray(ref, dtype=np.float64)
    scale = max(1.0, float(np.abs(ref).max())) if ref.size else 1.0
    return _check_close(np.asarray(got, dtype=np.float64) / scale, ref / scale, name)

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,T,Hq,Hkv,D,W", [(2, 320, 4, 2, 64, 64), (1, 400, 2, 2, 128, 96)])
def test_fused_layer_matches_the_oracle_chain(B, T, Hq, Hkv, D, W):
    from paper_2608_29539_gb300 import logo as L
    from paper_2608_29539_gb300.layer import LayerConfig, LogoAttention
    ratio, dm = 0.25, Hq * D
    g = torch.Generator().manual_seed(T + D)
    bf = lambda *s, scale=1.0: (scale * torch.randn(*s, generator=g)).bfloat16()  # noqa: E731
    x, qL, kL, vL, dO = bf(B, T, dm), bf(B, T, Hq, D), bf(B, T, Hkv, D), bf(B, T, Hkv, D), bf(B, T, Hq, D)
    w = (torch.randn(dm, generator=g) / dm ** 0.5).float()
    eye = lambda H: (torch.eye(D) + 0.05 * torch.randn(H, D, D, generator=g)).bfloat16()  # noqa: E731
    Aq, Ak, Av = eye(Hq), eye(Hkv), eye(Hkv)
    gl = (1 + 0.1 * torch.randn(Hq, D, generator=g)).float()
    gg = (1 + 0.1 * torch.randn(Hq, D, generator=g)).float()
    dev = torch.device("cuda")
    cfg = LayerConfig(B, T, Hq, Hkv, D, W, mode=L.LOGO_SELECT_RATIO, ratio=ratio)
    layer = LogoAttention(cfg, device=dev)
    d = lambda t: t.to(dev)  # noqa: E731
    args = (d(x), d(w), d(qL), d(kL), d(vL), {"a": d(Aq)}, {"a": d(Ak)}, {"a": d(Av)})
    o = layer.forward_fused(*args, gain_l=d(gl), gain_g=d(gg))
    grads = layer.backward_fused(d(dO), *args, gain_l=d(gl), gain_g=d(gg))
    torch.cuda.synchronize()

    # ---- the oracle chain
    f = np32
    p = oracle.gate(f(x), f(w))
    z = oracle.select_ratio(p.astype(np.float32), oracle.k_from_ratio(ratio, T))
    assert np.array_equal(z, layer.z.cpu().numpy())  # same selection
    np.testing.assert_allclose(f(layer.gate_p), p, atol=1e-5)
    pos, cu_q, row_of, n = oracle.compact(z)
    lb, lt = oracle.local_rows(B, T)
    gb, gt = oracle.global_rows(pos, cu_q)
    qG = oracle.branch_fwd(f(qL), A=f(Aq)).reshape(B, T, Hq, D)
    kG = oracle.branch_fwd(f(kL), A=f(Ak)).reshape(B, T, Hkv, D)
    vG = oracle.branch_fwd(f(vL), A=f(Av)).reshape(B, T, Hkv, D)
    oL, _ = oracle.attn_fwd(f(qL), f(kL), f(vL), lb, lt, W)
    oG, _ = oracle.attn_fwd(qG, kG, vG, gb, gt, 0)
    oL = oL.reshape(B, T, Hq, D)
    ro, _, _ = oracle.combine_fwd(oL, oG, p.astype(np.float32), z, row_of, f(gl), f(gg))
    check_close(f(o), ro, "o")
    dOL, dOG, dp = oracle.combine_bwd(f(dO), oL, oG, p.astype(np.float32), z, row_of, f(gl), f(gg))
    dgl, dgg = oracle.combine_dgain(f(dO), oL, oG, p.astype(np.float32), z, row_of)
    check_close(f(grads["dgain_l"]), dgl, "dgain_l")
    check_close(f(grads["dgain_g"]), dgg, "dgain_g")
    dqL, dkL, dvL = oracle.attn_bwd(f(qL), f(kL), f(vL), lb, lt, W, dOL)
    dqGc, dkG, dvG = oracle.attn_bwd(qG, kG, vG, gb, gt, 0, dOG)
    duq, dAq = oracle.branch_bwd(f(qL), dqGc, A=f(Aq), rows=(gb, gt))
    duk, dAk = oracle.branch_bwd(f(kL), dkG.reshape(-1, Hkv, D), A=f(Ak))
    duv, dAv = oracle.branch_bwd(f(vL), dvG.reshape(-1, Hkv, D), A=f(Av))
    dq_tot = dqL.reshape(B, T, Hq, D).copy()
    dq_tot[gb, gt] += duq
    check_close(f(grads["dqL"]), dq_tot, "dQ^L (local + transformed global)")
    check_close(f(grads["dkL"]), dkL + duk.reshape(B, T, Hkv, D), "dK^L")
    check_close(f(grads["dvL"]), dvL + duv.reshape(B, T, Hkv, D), "dV^L")
    check_close(f(grads["tq"]["dA"]), dAq, "dA_Q")
    check_close(f(grads["tk"]["dA"]), dAk, "dA_K")
    check_close(f(grads["tv"]["dA"]), dAv, "dA_V")
    dx, dw = oracle.gate_bwd(f(x), f(w), dp)
    check_close(f(grads["dx"]), dx, "dx")
    check_close(f(grads["dw_g"]), dw, "dw_g")
