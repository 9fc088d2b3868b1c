"""The fused layer path (LogoAttention.forward_fused / backward_fused): Eq. 7
gate + selection, Eq. 5 LP transforms (Q^G on the selected rows only), both
branches, Eq. 9/10, and every gradient back to x, w_g, Q^L/K^L/V^L, the
transform matrices and the ContextNorm gains.

Each stage of the chain is compared with the oracle on the inputs that stage
received on the GPU (the upstream GPU results, upcast), so every tensor is
held to the same bound as the unit tests: |got - ref| <= 2e-2 + 2^-8 |ref|
and relative L2 <= 1e-2.

One place rounds twice.  backward_fused adds the transforms' share of the
global gradient (b) into the local branch's bf16 gradient (a) in place:
dQ^L = bf16(bf16(a) + b), likewise dK^L and dV^L.  The two roundings move the
result by at most 2^-8 |a| + 2^-8 |a + b|, so those three tensors are held to
2e-2 + 2^-8 (|a| + |a + b|), with a and a + b the oracle's values."""
import numpy as np
import pytest
import torch

import oracle
from helpers import check_close, np32

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
    f = np32

    # Eq. 7 gate (float32 output) and the selection on the GPU's gate values
    p = f(layer.gate_p)
    check_close(p, oracle.gate(f(x), f(w)), "p", max_abs=1e-5, rel=0.0)
    z = oracle.select_ratio(p, oracle.k_from_ratio(ratio, T))
    assert np.array_equal(z, layer.z.cpu().numpy())
    pos, cu_q, row_of, n = oracle.compact(z)
    assert int(layer.n_sel[0]) == n and np.array_equal(f(layer.pos)[:n].astype(np.int32), pos)
    lb, lt = oracle.local_rows(B, T)
    gb, gt = oracle.global_rows(pos, cu_q)

    # Eq. 5 transforms: Q^G on the selected rows, K^G and V^G on every row
    qG, kG, vG = f(layer.qG), f(layer.kG), f(layer.vG)
    check_close(qG[gb, gt], oracle.branch_fwd(f(qL), A=f(Aq), rows=(gb, gt)), "Q^G (selected rows)")
    check_close(kG.reshape(-1, Hkv, D), oracle.branch_fwd(f(kL), A=f(Ak)), "K^G")
    check_close(vG.reshape(-1, Hkv, D), oracle.branch_fwd(f(vL), A=f(Av)), "V^G")

    # both branches on the GPU's branch inputs, then Eq. 9/10
    oL, _ = oracle.attn_fwd(f(qL), f(kL), f(vL), lb, lt, W)
    check_close(f(layer.o_l).reshape(-1, Hq, D), oL, "O^L")
    oG, _ = oracle.attn_fwd(qG, kG, vG, gb, gt, 0)
    o_c = f(layer.o_c)[:n]
    check_close(o_c, oG, "O^G")
    o_l = f(layer.o_l)
    ro, _, _ = oracle.combine_fwd(o_l, o_c, p, z, row_of, f(gl), f(gg))
    check_close(f(o), ro, "o")

    # combine backward with the gain gradients
    dOL, dOG, dp = oracle.combine_bwd(f(dO), o_l, o_c, p, z, row_of, f(gl), f(gg))
    check_close(f(layer.dO_l), dOL, "dO^L")
    check_close(f(layer.dO_c)[:n], dOG, "dO^G")
    check_close(f(layer.dgate), dp, "dp")
    dgl, dgg = oracle.combine_dgain(f(dO), o_l, o_c, p, z, row_of)
    check_close(f(grads["dgain_l"]), dgl, "dgain_l")
    check_close(f(grads["dgain_g"]), dgg, "dgain_g")

    # global backward on the GPU's transformed inputs; dQ^G zero off the selection
    dqGc, dkG, dvG = oracle.attn_bwd(qG, kG, vG, gb, gt, 0, f(layer.dO_c)[:n])
    dqG = f(layer.dqG)
    check_close(dqG[gb, gt], dqGc, "dQ^G (selected rows)")
    off = np.ones((B, T), dtype=bool)
    off[gb, gt] = False
    assert (dqG[off] == 0).all()
    check_close(f(layer.dkG), dkG, "dK^G")
    check_close(f(layer.dvG), dvG, "dV^G")

    # transform backward on the GPU's dQ^G / dK^G / dV^G, added into the local gradients
    dqL, dkL, dvL = oracle.attn_bwd(f(qL), f(kL), f(vL), lb, lt, W, f(layer.dO_l).reshape(-1, Hq, D))
    duq, dAq = oracle.branch_bwd(f(qL), dqG[gb, gt], A=f(Aq), rows=(gb, gt))
    duk, dAk = oracle.branch_bwd(f(kL), f(layer.dkG).reshape(-1, Hkv, D), A=f(Ak))
    duv, dAv = oracle.branch_bwd(f(vL), f(layer.dvG).reshape(-1, Hkv, D), A=f(Av))
    dq_a = dqL.reshape(B, T, Hq, D)
    dq_tot = dq_a.copy()
    dq_tot[gb, gt] += duq
    dk_a, dv_a = dkL, dvL
    dk_tot, dv_tot = dk_a + duk.reshape(B, T, Hkv, D), dv_a + duv.reshape(B, T, Hkv, D)
    two = lambda a, tot: np.abs(a) + np.abs(tot)  # noqa: E731  (two bf16 roundings: of a, then of a + b)
    check_close(f(grads["dqL"]), dq_tot, "dQ^L (local + transformed global)", scale_ref=two(dq_a, dq_tot))
    check_close(f(grads["dkL"]), dk_tot, "dK^L (local + transformed global)", scale_ref=two(dk_a, dk_tot))
    check_close(f(grads["dvL"]), dv_tot, "dV^L (local + transformed global)", scale_ref=two(dv_a, dv_tot))
    check_close(f(grads["tq"]["dA"]), dAq, "dA_Q")
    check_close(f(grads["tk"]["dA"]), dAk, "dA_K")
    check_close(f(grads["tv"]["dA"]), dAv, "dA_V")

    # gate backward on the GPU's dp
    dx, dw = oracle.gate_bwd(f(x), f(w), f(layer.dgate))
    check_close(f(grads["dx"]), dx, "dx")
    check_close(f(grads["dw_g"]), dw, "dw_g")
