"""Pins for the CPU oracle, independent of the oracle itself (CPU only).

Each pin ties an oracle function to something the paper or the mathematics
fixes: a library routine computing the same special case (torch SDPA and
autograd, torch rms_norm, numpy sorts), a closed form, an invariant the paper
states, finite differences, or a value the paper prints (tests/golden/).
"""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(12345)


def _rand(*shape, scale=1.0):
    return (rng.standard_normal(shape) * scale).astype(np.float32)


# ------------------------------------------------------------------ selection
def test_threshold_matches_numpy_compare():
    p = rng.random((3, 257)).astype(np.float32)
    for b in (0.0, 0.25, 0.5, float(p[1, 7]), 0.999):
        z = oracle.select_threshold(p, b)
        np.testing.assert_array_equal(z, (p > np.float32(b)).astype(np.uint8))


def test_threshold_strict_at_equality():
    p = np.array([[0.5, 0.5000001, 0.4999999, 0.5]], dtype=np.float32)
    z = oracle.select_threshold(p, 0.5)
    assert z.tolist() == [[0, 1, 0, 0]]  # Eq. 7 compares with '>'


def test_pmask_start_selects_everything():
    g = json.load(open(os.path.join(GOLDEN, "pmask_threshold.json")))
    b0 = g["gate_center"] - g["gamma"] * g["S"]
    assert b0 == pytest.approx(g["b_th0"])
    p = (1.0 / (1.0 + np.exp(-rng.standard_normal((2, 300)) * 4))).astype(np.float32)
    p = np.clip(p, np.float32(1e-7), np.float32(1 - 1e-7))
    assert oracle.select_threshold(p, g["b_th0"]).all() == g["all_selected"]
    assert not oracle.select_threshold(p, 1.0).any()


def test_pmask_start_value_of_app_c1():
    g = json.load(open(os.path.join(GOLDEN, "pmask_threshold.json")))
    assert oracle.pmask_threshold(g["gamma"], g["S"]) == pytest.approx(g["b_th0"], abs=1e-12)


def test_budget_update_moves_the_threshold_as_sec32_states():
    # Sec. 3.2: F > rho raises b_th (fewer tokens), F < rho lowers it; Eq. 3 F = N / |B|
    g = 2.0 ** -11
    b, F = oracle.budget_update(6, 10, 0.5, g, 0.25)
    assert F == 0.6 and b > np.float32(0.25) and b - np.float32(0.25) == np.float32(g)
    b, F = oracle.budget_update(4, 10, 0.5, g, 0.25)
    assert F == 0.4 and b < np.float32(0.25) and np.float32(0.25) - b == np.float32(g)
    b, F = oracle.budget_update(5, 10, 0.5, g, 0.25)  # F == rho exactly: sign(0) = 0
    assert F == 0.5 and b == np.float32(0.25)
    b, F = oracle.budget_update(0, 7, 0.0, g, 0.25)   # nothing selected at rho = 0: no move
    assert F == 0.0 and b == np.float32(0.25)


def test_pmask_phase_ends_at_the_gate_centre():
    # Sec. 3.2 / App. C.1: from the P-mask start every token is selected while
    # b_th < 0 < p (F = 1), and with the gates spread over (0, 1) F stays above
    # rho = 0.25 all the way up, so each step raises b_th by gamma and it reaches
    # the gate centre 0.5 after S steps.  gamma = 2^-11 and S = 4096 keep every
    # value a multiple of 2^-11 below 2 in magnitude, so float32 is exact here.
    gamma, S = 2.0 ** -11, 4096
    b = np.float32(oracle.pmask_threshold(gamma, S))
    assert b == np.float32(-1.5)
    p = np.linspace(0.001, 0.999, 777, dtype=np.float32).reshape(1, -1)
    for step in range(S):
        z = oracle.select_threshold(p, b)
        n = int(z.sum())
        if b < 0:
            assert n == p.size  # P-mask: every token takes the global branch
        b, F = oracle.budget_update(n, p.size, 0.25, gamma, b)
        assert F > 0.25
    assert b == np.float32(0.5)


def test_controller_settles_at_the_rho_quantile():
    # Gates on a uniform grid p_t = (t + 0.5) / T: F(b) = #{p > b} / T = 1 - b up to
    # 1/T, so Eq. 11 drives b_th to the (1 - rho) quantile and then stays within
    # gamma (+ 1/T) of it, with F within the same distance of rho.  A sign error
    # in the update runs away instead.
    T, rho, gamma = 1000, 0.3, 2.0 ** -10
    p = ((np.arange(T) + 0.5) / T).astype(np.float32).reshape(1, -1)
    b = np.float32(0.5)
    tail = []
    for step in range(1200):
        n = int(oracle.select_threshold(p, b).sum())
        b, F = oracle.budget_update(n, T, rho, gamma, b)
        if step >= 1000:
            tail.append((float(b), F))
    assert all(abs(bb - (1 - rho)) <= gamma + 1.0 / T for bb, _ in tail)
    assert all(abs(F - rho) <= gamma + 2.0 / T for _, F in tail)
    assert len({bb for bb, _ in tail}) >= 2  # it oscillates around the target


def test_tiny_workload_selects_exactly_128():
    from paper_2608_29539_gb300.workloads import WORKLOADS, make_inputs
    x = make_inputs(WORKLOADS["tiny"])
    z = oracle.select_threshold(x["p"].numpy(), x["b_th"])
    assert int(z.sum()) == 128


def _topk_numpy(p, k):
    z = np.zeros(p.shape, np.uint8)
    for b in range(p.shape[0]):
        T = p.shape[1]
        order = np.lexsort((np.arange(T), -p[b].astype(np.float64)))  # p desc, t asc
        z[b, order[:k]] = 1
    return z


@pytest.mark.parametrize("T,k", [(1, 0), (1, 1), (100, 13), (1000, 125), (257, 257), (64, 0)])
def test_ratio_matches_lexsort_topk(T, k):
    p = rng.random((2, T)).astype(np.float32)
    z = oracle.select_ratio(p, k)
    np.testing.assert_array_equal(z, _topk_numpy(p, k))
    assert (z.sum(axis=1) == k).all()


def test_ratio_ties_go_to_lower_position():
    p = np.full((1, 10), 0.5, dtype=np.float32)
    p[0, 7] = 0.9
    z = oracle.select_ratio(p, 4)
    assert z[0].nonzero()[0].tolist() == [0, 1, 2, 7]
    p = np.zeros((1, 6), np.float32)
    p[0, 3] = -0.0
    assert oracle.select_ratio(p, 2)[0].nonzero()[0].tolist() == [0, 1]  # -0 == +0


def test_k_from_ratio():
    assert oracle.k_from_ratio(0.125, 16384) == 2048
    assert oracle.k_from_ratio(0.0625, 65536) == 4096
    assert oracle.k_from_ratio(1.0 / 32, 32768) == 1024
    assert oracle.k_from_ratio(1.0, 777) == 777
    assert oracle.k_from_ratio(0.0, 777) == 0


def test_compact_matches_nonzero():
    z = (rng.random((3, 50)) < 0.3).astype(np.uint8)
    pos, cu_q, row_of, n = oracle.compact(z)
    assert n == int(z.sum())
    bb, tt = np.nonzero(z)  # row-major order = batch-major, ascending t
    np.testing.assert_array_equal(pos, tt)
    np.testing.assert_array_equal(np.diff(cu_q), z.sum(axis=1))
    assert cu_q[0] == 0 and cu_q[-1] == n
    ref = -np.ones_like(row_of)
    ref[bb, tt] = np.arange(n)
    np.testing.assert_array_equal(row_of, ref)


# ------------------------------------------------------------------ attention
def _sdpa_ref(q, k, v, window, rows_t=None, grad_out=None):
    """torch float64 SDPA with an explicit boolean mask; q,k,v [B,T,H,D]."""
    qt = torch.tensor(q, dtype=torch.float64).transpose(1, 2).requires_grad_(True)
    kt = torch.tensor(k, dtype=torch.float64).transpose(1, 2).requires_grad_(True)
    vt = torch.tensor(v, dtype=torch.float64).transpose(1, 2).requires_grad_(True)
    T = q.shape[1]
    grp = q.shape[2] // k.shape[2]
    kk = kt.repeat_interleave(grp, dim=1)
    vv = vt.repeat_interleave(grp, dim=1)
    t = torch.arange(T)
    allowed = t[None, :] <= t[:, None]
    if window > 0:
        allowed &= t[None, :] > t[:, None] - window
    o = F.scaled_dot_product_attention(qt, kk, vv, attn_mask=allowed)
    o = o.transpose(1, 2)  # [B,T,H,D]
    if grad_out is None:
        return o.detach().numpy(), None
    o.backward(torch.tensor(grad_out, dtype=torch.float64))
    return o.detach().numpy(), (qt.grad.transpose(1, 2).numpy(), kt.grad.transpose(1, 2).numpy(),
                                vt.grad.transpose(1, 2).numpy())


@pytest.mark.parametrize("window", [0, 1, 5, 16, 64])
@pytest.mark.parametrize("Hq,Hkv", [(2, 2), (4, 2)])
def test_attn_fwd_matches_torch_sdpa(window, Hq, Hkv):
    B, T, D = 2, 37, 16
    q, k, v = _rand(B, T, Hq, D), _rand(B, T, Hkv, D), _rand(B, T, Hkv, D)
    rb, rt = oracle.local_rows(B, T)
    o, lse = oracle.attn_fwd(q, k, v, rb, rt, window)
    ref, _ = _sdpa_ref(q, k, v, window)
    np.testing.assert_allclose(o.reshape(B, T, Hq, D), ref, rtol=1e-10, atol=1e-12)


def test_attn_lse_matches_logsumexp():
    B, T, H, D = 1, 20, 2, 8
    q, k, v = _rand(B, T, H, D), _rand(B, T, H, D), _rand(B, T, H, D)
    rb, rt = oracle.local_rows(B, T)
    for window in (0, 6):
        _, lse = oracle.attn_fwd(q, k, v, rb, rt, window)
        s = torch.einsum("bthd,bshd->bhts", torch.tensor(q, dtype=torch.float64),
                         torch.tensor(k, dtype=torch.float64)) / math.sqrt(D)
        t = torch.arange(T)
        allowed = (t[None, :] <= t[:, None]) & ((t[None, :] > t[:, None] - window) if window > 0 else True)
        ref = torch.logsumexp(s.masked_fill(~allowed, -math.inf), dim=-1)  # [B,H,T]
        np.testing.assert_allclose(lse.reshape(B, T, H), ref.permute(0, 2, 1).numpy(), rtol=1e-12, atol=1e-12)


def test_attn_closed_forms():
    B, T, H, D = 1, 30, 3, 8
    k, v = _rand(B, T, H, D), _rand(B, T, H, D)
    rb, rt = oracle.local_rows(B, T)
    # q = 0: uniform weights over the visible keys -> the mean of their values, lse = log(count)
    q0 = np.zeros((B, T, H, D), np.float32)
    for window in (0, 7):
        o, lse = oracle.attn_fwd(q0, k, v, rb, rt, window)
        for t in range(T):
            lo = max(0, t - window + 1) if window > 0 else 0
            np.testing.assert_allclose(o[t], v[0, lo:t + 1].astype(np.float64).mean(axis=0), rtol=1e-12, atol=1e-12)
            np.testing.assert_allclose(lse[t], math.log(t + 1 - lo), rtol=0, atol=1e-12)
    # constant values -> output is that constant whatever the weights
    q = _rand(B, T, H, D, scale=3.0)
    vc = np.broadcast_to(np.arange(D, dtype=np.float32), (B, T, H, D)).copy()
    o, _ = oracle.attn_fwd(q, k, vc, rb, rt, 0)
    np.testing.assert_allclose(o, np.broadcast_to(np.arange(D, dtype=np.float64), o.shape), atol=1e-10)
    # the first token sees only itself; window 1 sees only itself everywhere
    o, _ = oracle.attn_fwd(q, k, v, rb, rt, 1)
    np.testing.assert_allclose(o, v[0].astype(np.float64), atol=0)


def test_window_at_least_T_is_full_causal():
    B, T, H, D = 2, 25, 2, 8
    q, k, v = _rand(B, T, H, D), _rand(B, T, H, D), _rand(B, T, H, D)
    rb, rt = oracle.local_rows(B, T)
    o_full, l_full = oracle.attn_fwd(q, k, v, rb, rt, 0)
    for w in (T, T + 1, 10 * T):
        o_w, l_w = oracle.attn_fwd(q, k, v, rb, rt, w)
        np.testing.assert_array_equal(o_w, o_full)
        np.testing.assert_array_equal(l_w, l_full)


def test_global_rows_equal_dense_causal_rows():
    # Eq. 8: a selected row gets exactly the dense causal output of its position;
    # ratio = 1 selects every row and reproduces dense causal attention.
    B, T, H, D = 2, 33, 2, 16
    q, k, v = _rand(B, T, H, D), _rand(B, T, H, D), _rand(B, T, H, D)
    ref, _ = _sdpa_ref(q, k, v, 0)
    p = rng.random((B, T)).astype(np.float32)
    for kk in (0, 1, 9, T):
        z = oracle.select_ratio(p, kk)
        pos, cu_q, row_of, n = oracle.compact(z)
        rb, rt = oracle.global_rows(pos, cu_q)
        o, _ = oracle.attn_fwd(q, k, v, rb, rt, 0)
        assert o.shape[0] == n
        np.testing.assert_allclose(o, ref[rb, rt], rtol=1e-10, atol=1e-12)


def test_head_subset_leaves_other_heads_untouched():
    B, T, H, D = 1, 12, 4, 8
    q, k, v = _rand(B, T, H, D), _rand(B, T, H, D), _rand(B, T, H, D)
    rb, rt = oracle.local_rows(B, T)
    o_all, _ = oracle.attn_fwd(q, k, v, rb, rt, 0)
    o_sub, _ = oracle.attn_fwd(q, k, v, rb, rt, 0, heads=[2])
    np.testing.assert_array_equal(o_sub[:, 2], o_all[:, 2])
    assert not o_sub[:, [0, 1, 3]].any()


@pytest.mark.parametrize("window", [0, 4, 11])
@pytest.mark.parametrize("Hq,Hkv", [(2, 2), (4, 1)])
def test_attn_bwd_matches_torch_autograd(window, Hq, Hkv):
    B, T, D = 2, 23, 8
    q, k, v = _rand(B, T, Hq, D), _rand(B, T, Hkv, D), _rand(B, T, Hkv, D)
    dO = _rand(B, T, Hq, D)
    rb, rt = oracle.local_rows(B, T)
    dq, dk, dv = oracle.attn_bwd(q, k, v, rb, rt, window, dO.reshape(B * T, Hq, D))
    _, (rq, rk, rv) = _sdpa_ref(q, k, v, window, grad_out=dO)
    np.testing.assert_allclose(dq.reshape(B, T, Hq, D), rq, rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(dk, rk, rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(dv, rv, rtol=1e-9, atol=1e-11)


def test_attn_bwd_selected_rows_only():
    # Sec. 3.3: K/V gradients accumulate over the selected query rows only.
    B, T, H, D = 1, 19, 2, 8
    q, k, v = _rand(B, T, H, D), _rand(B, T, H, D), _rand(B, T, H, D)
    sel = np.array([2, 3, 11, 18])
    dO = _rand(len(sel), H, D)
    dq, dk, dv = oracle.attn_bwd(q, k, v, np.zeros(len(sel), np.int32), sel, 0, dO)
    full = np.zeros((B, T, H, D), np.float32)
    full[0, sel] = dO
    _, (rq, rk, rv) = _sdpa_ref(q, k, v, 0, grad_out=full)
    np.testing.assert_allclose(dq, rq[0, sel], rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(dk, rk, rtol=1e-9, atol=1e-11)
    np.testing.assert_allclose(dv, rv, rtol=1e-9, atol=1e-11)
    # keys after the last selected position receive no gradient
    assert not dk[0, sel.max() + 1:].any() and not dv[0, sel.max() + 1:].any()


def test_attn_bwd_finite_differences():
    B, T, H, D = 1, 9, 1, 4
    q, k, v = _rand(B, T, H, D), _rand(B, T, H, D), _rand(B, T, H, D)
    dO = _rand(B * T, H, D)
    rb, rt = oracle.local_rows(B, T)
    window = 4
    dq, dk, dv = oracle.attn_bwd(q, k, v, rb, rt, window, dO)

    def loss(q_, k_, v_):
        o, _ = oracle.attn_fwd(q_, k_, v_, rb, rt, window)
        return float((o * dO.astype(np.float64)).sum())

    for name, arr, grad in (("q", q, dq.reshape(B, T, H, D)), ("k", k, dk), ("v", v, dv)):
        for idx in [(0, 0, 0, 1), (0, 4, 0, 3), (0, 8, 0, 0)]:
            hi, lo = arr.copy(), arr.copy()
            hi[idx] += np.float32(1e-2)
            lo[idx] -= np.float32(1e-2)
            step = float(hi[idx]) - float(lo[idx])
            args_hi = {"q": q, "k": k, "v": v}
            args_lo = dict(args_hi)
            args_hi[name], args_lo[name] = hi, lo
            fd = (loss(**{f"{a}_": b for a, b in args_hi.items()}) -
                  loss(**{f"{a}_": b for a, b in args_lo.items()})) / step
            assert fd == pytest.approx(grad[idx], rel=2e-4, abs=1e-6), (name, idx)


# -------------------------------------------------------------------- combine
def _setup_combine(B=2, T=13, H=3, D=16, ratio_k=5, gains=True):
    oL = _rand(B, T, H, D)
    p = rng.random((B, T)).astype(np.float32)
    z = oracle.select_ratio(p, ratio_k)
    pos, cu_q, row_of, n = oracle.compact(z)
    oGc = _rand(n, H, D)
    gL = (1 + 0.2 * _rand(H, D)) if gains else None
    gG = (1 + 0.2 * _rand(H, D)) if gains else None
    return oL, oGc, p, z, row_of, gL, gG, n


def test_contextnorm_matches_torch_rms_norm():
    oL, oGc, p, z, row_of, gL, gG, n = _setup_combine()
    zero = np.zeros_like(z)
    o, rL, _ = oracle.combine_fwd(oL, oGc, p, zero, -np.ones_like(row_of), gL, gG, eps=1e-6)
    H, D = gL.shape
    for h in range(H):
        ref = F.rms_norm(torch.tensor(oL[:, :, h], dtype=torch.float64), (D,),
                         weight=torch.tensor(gL[h], dtype=torch.float64), eps=1e-6)
        np.testing.assert_allclose(o[:, :, h], ref.numpy(), rtol=1e-12, atol=1e-12)


def test_contextnorm_closed_form_unit_gain():
    oL, oGc, p, z, row_of, _, _, n = _setup_combine()
    eps = 1e-3
    _, rL, rG = oracle.combine_fwd(oL, oGc, p, z, row_of, None, None, eps=eps)
    m = (oL.astype(np.float64) ** 2).mean(axis=-1)
    # with gain 1: mean_d(o~^2) = m r^2 = m / (m + eps)
    np.testing.assert_allclose(m * rL ** 2, m / (m + eps), rtol=1e-12)
    mg = (oGc.astype(np.float64) ** 2).mean(axis=-1)
    np.testing.assert_allclose(mg * rG ** 2, mg / (mg + eps), rtol=1e-12)


def test_fusion_reductions():
    oL, oGc, p, z, row_of, gL, gG, n = _setup_combine()
    oL_only, _, _ = oracle.combine_fwd(oL, oGc, p, np.zeros_like(z), -np.ones_like(row_of), gL, gG)
    o, _, _ = oracle.combine_fwd(oL, oGc, p, z, row_of, gL, gG)
    # unselected tokens reduce exactly to the local output (Sec. 3.2, after Eq. 10)
    np.testing.assert_array_equal(o[z == 0], oL_only[z == 0])
    # p -> 0 on selected rows gives the local output, p -> 1 the global one
    o0, _, _ = oracle.combine_fwd(oL, oGc, np.zeros_like(p), z, row_of, gL, gG)
    np.testing.assert_allclose(o0, oL_only, atol=1e-12)
    o1, _, _ = oracle.combine_fwd(oL, oGc, np.ones_like(p), z, row_of, gL, gG)
    bb, tt = np.nonzero(z)
    H, D = gG.shape
    for h in range(H):
        ref = F.rms_norm(torch.tensor(oGc[:, h], dtype=torch.float64), (D,),
                         weight=torch.tensor(gG[h], dtype=torch.float64), eps=1e-6).numpy()
        np.testing.assert_allclose(o1[bb, tt, h], ref, atol=1e-12)
    # convex combination: o = (1-p) oL~ + p oG~ is linear in p
    ph = (0.5 * np.ones_like(p)).astype(np.float32)
    oh, _, _ = oracle.combine_fwd(oL, oGc, ph, z, row_of, gL, gG)
    np.testing.assert_allclose(oh, 0.5 * (o0 + o1), atol=1e-12)


def test_combine_bwd_finite_differences():
    oL, oGc, p, z, row_of, gL, gG, n = _setup_combine(B=1, T=7, H=2, D=8, ratio_k=3)
    dO = _rand(*oL.shape)
    dOL, dOG, dp = oracle.combine_bwd(dO, oL, oGc, p, z, row_of, gL, gG)

    def loss(oL_, oGc_, p_):
        o, _, _ = oracle.combine_fwd(oL_, oGc_, p_, z, row_of, gL, gG)
        return float((o * dO.astype(np.float64)).sum())

    h = np.float32(1e-2)
    for idx in [(0, 0, 0, 0), (0, 3, 1, 5), (0, 6, 0, 7)]:
        hi, lo = oL.copy(), oL.copy()
        hi[idx] += h
        lo[idx] -= h
        fd = (loss(hi, oGc, p) - loss(lo, oGc, p)) / (float(hi[idx]) - float(lo[idx]))
        assert fd == pytest.approx(dOL[idx], rel=1e-3, abs=1e-6)
    for idx in [(0, 0, 0), (n - 1, 1, 7)]:
        hi, lo = oGc.copy(), oGc.copy()
        hi[idx] += h
        lo[idx] -= h
        fd = (loss(oL, hi, p) - loss(oL, lo, p)) / (float(hi[idx]) - float(lo[idx]))
        assert fd == pytest.approx(dOG[idx], rel=1e-3, abs=1e-6)
    for t in range(oL.shape[1]):
        hi, lo = p.copy(), p.copy()
        hi[0, t] += h
        lo[0, t] -= h
        fd = (loss(oL, oGc, hi) - loss(oL, oGc, lo)) / (float(hi[0, t]) - float(lo[0, t]))
        assert fd == pytest.approx(dp[0, t], rel=1e-6, abs=1e-9)
    assert (dp[z == 0] == 0).all()


def test_combine_bwd_matches_torch_autograd():
    oL, oGc, p, z, row_of, gL, gG, n = _setup_combine()
    dO = _rand(*oL.shape)
    dOL, dOG, dp = oracle.combine_bwd(dO, oL, oGc, p, z, row_of, gL, gG)
    B, T, H, D = oL.shape
    tL = torch.tensor(oL, dtype=torch.float64, requires_grad=True)
    tG = torch.tensor(oGc, dtype=torch.float64, requires_grad=True)
    tp = torch.tensor(p, dtype=torch.float64, requires_grad=True)
    nL = torch.stack([F.rms_norm(tL[:, :, h], (D,), weight=torch.tensor(gL[h], dtype=torch.float64), eps=1e-6)
                      for h in range(H)], dim=2)
    nG = torch.stack([F.rms_norm(tG[:, h], (D,), weight=torch.tensor(gG[h], dtype=torch.float64), eps=1e-6)
                      for h in range(H)], dim=1)
    bb, tt = np.nonzero(z)
    full_g = torch.zeros_like(nL).index_put((torch.tensor(bb), torch.tensor(tt)), nG)
    zt = torch.tensor(z, dtype=torch.float64)[..., None, None]
    pp = tp[..., None, None]
    o = zt * ((1 - pp) * nL + pp * full_g) + (1 - zt) * nL
    o.backward(torch.tensor(dO, dtype=torch.float64))
    np.testing.assert_allclose(dOL, tL.grad.numpy(), rtol=1e-9, atol=1e-12)
    np.testing.assert_allclose(dOG, tG.grad.numpy(), rtol=1e-9, atol=1e-12)
    np.testing.assert_allclose(dp, tp.grad.numpy(), rtol=1e-9, atol=1e-12)


def test_gain_grads_match_torch_autograd():
    oL, oGc, p, z, row_of, gL, gG, n = _setup_combine()
    dO = _rand(*oL.shape)
    dgL, dgG = oracle.combine_dgain(dO, oL, oGc, p, z, row_of)
    B, T, H, D = oL.shape
    wL = torch.tensor(gL, dtype=torch.float64, requires_grad=True)
    wG = torch.tensor(gG, dtype=torch.float64, requires_grad=True)
    nL = torch.stack([F.rms_norm(torch.tensor(oL[:, :, h], dtype=torch.float64), (D,), weight=wL[h], eps=1e-6)
                      for h in range(H)], dim=2)
    nG = torch.stack([F.rms_norm(torch.tensor(oGc[:, h], dtype=torch.float64), (D,), weight=wG[h], eps=1e-6)
                      for h in range(H)], dim=1)
    bb, tt = np.nonzero(z)
    full_g = torch.zeros_like(nL).index_put((torch.tensor(bb), torch.tensor(tt)), nG)
    zt = torch.tensor(z, dtype=torch.float64)[..., None, None]
    pp = torch.tensor(p, dtype=torch.float64)[..., None, None]
    o = zt * ((1 - pp) * nL + pp * full_g) + (1 - zt) * nL
    o.backward(torch.tensor(dO, dtype=torch.float64))
    np.testing.assert_allclose(dgL, wL.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(dgG, wG.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_gain_grads_finite_differences_and_special_cases():
    oL, oGc, p, z, row_of, gL, gG, n = _setup_combine(B=1, T=7, H=2, D=8, ratio_k=3)
    dO = _rand(*oL.shape)
    dgL, dgG = oracle.combine_dgain(dO, oL, oGc, p, z, row_of)

    def loss(gL_, gG_):
        o, _, _ = oracle.combine_fwd(oL, oGc, p, z, row_of, gL_, gG_)
        return float((o * dO.astype(np.float64)).sum())

    for idx in [(0, 0), (1, 5), (0, 7)]:
        for which in (0, 1):
            hi = [gL.copy(), gG.copy()]
            lo = [gL.copy(), gG.copy()]
            hi[which][idx] += np.float32(0.25)
            lo[which][idx] -= np.float32(0.25)
            step = float(hi[which][idx]) - float(lo[which][idx])
            fd = (loss(*hi) - loss(*lo)) / step  # exact up to rounding: the output is linear in a gain
            assert fd == pytest.approx((dgL, dgG)[which][idx], rel=1e-9, abs=1e-12)
    # nothing selected: no gradient reaches the global gain; p = 0 on the selected
    # tokens: the local gain sees dO itself on every token
    dgL0, dgG0 = oracle.combine_dgain(dO, oL, oGc, p, np.zeros_like(z), row_of)
    assert (dgG0 == 0).all()
    _, rL, _ = oracle.combine_fwd(oL, oGc, p, np.zeros_like(z), row_of, None, None)
    ref = (dO.astype(np.float64) * oL.astype(np.float64) * rL[..., None]).sum(axis=(0, 1))
    np.testing.assert_allclose(dgL0, ref, rtol=1e-12, atol=1e-12)


def test_gate_matches_numpy_and_closed_forms():
    rng = np.random.default_rng(11)
    x = rng.standard_normal((3, 17, 64)).astype(np.float32)
    w = (0.1 * rng.standard_normal(64)).astype(np.float32)
    p = oracle.gate(x, w)
    logit = x.astype(np.float64) @ w.astype(np.float64)
    np.testing.assert_allclose(p, 1.0 / (1.0 + np.exp(-logit)), rtol=1e-14)
    np.testing.assert_allclose(p, torch.sigmoid(torch.tensor(logit)).numpy(), rtol=1e-14)
    # near-zero init of the gate (Sec. 3.2): w = 0 puts every p at exactly 0.5
    assert (oracle.gate(x, np.zeros(64, np.float32)) == 0.5).all()
    # one active coordinate: p = sigmoid(x_i w_i); opposite inputs give 1 - p
    e = np.zeros(64, np.float32)
    e[5] = 2.0
    np.testing.assert_allclose(oracle.gate(x, e), 1 / (1 + np.exp(-2.0 * x[..., 5].astype(np.float64))), rtol=1e-14)
    np.testing.assert_allclose(oracle.gate(-x, w), 1.0 - p, rtol=1e-12, atol=1e-15)


def test_gate_bwd_matches_torch_autograd_and_finite_differences():
    rng = np.random.default_rng(12)
    x = rng.standard_normal((2, 9, 32)).astype(np.float32)
    w = (0.2 * rng.standard_normal(32)).astype(np.float32)
    dp = rng.standard_normal((2, 9)).astype(np.float32)
    dx, dw = oracle.gate_bwd(x, w, dp)
    tx = torch.tensor(x, dtype=torch.float64, requires_grad=True)
    tw = torch.tensor(w, dtype=torch.float64, requires_grad=True)
    torch.sigmoid(tx @ tw).backward(torch.tensor(dp, dtype=torch.float64))
    np.testing.assert_allclose(dx, tx.grad.numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(dw, tw.grad.numpy(), rtol=1e-12, atol=1e-15)
    loss = lambda w_: float((oracle.gate(x, w_) * dp.astype(np.float64)).sum())  # noqa: E731
    for i in (0, 13, 31):
        hi, lo = w.copy(), w.copy()
        hi[i] += np.float32(1e-3)
        lo[i] -= np.float32(1e-3)
        fd = (loss(hi) - loss(lo)) / (float(hi[i]) - float(lo[i]))
        assert fd == pytest.approx(dw[i], rel=1e-5, abs=1e-9)
    # dp = 0 passes no gradient; w = 0 gives dlogit = dp / 4 and dx = 0
    dx0, dw0 = oracle.gate_bwd(x, w, np.zeros_like(dp))
    assert (dx0 == 0).all() and (dw0 == 0).all()
    dxz, dwz = oracle.gate_bwd(x, np.zeros_like(w), dp)
    assert (dxz == 0).all()
    np.testing.assert_allclose(dwz, (dp.astype(np.float64)[..., None] / 4 * x).sum(axis=(0, 1)), rtol=1e-12)


def test_branch_transform_matches_einsum_and_identity():
    rng = np.random.default_rng(21)
    u = rng.standard_normal((2, 9, 3, 16)).astype(np.float32)
    A = rng.standard_normal((3, 16, 16)).astype(np.float32)
    s_ = rng.standard_normal((3, 16)).astype(np.float32)
    b_ = rng.standard_normal((3, 16)).astype(np.float32)
    g = oracle.branch_fwd(u, A=A)
    ref = np.einsum("bthi,hij->bthj", u.astype(np.float64), A.astype(np.float64)).reshape(-1, 3, 16)
    np.testing.assert_allclose(g, ref, rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(oracle.branch_fwd(u, s=s_, b=b_),
                               (u.astype(np.float64) * s_ + b_).reshape(-1, 3, 16), rtol=1e-15, atol=1e-15)
    # identity initialisation (Sec. 3.2): both forms start as U^G = U^L exactly
    eye = np.broadcast_to(np.eye(16, dtype=np.float32), (3, 16, 16)).copy()
    assert (oracle.branch_fwd(u, A=eye) == u.reshape(-1, 3, 16)).all()
    assert (oracle.branch_fwd(u, s=np.ones((3, 16), np.float32), b=np.zeros((3, 16), np.float32))
            == u.reshape(-1, 3, 16)).all()
    # a row subset gives those rows of the full result, in the listed order
    rb, rt = np.array([1, 0, 1]), np.array([8, 2, 0])
    np.testing.assert_array_equal(oracle.branch_fwd(u, A=A, rows=(rb, rt)), g.reshape(2, 9, 3, 16)[rb, rt])


def test_branch_transform_bwd_matches_torch_autograd():
    rng = np.random.default_rng(22)
    u = rng.standard_normal((2, 7, 2, 8)).astype(np.float32)
    A = rng.standard_normal((2, 8, 8)).astype(np.float32)
    s_ = rng.standard_normal((2, 8)).astype(np.float32)
    b_ = rng.standard_normal((2, 8)).astype(np.float32)
    rb, rt = np.array([0, 0, 1, 1, 1]), np.array([1, 4, 0, 2, 6])
    dg = rng.standard_normal((5, 2, 8)).astype(np.float32)
    du, dA = oracle.branch_bwd(u, dg, A=A, rows=(rb, rt))
    tu = torch.tensor(u, dtype=torch.float64, requires_grad=True)
    tA = torch.tensor(A, dtype=torch.float64, requires_grad=True)
    torch.einsum("rhi,hij->rhj", tu[rb, rt], tA).backward(torch.tensor(dg, dtype=torch.float64))
    np.testing.assert_allclose(du, tu.grad.numpy()[rb, rt], rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(dA, tA.grad.numpy(), rtol=1e-12, atol=1e-13)
    du2, ds, db = oracle.branch_bwd(u, dg, s=s_, rows=(rb, rt))
    tu = torch.tensor(u, dtype=torch.float64, requires_grad=True)
    ts = torch.tensor(s_, dtype=torch.float64, requires_grad=True)
    tb = torch.tensor(b_, dtype=torch.float64, requires_grad=True)
    (tu[rb, rt] * ts + tb).backward(torch.tensor(dg, dtype=torch.float64))
    np.testing.assert_allclose(du2, tu.grad.numpy()[rb, rt], rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(ds, ts.grad.numpy(), rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(db, tb.grad.numpy(), rtol=1e-12, atol=1e-13)
    # finite difference on one entry of A (the loss is linear in A: exact up to rounding)
    loss = lambda A_: float((oracle.branch_fwd(u, A=A_, rows=(rb, rt)) * dg.astype(np.float64)).sum())  # noqa: E731
    hi, lo = A.copy(), A.copy()
    hi[1, 3, 5] += np.float32(0.5)
    lo[1, 3, 5] -= np.float32(0.5)
    step = float(hi[1, 3, 5]) - float(lo[1, 3, 5])
    assert (loss(hi) - loss(lo)) / step == pytest.approx(dA[1, 3, 5], rel=1e-10, abs=1e-12)


def test_ratio_zero_layer_is_pure_local():
    # rho = 0: no token is selected, the layer output is Norm^L(O^L) and no
    # gradient reaches the global branch or the gate.
    oL, _, p, _, _, gL, gG, _ = _setup_combine()
    z = oracle.select_ratio(p, 0)
    pos, cu_q, row_of, n = oracle.compact(z)
    assert n == 0
    o, _, _ = oracle.combine_fwd(oL, np.zeros((0,), np.float32), p, z, row_of, gL, gG)
    dO = _rand(*oL.shape)
    dOL, dOG, dp = oracle.combine_bwd(dO, oL, np.zeros((0,), np.float32), p, z, row_of, gL, gG)
    assert dOG.shape[0] == 0 and not dp.any()
    H, D = gL.shape
    for h in range(H):
        ref = F.rms_norm(torch.tensor(oL[:, :, h], dtype=torch.float64), (D,),
                         weight=torch.tensor(gL[h], dtype=torch.float64), eps=1e-6)
        np.testing.assert_allclose(o[:, :, h], ref.numpy(), rtol=1e-12, atol=1e-12)
