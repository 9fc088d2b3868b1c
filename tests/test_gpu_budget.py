"""Device-resident routing loop (Sec. 3.2 Budget Control): each step runs
logo_select_device_threshold (Eq. 7 with the threshold read on the device) and
logo_budget_update (Eq. 3 + Eq. 11 in place), with no host synchronisation
inside the loop.  Every step's routing, count, realised ratio and threshold
must equal the oracle's float32 recurrence bit for bit."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def _buffers(B, T, dev):
    from paper_2608_29539_gb300 import logo as L
    z = torch.empty((B, T), dtype=torch.uint8, device=dev)
    pos = torch.empty((B * T,), dtype=torch.int32, device=dev)
    cu_q = torch.empty((B + 1,), dtype=torch.int32, device=dev)
    row_of = torch.empty((B, T), dtype=torch.int32, device=dev)
    n_sel = torch.empty((1,), dtype=torch.int32, device=dev)
    ws = torch.empty(L.workspace_bytes("select", L.Dims(B, T, 1, 1, 64)), dtype=torch.uint8, device=dev)
    return z, pos, cu_q, row_of, n_sel, ws


def test_device_threshold_select_equals_host_threshold_select():
    from paper_2608_29539_gb300 import logo as L
    dev = torch.device("cuda")
    rng = np.random.default_rng(7)
    B, T = 2, 3001
    p = torch.from_numpy(rng.uniform(0, 1, (B, T)).astype(np.float32)).to(dev)
    for b in (0.37, -0.5, 1.0, float(p[1, 17])):
        ref = [t.clone() for t in L.logo_select(p, L.LOGO_SELECT_THRESHOLD, b_th=b)]
        got = L.logo_select_device_threshold(p, torch.tensor([b], dtype=torch.float32, device=dev))
        torch.cuda.synchronize()
        n = int(ref[4][0])
        assert int(got[4][0]) == n
        assert torch.equal(got[0], ref[0]) and torch.equal(got[2], ref[2]) and torch.equal(got[3], ref[3])
        assert torch.equal(got[1][:n], ref[1][:n])


def test_device_budget_loop_matches_oracle():
    from paper_2608_29539_gb300 import logo as L
    dev = torch.device("cuda")
    rng = np.random.default_rng(2608)
    B, T, K = 3, 2500, 48  # T is not a multiple of select's 1024-token chunk
    rho, gamma, pmask_steps = 0.2, 2.0 ** -5, 8
    # gates drift from step to step so that the controller moves both ways
    base = rng.uniform(0.0, 1.0, (B, T)).astype(np.float32)
    p_all = np.stack([
        np.clip(base + np.float32(0.15 * np.sin(k / 5.0)) + rng.normal(0.0, 0.02, (B, T)).astype(np.float32),
                1e-6, 1.0 - 1e-6).astype(np.float32)
        for k in range(K)
    ])
    b0 = L.logo_pmask_initial_threshold(gamma, pmask_steps)
    p_dev = torch.from_numpy(p_all).to(dev)
    b_th = torch.tensor([b0], dtype=torch.float32, device=dev)
    f_dev = torch.empty((1,), dtype=torch.float32, device=dev)
    z, pos, cu_q, row_of, n_sel, ws = _buffers(B, T, dev)
    z_all = torch.empty((K, B, T), dtype=torch.uint8, device=dev)
    n_all = torch.empty((K,), dtype=torch.int32, device=dev)
    b_traj = torch.empty((K,), dtype=torch.float32, device=dev)
    f_traj = torch.empty((K,), dtype=torch.float32, device=dev)
    for k in range(K):
        L.logo_select_device_threshold(p_dev[k], b_th, z, pos, cu_q, row_of, n_sel, workspace=ws)
        z_all[k].copy_(z)
        n_all[k].copy_(n_sel[0])
        L.logo_budget_update(n_sel, B, T, rho, gamma, b_th, f_out=f_dev)
        b_traj[k].copy_(b_th[0])
        f_traj[k].copy_(f_dev[0])
    torch.cuda.synchronize()
    zs, ns = z_all.cpu().numpy(), n_all.cpu().numpy()
    bt, ft = b_traj.cpu().numpy(), f_traj.cpu().numpy()

    b = np.float32(b0)
    up = down = 0
    for k in range(K):
        zo = oracle.select_threshold(p_all[k], b)
        np.testing.assert_array_equal(zs[k], zo)
        n = int(zo.sum())
        assert int(ns[k]) == n
        b_new, F = oracle.budget_update(n, B * T, rho, gamma, b)
        assert bt[k] == b_new, (k, bt[k], b_new)
        assert ft[k] == np.float32(F)
        up += int(b_new > b)
        down += int(b_new < b)
        b = b_new
    assert up > 0 and down > 0
    # packing of the last step
    pos_o, cu_o, row_o, n_o = oracle.compact(zs[-1])
    assert int(cu_q.cpu()[-1]) == n_o
    np.testing.assert_array_equal(cu_q.cpu().numpy(), cu_o)
    np.testing.assert_array_equal(row_of.cpu().numpy(), row_o)
    np.testing.assert_array_equal(pos.cpu().numpy()[:n_o], pos_o)
