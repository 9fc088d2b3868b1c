"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Every case feeds both sides the same seeded inputs (the bf16 values the GPU
gets, upcast for the oracle) and compares element by element: indices
bit-exact, floating outputs within max-abs <= 2e-2 and relative L2 <= 1e-2.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from helpers import check_close, np32, seeded

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_29539_gb300 import build
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    yield
    from paper_2608_29539_gb300 import logo as L
    assert L.logo_get_device_status() == 0


def L():
    from paper_2608_29539_gb300 import logo
    return logo


# ------------------------------------------------------------------- select
def gpu_select(p, mode, b_th=0.5, ratio=0.0):
    z, pos, cu_q, row_of, n = L().logo_select(p.cuda(), mode, b_th, ratio)
    torch.cuda.synchronize()
    n = int(n.item())
    return z.cpu().numpy(), pos[:n].cpu().numpy(), cu_q.cpu().numpy(), row_of.cpu().numpy(), n


def oracle_select(p, mode, b_th=0.5, ratio=0.0):
    p = np32(p)
    if mode == L().LOGO_SELECT_THRESHOLD:
        z = oracle.select_threshold(p, b_th)
    else:
        z = oracle.select_ratio(p, oracle.k_from_ratio(ratio, p.shape[1]))
    pos, cu_q, row_of, n = oracle.compact(z)
    return z, pos, cu_q, row_of, n


def _gates(kind, B, T, seed):
    g = torch.Generator().manual_seed(seed)
    if kind == "normal":
        return torch.sigmoid(torch.randn((B, T), generator=g))
    if kind == "ties":  # only 7 distinct values: many exact ties
        return (torch.randint(0, 7, (B, T), generator=g).float() / 8.0).contiguous()
    if kind == "signed_zero":
        x = torch.zeros((B, T))
        x[:, ::3] = -0.0
        x[:, 5::7] = 0.5
        return x
    if kind == "clustered":
        from paper_2608_29539_gb300.workloads import clustered_logits
        return torch.sigmoid(torch.stack([clustered_logits(T, g) for _ in range(B)]))
    raise ValueError(kind)


SELECT_CASES = [
    # kind, B, T, mode, b_th, ratio
    ("normal", 1, 512, 0, 0.6747, 0.0),
    ("normal", 3, 5000, 1, 0.0, 0.125),
    ("normal", 2, 1025, 1, 0.0, 0.3),
    ("ties", 2, 3000, 1, 0.0, 0.3),
    ("ties", 1, 2049, 0, 0.5, 0.0),
    ("signed_zero", 2, 100, 1, 0.0, 0.5),
    ("clustered", 1, 16384, 1, 0.0, 0.125),
    ("normal", 2, 777, 0, -2.0, 0.0),   # P-mask start: everything selected
    ("normal", 2, 777, 0, 1.0, 0.0),    # nothing selected
    ("normal", 2, 777, 1, 0.0, 0.0),
    ("normal", 2, 777, 1, 0.0, 1.0),
    ("normal", 1, 1, 1, 0.0, 1.0),
    ("normal", 1, 1, 0, 0.5, 0.0),
    ("normal", 4, 65536, 1, 0.0, 0.0625),
    ("ties", 3, 4097, 1, 0.0, 0.25),       # one-block ratio path: 16 tokens per thread, ragged
    ("ties", 2, 4096, 1, 0.0, 0.25),       # ... 4 tokens per thread, full
    ("normal", 1, 16385, 1, 0.0, 0.125),   # cluster path, 4 tokens per thread
    ("normal", 2, 5000, 1, 0.0, 0.0),      # cluster path, k = 0
    ("normal", 1, 9000, 1, 0.0, 1.0),      # cluster path, k = T
    ("ties", 2, 32768, 1, 0.0, 0.5),       # cluster path, ties spanning every CTA
    ("normal", 1, 131072, 1, 0.0, 0.125),  # largest cluster case, 16 tokens per thread
    ("normal", 1, 140000, 1, 0.0, 0.01),   # beyond the cluster path: multi-launch radix select
]


@pytest.mark.parametrize("kind,B,T,mode,b_th,ratio", SELECT_CASES)
def test_select_bit_exact(kind, B, T, mode, b_th, ratio):
    p = _gates(kind, B, T, seed=T + B).float().contiguous()
    gz, gpos, gcu, grow, gn = gpu_select(p, mode, b_th, ratio)
    oz, opos, ocu, orow, on = oracle_select(p, mode, b_th, ratio)
    assert gn == on
    np.testing.assert_array_equal(gz, oz)
    np.testing.assert_array_equal(gpos, opos)
    np.testing.assert_array_equal(gcu, ocu)
    np.testing.assert_array_equal(grow, orow)


def test_select_tiny_workload_exactly_128():
    from paper_2608_29539_gb300.workloads import WORKLOADS, make_inputs
    x = make_inputs(WORKLOADS["tiny"])
    gz, gpos, gcu, grow, gn = gpu_select(x["p"], 0, x["b_th"])
    assert gn == 128
    oz, opos, *_ = oracle_select(x["p"], 0, x["b_th"])
    np.testing.assert_array_equal(gpos, opos)


# ---------------------------------------------------------------- attention
def qkv(B, T, Hq, Hkv, D, seed, std=1.0):
    q = seeded((B, T, Hq, D), seed, torch.bfloat16, std)
    k = seeded((B, T, Hkv, D), seed + 1, torch.bfloat16, std)
    v = seeded((B, T, Hkv, D), seed + 2, torch.bfloat16)
    return q, k, v


LOCAL_CASES = [
    # B, T, Hq, Hkv, D, W
    (1, 512, 4, 4, 64, 64),
    (2, 300, 4, 2, 128, 17),
    (1, 257, 2, 2, 128, 1),
    (1, 200, 2, 1, 64, 1000),
    (2, 640, 2, 2, 128, 256),
    (1, 129, 1, 1, 128, 128),
    (1, 1, 1, 1, 64, 4),
]


@pytest.mark.parametrize("B,T,Hq,Hkv,D,W", LOCAL_CASES)
def test_local_fwd(B, T, Hq, Hkv, D, W):
    q, k, v = qkv(B, T, Hq, Hkv, D, seed=10 * T + W)
    o, lse = L().logo_local_attn_fwd(q.cuda(), k.cuda(), v.cuda(), W)
    torch.cuda.synchronize()
    rb, rt = oracle.local_rows(B, T)
    ro, rl = oracle.attn_fwd(np32(q), np32(k), np32(v), rb, rt, W)
    check_close(np32(o).reshape(B * T, Hq, D), ro, "o")
    check_close(np32(lse).transpose(0, 2, 1).reshape(B * T, Hq), rl, "lse", 1e-3, 1e-5, rel=0.0)


@pytest.mark.parametrize("B,T,Hq,Hkv,D,W", LOCAL_CASES)
def test_local_bwd(B, T, Hq, Hkv, D, W):
    q, k, v = qkv(B, T, Hq, Hkv, D, seed=7 * T + W)
    dO = seeded((B, T, Hq, D), 99 + T, torch.bfloat16)
    qc, kc, vc, dOc = q.cuda(), k.cuda(), v.cuda(), dO.cuda()
    o, lse = L().logo_local_attn_fwd(qc, kc, vc, W)
    dq, dk, dv = L().logo_local_attn_bwd(qc, kc, vc, o, lse, dOc, W)
    torch.cuda.synchronize()
    rb, rt = oracle.local_rows(B, T)
    rdq, rdk, rdv = oracle.attn_bwd(np32(q), np32(k), np32(v), rb, rt, W, np32(dO).reshape(B * T, Hq, D))
    check_close(np32(dq).reshape(B * T, Hq, D), rdq, "dq")
    check_close(np32(dk), rdk, "dk")
    check_close(np32(dv), rdv, "dv")


GLOBAL_CASES = [
    # B, T, Hq, Hkv, D, gate kind, ratio
    (1, 512, 4, 4, 64, "normal", 0.25),
    (2, 700, 4, 2, 128, "normal", 0.125),
    (1, 300, 2, 2, 128, "normal", 1.0),
    (2, 400, 2, 2, 128, "normal", 0.0),
    (1, 1000, 2, 1, 64, "clustered", 0.125),
    (3, 257, 2, 2, 128, "ties", 0.5),
    (1, 129, 1, 1, 128, "normal", 1.0 / 129),
    # few, long tiles: each tile's KV range is split into shares merged afterwards;
    # rows early in a tile see nothing of its later shares
    (1, 4096, 2, 1, 128, "normal", 0.05),
    (1, 6000, 1, 1, 64, "normal", 0.04),
]


def _global_setup(B, T, Hq, Hkv, D, kind, ratio, seed):
    q, k, v = qkv(B, T, Hq, Hkv, D, seed)
    p = _gates(kind, B, T, seed + 5).float().contiguous()
    z, pos, cu_q, row_of, n = L().logo_select(p.cuda(), L().LOGO_SELECT_RATIO, 0.0, ratio)
    torch.cuda.synchronize()
    nn = int(n.item())
    oz, opos, ocu, orow, on = oracle_select(p, 1, 0.0, ratio)
    assert nn == on
    np.testing.assert_array_equal(pos[:nn].cpu().numpy(), opos)
    return q, k, v, p, (z, pos, cu_q, row_of, n), nn, opos, ocu, orow


@pytest.mark.parametrize("B,T,Hq,Hkv,D,kind,ratio", GLOBAL_CASES)
def test_global_fwd(B, T, Hq, Hkv, D, kind, ratio):
    q, k, v, p, sel, n, opos, ocu, _ = _global_setup(B, T, Hq, Hkv, D, kind, ratio, seed=3 * T + 11)
    z, pos, cu_q, row_of, nt = sel
    o_c, lse_c = L().logo_global_sparse_attn_fwd(q.cuda(), k.cuda(), v.cuda(), pos, cu_q, nt)
    torch.cuda.synchronize()
    rb, rt = oracle.global_rows(opos, ocu)
    ro, rl = oracle.attn_fwd(np32(q), np32(k), np32(v), rb, rt, 0)
    check_close(np32(o_c)[:n], ro, "o_c")
    check_close(np32(lse_c)[:, :n].T, rl, "lse_c", 1e-3, 1e-5, rel=0.0)


@pytest.mark.parametrize("B,T,Hq,Hkv,D,kind,ratio", GLOBAL_CASES)
def test_global_bwd(B, T, Hq, Hkv, D, kind, ratio):
    q, k, v, p, sel, n, opos, ocu, _ = _global_setup(B, T, Hq, Hkv, D, kind, ratio, seed=5 * T + 3)
    z, pos, cu_q, row_of, nt = sel
    cap = B * T
    dO_c = torch.full((cap, Hq, D), float("nan"), dtype=torch.bfloat16)  # rows >= n must never be read
    dO_c[:n] = seeded((n, Hq, D), 77 + T, torch.bfloat16)
    qc, kc, vc = q.cuda(), k.cuda(), v.cuda()
    o_c, lse_c = L().logo_global_sparse_attn_fwd(qc, kc, vc, pos, cu_q, nt)
    # dq starts poisoned: every row, selected or not, must be written by the call
    dq0 = torch.full(qc.shape, float("nan"), dtype=torch.bfloat16, device=qc.device)
    dq, dk, dv = L().logo_global_sparse_attn_bwd(qc, kc, vc, pos, cu_q, nt, o_c, lse_c, dO_c.cuda(), dq=dq0)
    torch.cuda.synchronize()
    rb, rt = oracle.global_rows(opos, ocu)
    rdq_c, rdk, rdv = oracle.attn_bwd(np32(q), np32(k), np32(v), rb, rt, 0, np32(dO_c[:n]))
    rdq = np.zeros((B, T, Hq, D))
    rdq[rb, rt] = rdq_c
    gdq = np32(dq)
    # unselected rows: exactly zero (App. B)
    mask = np.ones((B, T), bool)
    mask[rb, rt] = False
    assert (gdq[mask] == 0).all()
    check_close(gdq, rdq, "dq")
    check_close(np32(dk), rdk, "dk")
    check_close(np32(dv), rdv, "dv")


# ------------------------------------------------------------------ combine
COMBINE_CASES = [
    # B, T, H, D, ratio, gains
    (2, 300, 4, 128, 0.25, True),
    (1, 513, 3, 64, 0.5, False),
    (2, 100, 2, 128, 0.0, True),
    (1, 64, 2, 64, 1.0, True),
    (1, 200, 32, 128, 0.125, False),  # unit gains, two vectors per thread (the 16K workload's width)
    (1, 100, 64, 128, 0.25, False),   # unit gains, four vectors per thread
]
# the widest rows the combine accepts (Hq*D = 16384, eight vectors per thread);
# beyond the gain-gradient variant's limit, so forward and backward only
WIDE_CASES = [(1, 50, 128, 128, 0.5, False), (1, 40, 128, 128, 0.5, True)]


def _combine_setup(B, T, H, D, ratio, gains, seed):
    p = _gates("normal", B, T, seed).float().contiguous()
    z, pos, cu_q, row_of, n = L().logo_select(p.cuda(), 1, 0.0, ratio)
    torch.cuda.synchronize()
    nn = int(n.item())
    o_l = seeded((B, T, H, D), seed + 1, torch.bfloat16, 0.3)
    o_c = seeded((B * T, H, D), seed + 2, torch.bfloat16, 0.3)
    gl = (1 + 0.1 * seeded((H, D), seed + 3)) if gains else None
    gg = (1 + 0.1 * seeded((H, D), seed + 4)) if gains else None
    return p, (z, row_of), nn, o_l, o_c, gl, gg


@pytest.mark.parametrize("B,T,H,D,ratio,gains", COMBINE_CASES + WIDE_CASES)
def test_combine_fwd(B, T, H, D, ratio, gains):
    p, (z, row_of), n, o_l, o_c, gl, gg = _combine_setup(B, T, H, D, ratio, gains, seed=T)
    cu = lambda t: None if t is None else t.cuda()  # noqa: E731
    o, rl, rg = L().logo_combine(o_l.cuda(), o_c.cuda(), p.cuda(), z, row_of, cu(gl), cu(gg), 1e-6)
    torch.cuda.synchronize()
    zn, rown = z.cpu().numpy(), row_of.cpu().numpy()
    ro, rrl, rrg = oracle.combine_fwd(np32(o_l), np32(o_c)[:n], np32(p), zn, rown,
                                      None if gl is None else np32(gl), None if gg is None else np32(gg), 1e-6)
    check_close(np32(o), ro, "o")
    check_close(np32(rl), rrl, "rstd_l", 1e-5, 1e-5, rel=1e-5)
    if n:
        check_close(np32(rg)[:n], rrg, "rstd_g", 1e-5, 1e-5, rel=1e-5)


@pytest.mark.parametrize("B,T,H,D,ratio,gains", COMBINE_CASES + WIDE_CASES)
def test_combine_bwd(B, T, H, D, ratio, gains):
    p, (z, row_of), n, o_l, o_c, gl, gg = _combine_setup(B, T, H, D, ratio, gains, seed=2 * T)
    dO = seeded((B, T, H, D), 5 * T, torch.bfloat16)
    cu = lambda t: None if t is None else t.cuda()  # noqa: E731
    dOl, dOc, dp = L().logo_combine_bwd(dO.cuda(), o_l.cuda(), o_c.cuda(), p.cuda(), z, row_of, cu(gl), cu(gg), 1e-6)
    torch.cuda.synchronize()
    zn, rown = z.cpu().numpy(), row_of.cpu().numpy()
    rdl, rdg, rdp = oracle.combine_bwd(np32(dO), np32(o_l), np32(o_c)[:n], np32(p), zn, rown,
                                       None if gl is None else np32(gl), None if gg is None else np32(gg), 1e-6)
    check_close(np32(dOl), rdl, "dO_l")
    if n:
        check_close(np32(dOc)[:n], rdg, "dO_c")
    check_close(np32(dp), rdp, "dgate_p")
    assert (np32(dp)[zn == 0] == 0).all()


GAIN_CASES = COMBINE_CASES + [
    (1, 700, 64, 128, 0.125, True),  # Hq*D = 8192, the largest supported: four vectors per thread
    (3, 77, 1, 64, 0.3, False),      # one head: most threads of a block idle
]


@pytest.mark.parametrize("B,T,H,D,ratio,gains", GAIN_CASES)
def test_combine_bwd_gains(B, T, H, D, ratio, gains):
    p, (z, row_of), n, o_l, o_c, gl, gg = _combine_setup(B, T, H, D, ratio, gains, seed=3 * T + H)
    dO = seeded((B, T, H, D), 7 * T, torch.bfloat16)
    cu = lambda t: None if t is None else t.cuda()  # noqa: E731
    args = (dO.cuda(), o_l.cuda(), o_c.cuda(), p.cuda(), z, row_of, cu(gl), cu(gg), 1e-6)
    plain = L().logo_combine_bwd(*args)
    with_gains = L().logo_combine_bwd_gains(*args)
    again = L().logo_combine_bwd_gains(*args)
    torch.cuda.synchronize()
    # the same input gradients as the plain call, bit for bit
    assert torch.equal(plain[0], with_gains[0]) and torch.equal(plain[2], with_gains[2])
    assert torch.equal(plain[1][:n], with_gains[1][:n])
    # deterministic: blocks are summed in a fixed order
    assert torch.equal(with_gains[3], again[3]) and torch.equal(with_gains[4], again[4])
    zn, rown = z.cpu().numpy(), row_of.cpu().numpy()
    rgl, rgg = oracle.combine_dgain(np32(dO), np32(o_l), np32(o_c)[:n], np32(p), zn, rown, 1e-6)
    check_close(np32(with_gains[3]), rgl, "dgain_l")
    check_close(np32(with_gains[4]), rgg, "dgain_g")
    if n == 0:
        assert bool((with_gains[4] == 0).all())


# --------------------------------------------------- whole step, small workload
def test_layer_step_4k_workload():
    """The 4K workload end to end through the layer chain; every call checked
    against the oracle on the same inputs it received."""
    from paper_2608_29539_gb300.layer import LayerConfig, LogoAttention
    from paper_2608_29539_gb300.workloads import WORKLOADS, make_inputs
    w = WORKLOADS["4k"]
    x = make_inputs(w)
    cfg = LayerConfig(B=w.B, T=w.T, Hq=w.Hq, Hkv=w.Hkv, D=w.D, window=w.window, mode=1, ratio=w.ratio)
    layer = LogoAttention(cfg)
    g = {k: x[k].cuda() for k in ("qL", "kL", "vL", "qG", "kG", "vG", "p", "dO")}
    layer.forward(g["qL"], g["kL"], g["vL"], g["qG"], g["kG"], g["vG"], g["p"])
    grads = layer.backward(g["dO"], g["qL"], g["kL"], g["vL"], g["qG"], g["kG"], g["vG"], g["p"])
    torch.cuda.synchronize()
    n = int(layer.n_sel.item())
    oz, opos, ocu, orow, on = oracle_select(x["p"], 1, 0.0, w.ratio)
    assert n == on == w.B * w.k_per_seq
    np.testing.assert_array_equal(layer.pos[:n].cpu().numpy(), opos)
    heads = [0, 5, 15]
    q, k, v = np32(x["qL"]), np32(x["kL"]), np32(x["vL"])
    rb, rt = oracle.local_rows(w.B, w.T)
    ro, _ = oracle.attn_fwd(q, k, v, rb, rt, w.window, heads=heads)
    check_close(np32(layer.o_l).reshape(-1, w.Hq, w.D)[:, heads], ro[:, heads], "o_l")
    gb, gt = oracle.global_rows(opos, ocu)
    qG, kG, vG = np32(x["qG"]), np32(x["kG"]), np32(x["vG"])
    rog, _ = oracle.attn_fwd(qG, kG, vG, gb, gt, 0, heads=heads)
    check_close(np32(layer.o_c)[:n][:, heads], rog[:, heads], "o_c")
    # combine on the device's own branch outputs
    rfo, _, _ = oracle.combine_fwd(np32(layer.o_l), np32(layer.o_c)[:n], np32(x["p"]), oz, orow)
    check_close(np32(layer.o), rfo, "o")
    rdl, rdg, rdp = oracle.combine_bwd(np32(x["dO"]), np32(layer.o_l), np32(layer.o_c)[:n], np32(x["p"]), oz, orow)
    check_close(np32(layer.dO_l), rdl, "dO_l")
    check_close(np32(layer.dO_c)[:n], rdg, "dO_c")
    # branch backward on the device's own upstream gradients, one head each
    h = [3]
    rdq, rdk, rdv = oracle.attn_bwd(q, k, v, rb, rt, w.window, np32(layer.dO_l).reshape(-1, w.Hq, w.D), heads=h)
    check_close(np32(grads["dqL"]).reshape(-1, w.Hq, w.D)[:, h], rdq[:, h], "dqL")
    check_close(np32(grads["dkL"])[:, :, h], rdk[:, :, h], "dkL")
    check_close(np32(grads["dvL"])[:, :, h], rdv[:, :, h], "dvL")
    rdq, rdk, rdv = oracle.attn_bwd(qG, kG, vG, gb, gt, 0, np32(layer.dO_c)[:n], heads=h)
    dense = np.zeros((w.B, w.T, w.Hq, w.D))
    dense[gb, gt] = rdq
    check_close(np32(grads["dqG"])[:, :, h], dense[:, :, h], "dqG")
    check_close(np32(grads["dkG"])[:, :, h], rdk[:, :, h], "dkG")
    check_close(np32(grads["dvG"])[:, :, h], rdv[:, :, h], "dvG")


def test_layer_two_streams_match_one_stream():
    """The local branch on the layer's side stream gives the results of the
    seven calls in order on one stream: every output bit-identical except dQ,
    whose fp32 reductions resolve in a run-dependent order (one bf16 ulp)."""
    from paper_2608_29539_gb300.layer import LayerConfig, LogoAttention
    from paper_2608_29539_gb300.workloads import WORKLOADS, make_inputs
    w = WORKLOADS["4k"]
    x = make_inputs(w, device="cuda")
    cfg = LayerConfig(B=w.B, T=w.T, Hq=w.Hq, Hkv=w.Hkv, D=w.D, window=w.window, mode=1, ratio=w.ratio)
    out = []
    for overlap in (False, True):
        layer = LogoAttention(cfg, overlap=overlap)
        args = (x["qL"], x["kL"], x["vL"], x["qG"], x["kG"], x["vG"], x["p"])
        for _ in range(2):
            layer.forward(*args)
            grads = layer.backward(x["dO"], *args)
        torch.cuda.synchronize()
        out.append(dict(o=layer.o.clone(), lse_l=layer.lse_l.clone(), **{k: v.clone() for k, v in grads.items()}))
    assert L().logo_get_device_status() == 0
    for k in out[0]:
        a, b = out[0][k].float(), out[1][k].float()
        if k in ("dqL", "dqG"):
            np.testing.assert_allclose(b.cpu().numpy(), a.cpu().numpy(), rtol=2 ** -7, atol=1e-3, err_msg=k)
        else:
            assert torch.equal(a, b), k


# ------------------------------------------- full size, the benchmark's launch
# Local backward shapes with several KV-block items per CTA on a 152-SM GPU
# (each CTA walks 5-7 items): item sequences crossing sequences and KV
# heads, GQA, a ragged last tile, a window of one.
LOCAL_MANY_ITEM_CASES = [
    # B, T, Hq, Hkv, D, W
    (1, 8192, 16, 16, 128, 64),
    (3, 5000, 16, 8, 128, 100),
    (1, 12000, 8, 8, 128, 1),
]


@pytest.mark.parametrize("B,T,Hq,Hkv,D,W", LOCAL_MANY_ITEM_CASES)
def test_local_bwd_many_items_per_cta(B, T, Hq, Hkv, D, W):
    test_local_bwd(B, T, Hq, Hkv, D, W)
    assert L().logo_get_device_status() == 0


def test_full_size_16k_workload_sampled():
    """The headline 16K workload (B=1, H=32, d=128, T=16384, W=1024, clustered
    selection at ratio 1/8) through the same layer object bench.py times.
    Selection checked in full; branch outputs on sampled rows of two heads;
    combine in full; gradients in full for one head of each branch."""
    import bench
    from paper_2608_29539_gb300.workloads import WORKLOADS, make_inputs
    w = WORKLOADS["16k"]
    x = make_inputs(w, device="cuda")
    layer = bench.layer_for(w, torch.device("cuda"))
    bench.run_step(layer, x)
    torch.cuda.synchronize()
    assert L().logo_get_device_status() == 0
    n = int(layer.n_sel.item())
    oz, opos, ocu, orow, on = oracle_select(x["p"].cpu(), 1, 0.0, w.ratio)
    assert n == on == w.k_per_seq
    np.testing.assert_array_equal(layer.pos[:n].cpu().numpy(), opos)
    np.testing.assert_array_equal(layer.z.cpu().numpy(), oz)
    np.testing.assert_array_equal(layer.row_of.cpu().numpy(), orow)
    f = lambda k: np32(x[k])  # noqa: E731
    qL, kL, vL, qG, kG, vG = (f(k) for k in ("qL", "kL", "vL", "qG", "kG", "vG"))
    rng = np.random.default_rng(0)
    heads = [0, 31]
    rows = np.sort(np.concatenate([rng.choice(w.T, 200, replace=False), [0, 1, 1023, 1024, w.T - 1]]))
    ro, _ = oracle.attn_fwd(qL, kL, vL, np.zeros_like(rows), rows, w.window, heads=heads)
    check_close(np32(layer.o_l)[0, rows][:, heads], ro[:, heads], "o_l sampled")
    grow = np.sort(np.concatenate([rng.choice(n, 200, replace=False), [0, n - 1]]))
    rog, _ = oracle.attn_fwd(qG, kG, vG, np.zeros_like(grow), opos[grow], 0, heads=heads)
    check_close(np32(layer.o_c)[grow][:, heads], rog[:, heads], "o_c sampled")
    rfo, _, _ = oracle.combine_fwd(np32(layer.o_l), np32(layer.o_c)[:n], f("p"), oz, orow)
    check_close(np32(layer.o), rfo, "o")
    h = [7]
    rb, rt = oracle.local_rows(w.B, w.T)
    rdq, rdk, rdv = oracle.attn_bwd(qL, kL, vL, rb, rt, w.window, np32(layer.dO_l).reshape(-1, w.Hq, w.D), heads=h)
    check_close(np32(layer.dqL).reshape(-1, w.Hq, w.D)[:, h], rdq[:, h], "dqL head 7")
    check_close(np32(layer.dkL)[:, :, h], rdk[:, :, h], "dkL head 7")
    check_close(np32(layer.dvL)[:, :, h], rdv[:, :, h], "dvL head 7")
    # dQ of every head on sampled rows
    dO_l = np32(layer.dO_l).reshape(-1, w.Hq, w.D)
    rdq, _, _ = oracle.attn_bwd(qL, kL, vL, np.zeros_like(rows), rows, w.window, dO_l[rows])
    check_close(np32(layer.dqL).reshape(-1, w.Hq, w.D)[rows], rdq, "dqL sampled rows, every head")
    gb, gt = oracle.global_rows(opos, ocu)
    rdq, rdk, rdv = oracle.attn_bwd(qG, kG, vG, gb, gt, 0, np32(layer.dO_c)[:n], heads=h)
    dense = np.zeros((w.B, w.T, w.Hq, w.D))
    dense[gb, gt] = rdq
    check_close(np32(layer.dqG)[:, :, h], dense[:, :, h], "dqG head 7")
    check_close(np32(layer.dkG)[:, :, h], rdk[:, :, h], "dkG head 7")
    check_close(np32(layer.dvG)[:, :, h], rdv[:, :, h], "dvG head 7")


def test_full_size_64k_gqa_sampled():
    """The 64K GQA workload (B=1, Hq=32, Hkv=8, d=128, T=65536, W=2048, ratio
    1/16) through the benchmark's layer object.  Selection in full; forward
    rows sampled; combine on a token subset; dQ on sampled rows (a row's dQ
    depends only on its own keys); dK/dV on a 64-key range, computed by the
    oracle from every query row that can see those keys (so they are
    complete), for one KV head (its whole query group)."""
    import bench
    from paper_2608_29539_gb300.workloads import WORKLOADS, make_inputs
    w = WORKLOADS["64k"]
    x = make_inputs(w, device="cuda")
    layer = bench.layer_for(w, torch.device("cuda"))
    bench.run_step(layer, x)
    torch.cuda.synchronize()
    assert L().logo_get_device_status() == 0
    n = int(layer.n_sel.item())
    oz, opos, ocu, orow, on = oracle_select(x["p"].cpu(), 1, 0.0, w.ratio)
    assert n == on == w.k_per_seq
    np.testing.assert_array_equal(layer.pos[:n].cpu().numpy(), opos)
    np.testing.assert_array_equal(layer.row_of.cpu().numpy(), orow)
    f = lambda k: np32(x[k])  # noqa: E731
    qL, kL, vL, qG, kG, vG = (f(k) for k in ("qL", "kL", "vL", "qG", "kG", "vG"))
    rng = np.random.default_rng(1)
    heads = [0, 5, 31]
    rows = np.sort(np.concatenate([rng.choice(w.T, 96, replace=False), [0, 2047, 2048, w.T - 1]])).astype(np.int32)
    ro, _ = oracle.attn_fwd(qL, kL, vL, np.zeros_like(rows), rows, w.window, heads=heads)
    check_close(np32(layer.o_l)[0, rows][:, heads], ro[:, heads], "o_l sampled")
    grow = np.sort(np.concatenate([rng.choice(n, 96, replace=False), [0, n - 1]]))
    rog, _ = oracle.attn_fwd(qG, kG, vG, np.zeros(len(grow), np.int32), opos[grow], 0, heads=heads)
    check_close(np32(layer.o_c)[grow][:, heads], rog[:, heads], "o_c sampled")
    # combine on the first 4096 tokens (their selected rows re-packed)
    tt = 4096
    z_sub = oz[:, :tt]
    sel_rows = orow[0, :tt][z_sub[0] == 1]
    row_sub = -np.ones((1, tt), np.int32)
    row_sub[0, z_sub[0] == 1] = np.arange(len(sel_rows), dtype=np.int32)
    o_l = np32(layer.o_l)[:, :tt]
    rfo, _, _ = oracle.combine_fwd(o_l, np32(layer.o_c)[sel_rows], f("p")[:, :tt], z_sub, row_sub)
    check_close(np32(layer.o)[:, :tt], rfo, "o (first 4096 tokens)")
    group = w.Hq // w.Hkv
    kvh = 2
    hs = list(range(kvh * group, (kvh + 1) * group))
    dOL = np32(layer.dO_l)[0]
    # local: dq on sampled rows; dK/dV on keys [s0, s0+64) from every row that sees them
    s0 = 20000
    lrows = np.arange(s0, s0 + 64 + w.window - 1, dtype=np.int32)
    rdq, rdk, rdv = oracle.attn_bwd(qL, kL, vL, np.zeros_like(lrows), lrows, w.window, dOL[lrows], heads=hs)
    check_close(np32(layer.dkL)[0, s0:s0 + 64, kvh], rdk[0, s0:s0 + 64, kvh], "dkL key range")
    check_close(np32(layer.dvL)[0, s0:s0 + 64, kvh], rdv[0, s0:s0 + 64, kvh], "dvL key range")
    check_close(np32(layer.dqL)[0, lrows][:, hs], rdq[:, hs], "dqL rows")
    # global: keys near the end so that few selected rows see them
    s1 = w.T - 1024
    grows = np.nonzero(opos >= s1)[0]
    dOc = np32(layer.dO_c)[:n]
    rdq, rdk, rdv = oracle.attn_bwd(qG, kG, vG, np.zeros(len(grows), np.int32), opos[grows], 0, dOc[grows], heads=hs)
    check_close(np32(layer.dkG)[0, s1:s1 + 64, kvh], rdk[0, s1:s1 + 64, kvh], "dkG key range")
    check_close(np32(layer.dvG)[0, s1:s1 + 64, kvh], rdv[0, s1:s1 + 64, kvh], "dvG key range")
    check_close(np32(layer.dqG)[0, opos[grows]][:, hs], rdq[:, hs], "dqG rows")
    # unselected rows of the dense global dQ are exactly zero
    unsel = np.setdiff1d(np.arange(w.T), opos)[:4096]
    assert not np32(layer.dqG)[0, unsel].any()
