"""Head-sharded replicas through the CUDA path, checked against the oracle.

Row sparsity is shared by all heads (Sec. 3.3, App. B): the selection of
Eq. 7 depends only on the gate values, so every shard selects the same rows
and the attention of a shard's heads needs nothing from the other shards.
The one exchange is the gate gradient dp_t of Eq. 10, a sum over every head.

Two tests:
- one process, shards run one after the other on the one GPU: every shard's
  outputs and gradients against the oracle on that shard's heads (stage by
  stage, each stage on the inputs it received), and against the unsharded
  CUDA run (per-head results bit for bit, dQ and dp to rounding);
- two gloo ranks, each a process running the CUDA layer on its shard on the
  one GPU (the ranks' kernels never wait on each other; the only exchange is
  the host-side all-reduce of dp), with dp all-reduced; every rank's results,
  the all-reduced dp included, against the oracle.
"""
import os
import socket
import tempfile

import numpy as np
import pytest
import torch

import oracle
from helpers import check_close, np32, seeded
from paper_2608_29539_gb300 import logo as L
from paper_2608_29539_gb300.layer import LayerConfig, LogoAttention
from paper_2608_29539_gb300.shard import HeadShardedLogoAttention, head_shard, take_heads

pytestmark = pytest.mark.gpu

SHAPE = dict(B=2, T=1000, Hq=8, Hkv=4, D=128)
WINDOW, RATIO = 256, 0.25


def _cfg():
    s = SHAPE
    return LayerConfig(s["B"], s["T"], s["Hq"], s["Hkv"], s["D"], window=WINDOW, mode=L.LOGO_SELECT_RATIO,
                       ratio=RATIO)


def _inputs(dev):
    B, T, Hq, Hkv, D = (SHAPE[k] for k in ("B", "T", "Hq", "Hkv", "D"))
    x = dict(qL=seeded((B, T, Hq, D), 1), kL=seeded((B, T, Hkv, D), 2), vL=seeded((B, T, Hkv, D), 3),
             qG=seeded((B, T, Hq, D), 4), kG=seeded((B, T, Hkv, D), 5), vG=seeded((B, T, Hkv, D), 6),
             dO=seeded((B, T, Hq, D), 7))
    x = {k: v.to(torch.bfloat16).to(dev) for k, v in x.items()}
    g = torch.Generator().manual_seed(8)
    x["p"] = torch.rand(B, T, generator=g).to(dev)
    x["gain_l"] = (1.0 + 0.1 * torch.randn(Hq, D, generator=g)).to(dev)
    x["gain_g"] = (1.0 + 0.1 * torch.randn(Hq, D, generator=g)).to(dev)
    return x


def _step(layer, x, q0, q1, kv0, kv1):
    q = lambda k: take_heads(x[k], q0, q1)  # noqa: E731
    kv = lambda k: take_heads(x[k], kv0, kv1)  # noqa: E731
    args = (q("qL"), kv("kL"), kv("vL"), q("qG"), kv("kG"), kv("vG"), x["p"])
    gains = (take_heads(x["gain_l"], q0, q1, axis=0), take_heads(x["gain_g"], q0, q1, axis=0))
    o = layer.forward(*args, *gains).clone()
    g = {k: v.clone() for k, v in layer.backward(q("dO"), *args, *gains).items()}
    return o, g


def _record(inner, o, g):
    """What one shard produced, on the host: outputs, gradients and the
    intermediates the next stage consumed."""
    n = int(inner.n_sel[0])
    rec = {k: np32(v) for k, v in g.items()}
    rec.update(o=np32(o), o_l=np32(inner.o_l), o_c=np32(inner.o_c)[:n], dO_l=np32(inner.dO_l),
               dO_c=np32(inner.dO_c)[:n], z=inner.z.cpu().numpy(), n=n)
    return rec


def _check_shard_against_oracle(rec, x, sh, dp_total=None):
    """Stage by stage on the shard's heads [q0, q1) / [kv0, kv1).  dp is the
    shard's partial sum over its heads, or (dp_total) the all-reduced sum over
    every head."""
    c = _cfg()
    h = lambda k, a, b: np32(take_heads(x[k], a, b))  # noqa: E731
    qL, kL, vL = h("qL", sh.q0, sh.q1), h("kL", sh.kv0, sh.kv1), h("vL", sh.kv0, sh.kv1)
    qG, kG, vG = h("qG", sh.q0, sh.q1), h("kG", sh.kv0, sh.kv1), h("vG", sh.kv0, sh.kv1)
    dO = h("dO", sh.q0, sh.q1)
    gl, gg = (np32(take_heads(x[k], sh.q0, sh.q1, axis=0)) for k in ("gain_l", "gain_g"))
    p = np32(x["p"])
    hq = sh.hq
    z = oracle.select_ratio(p, oracle.k_from_ratio(RATIO, c.T))
    assert np.array_equal(z, rec["z"])
    pos, cu_q, row_of, n = oracle.compact(z)
    assert rec["n"] == n
    lb, lt = oracle.local_rows(c.B, c.T)
    gb, gt = oracle.global_rows(pos, cu_q)
    tag = f"shard {sh.rank}/{sh.world}"
    ro_l, _ = oracle.attn_fwd(qL, kL, vL, lb, lt, WINDOW)
    check_close(rec["o_l"].reshape(-1, hq, c.D), ro_l, f"{tag} O^L")
    ro_c, _ = oracle.attn_fwd(qG, kG, vG, gb, gt, 0)
    check_close(rec["o_c"], ro_c, f"{tag} O^G")
    ro, _, _ = oracle.combine_fwd(rec["o_l"], rec["o_c"], p, z, row_of, gl, gg)
    check_close(rec["o"], ro, f"{tag} o")
    rdOL, rdOG, rdp = oracle.combine_bwd(dO, rec["o_l"], rec["o_c"], p, z, row_of, gl, gg)
    check_close(rec["dO_l"], rdOL, f"{tag} dO^L")
    check_close(rec["dO_c"], rdOG, f"{tag} dO^G")
    check_close(rec["dgate_p"], rdp if dp_total is None else dp_total, f"{tag} dp")
    rdq, rdk, rdv = oracle.attn_bwd(qL, kL, vL, lb, lt, WINDOW, rec["dO_l"].reshape(-1, hq, c.D))
    check_close(rec["dqL"].reshape(-1, hq, c.D), rdq, f"{tag} dQ^L")
    check_close(rec["dkL"], rdk, f"{tag} dK^L")
    check_close(rec["dvL"], rdv, f"{tag} dV^L")
    rdq, rdk, rdv = oracle.attn_bwd(qG, kG, vG, gb, gt, 0, rec["dO_c"])
    dense = np.zeros((c.B, c.T, hq, c.D))
    dense[gb, gt] = rdq
    check_close(rec["dqG"], dense, f"{tag} dQ^G")
    assert (rec["dqG"][z == 0] == 0).all()
    check_close(rec["dkG"], rdk, f"{tag} dK^G")
    check_close(rec["dvG"], rdv, f"{tag} dV^G")
    return rdp


@pytest.mark.parametrize("world", [2, 4])
def test_head_sharded_layer_matches_oracle_and_unsharded(world):
    c = _cfg()
    dev = torch.device("cuda")
    x = _inputs(dev)
    full = LogoAttention(c, device=dev)
    o_ref, g_ref = _step(full, x, 0, c.Hq, 0, c.Hkv)
    n = int(full.n_sel[0])
    ref_ol, ref_oc = full.o_l.clone(), full.o_c[:n].clone()
    outs, grads, ols, ocs = [], [], [], []
    dp_parts = []
    for r in range(world):
        sh = head_shard(c.Hq, c.Hkv, r, world)
        layer = HeadShardedLogoAttention(c, sh, device=dev)  # no process group: dp summed below
        o, g = _step(layer, x, sh.q0, sh.q1, sh.kv0, sh.kv1)
        torch.cuda.synchronize()
        assert int(layer.inner.n_sel[0]) == n  # the same selection on every shard
        dp_parts.append(_check_shard_against_oracle(_record(layer.inner, o, g), x, sh))
        outs.append(o)
        grads.append(g)
        ols.append(layer.inner.o_l.clone())
        ocs.append(layer.inner.o_c[:n].clone())
    torch.cuda.synchronize()
    # against the unsharded CUDA run: per-head results are the same arithmetic on the same data
    assert torch.equal(torch.cat(ols, dim=2), ref_ol)
    assert torch.equal(torch.cat(ocs, dim=1), ref_oc)
    for k in ("dkL", "dvL", "dkG", "dvG"):
        assert torch.equal(torch.cat([g[k] for g in grads], dim=2), g_ref[k]), k
    o = torch.cat(outs, dim=2).float()
    assert ((o - o_ref.float()).abs() <= 2.0 ** -8 * o_ref.float().abs().clamp(min=1.0)).all()
    for k in ("dqL", "dqG"):
        got, ref = torch.cat([g[k] for g in grads], dim=2).float(), g_ref[k].float()
        assert ((got - ref).abs() <= 2.0 ** -7 * ref.abs().clamp(min=1.0)).all(), k
    # the head-summed gate gradient: the sum of the shards' partial sums
    dp = sum(g["dgate_p"] for g in grads)
    assert float(g_ref["dgate_p"].abs().sum()) > 0
    check_close(np32(dp), sum(dp_parts), "dp summed over shards")
    assert ((dp - g_ref["dgate_p"]).abs() <= 1e-4 * g_ref["dgate_p"].abs().clamp(min=1.0)).all()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _gloo_cuda_worker(rank, world, port, outdir):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dev = torch.device("cuda:0")
        x = _inputs(dev)
        c = _cfg()
        sh = head_shard(c.Hq, c.Hkv, rank, world)
        layer = HeadShardedLogoAttention(c, sh, device=dev)  # the CUDA layer; dp all-reduced over gloo
        o, g = _step(layer, x, sh.q0, sh.q1, sh.kv0, sh.kv1)
        torch.cuda.synchronize()
        if L.logo_get_device_status() != 0:
            raise RuntimeError("device reported an error")
        np.savez(os.path.join(outdir, f"rank{rank}.npz"), **_record(layer.inner, o, g))
    finally:
        dist.destroy_process_group()


def test_head_sharded_layer_two_gloo_ranks_cuda_against_oracle():
    import torch.multiprocessing as mp
    world = 2
    c = _cfg()
    x = _inputs(torch.device("cpu"))
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(_gloo_cuda_worker, args=(world, _free_port(), d), nprocs=world, join=True,
                           start_method="spawn")
        recs = [dict(np.load(os.path.join(d, f"rank{r}.npz"))) for r in range(world)]
    for r in recs:
        r["n"] = int(r["n"])
    # the all-reduced dp every rank holds: the oracle's dp of each shard's heads, summed
    z = oracle.select_ratio(np32(x["p"]), oracle.k_from_ratio(RATIO, c.T))
    pos, cu_q, row_of, n = oracle.compact(z)
    o_l = np.concatenate([r["o_l"] for r in recs], axis=2)
    o_c = np.concatenate([r["o_c"] for r in recs], axis=1)
    _, _, dp_total = oracle.combine_bwd(np32(x["dO"]), o_l, o_c, np32(x["p"]), z, row_of, np32(x["gain_l"]),
                                        np32(x["gain_g"]))
    assert float(np.abs(dp_total).sum()) > 0
    for r, rec in enumerate(recs):
        _check_shard_against_oracle(rec, x, head_shard(c.Hq, c.Hkv, r, world), dp_total=dp_total)
    assert np.array_equal(recs[0]["dgate_p"], recs[1]["dgate_p"])  # every rank holds the same total
