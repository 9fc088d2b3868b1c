"""Head-sharded replicas on the host: two gloo ranks, each running the layer on
its own heads (the oracle stands in for the per-shard CUDA path), give the
unsharded layer's outputs and gradients; the gate gradient, a sum over every
head, is the one exchange (all-reduced across the shards).  Also the head
partition rules and bench.py's max/sum-over-ranks timing helpers."""
import os
import socket
import tempfile

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2608_29539_gb300 import logo as L
from paper_2608_29539_gb300.layer import LayerConfig
from paper_2608_29539_gb300.shard import (HeadShardedLogoAttention, head_shard, shard_config,
                                          take_heads)

B, T, HQ, HKV, D, W, RATIO = 2, 40, 4, 2, 16, 12, 0.25


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _inputs():
    """Seeded full-head inputs, bf16-rounded values held in float32 tensors."""
    g = torch.Generator().manual_seed(2024)
    r = lambda *shape: torch.randn(*shape, generator=g).bfloat16().float()  # noqa: E731
    x = dict(qL=r(B, T, HQ, D), kL=r(B, T, HKV, D), vL=r(B, T, HKV, D),
             qG=r(B, T, HQ, D), kG=r(B, T, HKV, D), vG=r(B, T, HKV, D), dO=r(B, T, HQ, D))
    x["p"] = torch.rand(B, T, generator=g)
    x["gain_l"] = (1.0 + 0.1 * torch.randn(HQ, D, generator=g)).bfloat16().float()
    x["gain_g"] = (1.0 + 0.1 * torch.randn(HQ, D, generator=g)).bfloat16().float()
    return x


class _OracleLayer:
    """The layer's forward / backward on the host, through the oracle, with the
    same method signatures as the CUDA layer (test stand-in for one shard)."""

    def __init__(self, cfg: LayerConfig):
        self.cfg = cfg

    def forward(self, qL, kL, vL, qG, kG, vG, gate_p, gain_l=None, gain_g=None):
        c = self.cfg
        z = oracle.select_ratio(gate_p.numpy(), oracle.k_from_ratio(c.ratio, c.T))
        self.z = z
        self.pos, self.cu_q, self.row_of, n = oracle.compact(z)
        lb, lt = oracle.local_rows(c.B, c.T)
        gb, gt = oracle.global_rows(self.pos, self.cu_q)
        self.oL, _ = oracle.attn_fwd(qL.numpy(), kL.numpy(), vL.numpy(), lb, lt, c.window)
        self.oG, _ = oracle.attn_fwd(qG.numpy(), kG.numpy(), vG.numpy(), gb, gt, 0)
        self.oL = self.oL.reshape(c.B, c.T, c.Hq, c.D)
        o, _, _ = oracle.combine_fwd(self.oL, self.oG, gate_p.numpy(), z, self.row_of,
                                     None if gain_l is None else gain_l.numpy(),
                                     None if gain_g is None else gain_g.numpy(), c.eps)
        return torch.from_numpy(o)

    def backward(self, dO, qL, kL, vL, qG, kG, vG, gate_p, gain_l=None, gain_g=None):
        c = self.cfg
        dOL, dOG, dp = oracle.combine_bwd(dO.numpy(), self.oL, self.oG, gate_p.numpy(), self.z, self.row_of,
                                          None if gain_l is None else gain_l.numpy(),
                                          None if gain_g is None else gain_g.numpy(), c.eps)
        lb, lt = oracle.local_rows(c.B, c.T)
        gb, gt = oracle.global_rows(self.pos, self.cu_q)
        dqL, dkL, dvL = oracle.attn_bwd(qL.numpy(), kL.numpy(), vL.numpy(), lb, lt, c.window, dOL)
        dqGc, dkG, dvG = oracle.attn_bwd(qG.numpy(), kG.numpy(), vG.numpy(), gb, gt, 0, dOG)
        dqG = np.zeros((c.B, c.T, c.Hq, c.D))
        dqG[gb, gt] = dqGc
        t = torch.from_numpy
        return dict(dqL=t(dqL.reshape(c.B, c.T, c.Hq, c.D)), dkL=t(dkL), dvL=t(dvL), dqG=t(dqG), dkG=t(dkG),
                    dvG=t(dvG), dgate_p=t(dp))


def _cfg():
    return LayerConfig(B, T, HQ, HKV, D, W, mode=L.LOGO_SELECT_RATIO, ratio=RATIO)


def _run_shard(layer, x, sh):
    q = lambda k: take_heads(x[k], sh.q0, sh.q1)  # noqa: E731
    kv = lambda k: take_heads(x[k], sh.kv0, sh.kv1)  # noqa: E731
    args = (q("qL"), kv("kL"), kv("vL"), q("qG"), kv("kG"), kv("vG"), x["p"])
    gains = (take_heads(x["gain_l"], sh.q0, sh.q1, axis=0), take_heads(x["gain_g"], sh.q0, sh.q1, axis=0))
    o = layer.forward(*args, *gains)
    g = layer.backward(q("dO"), *args, *gains)
    return o, g


def _worker(rank, world, port, outdir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        x = _inputs()
        cfg = _cfg()
        sh = head_shard(HQ, HKV, rank, world)
        layer = HeadShardedLogoAttention(cfg, sh, device="cpu", inner=_OracleLayer(shard_config(cfg, sh)))
        o, g = _run_shard(layer, x, sh)
        torch.save({"o": o, **g}, os.path.join(outdir, f"rank{rank}.pt"))
    finally:
        dist.destroy_process_group()


def test_head_shard_partition():
    for Hq, Hkv, world in [(32, 8, 2), (32, 8, 4), (32, 8, 8), (16, 16, 4), (8, 2, 1)]:
        shards = [head_shard(Hq, Hkv, r, world) for r in range(world)]
        assert shards[0].q0 == 0 and shards[-1].q1 == Hq and shards[0].kv0 == 0 and shards[-1].kv1 == Hkv
        for a, b in zip(shards, shards[1:]):
            assert a.q1 == b.q0 and a.kv1 == b.kv0
        g = Hq // Hkv
        for s in shards:
            assert s.q0 == s.kv0 * g and s.q1 == s.kv1 * g  # whole GQA groups
    for bad in [(32, 8, 3), (32, 6, 4), (30, 8, 2)]:
        with pytest.raises(ValueError):
            head_shard(bad[0], bad[1], 0, bad[2])
    with pytest.raises(ValueError):
        head_shard(32, 8, 2, 2)


def test_head_sharded_layer_two_gloo_ranks_matches_unsharded():
    world = 2
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(_worker, args=(world, _free_port(), d), nprocs=world, join=True, start_method="spawn")
        parts = [torch.load(os.path.join(d, f"rank{r}.pt")) for r in range(world)]
    x = _inputs()
    full = HeadShardedLogoAttention(_cfg(), head_shard(HQ, HKV, 0, 1), device="cpu", inner=_OracleLayer(_cfg()))
    o_ref, g_ref = _run_shard(full, x, head_shard(HQ, HKV, 0, 1))
    # per-head tensors: each head's arithmetic is the same on its shard, so they match exactly
    o = torch.cat([p["o"] for p in parts], dim=2)
    assert torch.equal(o, o_ref)
    for k in ("dqL", "dqG", "dkL", "dvL", "dkG", "dvG"):
        got = torch.cat([p[k] for p in parts], dim=2)
        assert torch.equal(got, g_ref[k]), k
    # the gate gradient sums over every head: every rank holds the all-reduced total
    for p in parts:
        np.testing.assert_allclose(p["dgate_p"].numpy(), g_ref["dgate_p"].numpy(), rtol=1e-12, atol=1e-12)
    assert float(g_ref["dgate_p"].abs().sum()) > 0


def _timing_worker(rank, world, port, outdir):
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(True)
        mx = bench.max_over_ranks(1.5 + rank, True)
        sm = bench.sum_over_ranks(10.0 * (rank + 1), True)
        torch.save({"max": mx, "sum": sm}, os.path.join(outdir, f"t{rank}.pt"))
    finally:
        dist.destroy_process_group()


def test_bench_timing_reductions_two_gloo_ranks():
    """bench.py times K steps per rank and reports the slowest rank's time and
    the units of all ranks: max / sum over ranks."""
    world = 2
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(_timing_worker, args=(world, _free_port(), d), nprocs=world, join=True,
                           start_method="spawn")
        res = [torch.load(os.path.join(d, f"t{r}.pt")) for r in range(world)]
    for r in res:
        assert r["max"] == 2.5 and r["sum"] == 30.0
