"""Head-sharded replicas through the CUDA path on one GPU: the layer run on two
head shards, one after the other, against the unsharded layer on the same
inputs.  Per-head results are the same arithmetic on the same data, so the
branch outputs and dK/dV match bit for bit; dQ (fp32 atomics in whatever
order the blocks finish) and the head-summed gate gradient (Eq. 10's dp, the
one quantity the shards exchange) match to rounding."""
import pytest
import torch

from helpers import seeded
from paper_2608_29539_gb300 import logo as L
from paper_2608_29539_gb300.layer import LayerConfig, LogoAttention
from paper_2608_29539_gb300.shard import HeadShardedLogoAttention, head_shard, take_heads

pytestmark = pytest.mark.gpu


def _inputs(B, T, Hq, Hkv, D, dev):
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


@pytest.mark.parametrize("world", [2, 4])
def test_head_sharded_layer_matches_unsharded(world):
    B, T, Hq, Hkv, D = 2, 1000, 8, 4, 128
    cfg = LayerConfig(B, T, Hq, Hkv, D, window=256, mode=L.LOGO_SELECT_RATIO, ratio=0.25)
    dev = torch.device("cuda")
    x = _inputs(B, T, Hq, Hkv, D, dev)
    full = LogoAttention(cfg, device=dev)
    o_ref, g_ref = _step(full, x, 0, Hq, 0, Hkv)
    n = int(full.n_sel[0])
    ref_ol, ref_oc = full.o_l.clone(), full.o_c[:n].clone()
    outs, grads, ols, ocs = [], [], [], []
    for r in range(world):
        sh = head_shard(Hq, Hkv, r, world)
        layer = HeadShardedLogoAttention(cfg, sh, device=dev)  # no process group: dp summed below
        o, g = _step(layer, x, sh.q0, sh.q1, sh.kv0, sh.kv1)
        assert int(layer.inner.n_sel[0]) == n  # the same selection on every shard
        outs.append(o)
        grads.append(g)
        ols.append(layer.inner.o_l.clone())
        ocs.append(layer.inner.o_c[:n].clone())
    torch.cuda.synchronize()
    assert torch.equal(torch.cat(ols, dim=2), ref_ol)
    assert torch.equal(torch.cat(ocs, dim=1), ref_oc)
    for k in ("dkL", "dvL", "dkG", "dvG"):
        assert torch.equal(torch.cat([g[k] for g in grads], dim=2), g_ref[k]), k
    # combine output: per (token, head) arithmetic, compared to one bf16 rounding
    o = torch.cat(outs, dim=2).float()
    assert ((o - o_ref.float()).abs() <= 2.0 ** -8 * o_ref.float().abs().clamp(min=1.0)).all()
    for k in ("dqL", "dqG"):
        got, ref = torch.cat([g[k] for g in grads], dim=2).float(), g_ref[k].float()
        assert ((got - ref).abs() <= 2.0 ** -7 * ref.abs().clamp(min=1.0)).all(), k
    dp = sum(g["dgate_p"] for g in grads)
    ref = g_ref["dgate_p"]
    assert float(ref.abs().sum()) > 0
    assert ((dp - ref).abs() <= 1e-4 * ref.abs().clamp(min=1.0)).all()
