"""Head-sharded replicas of the layer: rank r of N runs the hot path on its own
contiguous block of heads.

Every head of Eq. 6 and Eq. 8 is independent once the token selection of
Eq. 7 is fixed, and the selection depends only on the gate values p_t, which
every rank holds whole: each rank computes the same selection locally, so
the forward needs no exchange.  The backward has one: p_t is shared by all
heads, so dp_t = z_t * sum over (h, d) of dO * (O~^G - O~^L) (the derivative
of Eq. 10) is a sum over every head, and each rank's partial sum over its
heads is all-reduced (a [B, T] float32 vector per step).

KV heads are split evenly (Hkv % N == 0) and each rank keeps the query heads
of its KV heads' groups, so a GQA group never straddles two ranks.
"""
from __future__ import annotations

import dataclasses

import torch

from .layer import LayerConfig, LogoAttention


@dataclasses.dataclass(frozen=True)
class HeadShard:
    """Heads [q0, q1) of Hq and [kv0, kv1) of Hkv held by `rank` of `world`."""
    rank: int
    world: int
    q0: int
    q1: int
    kv0: int
    kv1: int

    @property
    def hq(self) -> int:
        return self.q1 - self.q0

    @property
    def hkv(self) -> int:
        return self.kv1 - self.kv0


def head_shard(Hq: int, Hkv: int, rank: int, world: int) -> HeadShard:
    """The contiguous head block of `rank`.  Raises ValueError when the heads do
    not split into whole GQA groups per rank."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} out of range for world size {world}")
    if Hkv < 1 or Hq % Hkv != 0:
        raise ValueError(f"Hq={Hq} is not a multiple of Hkv={Hkv}")
    if Hkv % world != 0:
        raise ValueError(f"Hkv={Hkv} KV heads do not split evenly over {world} ranks")
    per_kv = Hkv // world
    group = Hq // Hkv
    kv0 = rank * per_kv
    return HeadShard(rank, world, kv0 * group, (kv0 + per_kv) * group, kv0, kv0 + per_kv)


def take_heads(t: torch.Tensor | None, h0: int, h1: int, axis: int = 2) -> torch.Tensor | None:
    """Heads [h0, h1) of a head-major tensor ([B, T, H, D] by default; axis 0 for
    per-head gains [H, D]), contiguous."""
    if t is None:
        return None
    return t.narrow(axis, h0, h1 - h0).contiguous()


def shard_config(cfg: LayerConfig, shard: HeadShard) -> LayerConfig:
    """The layer configuration of one shard: same tokens and selection, fewer heads."""
    return dataclasses.replace(cfg, Hq=shard.hq, Hkv=shard.hkv)


def all_reduce_gate_grad(dgate: torch.Tensor, process_group=None) -> torch.Tensor:
    """Sum the per-rank partial dp over the head shards, in place."""
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(process_group) > 1:
        if dgate.is_cuda and dist.get_backend(process_group) == "gloo":
            host = dgate.cpu()  # gloo reduces host memory; the vector is B*T floats
            dist.all_reduce(host, op=dist.ReduceOp.SUM, group=process_group)
            dgate.copy_(host)
        else:
            dist.all_reduce(dgate, op=dist.ReduceOp.SUM, group=process_group)
    return dgate


class HeadShardedLogoAttention:
    """The layer on one head shard.  Inputs are the rank's own heads (a head-
    sharded projection produces them); gate_p is the full [B, T] gate.

    `inner` is the per-shard layer; by default the CUDA path (`LogoAttention`
    on the shard's configuration).  Another object with the same forward /
    backward methods may be passed (the multi-process tests use one on the
    host)."""

    def __init__(self, cfg: LayerConfig, shard: HeadShard, device="cuda", process_group=None, inner=None):
        self.cfg = cfg
        self.shard = shard
        self.local_cfg = shard_config(cfg, shard)
        self.process_group = process_group
        self.inner = inner if inner is not None else LogoAttention(self.local_cfg, device=device)

    def forward(self, qL, kL, vL, qG, kG, vG, gate_p, gain_l=None, gain_g=None):
        return self.inner.forward(qL, kL, vL, qG, kG, vG, gate_p, gain_l, gain_g)

    def backward(self, dO, qL, kL, vL, qG, kG, vG, gate_p, gain_l=None, gain_g=None):
        grads = self.inner.backward(dO, qL, kL, vL, qG, kG, vG, gate_p, gain_l, gain_g)
        all_reduce_gate_grad(grads["dgate_p"], self.process_group)
        return grads
