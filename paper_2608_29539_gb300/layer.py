"""One training step of the LoGo attention layer's hot path, chained from the
C-ABI entry points (forward: select, local, global, combine; backward:
combine_bwd, global_bwd, local_bwd).  Buffers and workspaces are allocated
once per shape and reused, so a step launches kernels only.

The caller owns everything outside the path: the projections of Eq. 4/5, the
gate logits and their sigmoid (Eq. 7), the output projection, and the chain
rule through the sigmoid for ``dgate_p``.
"""
from __future__ import annotations

import dataclasses

import torch

from . import logo as L


@dataclasses.dataclass
class LayerConfig:
    B: int
    T: int
    Hq: int
    Hkv: int
    D: int
    window: int
    mode: int = L.LOGO_SELECT_RATIO
    b_th: float = 0.5
    ratio: float = 0.125
    eps: float = 1e-6
    scale: float = 0.0  # 0 -> 1/sqrt(D)


class LogoAttention:
    """Preallocated forward/backward of the layer for one shape on one device."""

    def __init__(self, cfg: LayerConfig, device="cuda"):
        self.cfg = c = cfg
        dev = torch.device(device)
        self.dims = L.Dims(c.B, c.T, c.Hq, c.Hkv, c.D)
        cap = c.B * c.T
        bf, f32, i32 = torch.bfloat16, torch.float32, torch.int32
        e = lambda shape, dt: torch.empty(shape, dtype=dt, device=dev)  # noqa: E731
        # selection
        self.z = e((c.B, c.T), torch.uint8)
        self.pos = e((cap,), i32)
        self.cu_q = e((c.B + 1,), i32)
        self.row_of = e((c.B, c.T), i32)
        self.n_sel = e((1,), i32)
        # forward activations
        self.o_l = e((c.B, c.T, c.Hq, c.D), bf)
        self.lse_l = e((c.B, c.Hq, c.T), f32)
        self.o_c = e((cap, c.Hq, c.D), bf)
        self.lse_c = e((c.Hq, cap), f32)
        self.o = e((c.B, c.T, c.Hq, c.D), bf)
        self.rstd_l = e((c.B, c.T, c.Hq), f32)
        self.rstd_g = e((cap, c.Hq), f32)
        # backward
        self.dO_l = e((c.B, c.T, c.Hq, c.D), bf)
        self.dO_c = e((cap, c.Hq, c.D), bf)
        self.dgate = e((c.B, c.T), f32)
        self.dqL = e((c.B, c.T, c.Hq, c.D), bf)
        self.dkL = e((c.B, c.T, c.Hkv, c.D), bf)
        self.dvL = e((c.B, c.T, c.Hkv, c.D), bf)
        self.dqG = e((c.B, c.T, c.Hq, c.D), bf)
        self.dkG = e((c.B, c.T, c.Hkv, c.D), bf)
        self.dvG = e((c.B, c.T, c.Hkv, c.D), bf)
        # workspaces: the largest of the calls, shared (calls are stream-ordered)
        nbytes = max(L.workspace_bytes(k, self.dims) for k in ("select", "local_bwd", "global_fwd", "global_bwd"))
        self.ws = e((nbytes,), torch.uint8)

    def forward(self, qL, kL, vL, qG, kG, vG, gate_p, gain_l=None, gain_g=None):
        c = self.cfg
        L.logo_select(gate_p, c.mode, c.b_th, c.ratio, self.z, self.pos, self.cu_q, self.row_of, self.n_sel,
                      workspace=self.ws)
        L.logo_local_attn_fwd(qL, kL, vL, c.window, c.scale, self.o_l, self.lse_l)
        L.logo_global_sparse_attn_fwd(qG, kG, vG, self.pos, self.cu_q, self.n_sel, c.scale, self.o_c, self.lse_c,
                                      workspace=self.ws)
        L.logo_combine(self.o_l, self.o_c, gate_p, self.z, self.row_of, gain_l, gain_g, c.eps, self.o, self.rstd_l,
                       self.rstd_g)
        return self.o

    def backward(self, dO, qL, kL, vL, qG, kG, vG, gate_p, gain_l=None, gain_g=None):
        c = self.cfg
        L.logo_combine_bwd(dO, self.o_l, self.o_c, gate_p, self.z, self.row_of, gain_l, gain_g, c.eps, self.dO_l,
                           self.dO_c, self.dgate)
        L.logo_global_sparse_attn_bwd(qG, kG, vG, self.pos, self.cu_q, self.n_sel, self.o_c, self.lse_c, self.dO_c,
                                      c.scale, self.dqG, self.dkG, self.dvG, workspace=self.ws)
        L.logo_local_attn_bwd(qL, kL, vL, self.o_l, self.lse_l, self.dO_l, c.window, c.scale, self.dqL, self.dkL,
                              self.dvL, workspace=self.ws)
        return dict(dqL=self.dqL, dkL=self.dkL, dvL=self.dvL, dqG=self.dqG, dkG=self.dkG, dvG=self.dvG,
                    dgate_p=self.dgate)
