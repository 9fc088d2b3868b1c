"""One training step of the LoGo attention layer's hot path, chained from the
C-ABI entry points (forward: select, local, global, combine; backward:
combine_bwd, global_bwd, local_bwd).  Buffers and workspaces are allocated
once per shape and reused, so a step launches kernels only.

The two branches are independent between the selection and the combine, and
again after the combine's backward, so the local calls run on a side stream
(forked from and joined back into the caller's stream) beside the global
calls: the kernel launched second fills the SMs the first one's tail leaves
idle, and the HBM-bound passes of one branch overlap the tensor-core work of
the other.  The local call is issued first on each fork: its persistent
kernel is the longer one, and with the global kernel launched first the local
kernel's late CTAs stretched the step.  The local backward has a
workspace of its own for that reason.  `overlap=False` keeps every call on
the caller's stream.

`forward` / `backward` take the branch inputs and the gate values as the
caller made them (the projections of Eq. 4/5, the gate of Eq. 7 and the
output projection stay outside).  `forward_fused` / `backward_fused` also
run the gate of Eq. 7 from the layer input, the Eq. 5 branch transforms
(Q^G on the selected rows only) and the ContextNorm gain gradients, so the
caller passes x, w_g, Q^L/K^L/V^L and the transform parameters, and gets back
every gradient of those.
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

    def __init__(self, cfg: LayerConfig, device="cuda", overlap: bool = True):
        self.cfg = c = cfg
        dev = torch.device(device)
        self.overlap = overlap
        self.side = torch.cuda.Stream(device=dev) if overlap and dev.type == "cuda" else None
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
        # workspaces: one shared by the calls on the caller's stream (they are
        # stream-ordered), one for the local backward on the side stream
        nbytes = max(L.workspace_bytes(k, self.dims) for k in ("select", "global_fwd", "global_bwd"))
        self.ws = e((nbytes,), torch.uint8)
        self.ws_l = e((L.workspace_bytes("local_bwd", self.dims),), torch.uint8)

    def _fork(self):
        """Side stream for the local branch (None: run it in order)."""
        if self.side is None:
            return None
        self.side.wait_stream(torch.cuda.current_stream())
        return torch.cuda.stream(self.side)

    def _join(self):
        if self.side is not None:
            torch.cuda.current_stream().wait_stream(self.side)

    def _local_fwd(self, qL, kL, vL):
        c = self.cfg
        L.logo_local_attn_fwd(qL, kL, vL, c.window, c.scale, self.o_l, self.lse_l)

    def _local_bwd(self, qL, kL, vL):
        c = self.cfg
        L.logo_local_attn_bwd(qL, kL, vL, self.o_l, self.lse_l, self.dO_l, c.window, c.scale, self.dqL, self.dkL,
                              self.dvL, workspace=self.ws_l)

    def _branches(self, local, other):
        """local() on the side stream beside other() on the caller's stream,
        joined before returning; both in order without a side stream."""
        ctx = self._fork()
        if ctx is None:
            other()
            local()
            return
        with ctx:
            local()
        other()
        self._join()

    def forward(self, qL, kL, vL, qG, kG, vG, gate_p, gain_l=None, gain_g=None):
        c = self.cfg
        # the fork follows the selection: captured in a CUDA graph, a local
        # branch forked at the very start would be a second root node, and
        # the graph then launched the global backward ahead of the local one
        # (measured at 16K: 2.39 ms a step against 2.23 with this order)
        L.logo_select(gate_p, c.mode, c.b_th, c.ratio, self.z, self.pos, self.cu_q, self.row_of, self.n_sel,
                      workspace=self.ws)
        self._branches(lambda: self._local_fwd(qL, kL, vL),
                       lambda: L.logo_global_sparse_attn_fwd(qG, kG, vG, self.pos, self.cu_q, self.n_sel, c.scale,
                                                             self.o_c, self.lse_c, workspace=self.ws))
        L.logo_combine(self.o_l, self.o_c, gate_p, self.z, self.row_of, gain_l, gain_g, c.eps, self.o, self.rstd_l,
                       self.rstd_g)
        return self.o

    def backward(self, dO, qL, kL, vL, qG, kG, vG, gate_p, gain_l=None, gain_g=None):
        c = self.cfg
        L.logo_combine_bwd(dO, self.o_l, self.o_c, gate_p, self.z, self.row_of, gain_l, gain_g, c.eps, self.dO_l,
                           self.dO_c, self.dgate)
        self._branches(lambda: self._local_bwd(qL, kL, vL),
                       lambda: L.logo_global_sparse_attn_bwd(qG, kG, vG, self.pos, self.cu_q, self.n_sel, self.o_c,
                                                             self.lse_c, self.dO_c, c.scale, self.dqG, self.dkG,
                                                             self.dvG, workspace=self.ws))
        return dict(dqL=self.dqL, dkL=self.dkL, dvL=self.dvL, dqG=self.dqG, dkG=self.dkG, dvG=self.dvG,
                    dgate_p=self.dgate)

    # ------------------------------------------------------------ fused path
    def forward_fused(self, x, w_g, qL, kL, vL, tq, tk, tv, gain_l=None, gain_g=None):
        """Eq. 7 gate + select, Eq. 5 transforms, both branches, Eq. 9/10.

        x [B, T, d_model] bf16 and w_g [d_model] float32 feed the gate; tq, tk,
        tv are the Eq. 5 parameters of Q, K, V: a dict {"a": [H, D, D] bf16}
        (LP) or {"s": [H, D], "b": [H, D] float32} (SO).  Returns o."""
        c = self.cfg
        if not hasattr(self, "gate_p"):
            self.gate_p = torch.empty((c.B, c.T), dtype=torch.float32, device=qL.device)
            self.qG = torch.empty_like(qL)
            self.kG = torch.empty_like(kL)
            self.vG = torch.empty_like(vL)
        L.logo_gate_select(x, w_g, c.mode, c.b_th, c.ratio, self.gate_p, self.z, self.pos, self.cu_q, self.row_of,
                           self.n_sel, workspace=self.ws)
        rows = (self.pos, self.cu_q, self.n_sel)
        L.logo_branch_transform(qL, rows=rows, u_g=self.qG, **tq)  # Q^G on the selected rows only
        L.logo_branch_transform(kL, u_g=self.kG, **tk)
        L.logo_branch_transform(vL, u_g=self.vG, **tv)
        return self.forward(qL, kL, vL, self.qG, self.kG, self.vG, self.gate_p, gain_l, gain_g)

    def backward_fused(self, dO, x, w_g, qL, kL, vL, tq, tk, tv, gain_l=None, gain_g=None):
        """Gradients of forward_fused: dqL/dkL/dvL (local branch plus the
        transforms' share of the global one), the transform parameters (dA or
        ds/db for q, k, v), the ContextNorm gains, x (the gate's share) and w_g."""
        c = self.cfg
        if not hasattr(self, "dgain_l"):
            self.dgain_l = torch.empty((c.Hq, c.D), dtype=torch.float32, device=dO.device)
            self.dgain_g = torch.empty_like(self.dgain_l)
            self.dx = torch.empty_like(x)
            self.dw_g = torch.empty_like(w_g)
        L.logo_combine_bwd_gains(dO, self.o_l, self.o_c, self.gate_p, self.z, self.row_of, gain_l, gain_g, c.eps,
                                 self.dO_l, self.dO_c, self.dgate, self.dgain_l, self.dgain_g)
        self._branches(lambda: self._local_bwd(qL, kL, vL),
                       lambda: L.logo_global_sparse_attn_bwd(self.qG, self.kG, self.vG, self.pos, self.cu_q,
                                                             self.n_sel, self.o_c, self.lse_c, self.dO_c, c.scale,
                                                             self.dqG, self.dkG, self.dvG, workspace=self.ws))
        rows = (self.pos, self.cu_q, self.n_sel)
        back = lambda t: {k: v for k, v in t.items() if k != "b"}  # noqa: E731  (b does not enter the backward)
        tqg = L.logo_branch_transform_bwd(qL, self.dqG, rows=rows, du_l=self.dqL, accumulate=True, **back(tq))
        tkg = L.logo_branch_transform_bwd(kL, self.dkG, du_l=self.dkL, accumulate=True, **back(tk))
        tvg = L.logo_branch_transform_bwd(vL, self.dvG, du_l=self.dvL, accumulate=True, **back(tv))
        L.logo_gate_bwd(x, w_g, self.gate_p, self.dgate, dx=self.dx, dw_g=self.dw_g)
        names = lambda t, g: ({"dA": g[1]} if "a" in t else {"ds": g[1], "db": g[2]})  # noqa: E731
        return dict(dqL=self.dqL, dkL=self.dkL, dvL=self.dvL, tq=names(tq, tqg), tk=names(tk, tkg),
                    tv=names(tv, tvg), dgain_l=self.dgain_l, dgain_g=self.dgain_g, dx=self.dx, dw_g=self.dw_g,
                    dgate_p=self.dgate)
