"""Seeded synthetic inputs shaped like the paper's long-context workloads.

This module only draws random numbers: it holds none of the layer's arithmetic
and is the one piece shared by the CUDA path's tests and the CPU oracle.  The
gate p_t is produced the way a caller of the layer produces it (Eq. 7 puts a
sigmoid on a gate logit); here the logits are synthetic.

Draw order (fixed, per workload seed): Q, K, V of the local branch, then Q, K,
V of the global branch, then gate logits, then the upstream gradient dO.  Every
tensor is drawn in float32 and rounded to bf16 for the device.  There is no
dataset: these tensors stand in for the paper's 8k-128k training contexts
(Sec. 4.1-4.2) and for the operator benchmark shapes of Sec. 4.3.
"""
from __future__ import annotations

import dataclasses
import math

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    T: int
    Hq: int
    Hkv: int
    D: int
    window: int
    ratio: float
    seed: int
    mode: str = "ratio"            # "ratio" (top-k per sequence) or "threshold" (Eq. 7)
    selection: str = "normal"      # "normal" logits ~ N(0,1) or "clustered" runs
    backward: bool = True
    qkv_std: float = 1.0           # std of the Q/K/V draws

    @property
    def k_per_seq(self) -> int:
        return int(math.floor(float(torch.tensor(self.ratio, dtype=torch.float32)) * self.T))

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads of the benchmark plan.  "tiny" is the small case the
# oracle finishes in seconds; "16k" is the headline long-context case.
WORKLOADS = {
    "tiny": Workload("tiny", B=1, T=512, Hq=4, Hkv=4, D=64, window=64, ratio=0.25, seed=0,
                     mode="threshold", backward=False, qkv_std=1.0 / math.sqrt(64)),
    "4k": Workload("4k", B=2, T=4096, Hq=16, Hkv=16, D=128, window=512, ratio=0.125, seed=1),
    "16k": Workload("16k", B=1, T=16384, Hq=32, Hkv=32, D=128, window=1024, ratio=0.125, seed=2,
                    selection="clustered"),
    "64k": Workload("64k", B=1, T=65536, Hq=32, Hkv=8, D=128, window=2048, ratio=0.0625, seed=3),
}
SWEEP_RATIOS = (0.0, 1.0 / 32, 0.125, 0.5, 1.0)


def sweep(ratio: float) -> Workload:
    """Ratio sweep at B=1, H=16, d=128, T=32768, W=1024."""
    return Workload(f"sweep{ratio:g}", B=1, T=32768, Hq=16, Hkv=16, D=128, window=1024,
                    ratio=ratio, seed=4)


def clustered_states(T: int, gen: torch.Generator, mean_run: float = 16.0, frac: float = 0.125) -> torch.Tensor:
    """The on/off states behind clustered gates: a two-state Markov chain whose
    'on' runs have mean length ``mean_run`` (leave with probability 1/mean_run)
    and whose stationary 'on' share is ``frac`` (enter with probability
    (1/mean_run) * frac / (1 - frac)); the first state is drawn from the
    stationary distribution.  Returns float32 0/1 of length T."""
    p_off = 1.0 / mean_run
    p_on = p_off * frac / (1.0 - frac)
    u = torch.rand(T, generator=gen, dtype=torch.float64)
    ul = u.tolist()
    s = 1 if ul[0] < frac else 0
    st = [0.0] * T
    for t in range(T):
        if t > 0:
            if s == 1 and ul[t] < p_off:
                s = 0
            elif s == 0 and ul[t] < p_on:
                s = 1
        st[t] = float(s)
    return torch.tensor(st, dtype=torch.float32)


def clustered_logits(T: int, gen: torch.Generator, mean_run: float = 16.0, frac: float = 0.125):
    """Gate logits with clustered high values: N(0,1) + 4 * state, the state
    from ``clustered_states`` (drawn first, then the noise)."""
    state = clustered_states(T, gen, mean_run, frac)
    noise = torch.randn(T, generator=gen, dtype=torch.float32)
    return noise + 4.0 * state


def make_inputs(w: Workload, device: str = "cpu", need_grad_inputs: bool | None = None):
    """Draw one workload's tensors.

    Returns a dict with bf16 ``qL, kL, vL, qG, kG, vG`` ([B,T,H,D]), float32 gate
    ``p`` ([B,T]) in (0,1), the selection control (``mode``, ``b_th``,
    ``ratio``), and bf16 ``dO`` ([B,T,Hq,D]) when the workload has a backward.
    ``device='cuda'`` draws on the GPU with a CUDA generator (a different but
    equally seeded stream) for large shapes."""
    gen = torch.Generator(device=device)
    gen.manual_seed(w.seed)
    shp_q = (w.B, w.T, w.Hq, w.D)
    shp_kv = (w.B, w.T, w.Hkv, w.D)

    def draw(shape):
        x = torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
        if w.qkv_std != 1.0:
            x.mul_(w.qkv_std)
        return x.to(torch.bfloat16)

    out = {}
    out["qL"], out["kL"], out["vL"] = draw(shp_q), draw(shp_kv), draw(shp_kv)
    out["qG"], out["kG"], out["vG"] = draw(shp_q), draw(shp_kv), draw(shp_kv)
    if w.selection == "clustered":
        cpu_gen = torch.Generator()
        cpu_gen.manual_seed(w.seed + 1000)
        g = torch.stack([clustered_logits(w.T, cpu_gen) for _ in range(w.B)]).to(device)
    else:
        g = torch.randn((w.B, w.T), generator=gen, device=device, dtype=torch.float32)
    p = torch.sigmoid(g).to(torch.float32)
    out["p"] = p.contiguous()
    out["mode"] = w.mode
    out["ratio"] = w.ratio
    if w.mode == "threshold":
        # b_th = the (T-k)-th smallest gate of the batch: with distinct gates
        # exactly k tokens lie strictly above it (B == 1 in the tiny workload).
        k = w.k_per_seq
        srt = torch.sort(p.reshape(-1).cpu()).values
        out["b_th"] = float(srt[p.numel() - k - 1]) if k < p.numel() else -1.0
    else:
        out["b_th"] = 0.5
    want_grad = w.backward if need_grad_inputs is None else need_grad_inputs
    if want_grad:
        out["dO"] = torch.randn(shp_q, generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)
    return out


def random_gains(H: int, D: int, seed: int, device: str = "cpu"):
    """ContextNorm gains near 1 (two per layer: local and global), float32 [H, D]."""
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    gl = 1.0 + 0.1 * torch.randn((H, D), generator=gen, device=device, dtype=torch.float32)
    gg = 1.0 + 0.1 * torch.randn((H, D), generator=gen, device=device, dtype=torch.float32)
    return gl, gg
