#!/usr/bin/env python
"""Benchmark of the LoGo attention layer's hot path on GB300.

One step = one training pass of the layer over one batch of synthetic input:
select -> local fwd -> global fwd -> combine -> combine bwd -> global bwd ->
local bwd (every call through the C ABI, inputs resident in HBM; the local
calls run on a second stream beside the global calls, forked after the
selection and after the combine bwd, joined before the combine and at the end
of the step).

Metric: useful TFLOP/s of the whole step.  Useful FLOPs count only the
query-key pairs the method must compute, 14*d per pair per head (4*d forward:
Q.K^T and P.V; 10*d backward: S recompute, dP, dV, dQ, dK):
  local pairs per head  = sum_t min(t+1, W)
  global pairs per head = sum over selected t of (t+1)   (realised selection)

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Prints one JSON line (rank 0).  For N > 1 (torchrun) every rank runs its own
replica of the workload (the path shards over sequences/heads with no
exchange): value = all ranks' useful FLOPs / the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "LoGo attn fwd+bwd useful TFLOP/s & % bf16 TC peak, T=16K r=0.125"
WORKLOAD = "16k"
L2_BYTES = 129 * 1024 * 1024

# DRAM traffic per launch of the dominant kernel from an ncu capture, keyed by
# the SHA-256 of the kernel source it was taken on; reported only while the
# source is unchanged (see profiles/).
TRAFFIC = {
    # attn_bwd2_kernel, 16K workload (ncu dram__bytes_read.sum + dram__bytes_write.sum, one launch each)
    ("local_bwd", "f716c69b384b4931"): 824986112 + 482090752,
    ("global_bwd", "f716c69b384b4931"): 476076288 + 432424704,
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", default=WORKLOAD,
                    help="16k (headline), 4k, 64k, or sweep:<ratio> (T=32K, H=16, W=1024)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-dense", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-routing", action="store_true")
    ap.add_argument("--no-fusions", action="store_true")
    ap.add_argument("--eager", action="store_true",
                    help="time eager launches instead of one CUDA graph replay per step")
    ap.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle work for cpu_baseline")
    return ap.parse_args()


# ------------------------------------------------------------------ helpers
def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return {"hbm": float(p["hbm_gbs"]), "bf16": float(p["bf16_tflops"]),
                "bf16_sus": float(p["bf16_tflops_sustained"]), "src": "measured"}
    except Exception:
        return {"hbm": 6800.0, "bf16": 1900.0, "bf16_sus": 1700.0, "src": "fallback"}


def local_pairs(T, W):
    W = min(W, T)
    return W * (W + 1) // 2 + (T - W) * W


def useful_flops(w, pos_by_seq):
    lp = local_pairs(w.T, w.window) * w.B
    gp = sum(int((p.astype(np.int64) + 1).sum()) for p in pos_by_seq)
    per_pair = 14 * w.D * w.Hq
    return lp * per_pair, gp * per_pair, lp, gp


def src_hash(path):
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    FIELDS = ["index", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={','.join(self.FIELDS)}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(self.idx)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------ the step
def make_device_inputs(w, device):
    from paper_2608_29539_gb300.workloads import make_inputs
    x = make_inputs(w, device=device)
    return {k: v for k, v in x.items()}


CALLS = ["select", "local_fwd", "global_fwd", "combine", "combine_bwd", "global_bwd", "local_bwd"]
LAUNCHES_PER_STEP = {"select": 4, "local_fwd": 1, "global_fwd": 4, "combine": 1, "combine_bwd": 1,
                     "global_bwd": 3, "local_bwd": 3}


def launches_per_step(w):
    """Kernels one step launches: select takes one launch in ratio mode for
    sequences of at most 128K tokens, four otherwise."""
    n = sum(LAUNCHES_PER_STEP.values())
    if w.mode == "ratio" and w.T <= 131072:
        n -= LAUNCHES_PER_STEP["select"] - 1
    return n


def step_calls(layer, g):
    """The seven calls of one step, in order, as (name, thunk) pairs."""
    from paper_2608_29539_gb300 import logo as L
    c = layer.cfg
    return [
        ("select", lambda: L.logo_select(g["p"], c.mode, c.b_th, c.ratio, layer.z, layer.pos, layer.cu_q,
                                         layer.row_of, layer.n_sel, workspace=layer.ws)),
        ("local_fwd", lambda: L.logo_local_attn_fwd(g["qL"], g["kL"], g["vL"], c.window, c.scale, layer.o_l,
                                                    layer.lse_l)),
        ("global_fwd", lambda: L.logo_global_sparse_attn_fwd(g["qG"], g["kG"], g["vG"], layer.pos, layer.cu_q,
                                                             layer.n_sel, c.scale, layer.o_c, layer.lse_c,
                                                             workspace=layer.ws)),
        ("combine", lambda: L.logo_combine(layer.o_l, layer.o_c, g["p"], layer.z, layer.row_of, None, None, c.eps,
                                           layer.o, layer.rstd_l, layer.rstd_g)),
        ("combine_bwd", lambda: L.logo_combine_bwd(g["dO"], layer.o_l, layer.o_c, g["p"], layer.z, layer.row_of,
                                                   None, None, c.eps, layer.dO_l, layer.dO_c, layer.dgate)),
        ("global_bwd", lambda: L.logo_global_sparse_attn_bwd(g["qG"], g["kG"], g["vG"], layer.pos, layer.cu_q,
                                                             layer.n_sel, layer.o_c, layer.lse_c, layer.dO_c,
                                                             c.scale, layer.dqG, layer.dkG, layer.dvG,
                                                             workspace=layer.ws)),
        ("local_bwd", lambda: L.logo_local_attn_bwd(g["qL"], g["kL"], g["vL"], layer.o_l, layer.lse_l, layer.dO_l,
                                                    c.window, c.scale, layer.dqL, layer.dkL, layer.dvL,
                                                    workspace=layer.ws_l)),
    ]


def run_step(layer, g, ev=None):
    """One full step through the layer: the local branch on the layer's side
    stream beside the global branch.  If ev is given, the
    seven calls run in order on one stream instead, with an event recorded
    after each (per-call times)."""
    if ev is None:
        args = (g["qL"], g["kL"], g["vL"], g["qG"], g["kG"], g["vG"], g["p"])
        layer.forward(*args)
        layer.backward(g["dO"], *args)
        return
    ev[0].record()
    for i, (_, call) in enumerate(step_calls(layer, g)):
        call()
        ev[i + 1].record()


def graph_ms(call, reps=20):
    """Device time of call(): one eager call on a side stream, then the call
    captured `reps` times back to back as one CUDA graph, one warm-up replay and
    one replay timed with CUDA events on the launching stream, divided by
    `reps`.  (Timing eager calls would add the host's launch time of a small
    call to its duration.)"""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        call()
    torch.cuda.current_stream().wait_stream(side)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        for _ in range(reps):
            call()
    graph.replay()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record()
    graph.replay()
    e1.record()
    torch.cuda.synchronize()
    del graph
    return e0.elapsed_time(e1) / reps


def per_call_device_ms(layer, g, reps):
    """Device time of each call of the step (graph_ms).  Every call is
    idempotent on the step's buffers, so repeating it leaves the state of the
    step unchanged."""
    return {name: graph_ms(call, reps) for name, call in step_calls(layer, g)}


def layer_for(w, device):
    from paper_2608_29539_gb300 import logo as L
    from paper_2608_29539_gb300.layer import LayerConfig, LogoAttention
    mode = L.LOGO_SELECT_RATIO if w.mode == "ratio" else L.LOGO_SELECT_THRESHOLD
    cfg = LayerConfig(w.B, w.T, w.Hq, w.Hkv, w.D, w.window, mode=mode, ratio=w.ratio)
    return LogoAttention(cfg, device=device)


def barrier(dist_on):
    if dist_on:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, dist_on):
    if not dist_on:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x, dist_on):
    if not dist_on:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ------------------------------------------------------------------ cpu side
def oracle_sample(w, x, budget_s, pos_by_seq, rows=None):
    """Time the oracle on a bounded sample of the workload: the first
    `nh` heads, the last `r` query rows of each branch of sequence 0 (the most
    expensive rows), forward + backward.  Returns (useful TFLOP/s, seconds,
    threads, description)."""
    import oracle
    nth = oracle.num_threads()
    f = lambda t: t.detach().float().cpu().numpy()  # noqa: E731
    qL, kL, vL = f(x["qL"][:1]), f(x["kL"][:1]), f(x["vL"][:1])
    qG, kG, vG = f(x["qG"][:1]), f(x["kG"][:1]), f(x["vG"][:1])
    group = w.Hq // w.Hkv
    nh = max(group, min(w.Hq, (nth // group) * group))
    heads = np.arange(nh, dtype=np.int32)
    sel = pos_by_seq[0]
    T = w.T

    def run(r_local, r_global):
        lt = np.arange(T - r_local, T, dtype=np.int32)
        gt = sel[len(sel) - r_global:].astype(np.int32) if r_global else np.zeros(0, np.int32)
        rng = np.random.default_rng(0)
        t0 = time.perf_counter()
        if r_local:
            oracle.attn_fwd(qL, kL, vL, np.zeros_like(lt), lt, w.window, heads=heads)
            dO = rng.standard_normal((r_local, w.Hq, w.D)).astype(np.float32)
            oracle.attn_bwd(qL, kL, vL, np.zeros_like(lt), lt, w.window, dO, heads=heads)
        if r_global:
            oracle.attn_fwd(qG, kG, vG, np.zeros_like(gt), gt, 0, heads=heads)
            dO = rng.standard_normal((r_global, w.Hq, w.D)).astype(np.float32)
            oracle.attn_bwd(qG, kG, vG, np.zeros_like(gt), gt, 0, dO, heads=heads)
        dt = time.perf_counter() - t0
        pairs = sum(min(t + 1, w.window) for t in lt.tolist()) + int((gt.astype(np.int64) + 1).sum())
        return dt, pairs * nh * 14 * w.D

    if rows is None:
        # grow the sample (doubling the rows) until one run fills about a
        # quarter of the budget, then size the final run to the budget
        r, dt = 8, 0.0
        while True:
            dt, _ = run(min(r, T), min(r, len(sel)))
            if dt >= budget_s / 4 or (r >= T and r >= len(sel)):
                break
            r *= 2
        scale = max(1.0, budget_s / max(dt, 1e-3))
        r = int(min(T, r * scale))
        rg = int(min(len(sel), r))
    else:
        r, rg = rows
    dt, flops = run(r, rg)
    desc = (f"oracle fp64 fwd+bwd on heads 0..{nh - 1} of sequence 0: the last {r} local query rows and the last "
            f"{rg} selected global rows (the most expensive rows); useful FLOPs counted as on the GPU")
    return flops / dt / 1e12, dt, nth, desc, (r, rg)


# ------------------------------------------------------------------ arms
def workload_named(name):
    from paper_2608_29539_gb300.workloads import WORKLOADS, sweep
    if name.startswith("sweep:"):
        return sweep(float(name.split(":", 1)[1]))
    return WORKLOADS[name]


def reference_arm(a, rank, world):
    """The oracle, as it stands, on the host cores: same metric and config."""
    if rank != 0:
        return
    from paper_2608_29539_gb300.workloads import make_inputs
    import oracle
    w = workload_named(a.workload)
    x = make_inputs(w, device="cpu")
    p = x["p"].numpy()
    z = oracle.select_ratio(p, w.k_per_seq) if w.mode == "ratio" else oracle.select_threshold(p, x["b_th"])
    pos, cu_q, _, n = oracle.compact(z)
    pos_by_seq = [pos[cu_q[b]:cu_q[b + 1]] for b in range(w.B)]
    per_step = max(2.0, 150.0 / max(1, a.steps + a.warmup))
    vals, secs = [], []
    rows = None  # sized once (first warm-up step), then fixed
    for i in range(a.warmup + a.steps):
        v, dt, nth, desc, rows = oracle_sample(w, x, per_step, pos_by_seq, rows)
        if i >= a.warmup:
            vals.append(v)
            secs.append(dt)
    value = float(np.mean(vals))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
            "steps": a.steps, "warmup": a.warmup, "ms_per_step": 1e3 * float(np.mean(secs)),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_of(w),
            "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": nth, "kind": "oracle", "sample": desc},
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def config_of(w):
    return {"workload": f"{w.name}: B={w.B} Hq={w.Hq} Hkv={w.Hkv} d={w.D} T={w.T} W={w.window} ratio={w.ratio} "
                        f"({w.selection} selection), fwd+bwd",
            "B": w.B, "T": w.T, "Hq": w.Hq, "Hkv": w.Hkv, "D": w.D, "window": w.window, "ratio": w.ratio,
            "selection": w.selection, "mode": w.mode,
            "l2": "inputs larger than L2 (6 x {:.0f} MiB bf16 Q/K/V tensors vs 129 MB L2); no flush".format(
                w.B * w.T * w.Hq * w.D * 2 / 2**20)}


def routing_bench(layer, x, w, dev):
    """Device-resident routing loop: logo_select_device_threshold then
    logo_budget_update, 50 steps on the workload's gates, no host sync."""
    from paper_2608_29539_gb300 import logo as L
    b_dev = torch.tensor([0.5], dtype=torch.float32, device=dev)
    f_dev = torch.empty((1,), dtype=torch.float32, device=dev)
    rl_bufs = (torch.empty_like(layer.z), torch.empty_like(layer.pos), torch.empty_like(layer.cu_q),
               torch.empty_like(layer.row_of), torch.empty_like(layer.n_sel))

    def routing_step():
        L.logo_select_device_threshold(x["p"], b_dev, *rl_bufs, workspace=layer.ws)
        L.logo_budget_update(rl_bufs[4], w.B, w.T, w.ratio, 2.0 ** -11, b_dev, f_out=f_dev)

    # each step reads the threshold the previous one wrote: 50 steps in one graph
    return {"us_per_step": graph_ms(routing_step, 50) * 1e3, "launches_per_step": 4,
            "note": "logo_select_device_threshold + logo_budget_update, no host sync; device time per step "
                    "(50 steps captured as one CUDA graph)"}


def fusions_bench(layer, x, w, dev, pk):
    """The fused pieces around the attention: the Eq. 7 gate + select on a
    [B, T, d_model = Hq*D] input, the gate backward (dx accumulated into the
    caller's gradient, dw_g), and the combine backward with the ContextNorm
    gain gradients against the one without.  Bytes are the HBM bytes each call
    must move at least; every operand is at least 128 MiB (about L2's size)."""
    from paper_2608_29539_gb300 import logo as L
    dm = w.Hq * w.D
    g = torch.Generator(device=dev).manual_seed(5)
    xin = torch.randn((w.B, w.T, dm), generator=g, device=dev).to(torch.bfloat16)
    wg = torch.randn((dm,), generator=g, device=dev) / dm ** 0.5
    dxin = torch.randn((w.B, w.T, dm), generator=g, device=dev).to(torch.bfloat16)
    bufs = (torch.empty((w.B, w.T), dtype=torch.float32, device=dev), torch.empty_like(layer.z),
            torch.empty_like(layer.pos), torch.empty_like(layer.cu_q), torch.empty_like(layer.row_of),
            torch.empty_like(layer.n_sel))
    c = layer.cfg
    dw = torch.empty((dm,), dtype=torch.float32, device=dev)
    gws = torch.empty((int(L.lib().logo_gate_bwd_workspace_size(L.Dims(w.B, w.T, 1, 1, 64), dm)),), dtype=torch.uint8,
                      device=dev)
    cws = torch.empty((L.workspace_bytes("combine_bwd_gains", layer.dims),), dtype=torch.uint8, device=dev)
    dgl = torch.empty((w.Hq, w.D), dtype=torch.float32, device=dev)
    dgg = torch.empty_like(dgl)
    n = int(layer.n_sel[0])

    timed = graph_ms  # device time per call

    gate = lambda: L.logo_gate_select(xin, wg, c.mode, c.b_th, c.ratio, *bufs, workspace=layer.ws)  # noqa: E731
    gate_bwd = lambda: L.logo_gate_bwd(xin, wg, bufs[0], layer.dgate, dx=dxin, accumulate=True, dw_g=dw,  # noqa: E731
                                       workspace=gws)
    cargs = (x["dO"], layer.o_l, layer.o_c, x["p"], layer.z, layer.row_of, None, None, c.eps, layer.dO_l, layer.dO_c,
             layer.dgate)
    cplain = lambda: L.logo_combine_bwd(*cargs)  # noqa: E731
    cgains = lambda: L.logo_combine_bwd_gains(*cargs, dgain_l=dgl, dgain_g=dgg, workspace=cws)  # noqa: E731
    tok_row = w.Hq * w.D * 2
    ntok = w.B * w.T
    out = {}
    ms = timed(gate)
    byts = ntok * dm * 2 + ntok * 4
    out["gate_select"] = {"ms": ms, "GB_per_s": byts / ms / 1e6, "frac_of_hbm_peak": byts / ms / 1e6 / pk["hbm"],
                          "bytes": byts, "d_model": dm, "launches": 5}
    ms = timed(gate_bwd)
    byts = 3 * ntok * dm * 2 + 2 * ntok * 4
    out["gate_bwd"] = {"ms": ms, "GB_per_s": byts / ms / 1e6, "frac_of_hbm_peak": byts / ms / 1e6 / pk["hbm"],
                       "bytes": byts, "note": "x read, dx read and written (accumulated), dw_g", "launches": 2}
    ms_p, ms_g = timed(cplain), timed(cgains)
    byts = 3 * ntok * tok_row + 2 * n * tok_row
    out["combine_bwd_gains"] = {"ms": ms_g, "ms_without_gains": ms_p, "GB_per_s": byts / ms_g / 1e6,
                                "frac_of_hbm_peak": byts / ms_g / 1e6 / pk["hbm"], "bytes": byts, "launches": 2}
    # Eq. 5 LP transforms: Q^G on the selected rows only, K^G on every row, and
    # the backward of the K transform (dK^L accumulated, dA)
    A = (torch.randn((w.Hkv, w.D, w.D), generator=g, device=dev) / w.D ** 0.5).to(torch.bfloat16)
    Aq = (torch.randn((w.Hq, w.D, w.D), generator=g, device=dev) / w.D ** 0.5).to(torch.bfloat16)
    qg, kg = torch.empty_like(x["qL"]), torch.empty_like(x["kL"])
    dkl = torch.zeros_like(x["kL"])
    tws = torch.empty((int(L.lib().logo_branch_transform_bwd_workspace_size(
        L.Dims(w.B, w.T, w.Hkv, w.Hkv, w.D))),), dtype=torch.uint8, device=dev)
    rows = (layer.pos, layer.cu_q, layer.n_sel)
    lp_q = lambda: L.logo_branch_transform(x["qL"], a=Aq, rows=rows, u_g=qg)  # noqa: E731
    lp_k = lambda: L.logo_branch_transform(x["kL"], a=A, u_g=kg)  # noqa: E731
    dkg = x["dO"][:, :, :w.Hkv].contiguous()  # a stand-in dK^G of the right shape
    lp_kb = lambda: L.logo_branch_transform_bwd(x["kL"], dkg, a=A, du_l=dkl, accumulate=True,  # noqa: E731
                                                workspace=tws)
    kv_row = w.Hkv * w.D * 2
    for name, fn, rows_n, row_b, heads, passes in (("lp_q_selected_rows", lp_q, n, tok_row, w.Hq, 2),
                                                   ("lp_k_all_rows", lp_k, ntok, kv_row, w.Hkv, 2),
                                                   ("lp_k_backward", lp_kb, ntok, kv_row, w.Hkv, 4)):
        ms = timed(fn)
        byts = passes * rows_n * row_b
        fl = (2 if passes == 2 else 4) * rows_n * heads * w.D * w.D
        out[name] = {"ms": ms, "rows": rows_n, "GB_per_s": byts / ms / 1e6,
                     "frac_of_hbm_peak": byts / ms / 1e6 / pk["hbm"], "tflops": fl / ms / 1e9, "bytes": byts}
    return out


def decode_bench(dev, pk):
    """Time one decoding step's attention (local branch from ring caches, global
    branch for the selected sequences only, fusion) and the same step under the
    paper's dense policy (every sequence runs the global call).  Inputs are
    synthetic and seeded; the caches are larger than L2."""
    from paper_2608_29539_gb300 import logo as L
    B, Lc, Hq, Hkv, D, W = 32, 16384, 32, 8, 128, 1024
    g = torch.Generator(device=dev).manual_seed(9)
    kG = torch.randn((B, Lc, Hkv, D), generator=g, device=dev).to(torch.bfloat16)
    vG = torch.randn((B, Lc, Hkv, D), generator=g, device=dev).to(torch.bfloat16)
    kR = torch.randn((B, W, Hkv, D), generator=g, device=dev).to(torch.bfloat16)
    vR = torch.randn((B, W, Hkv, D), generator=g, device=dev).to(torch.bfloat16)
    qL = torch.randn((B, Hq, D), generator=g, device=dev).to(torch.bfloat16)
    qG = torch.randn((B, Hq, D), generator=g, device=dev).to(torch.bfloat16)
    seq_len = torch.full((B,), Lc, dtype=torch.int32, device=dev)
    p = torch.rand((B, 1), generator=g, device=dev)
    b_th = float(torch.quantile(p.flatten().cpu(), 7.0 / 8.0))
    sparse_sel = L.logo_select(p, L.LOGO_SELECT_THRESHOLD, b_th=b_th)
    dense_sel = L.logo_select(p, L.LOGO_SELECT_THRESHOLD, b_th=-1.0)
    n = int(sparse_sel[4][0])
    ws = torch.empty(int(L.lib().logo_decode_workspace_size(L.Dims(B, Lc, Hq, Hkv, D))), dtype=torch.uint8,
                     device=dev)
    ws_l = torch.empty(int(L.lib().logo_decode_workspace_size(L.Dims(B, W, Hq, Hkv, D))), dtype=torch.uint8,
                       device=dev)
    aux = torch.cuda.Stream(device=dev)
    o_l = torch.empty((B, Hq, D), dtype=torch.bfloat16, device=dev)
    o_c = torch.empty((B, Hq, D), dtype=torch.bfloat16, device=dev)
    o = torch.empty((B, 1, Hq, D), dtype=torch.bfloat16, device=dev)
    rl = torch.empty((B, 1, Hq), dtype=torch.float32, device=dev)
    rg = torch.empty((B, Hq), dtype=torch.float32, device=dev)

    def step(sel):
        # the two branches are independent: the local call runs on a second
        # stream beside the global one (their items fill the GPU together),
        # joined before the fusion
        zz, _, cq, ro, ns = sel
        main = torch.cuda.current_stream(dev)
        aux.wait_stream(main)
        with torch.cuda.stream(aux):
            L.logo_decode_local_attn(qL, kR, vR, seq_len, W, o=o_l, workspace=ws_l)
        L.logo_decode_global_sparse_attn(qG, kG, vG, seq_len, cq, ns, o_c=o_c, workspace=ws)
        main.wait_stream(aux)
        L.logo_combine(o_l.view(B, 1, Hq, D), o_c, p, zz, ro, None, None, 1e-6, o, rl, rg)

    def timed(sel, reps=20):  # device time per step, both streams inside one graph
        return graph_ms(lambda: step(sel), reps)

    sparse_ms = timed(sparse_sel)
    dense_ms = timed(dense_sel)
    row_bytes = Hkv * D * 2 * 2  # K and V of one position, bf16
    bytes_sparse = B * W * row_bytes + n * Lc * row_bytes
    bytes_dense = B * W * row_bytes + B * Lc * row_bytes
    gbs = bytes_sparse / (sparse_ms / 1e3) / 1e9
    gbs_dense = bytes_dense / (dense_ms / 1e3) / 1e9
    del kG, vG
    return {"workload": f"B{B} cache {Lc} Hq{Hq}/Hkv{Hkv} d{D} W{W}, {n}/{B} sequences selected",
            "ms_per_step": sparse_ms, "cache_GB_per_s": gbs, "frac_of_hbm_peak": gbs / pk["hbm"],
            "dense_policy_ms": dense_ms, "dense_policy_GB_per_s": gbs_dense,
            "speedup_vs_dense_policy": dense_ms / sparse_ms, "ideal_speedup": bytes_dense / bytes_sparse,
            "launches_per_step": 4,
            "note": "routing on (B, 1) is outside the timed loop; bytes = K and V cache rows read; launches: "
                    "local attention (on a second stream, beside the global call), the global call's counter clear "
                    "and attention, the fusion"}


def native_arm(a, rank, world, local_rank, dist_on):
    from paper_2608_29539_gb300 import logo as L
    w = workload_named(a.workload)
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    pk = peaks()
    x = make_device_inputs(w, "cuda")
    layer = layer_for(w, dev)
    run_step(layer, x)
    torch.cuda.synchronize()
    n = int(layer.n_sel.item())
    cu = layer.cu_q.cpu().numpy()
    pos = layer.pos[:n].cpu().numpy()
    pos_by_seq = [pos[cu[b]:cu[b + 1]] for b in range(w.B)]
    fl_local, fl_global, lp, gp = useful_flops(w, pos_by_seq)
    fl_step = fl_local + fl_global

    for _ in range(max(0, a.warmup - 1)):
        run_step(layer, x)
    torch.cuda.synchronize()
    # The step has fixed shapes and keeps every count on the device, so it is
    # captured once as a CUDA graph and replayed: one launch of the graph per
    # step instead of eight host-side calls.
    graph = None
    if not a.eager:
        side = torch.cuda.Stream(device=dev)
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            run_step(layer, x)
        torch.cuda.current_stream().wait_stream(side)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            run_step(layer, x)
        for _ in range(max(1, a.warmup)):
            graph.replay()
    # ---- timed region: K steps (graph replays, or eager calls with per-call
    # events); then K eager steps with an event after each call on the
    # launching stream, which give the per-call times and the roofline
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(8)] for _ in range(a.steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    barrier(dist_on)
    with ClockSampler(local_rank) as clk:
        time.sleep(0.25)
        t_start.record()
        for s in range(a.steps):
            if graph is not None:
                graph.replay()
            else:
                run_step(layer, x, evs[s])
        t_end.record()
        torch.cuda.synchronize()
        if graph is not None:
            for s in range(a.steps):
                run_step(layer, x, evs[s])
            torch.cuda.synchronize()
        time.sleep(0.25)
    barrier(dist_on)
    st = L.logo_get_device_status()
    if st != 0:
        raise RuntimeError(f"device status {st} after the timed region")
    total_ms = t_start.elapsed_time(t_end)
    total_ms = max_over_ranks(total_ms, dist_on)
    ms_step = total_ms / a.steps
    per_call_eager = {c: float(np.mean([evs[s][i].elapsed_time(evs[s][i + 1]) for s in range(a.steps)]))
                      for i, c in enumerate(CALLS)}
    eager_ms = float(np.mean([evs[s][0].elapsed_time(evs[s][7]) for s in range(a.steps)]))
    per_call = per_call_device_ms(layer, x, reps=max(3, a.steps))
    flops_all = sum_over_ranks(fl_step * a.steps, dist_on)
    value = flops_all / (total_ms / 1e3) / 1e12

    # roofline of the dominant call (its tensor-core kernel dominates the call)
    flops_call = {"local_fwd": fl_local * 4 / 14, "local_bwd": fl_local * 10 / 14,
                  "global_fwd": fl_global * 4 / 14, "global_bwd": fl_global * 10 / 14}
    g_ms = per_call["global_fwd"] + per_call["global_bwd"]
    dom = max(flops_call, key=lambda c: per_call[c])
    achieved = flops_call[dom] / (per_call[dom] / 1e3) / 1e12
    kernel_src = os.path.join(ROOT, "paper_2608_29539_gb300", "csrc",
                              "attn_bwd.cu" if dom.endswith("bwd") else "attn_fwd.cu")
    tr = TRAFFIC.get((dom, src_hash(kernel_src)))
    roof = {"bound": "tensor", "kernel": dom, "achieved": achieved, "peak": pk["bf16"], "unit": "TFLOP/s",
            "frac": achieved / pk["bf16"], "traffic": tr,
            "peak_note": f"{pk['src']} burst bf16 (the call runs for about a millisecond at the maximum SM "
                         f"clock); frac of the sustained peak {achieved / pk['bf16_sus']:.3f}",
            "frac_of_sustained": achieved / pk["bf16_sus"],
            "timing": "CUDA events on the launching stream around one replay of a CUDA graph holding the "
                      "call K times back to back, divided by K"}
    l_ms = per_call["local_fwd"] + per_call["local_bwd"]
    breakdown = {c: {"ms": per_call[c], "ms_eager_call": per_call_eager[c]} for c in CALLS}
    for c, fl in flops_call.items():
        breakdown[c]["tflops"] = fl / (per_call[c] / 1e3) / 1e12
    line = {"metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": a.steps,
            "warmup": a.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded; no dataset)", "config": config_of(w),
            "frac_of_peak": value / pk["bf16"], "frac_of_sustained_peak": value / pk["bf16_sus"],
            "global_fwd_bwd": {"tflops": fl_global / (g_ms / 1e3) / 1e12,
                               "frac_of_peak": fl_global / (g_ms / 1e3) / 1e12 / pk["bf16"],
                               "frac_of_sustained_peak": fl_global / (g_ms / 1e3) / 1e12 / pk["bf16_sus"],
                               "ms": g_ms},
            "local_fwd_bwd": {"tflops": fl_local / (l_ms / 1e3) / 1e12, "ms": l_ms},
            "useful_flops_per_step": fl_step, "pairs_per_head": {"local": lp, "global": gp},
            "selected": n, "per_call": breakdown, "roofline": roof,
            "launch": ("one CUDA graph replay per step; the local calls on a second stream beside the "
                       "global calls" if graph is not None else "eager calls, one stream"),
            "eager_ms_per_step": eager_ms,
            "gpu_launches": launches_per_step(w) * a.steps, "clocks": clk.summary()}

    # ---- dense comparison: the same global kernels with every token selected
    if not a.no_dense:
        from paper_2608_29539_gb300.layer import LayerConfig, LogoAttention
        dl = layer_for(w.with_(ratio=1.0), dev)
        run_step(dl, x)
        reps = 3
        e = [torch.cuda.Event(enable_timing=True) for _ in range(8)]
        tt = []
        for _ in range(reps):
            run_step(dl, x, e)
            torch.cuda.synchronize()
            tt.append(e[2].elapsed_time(e[3]) + e[5].elapsed_time(e[6]))
        dense_ms = float(np.median(tt))
        dense_flops = w.B * w.T * (w.T + 1) // 2 * 14 * w.D * w.Hq
        line["dense_global_fwd_bwd"] = {"ms": dense_ms, "tflops": dense_flops / (dense_ms / 1e3) / 1e12,
                                        "speedup_sparse_vs_dense": dense_ms / max(g_ms, 1e-9),
                                        "ideal_speedup": dense_flops / max(fl_global, 1)}
        del dl

    # ---- device-resident routing loop (Sec. 3.2): threshold select with the
    # threshold on the device, then the Eq. 11 update, on this workload's gates
    if not a.no_routing:
        line["device_routing_loop"] = routing_bench(layer, x, w, dev)

    # ---- the fused gate (Eq. 7) + select, its backward, and the combine
    # backward with the ContextNorm gain gradients
    if not a.no_fusions:
        line["fusions"] = fusions_bench(layer, x, w, dev, pk)

    # ---- one decoding step (Sec. 3.3): 32 sequences with 16K-token caches,
    # GQA 32/8, d = 128, W = 1024, about 1/8 of the new tokens selected
    if not a.no_decode and rank == 0:
        line["decode"] = decode_bench(dev, pk)

    # ---- end to end through host buffers: every step copies its inputs in from
    # pinned host memory and reads O and dL/dp back.  The inputs are double
    # buffered on the device: step i+1's are copied in on a copy stream while
    # step i computes from the other buffer (the host-to-device link, not the
    # GPU, bounds this loop); the readback follows each step on its stream.
    if not a.no_e2e:
        host = {k: x[k].cpu().pin_memory() for k in ("qL", "kL", "vL", "qG", "kG", "vG", "p", "dO")}
        dev_in = [{k: torch.empty_like(x[k]) for k in host} for _ in range(2)]
        out_o = torch.empty(layer.o.shape, dtype=layer.o.dtype).pin_memory()
        out_dp = torch.empty(layer.dgate.shape, dtype=layer.dgate.dtype).pin_memory()
        h2d = sum(t.numel() * t.element_size() for t in host.values())
        d2h = out_o.numel() * out_o.element_size() + out_dp.numel() * out_dp.element_size()
        main = torch.cuda.current_stream(dev)
        copy_stream = torch.cuda.Stream(device=dev)
        copied = [torch.cuda.Event() for _ in range(2)]
        consumed = [torch.cuda.Event() for _ in range(2)]

        def copy_in(slot):
            copy_stream.wait_event(consumed[slot])  # the step that read this buffer is done
            with torch.cuda.stream(copy_stream):
                for k in host:
                    dev_in[slot][k].copy_(host[k], non_blocking=True)
            copied[slot].record(copy_stream)

        def e2e_steps(n):
            copy_stream.wait_stream(main)  # no copy starts before the region's first event
            copy_in(0)
            for i in range(n):
                s = i & 1
                if i + 1 < n:
                    copy_in(s ^ 1)
                main.wait_event(copied[s])
                run_step(layer, dev_in[s])
                consumed[s].record(main)
                out_o.copy_(layer.o, non_blocking=True)
                out_dp.copy_(layer.dgate, non_blocking=True)
            main.wait_stream(copy_stream)

        e2e_steps(2)
        torch.cuda.synchronize()
        barrier(dist_on)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        e2e_steps(a.steps)
        e1.record()
        torch.cuda.synchronize()
        e2e_ms = max_over_ranks(e0.elapsed_time(e1), dist_on)
        line["e2e"] = {"value": flops_all / (e2e_ms / 1e3) / 1e12, "unit": "TFLOP/s", "h2d_bytes_per_step": h2d,
                       "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms / a.steps,
                       "note": "pinned host inputs copied in and the layer output O plus dL/dp copied out each step; "
                               "the inputs double buffered on the device, step i+1's copied in on a copy stream "
                               "while step i computes"}
    else:
        line["e2e"] = None

    # ---- the oracle on the host cores (rank 0, N = 1 only)
    if rank == 0 and world == 1 and not a.no_cpu_baseline:
        xc = {k: x[k][:1].cpu() for k in ("qL", "kL", "vL", "qG", "kG", "vG")}
        v, dt, nth, desc, _ = oracle_sample(w, xc, a.cpu_budget, pos_by_seq)
        line["cpu_baseline"] = {"value": v, "unit": "TFLOP/s", "cores": nth, "kind": "oracle", "sample": desc,
                                "seconds": dt}
    if rank == 0:
        print(json.dumps(line), flush=True)


def main():
    a = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    dist_on = world > 1
    if dist_on:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        if a.impl == "reference":
            reference_arm(a, rank, world)
        else:
            import __graft_entry__
            __graft_entry__.build()
            native_arm(a, rank, world, local_rank, dist_on)
    finally:
        if dist_on:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
