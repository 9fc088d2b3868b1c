"""The seeded input recipe on CPU: the clustered gate chain behind the 16K
workload has the stated statistics (stationary 'on' share 1/8, mean 'on' run 16
tokens), the generators are reproducible from their seed, and the workload
table holds the shapes the design names."""
import numpy as np
import torch

from paper_2608_29539_gb300.workloads import WORKLOADS, clustered_logits, clustered_states


def _runs(state):
    s = state.numpy().astype(np.int8)
    edges = np.diff(np.concatenate(([0], s, [0])))
    starts, ends = np.flatnonzero(edges == 1), np.flatnonzero(edges == -1)
    return ends - starts


def test_clustered_chain_statistics():
    st = clustered_states(1_000_000, torch.Generator().manual_seed(123))
    share = float(st.mean())
    runs = _runs(st)
    # 1e6 tokens: ~7800 runs; the standard errors are ~0.004 (share) and ~0.2 (mean run)
    assert abs(share - 0.125) < 0.012, share
    assert abs(float(runs.mean()) - 16.0) < 1.0, runs.mean()
    # geometric run lengths: P(run = 1) = 1/16
    assert abs(float((runs == 1).mean()) - 1.0 / 16.0) < 0.015


def test_clustered_logits_are_noise_plus_four_times_the_state():
    g1, g2 = torch.Generator().manual_seed(7), torch.Generator().manual_seed(7)
    lg = clustered_logits(4096, g1)
    st = clustered_states(4096, g2)
    noise = torch.randn(4096, generator=g2, dtype=torch.float32)
    assert torch.equal(lg, noise + 4.0 * st)


def test_generators_are_reproducible():
    a = clustered_logits(1000, torch.Generator().manual_seed(5))
    b = clustered_logits(1000, torch.Generator().manual_seed(5))
    c = clustered_logits(1000, torch.Generator().manual_seed(6))
    assert torch.equal(a, b) and not torch.equal(a, c)


def test_workload_shapes():
    w = WORKLOADS["16k"]
    assert (w.B, w.T, w.Hq, w.Hkv, w.D, w.window, w.ratio) == (1, 16384, 32, 32, 128, 1024, 0.125)
    w = WORKLOADS["64k"]
    assert (w.B, w.T, w.Hq, w.Hkv, w.D, w.window, w.ratio) == (1, 65536, 32, 8, 128, 2048, 0.0625)
    w = WORKLOADS["4k"]
    assert (w.B, w.T, w.Hq, w.Hkv, w.D, w.window, w.ratio) == (2, 4096, 16, 16, 128, 512, 0.125)
