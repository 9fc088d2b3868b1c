"""Host logic of bench.py on CPU: the useful-FLOP count behind the headline
metric (computed (query, key) pairs x 14 d per head, never masked ones) against
brute-force pair counting, and the per-step launch count the JSON line claims."""
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402
from paper_2608_29539_gb300.workloads import WORKLOADS  # noqa: E402


def _brute_local_pairs(T, W):
    # keys s visible from query t in the window: max(0, t - W + 1) <= s <= t (Eq. 6)
    return sum(t - max(0, t - W + 1) + 1 for t in range(T))


@pytest.mark.parametrize("T,W", [(1, 1), (5, 3), (64, 64), (100, 7), (100, 200), (1000, 128)])
def test_local_pairs_is_the_window_count(T, W):
    assert bench.local_pairs(T, W) == _brute_local_pairs(T, W)


def test_useful_flops_count_visible_pairs_only():
    w = WORKLOADS["4k"].with_(T=300, window=50, B=2)
    rng = np.random.default_rng(0)
    pos_by_seq = [np.sort(rng.choice(300, size=k, replace=False)).astype(np.int32) for k in (40, 7)]
    fl_local, fl_global, lp, gp = bench.useful_flops(w, pos_by_seq)
    # global: a selected query at position t sees keys 0..t (Eq. 8, causal on real positions)
    brute_gp = sum(len(range(0, int(t) + 1)) for pos in pos_by_seq for t in pos)
    assert gp == brute_gp
    assert lp == w.B * _brute_local_pairs(w.T, w.window)
    per_pair = 14 * w.D * w.Hq  # 4 d forward (QK^T, PV) + 10 d backward, per head
    assert fl_local == lp * per_pair and fl_global == gp * per_pair


def test_launch_count_per_step():
    # 16K ratio workload: select 1, local fwd 1, global fwd 4 (gather, schedule,
    # attention, merge of split KV ranges), combine 1, combine bwd 1, global bwd 3
    # (pre, attention, post), local bwd 3 (pre, attention, post)
    assert bench.launches_per_step(WORKLOADS["16k"]) == 14
    # up to 128K tokens the selection is one cluster launch
    assert bench.launches_per_step(WORKLOADS["64k"]) == 14
    # longer sequences take the four-launch selection
    assert bench.launches_per_step(WORKLOADS["64k"].with_(T=262144)) == 17
