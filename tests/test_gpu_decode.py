"""One autoregressive decoding step (Sec. 3.3 Autoregressive Decoding):
logo_decode_local_attn over a ring cache (Eq. 6) and
logo_decode_global_sparse_attn over dense caches for the selected sequences
only (Eq. 8), against the oracle's dense attention for the new token.  Cache
rows the step must not see are poisoned with NaN."""
import numpy as np
import pytest
import torch

import oracle
from helpers import check_close, np32, seeded

pytestmark = pytest.mark.gpu

LENS = [1, 127, 128, 129, 1024, 1025, 1500, 3000]  # chunk edges, ring edges, the full cache


def _caches(B, L, Hq, Hkv, D, seed):
    kL = seeded((B, L, Hkv, D), seed, torch.bfloat16)
    vL = seeded((B, L, Hkv, D), seed + 1, torch.bfloat16)
    kG = seeded((B, L, Hkv, D), seed + 2, torch.bfloat16)
    vG = seeded((B, L, Hkv, D), seed + 3, torch.bfloat16)
    qL = seeded((B, Hq, D), seed + 4, torch.bfloat16)
    qG = seeded((B, Hq, D), seed + 5, torch.bfloat16)
    return kL, vL, kG, vG, qL, qG


def _ring(dense, lens, R, W=None):
    """Ring cache of R slots: position s of the last R positions in slot s mod R.
    Slots never written, and (if W is given) slots holding positions outside
    the window, are NaN: the step must not see them."""
    B, L, H, D = dense.shape
    ring = torch.full((B, R, H, D), float("nan"), dtype=torch.bfloat16)
    for b, n in enumerate(lens):
        lo = max(0, n - R) if W is None else max(0, n - min(R, W))
        s = torch.arange(lo, n)
        ring[b, s % R] = dense[b, s]
    return ring


def _poisoned(dense, lens):
    """Dense cache with the rows at and past each sequence's length poisoned."""
    out = dense.clone()
    for b, n in enumerate(lens):
        out[b, n:] = float("nan")
    return out


def _oracle_new_token(q, k, v, lens, window, rows):
    """Eq. 1 for the new token (position len_b - 1) of the sequences in `rows`."""
    B, Hq, D = q.shape
    L = k.shape[1]
    qf = np.zeros((B, L, Hq, D), dtype=np.float32)
    for b in range(B):
        qf[b, lens[b] - 1] = np32(q[b])
    o, _ = oracle.attn_fwd(qf, np32(k), np32(v), np.array(rows, np.int32),
                           np.array([lens[b] - 1 for b in rows], np.int32), window)
    return o


@pytest.mark.parametrize("D,Hq,Hkv,R", [(128, 8, 2, 1024), (64, 4, 4, 1024), (128, 16, 1, 1152)])
def test_decode_local_ring(D, Hq, Hkv, R):
    from paper_2608_29539_gb300 import logo as L
    W = 1024
    B, Lmax = len(LENS), max(LENS)
    kL, vL, _, _, qL, _ = _caches(B, Lmax, Hq, Hkv, D, seed=41 + D + Hq)
    dev = torch.device("cuda")
    k_ring, v_ring = _ring(kL, LENS, R, W).to(dev), _ring(vL, LENS, R, W).to(dev)
    seq_len = torch.tensor(LENS, dtype=torch.int32, device=dev)
    o = L.logo_decode_local_attn(qL.to(dev), k_ring, v_ring, seq_len, W)
    torch.cuda.synchronize()
    ref = _oracle_new_token(qL, kL, vL, LENS, W, list(range(B)))
    check_close(np32(o), ref, f"decode local D{D} Hq{Hq} Hkv{Hkv} R{R}")


@pytest.mark.parametrize("D,Hq,Hkv", [(128, 8, 2), (64, 4, 4), (128, 16, 1)])
def test_decode_global_selected_rows_only(D, Hq, Hkv):
    from paper_2608_29539_gb300 import logo as L
    B, Lmax = len(LENS), max(LENS)
    _, _, kG, vG, _, qG = _caches(B, Lmax, Hq, Hkv, D, seed=77 + D + Hq)
    dev = torch.device("cuda")
    chosen = [0, 2, 3, 6, 7]
    p = torch.full((B, 1), 0.2, dtype=torch.float32)
    p[chosen, 0] = 0.9
    z, pos, cu_q, row_of, n_sel = L.logo_select(p.to(dev), L.LOGO_SELECT_THRESHOLD, b_th=0.5)
    k_cache, v_cache = _poisoned(kG, LENS).to(dev), _poisoned(vG, LENS).to(dev)
    seq_len = torch.tensor(LENS, dtype=torch.int32, device=dev)
    o_c = torch.full((B, Hq, D), 7.0, dtype=torch.bfloat16, device=dev)  # sentinel for untouched rows
    L.logo_decode_global_sparse_attn(qG.to(dev), k_cache, v_cache, seq_len, cu_q, n_sel, o_c=o_c)
    torch.cuda.synchronize()
    n = int(n_sel[0])
    assert n == len(chosen)
    ref = _oracle_new_token(qG, kG, vG, LENS, 0, chosen)
    check_close(np32(o_c[:n]), ref, f"decode global D{D} Hq{Hq} Hkv{Hkv}")
    assert bool((o_c[n:] == 7.0).all())


def test_decode_global_with_nothing_selected_writes_nothing():
    from paper_2608_29539_gb300 import logo as L
    B, Lmax, Hq, Hkv, D = 4, 600, 4, 2, 128
    _, _, kG, vG, _, qG = _caches(B, Lmax, Hq, Hkv, D, seed=5)
    dev = torch.device("cuda")
    p = torch.full((B, 1), 0.1, dtype=torch.float32, device=dev)
    z, pos, cu_q, row_of, n_sel = L.logo_select(p, L.LOGO_SELECT_THRESHOLD, b_th=0.5)
    o_c = torch.full((B, Hq, D), 3.0, dtype=torch.bfloat16, device=dev)
    seq_len = torch.tensor([600, 1, 300, 599], dtype=torch.int32, device=dev)
    L.logo_decode_global_sparse_attn(qG.to(dev), kG.to(dev), vG.to(dev), seq_len, cu_q, n_sel, o_c=o_c)
    torch.cuda.synchronize()
    assert int(n_sel[0]) == 0
    assert bool((o_c == 3.0).all())


def test_decode_step_fused_through_combine():
    """A whole step: gate routing on (B, 1), both branches, Eq. 9 + Eq. 10 fusion."""
    from paper_2608_29539_gb300 import logo as L
    W, R, Hq, Hkv, D = 1024, 1024, 8, 2, 128
    B, Lmax = len(LENS), max(LENS)
    kL, vL, kG, vG, qL, qG = _caches(B, Lmax, Hq, Hkv, D, seed=123)
    dev = torch.device("cuda")
    p = torch.from_numpy(np.random.default_rng(3).uniform(0, 1, (B, 1)).astype(np.float32))
    z, pos, cu_q, row_of, n_sel = L.logo_select(p.to(dev), L.LOGO_SELECT_THRESHOLD, b_th=0.45)
    seq_len = torch.tensor(LENS, dtype=torch.int32, device=dev)
    o_l = L.logo_decode_local_attn(qL.to(dev), _ring(kL, LENS, R).to(dev), _ring(vL, LENS, R).to(dev), seq_len, W)
    o_c = torch.zeros((B, Hq, D), dtype=torch.bfloat16, device=dev)
    L.logo_decode_global_sparse_attn(qG.to(dev), _poisoned(kG, LENS).to(dev), _poisoned(vG, LENS).to(dev), seq_len,
                                     cu_q, n_sel, o_c=o_c)
    o = torch.empty((B, 1, Hq, D), dtype=torch.bfloat16, device=dev)
    rl = torch.empty((B, 1, Hq), dtype=torch.float32, device=dev)
    rg = torch.empty((B, Hq), dtype=torch.float32, device=dev)
    L.logo_combine(o_l.view(B, 1, Hq, D), o_c, p.to(dev), z, row_of, None, None, 1e-6, o, rl, rg)
    torch.cuda.synchronize()
    zc = z.cpu().numpy()
    sel = [b for b in range(B) if zc[b, 0]]
    assert len(sel) == int(n_sel[0]) and 0 < len(sel) < B
    ref_l = _oracle_new_token(qL, kL, vL, LENS, W, list(range(B)))
    ref_g = _oracle_new_token(qG, kG, vG, LENS, 0, sel)
    check_close(np32(o_l), ref_l, "step local")
    check_close(np32(o_c[:len(sel)]), ref_g, "step global")
    # fusion on the outputs the call received (unit parity)
    ref_o, _, _ = oracle.combine_fwd(np32(o_l).reshape(B, 1, Hq, D), np32(o_c[:len(sel)]), p.numpy(), zc,
                                     row_of.cpu().numpy(), None, None, 1e-6)
    check_close(np32(o), ref_o, "step fused output")


@pytest.mark.parametrize("D,Hq,Hkv", [(128, 4, 2), (64, 8, 2)])
def test_decode_long_caches_many_chunks(D, Hq, Hkv):
    """Few rows and long caches: each (row, KV head) is cut into many chunks
    (for parallelism) whose partial results the last chunk to finish merges;
    both the dense cache of the global call and a long ring of the local one."""
    from paper_2608_29539_gb300 import logo as L
    lens = [20000, 9000]
    B, Lmax, W, R = len(lens), max(lens), 4096, 4096
    kL, vL, kG, vG, qL, qG = _caches(B, Lmax, Hq, Hkv, D, seed=314 + D)
    dev = torch.device("cuda")
    seq_len = torch.tensor(lens, dtype=torch.int32, device=dev)
    o_l = L.logo_decode_local_attn(qL.to(dev), _ring(kL, lens, R, W).to(dev), _ring(vL, lens, R, W).to(dev),
                                   seq_len, W)
    p = torch.full((B, 1), 0.9, dtype=torch.float32, device=dev)
    z, pos, cu_q, row_of, n_sel = L.logo_select(p, L.LOGO_SELECT_THRESHOLD, b_th=0.5)
    o_c = torch.zeros((B, Hq, D), dtype=torch.bfloat16, device=dev)
    L.logo_decode_global_sparse_attn(qG.to(dev), _poisoned(kG, lens).to(dev), _poisoned(vG, lens).to(dev), seq_len,
                                     cu_q, n_sel, o_c=o_c)
    torch.cuda.synchronize()
    check_close(np32(o_l), _oracle_new_token(qL, kL, vL, lens, W, [0, 1]), f"decode local long D{D}")
    check_close(np32(o_c), _oracle_new_token(qG, kG, vG, lens, 0, [0, 1]), f"decode global long D{D}")
