"""Plain CPU oracle of the LoGo attention layer's hot path (arXiv 2608.29539).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` (its ``cpu_baseline`` leg and ``--impl reference`` arm) may import
this package.  It shares no code with the CUDA path and never calls it.

The arithmetic lives in ``logo_oracle.c`` (IEEE double, OpenMP over rows or
(batch, KV head)); this module compiles it with gcc on first use and marshals
numpy arrays.  Each function names the passage of the paper it follows:

* ``select_threshold``  -- Eq. 7, z_t = 1[p_t > b_th] (float32 compare)
* ``select_ratio``      -- per-sequence top-k reading of the target ratio rho
* ``compact``           -- the selected set I (Sec. 3.2) packed ascending (App. B)
* ``budget_update``     -- Eq. 3 realised ratio and the Eq. 11 threshold update
* ``pmask_threshold``   -- the P-mask start value of Sec. 3.2 / App. C.1
* ``attn_fwd/attn_bwd`` -- Eq. 1 over C^w_t (Eq. 6, local) or C^inf_t (Eq. 8,
                           global, selected rows only)
* ``combine_fwd/bwd``   -- Eq. 9 ContextNorm + Eq. 10 fusion
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "logo_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "liblogo_oracle.so")
_lock = threading.Lock()
_lib = None

_f32p = np.ctypeslib.ndpointer(dtype=np.float32, flags="C_CONTIGUOUS")
_f64p = np.ctypeslib.ndpointer(dtype=np.float64, flags="C_CONTIGUOUS")
_i32p = np.ctypeslib.ndpointer(dtype=np.int32, flags="C_CONTIGUOUS")
_u8p = np.ctypeslib.ndpointer(dtype=np.uint8, flags="C_CONTIGUOUS")
_i64 = ctypes.c_int64
_int = ctypes.c_int


def build(force: bool = False) -> str:
    """Compile the oracle shared library (gcc, -O2, OpenMP).  Returns its path."""
    os.makedirs(_BUILD, exist_ok=True)
    stale = (not os.path.exists(_LIB)) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.oracle_select_threshold.argtypes = [_f32p, _i64, ctypes.c_float, _u8p]
            lib.oracle_select_ratio.argtypes = [_f32p, _int, _int, _int, _u8p]
            lib.oracle_compact.argtypes = [_u8p, _int, _int, _i32p, _i32p, _i32p]
            lib.oracle_compact.restype = _i64
            lib.oracle_budget_update.argtypes = [_i64, _i64, ctypes.c_float, ctypes.c_float, ctypes.c_float,
                                                 ctypes.POINTER(ctypes.c_double)]
            lib.oracle_budget_update.restype = ctypes.c_float
            lib.oracle_pmask_threshold.argtypes = [ctypes.c_double, _i64]
            lib.oracle_pmask_threshold.restype = ctypes.c_double
            lib.oracle_attn_fwd.argtypes = [_f32p, _f32p, _f32p, _int, _int, _int, _int, _int,
                                            _i64, _i32p, _i32p, _int, _i32p, _int, ctypes.c_double,
                                            _f64p, _f64p]
            lib.oracle_attn_bwd.argtypes = [_f32p, _f32p, _f32p, _int, _int, _int, _int, _int,
                                            _i64, _i32p, _i32p, _int, _i32p, _int, ctypes.c_double,
                                            _f32p, _f64p, _f64p, _f64p]
            lib.oracle_combine_fwd.argtypes = [_f32p, _f32p, _f32p, _u8p, _i32p, ctypes.c_void_p,
                                               ctypes.c_void_p, ctypes.c_double, _int, _int, _int, _int,
                                               _f64p, _f64p, _f64p]
            lib.oracle_combine_bwd.argtypes = [_f32p, _f32p, _f32p, _f32p, _u8p, _i32p, ctypes.c_void_p,
                                               ctypes.c_void_p, ctypes.c_double, _int, _int, _int, _int,
                                               _f64p, _f64p, _f64p]
            lib.oracle_combine_dgain.argtypes = [_f32p, _f32p, _f32p, _f32p, _u8p, _i32p, ctypes.c_double,
                                                 _int, _int, _int, _int, _f64p, _f64p]
            lib.oracle_gate.argtypes = [_f32p, _f32p, _i64, _int, _f64p]
            lib.oracle_gate_bwd.argtypes = [_f32p, _f32p, _f32p, _i64, _int, _f64p, _f64p]
            _i64p = np.ctypeslib.ndpointer(dtype=np.int64, flags="C_CONTIGUOUS")
            lib.oracle_branch_fwd.argtypes = [_f32p, _int, _int, _i64p, _i64, ctypes.c_void_p, ctypes.c_void_p,
                                              ctypes.c_void_p, _f64p]
            lib.oracle_branch_bwd.argtypes = [_f32p, _int, _int, _i64p, _i64, ctypes.c_void_p, ctypes.c_void_p,
                                              _f32p, _f64p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
            lib.oracle_num_threads.restype = _int
            _lib = lib
    return _lib


def num_threads() -> int:
    """OpenMP threads the oracle uses (the cores it runs on)."""
    return int(_load().oracle_num_threads())


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


# --------------------------------------------------------------------- select
def k_from_ratio(ratio: float, T: int) -> int:
    """Tokens selected per sequence in ratio mode: floor(rho * T), rho read as float32."""
    return int(math.floor(float(np.float32(ratio)) * T))


def select_threshold(p, b_th: float) -> np.ndarray:
    """Eq. 7: z = 1[p > b_th], compared in float32.  p: [B, T] float32."""
    p = _f32(p)
    z = np.zeros(p.shape, dtype=np.uint8)
    _load().oracle_select_threshold(p, p.size, ctypes.c_float(np.float32(b_th)), z)
    return z


def select_ratio(p, k: int) -> np.ndarray:
    """Top-k gates per sequence, ties to the lower position.  p: [B, T] float32."""
    p = _f32(p)
    B, T = p.shape
    z = np.zeros(p.shape, dtype=np.uint8)
    _load().oracle_select_ratio(p, B, T, int(k), z)
    return z


def compact(z):
    """Pack I ascending per sequence: returns (pos[N], cu_q[B+1], row_of[B,T], N)."""
    z = np.ascontiguousarray(z, dtype=np.uint8)
    B, T = z.shape
    pos = np.zeros(max(B * T, 1), dtype=np.int32)
    cu_q = np.zeros(B + 1, dtype=np.int32)
    row_of = np.zeros((B, T), dtype=np.int32)
    n = int(_load().oracle_compact(z, B, T, pos, cu_q, row_of))
    return pos[:n].copy(), cu_q, row_of, n


def budget_update(n_sel: int, n_valid: int, rho: float, gamma: float, b_th: float):
    """Eq. 3 + Eq. 11: returns (new b_th as float32, F).  See oracle_budget_update."""
    F = ctypes.c_double(0.0)
    b = _load().oracle_budget_update(int(n_sel), int(n_valid), ctypes.c_float(np.float32(rho)),
                                     ctypes.c_float(np.float32(gamma)), ctypes.c_float(np.float32(b_th)),
                                     ctypes.byref(F))
    return np.float32(b), float(F.value)


def pmask_threshold(gamma: float, steps: int) -> float:
    """P-mask start b_th,0 = 0.5 - gamma * S (Sec. 3.2, App. C.1), in double."""
    return float(_load().oracle_pmask_threshold(float(gamma), int(steps)))


# ------------------------------------------------------------------ attention
def _rows(row_b, row_t):
    row_b = _i32(row_b).reshape(-1)
    row_t = _i32(row_t).reshape(-1)
    assert row_b.shape == row_t.shape
    return row_b, row_t


def _heads(heads, Hq):
    if heads is None:
        heads = np.arange(Hq, dtype=np.int32)
    return _i32(heads).reshape(-1)


def attn_fwd(q, k, v, row_b, row_t, window: int, scale: float | None = None, heads=None):
    """Eq. 1 for query rows (row_b[r], row_t[r]).

    q: [B, T, Hq, D]; k, v: [B, T, Hkv, D] (float32 holding the device values).
    window > 0: local C^w_t (Eq. 6); window <= 0: global C^inf_t (Eq. 8).
    Returns o [nrows, Hq, D] and lse [nrows, Hq] (natural log), float64; rows of
    heads not listed stay 0."""
    q, k, v = _f32(q), _f32(k), _f32(v)
    B, T, Hq, D = q.shape
    Hkv = k.shape[2]
    row_b, row_t = _rows(row_b, row_t)
    hs = _heads(heads, Hq)
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    n = row_b.size
    o = np.zeros((n, Hq, D), dtype=np.float64)
    lse = np.zeros((n, Hq), dtype=np.float64)
    if n:
        _load().oracle_attn_fwd(q, k, v, B, T, Hq, Hkv, D, n, row_b, row_t, hs.size, hs,
                                int(window), scale, o, lse)
    return o, lse


def attn_bwd(q, k, v, row_b, row_t, window: int, dO, scale: float | None = None, heads=None):
    """Gradients of attn_fwd with the row set fixed.

    dO: [nrows, Hq, D].  Returns dq [nrows, Hq, D], dk, dv [B, T, Hkv, D]
    (float64).  dk/dv sum over the listed query heads of each group."""
    q, k, v = _f32(q), _f32(k), _f32(v)
    B, T, Hq, D = q.shape
    Hkv = k.shape[2]
    row_b, row_t = _rows(row_b, row_t)
    hs = _heads(heads, Hq)
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    n = row_b.size
    dO = _f32(dO).reshape(n, Hq, D) if n else np.zeros((0, Hq, D), np.float32)
    dq = np.zeros((n, Hq, D), dtype=np.float64)
    dk = np.zeros((B, T, Hkv, D), dtype=np.float64)
    dv = np.zeros((B, T, Hkv, D), dtype=np.float64)
    if n:
        _load().oracle_attn_bwd(q, k, v, B, T, Hq, Hkv, D, n, row_b, row_t, hs.size, hs,
                                int(window), scale, dO, dq, dk, dv)
    return dq, dk, dv


def local_rows(B: int, T: int):
    """Every token (b, t) in order: the local branch's query rows (Eq. 6)."""
    b = np.repeat(np.arange(B, dtype=np.int32), T)
    t = np.tile(np.arange(T, dtype=np.int32), B)
    return b, t


def global_rows(pos, cu_q):
    """Packed selected rows (App. B layout) as (row_b, row_t)."""
    cu_q = np.asarray(cu_q)
    B = cu_q.size - 1
    b = np.repeat(np.arange(B, dtype=np.int32), np.diff(cu_q))
    return b, _i32(pos)


# -------------------------------------------------------------------- combine
def _gain(g):
    if g is None:
        return None, None
    g = _f32(g)
    return g, g.ctypes.data_as(ctypes.c_void_p)


def combine_fwd(oL, oGc, p, z, row_of, gL=None, gG=None, eps: float = 1e-6):
    """Eq. 9 + Eq. 10.  Returns o [B,T,H,D], rstdL [B,T,H], rstdG [N,H] (float64)."""
    oL = _f32(oL)
    B, T, H, D = oL.shape
    n = int(np.asarray(z).sum())
    oGc = _f32(oGc).reshape(-1, H, D) if n else np.zeros((1, H, D), np.float32)
    gL_a, gL_p = _gain(gL)
    gG_a, gG_p = _gain(gG)
    o = np.zeros((B, T, H, D), dtype=np.float64)
    rL = np.zeros((B, T, H), dtype=np.float64)
    rG = np.zeros((max(n, 1), H), dtype=np.float64)
    _load().oracle_combine_fwd(oL, oGc, _f32(p), np.ascontiguousarray(z, dtype=np.uint8), _i32(row_of),
                               gL_p, gG_p, float(eps), B, T, H, D, o, rL, rG)
    return o, rL, rG[:n]


def combine_bwd(dO, oL, oGc, p, z, row_of, gL=None, gG=None, eps: float = 1e-6):
    """Backward of combine_fwd with z fixed: dOL [B,T,H,D], dOGc [N,H,D], dp [B,T]."""
    oL = _f32(oL)
    B, T, H, D = oL.shape
    n = int(np.asarray(z).sum())
    oGc = _f32(oGc).reshape(-1, H, D) if n else np.zeros((1, H, D), np.float32)
    gL_a, gL_p = _gain(gL)
    gG_a, gG_p = _gain(gG)
    dOL = np.zeros((B, T, H, D), dtype=np.float64)
    dOG = np.zeros((max(n, 1), H, D), dtype=np.float64)
    dp = np.zeros((B, T), dtype=np.float64)
    _load().oracle_combine_bwd(_f32(dO), oL, oGc, _f32(p), np.ascontiguousarray(z, dtype=np.uint8),
                               _i32(row_of), gL_p, gG_p, float(eps), B, T, H, D, dOL, dOG, dp)
    return dOL, dOG[:n], dp


def combine_dgain(dO, oL, oGc, p, z, row_of, eps: float = 1e-6):
    """Gradients of the ContextNorm gains of Eq. 9 with z fixed: (dgL, dgG),
    each [H, D] float64 (the gains' own values do not enter: o~ is linear in
    them)."""
    oL = _f32(oL)
    B, T, H, D = oL.shape
    n = int(np.asarray(z).sum())
    oGc = _f32(oGc).reshape(-1, H, D) if n else np.zeros((1, H, D), np.float32)
    dgL = np.zeros((H, D), dtype=np.float64)
    dgG = np.zeros((H, D), dtype=np.float64)
    _load().oracle_combine_dgain(_f32(dO), oL, oGc, _f32(p), np.ascontiguousarray(z, dtype=np.uint8),
                                 _i32(row_of), float(eps), B, T, H, D, dgL, dgG)
    return dgL, dgG


def gate(x, w):
    """Eq. 7: p = sigmoid(x . w_g) per token.  x [..., dm], w [dm]; returns p
    [...] float64."""
    x = _f32(x)
    dm = x.shape[-1]
    n = x.size // dm if dm else 0
    p = np.zeros(n, dtype=np.float64)
    if n:
        _load().oracle_gate(x.reshape(n, dm), _f32(w).reshape(dm), n, dm, p)
    return p.reshape(x.shape[:-1])


def gate_bwd(x, w, dp):
    """Backward of gate for the given dp: (dx [..., dm], dw [dm]) float64."""
    x = _f32(x)
    dm = x.shape[-1]
    n = x.size // dm
    dx = np.zeros((n, dm), dtype=np.float64)
    dw = np.zeros(dm, dtype=np.float64)
    if n:
        _load().oracle_gate_bwd(x.reshape(n, dm), _f32(w).reshape(dm), _f32(dp).reshape(n), n, dm, dx, dw)
    return dx.reshape(x.shape), dw


def _branch_rows(B, T, rows):
    if rows is None:
        return np.arange(B * T, dtype=np.int64)
    rb, rt = rows
    return (np.asarray(rb, dtype=np.int64) * T + np.asarray(rt, dtype=np.int64)).reshape(-1)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def branch_fwd(u, A=None, s=None, b=None, rows=None):
    """Eq. 5 on the rows (row_b, row_t) of u [B, T, H, D] (all rows if None):
    LP with A [H, D, D], else SO with s, b [H, D].  Returns [nrows, H, D] float64."""
    u = _f32(u)
    B, T, H, D = u.shape
    r = _branch_rows(B, T, rows)
    A = None if A is None else _f32(A)
    s = None if s is None else _f32(s)
    b = None if b is None else _f32(b)
    g = np.zeros((r.size, H, D), dtype=np.float64)
    if r.size:
        _load().oracle_branch_fwd(u, H, D, r, r.size, _ptr(A), _ptr(s), _ptr(b), g)
    return g


def branch_bwd(u, dg, A=None, s=None, rows=None):
    """Gradients of branch_fwd for dg [nrows, H, D]: (du [nrows, H, D], dA) for LP,
    (du, ds, db) for SO, float64."""
    u = _f32(u)
    B, T, H, D = u.shape
    r = _branch_rows(B, T, rows)
    dg = _f32(dg).reshape(r.size, H, D)
    du = np.zeros((r.size, H, D), dtype=np.float64)
    if A is not None:
        A = _f32(A)
        dA = np.zeros((H, D, D), dtype=np.float64)
        if r.size:
            _load().oracle_branch_bwd(u, H, D, r, r.size, _ptr(A), None, dg, du, _ptr(dA), None, None)
        return du, dA
    s = _f32(s)
    ds = np.zeros((H, D), dtype=np.float64)
    db = np.zeros((H, D), dtype=np.float64)
    if r.size:
        _load().oracle_branch_bwd(u, H, D, r, r.size, None, _ptr(s), dg, du, None, _ptr(ds), _ptr(db))
    return du, ds, db
