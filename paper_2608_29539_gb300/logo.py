"""Thin Python binding of the LoGo C ABI (``include/logo.h``).

Argument marshalling only: every function here checks dtypes/shapes, allocates
missing outputs and workspaces through torch (device memory is torch's job),
and calls the entry point of the same name in ``_lib/liblogo.so`` on the
current CUDA stream.  All computation runs in the library's CUDA kernels;
there is no CPU path.  If the library has not been built, every call raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

_c_int = ctypes.c_int
_c_float = ctypes.c_float
_c_size = ctypes.c_size_t
_vp = ctypes.c_void_p

LOGO_OK = 0
LOGO_ERR_INVALID_ARG = -1
LOGO_ERR_UNSUPPORTED = -2
LOGO_ERR_CUDA = -3
LOGO_ERR_TIMEOUT = -4
LOGO_ERR_WORKSPACE = -5
LOGO_ERR_SCRATCH_LIMIT = -6
LOGO_SELECT_THRESHOLD = 0
LOGO_SELECT_RATIO = 1

_ERR_NAMES = {
    LOGO_ERR_INVALID_ARG: "LOGO_ERR_INVALID_ARG",
    LOGO_ERR_UNSUPPORTED: "LOGO_ERR_UNSUPPORTED",
    LOGO_ERR_CUDA: "LOGO_ERR_CUDA",
    LOGO_ERR_TIMEOUT: "LOGO_ERR_TIMEOUT",
    LOGO_ERR_WORKSPACE: "LOGO_ERR_WORKSPACE",
    LOGO_ERR_SCRATCH_LIMIT: "LOGO_ERR_SCRATCH_LIMIT",
}


class LogoError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} returned {_ERR_NAMES.get(code, code)}")
        self.code = code


class Dims(ctypes.Structure):
    _fields_ = [("B", _c_int), ("T", _c_int), ("Hq", _c_int), ("Hkv", _c_int), ("D", _c_int)]


_lib = None

_SIGS = {
    "logo_get_device_status": (_c_int, [ctypes.POINTER(_c_int)]),
    "logo_num_sms": (_c_int, []),
    "logo_selftest_wait_expiry": (_c_int, [ctypes.c_uint64, _vp]),
    "logo_select_workspace_size": (_c_size, [Dims]),
    "logo_select": (_c_int, [_vp, Dims, _c_int, _c_float, _c_float, _vp, _vp, _vp, _vp, _vp, _vp, _c_size, _vp]),
    "logo_gate_select": (_c_int, [_vp, _vp, _c_int, Dims, _c_int, _c_float, _c_float, _vp, _vp, _vp, _vp, _vp, _vp,
                                  _vp, _c_size, _vp]),
    "logo_gate_bwd_workspace_size": (_c_size, [Dims, _c_int]),
    "logo_branch_transform": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, Dims, _vp]),
    "logo_branch_transform_bwd_workspace_size": (_c_size, [Dims]),
    "logo_branch_transform_bwd": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _c_int, _vp, _vp, _vp, Dims, _vp,
                                           _c_size, _vp]),
    "logo_gate_bwd": (_c_int, [_vp, _vp, _vp, _vp, _c_int, Dims, _vp, _c_int, _vp, _vp, _c_size, _vp]),
    "logo_select_noalloc": (_c_int, [_vp, Dims, _c_int, _c_float, _c_float, _vp, _vp, _vp, _vp, _vp, _vp]),
    "logo_select_device_threshold": (_c_int, [_vp, Dims, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _c_size, _vp]),
    "logo_budget_update": (_c_int, [_vp, Dims, _c_float, _c_float, _vp, _vp, _vp]),
    "logo_pmask_initial_threshold": (_c_float, [_c_float, ctypes.c_longlong]),
    "logo_decode_workspace_size": (_c_size, [Dims]),
    "logo_decode_local_attn": (_c_int, [_vp, _vp, _vp, _vp, _vp, Dims, _c_int, _c_float, _vp, _c_size, _vp]),
    "logo_decode_global_sparse_attn": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, Dims, _c_float, _vp, _c_size,
                                                _vp]),
    "logo_local_attn_fwd": (_c_int, [_vp, _vp, _vp, _vp, _vp, Dims, _c_int, _c_float, _vp]),
    "logo_local_attn_bwd_workspace_size": (_c_size, [Dims]),
    "logo_local_attn_bwd": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, Dims, _c_int, _c_float, _vp,
                                     _c_size, _vp]),
    "logo_global_attn_fwd_workspace_size": (_c_size, [Dims]),
    "logo_global_sparse_attn_fwd": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, Dims, _c_float, _vp, _c_size,
                                             _vp]),
    "logo_global_attn_bwd_workspace_size": (_c_size, [Dims]),
    "logo_global_sparse_attn_bwd": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, Dims,
                                             _c_float, _vp, _c_size, _vp]),
    "logo_combine": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _c_float, _vp, _vp, _vp, Dims, _vp]),
    "logo_combine_bwd": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _c_float, _vp, _vp, _vp, Dims, _vp]),
    "logo_combine_bwd_workspace_size": (_c_size, [Dims]),
    "logo_combine_bwd_gains": (_c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _c_float, _vp, _vp, _vp, _vp, _vp,
                                        Dims, _vp, _c_size, _vp]),
}


def library_path() -> str:
    return _build.LIB


def lib():
    """Load liblogo.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        path = _build.LIB
        if not os.path.exists(path):
            raise RuntimeError(f"LoGo CUDA library not built ({path}); run python -m paper_2608_29539_gb300.build")
        L = ctypes.CDLL(path)
        for name, (res, args) in _SIGS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _p(t):
    return None if t is None else _vp(t.data_ptr())


def _stream():
    return _vp(torch.cuda.current_stream().cuda_stream)


def _call(name, *args):
    rc = getattr(lib(), name)(*args)
    if rc != LOGO_OK:
        raise LogoError(name, rc)


def _need(t, dtype, name, shape=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t


def dims_of(q: torch.Tensor, k: torch.Tensor) -> Dims:
    B, T, Hq, D = q.shape
    return Dims(B, T, Hq, k.shape[2], D)


def _workspace(nbytes: int, device, ws=None):
    if ws is not None:
        if ws.numel() * ws.element_size() < nbytes:
            raise ValueError("workspace too small")
        return ws
    return torch.empty(max(int(nbytes), 16), dtype=torch.uint8, device=device)


def workspace_bytes(kind: str, dims: Dims) -> int:
    fn = {"select": "logo_select_workspace_size", "local_bwd": "logo_local_attn_bwd_workspace_size",
          "global_fwd": "logo_global_attn_fwd_workspace_size",
          "global_bwd": "logo_global_attn_bwd_workspace_size",
          "combine_bwd_gains": "logo_combine_bwd_workspace_size"}[kind]
    return int(getattr(lib(), fn)(dims))


# ----------------------------------------------------------------------- API
def logo_get_device_status() -> int:
    st = _c_int(0)
    _call("logo_get_device_status", ctypes.byref(st))
    return st.value


def logo_num_sms() -> int:
    return int(lib().logo_num_sms())


def logo_selftest_wait_expiry(budget_ns: int) -> None:
    """Launch one warp whose bounded mbarrier wait can never complete; after
    budget_ns it records LOGO_ERR_TIMEOUT (read it with logo_get_device_status)."""
    _call("logo_selftest_wait_expiry", int(budget_ns), _stream())


def logo_select(gate_p, mode: int, b_th: float = 0.5, ratio: float = 0.0, z=None, pos=None, cu_q=None,
                row_of=None, n_sel_total=None, workspace=None):
    """Eq. 7 routing and packing of I.  Returns (z, pos, cu_q, row_of, n_sel_total)."""
    _need(gate_p, torch.float32, "gate_p")
    B, T = gate_p.shape
    dev = gate_p.device
    dims = Dims(B, T, 1, 1, 64)
    z = z if z is not None else torch.empty((B, T), dtype=torch.uint8, device=dev)
    pos = pos if pos is not None else torch.empty((B * T,), dtype=torch.int32, device=dev)
    cu_q = cu_q if cu_q is not None else torch.empty((B + 1,), dtype=torch.int32, device=dev)
    row_of = row_of if row_of is not None else torch.empty((B, T), dtype=torch.int32, device=dev)
    n_sel_total = n_sel_total if n_sel_total is not None else torch.empty((1,), dtype=torch.int32, device=dev)
    nbytes = workspace_bytes("select", dims)
    ws = _workspace(nbytes, dev, workspace)
    _call("logo_select", _p(gate_p), dims, int(mode), float(b_th), float(ratio), _p(z), _p(pos), _p(cu_q),
          _p(row_of), _p(n_sel_total), _p(ws), nbytes, _stream())
    return z, pos, cu_q, row_of, n_sel_total


def logo_gate_select(x, w_g, mode: int, b_th: float = 0.5, ratio: float = 0.0, gate_p=None, z=None, pos=None,
                     cu_q=None, row_of=None, n_sel_total=None, workspace=None):
    """Eq. 7 gate p = sigmoid(x . w_g) (x [B, T, d_model] bf16, w_g [d_model]
    float32) followed by the routing of logo_select.  Returns
    (gate_p, z, pos, cu_q, row_of, n_sel_total)."""
    _need(x, torch.bfloat16, "x")
    _need(w_g, torch.float32, "w_g")
    B, T, dm = x.shape
    dev = x.device
    dims = Dims(B, T, 1, 1, 64)
    gate_p = gate_p if gate_p is not None else torch.empty((B, T), dtype=torch.float32, device=dev)
    z = z if z is not None else torch.empty((B, T), dtype=torch.uint8, device=dev)
    pos = pos if pos is not None else torch.empty((B * T,), dtype=torch.int32, device=dev)
    cu_q = cu_q if cu_q is not None else torch.empty((B + 1,), dtype=torch.int32, device=dev)
    row_of = row_of if row_of is not None else torch.empty((B, T), dtype=torch.int32, device=dev)
    n_sel_total = n_sel_total if n_sel_total is not None else torch.empty((1,), dtype=torch.int32, device=dev)
    nbytes = workspace_bytes("select", dims)
    ws = _workspace(nbytes, dev, workspace)
    _call("logo_gate_select", _p(x), _p(w_g), int(dm), dims, int(mode), float(b_th), float(ratio), _p(gate_p), _p(z),
          _p(pos), _p(cu_q), _p(row_of), _p(n_sel_total), _p(ws), nbytes, _stream())
    return gate_p, z, pos, cu_q, row_of, n_sel_total


def logo_gate_bwd(x, w_g, gate_p, dgate_p, dx=None, accumulate: bool = False, dw_g=None, want_dx: bool = True,
                  want_dw: bool = True, workspace=None):
    """Backward of the gate: dx = dlogit w_g (written, or added to dx when
    accumulate), dw_g = sum_t dlogit_t x_t with dlogit = dp p (1 - p).
    Returns (dx, dw_g) (None for a part not asked for)."""
    _need(x, torch.bfloat16, "x")
    B, T, dm = x.shape
    dev = x.device
    dims = Dims(B, T, 1, 1, 64)
    if want_dx and dx is None:
        if accumulate:
            raise ValueError("accumulate needs the dx to add to")
        dx = torch.empty_like(x)
    if not want_dx:
        dx = None
    dw_g = (dw_g if dw_g is not None else torch.empty((dm,), dtype=torch.float32, device=dev)) if want_dw else None
    nbytes = int(lib().logo_gate_bwd_workspace_size(dims, dm)) if want_dw else 0
    ws = _workspace(nbytes, dev, workspace) if want_dw else None
    _call("logo_gate_bwd", _p(x), _p(w_g), _p(gate_p), _p(dgate_p), int(dm), dims, _p(dx), int(bool(accumulate)),
          _p(dw_g), _p(ws), nbytes, _stream())
    return dx, dw_g


def _transform_rows(rows):
    if rows is None:
        return None, None, None
    pos, cu_q, n_sel_total = rows
    return pos, cu_q, n_sel_total


def logo_branch_transform(u_l, a=None, s=None, b=None, rows=None, u_g=None):
    """Eq. 5: U^G = U^L A (LP, a [H, D, D] bf16) or U^L * s + b (SO, s and b
    [H, D] float32), on every row, or on the packed selected rows when rows =
    (pos, cu_q, n_sel_total).  u_l [B, T, H, D] bf16.  Returns u_g."""
    _need(u_l, torch.bfloat16, "u_l")
    B, T, H, D = u_l.shape
    u_g = u_g if u_g is not None else torch.empty_like(u_l)
    pos, cu_q, n_sel = _transform_rows(rows)
    _call("logo_branch_transform", _p(u_l), _p(a), _p(s), _p(b), _p(pos), _p(cu_q), _p(n_sel), _p(u_g),
          Dims(B, T, H, H, D), _stream())
    return u_g


def logo_branch_transform_bwd(u_l, du_g, a=None, s=None, rows=None, du_l=None, accumulate: bool = False,
                              workspace=None):
    """Gradients of logo_branch_transform.  Returns (du_l, da) for LP and
    (du_l, ds, db) for SO."""
    _need(u_l, torch.bfloat16, "u_l")
    B, T, H, D = u_l.shape
    dev = u_l.device
    dims = Dims(B, T, H, H, D)
    if du_l is None:
        if accumulate:
            raise ValueError("accumulate needs the du_l to add to")
        du_l = torch.empty_like(u_l)
    da = torch.empty((H, D, D), dtype=torch.float32, device=dev) if a is not None else None
    ds = torch.empty((H, D), dtype=torch.float32, device=dev) if a is None else None
    db = torch.empty((H, D), dtype=torch.float32, device=dev) if a is None else None
    nbytes = int(lib().logo_branch_transform_bwd_workspace_size(dims))
    ws = _workspace(nbytes, dev, workspace)
    pos, cu_q, n_sel = _transform_rows(rows)
    _call("logo_branch_transform_bwd", _p(u_l), _p(a), _p(s), _p(pos), _p(cu_q), _p(n_sel), _p(du_g), _p(du_l),
          int(bool(accumulate)), _p(da), _p(ds), _p(db), dims, _p(ws), nbytes, _stream())
    return (du_l, da) if a is not None else (du_l, ds, db)


def logo_select_device_threshold(gate_p, b_th, z=None, pos=None, cu_q=None, row_of=None, n_sel_total=None,
                                 workspace=None):
    """Eq. 7 routing with the threshold read on the device from b_th (a
    one-element float32 CUDA tensor).  Returns (z, pos, cu_q, row_of, n_sel_total)."""
    _need(gate_p, torch.float32, "gate_p")
    _need(b_th, torch.float32, "b_th", (1,))
    B, T = gate_p.shape
    dev = gate_p.device
    dims = Dims(B, T, 1, 1, 64)
    z = z if z is not None else torch.empty((B, T), dtype=torch.uint8, device=dev)
    pos = pos if pos is not None else torch.empty((B * T,), dtype=torch.int32, device=dev)
    cu_q = cu_q if cu_q is not None else torch.empty((B + 1,), dtype=torch.int32, device=dev)
    row_of = row_of if row_of is not None else torch.empty((B, T), dtype=torch.int32, device=dev)
    n_sel_total = n_sel_total if n_sel_total is not None else torch.empty((1,), dtype=torch.int32, device=dev)
    nbytes = workspace_bytes("select", dims)
    ws = _workspace(nbytes, dev, workspace)
    _call("logo_select_device_threshold", _p(gate_p), dims, _p(b_th), _p(z), _p(pos), _p(cu_q), _p(row_of),
          _p(n_sel_total), _p(ws), nbytes, _stream())
    return z, pos, cu_q, row_of, n_sel_total


def logo_budget_update(n_sel_total, B: int, T: int, rho: float, gamma: float, b_th, f_out=None):
    """Eq. 3 + Eq. 11 on the device: b_th (one-element float32 CUDA tensor) is
    moved by gamma * sign(N / (B*T) - rho) in place; f_out (optional, same
    kind) receives F.  Returns b_th."""
    _need(n_sel_total, torch.int32, "n_sel_total", (1,))
    _need(b_th, torch.float32, "b_th", (1,))
    if f_out is not None:
        _need(f_out, torch.float32, "f_out", (1,))
    _call("logo_budget_update", _p(n_sel_total), Dims(int(B), int(T), 1, 1, 64), float(rho), float(gamma),
          _p(b_th), _p(f_out), _stream())
    return b_th


def logo_pmask_initial_threshold(gamma: float, pmask_steps: int) -> float:
    """P-mask start value 0.5 - gamma * steps (Sec. 3.2, App. C.1); host only."""
    return float(lib().logo_pmask_initial_threshold(float(gamma), int(pmask_steps)))


def _decode_dims(q, k):
    B, Hq, D = q.shape
    return Dims(B, k.shape[1], Hq, k.shape[2], D)


def logo_decode_local_attn(q, k_ring, v_ring, seq_len, window: int, scale: float = 0.0, o=None, workspace=None):
    """One decoding step of the local branch (Eq. 6) from ring caches
    [B, R, Hkv, D] (position s in slot s mod R).  q [B, Hq, D]; seq_len [B]
    int32 (cache length, the new token included).  Returns o [B, Hq, D]."""
    _need(q, torch.bfloat16, "q")
    _need(k_ring, torch.bfloat16, "k_ring")
    _need(v_ring, torch.bfloat16, "v_ring", k_ring.shape)
    _need(seq_len, torch.int32, "seq_len", (q.shape[0],))
    dims = _decode_dims(q, k_ring)
    o = o if o is not None else torch.empty_like(q)
    nbytes = int(lib().logo_decode_workspace_size(dims))
    ws = _workspace(nbytes, q.device, workspace)
    _call("logo_decode_local_attn", _p(q), _p(k_ring), _p(v_ring), _p(seq_len), _p(o), dims, int(window),
          float(scale), _p(ws), nbytes, _stream())
    return o


def logo_decode_global_sparse_attn(q, k_cache, v_cache, seq_len, cu_q, n_sel_total, scale: float = 0.0, o_c=None,
                                   workspace=None):
    """One decoding step of the global branch (Eq. 8) for the selected
    sequences only (packed rows of a (B, 1) selection), from dense caches
    [B, L, Hkv, D].  Returns o_c [B, Hq, D] (packed rows; rows >= n_sel untouched)."""
    _need(q, torch.bfloat16, "q")
    _need(k_cache, torch.bfloat16, "k_cache")
    _need(v_cache, torch.bfloat16, "v_cache", k_cache.shape)
    _need(seq_len, torch.int32, "seq_len", (q.shape[0],))
    _need(cu_q, torch.int32, "cu_q", (q.shape[0] + 1,))
    _need(n_sel_total, torch.int32, "n_sel_total", (1,))
    dims = _decode_dims(q, k_cache)
    o_c = o_c if o_c is not None else torch.empty_like(q)
    nbytes = int(lib().logo_decode_workspace_size(dims))
    ws = _workspace(nbytes, q.device, workspace)
    _call("logo_decode_global_sparse_attn", _p(q), _p(k_cache), _p(v_cache), _p(seq_len), _p(cu_q),
          _p(n_sel_total), _p(o_c), dims, float(scale), _p(ws), nbytes, _stream())
    return o_c


def logo_select_noalloc(gate_p, mode: int, b_th: float = 0.5, ratio: float = 0.0, z=None, pos=None, cu_q=None,
                        row_of=None, n_sel_total=None):
    """logo_select without a workspace, for callers that cannot allocate
    scratch (its scratch is a static device array inside the library; see
    include/logo.h for the size limits).  The outputs must be given or are
    allocated here by torch.  Returns (z, pos, cu_q, row_of, n_sel_total)."""
    _need(gate_p, torch.float32, "gate_p")
    B, T = gate_p.shape
    dev = gate_p.device
    dims = Dims(B, T, 1, 1, 64)
    z = z if z is not None else torch.empty((B, T), dtype=torch.uint8, device=dev)
    pos = pos if pos is not None else torch.empty((B * T,), dtype=torch.int32, device=dev)
    cu_q = cu_q if cu_q is not None else torch.empty((B + 1,), dtype=torch.int32, device=dev)
    row_of = row_of if row_of is not None else torch.empty((B, T), dtype=torch.int32, device=dev)
    n_sel_total = n_sel_total if n_sel_total is not None else torch.empty((1,), dtype=torch.int32, device=dev)
    _call("logo_select_noalloc", _p(gate_p), dims, int(mode), float(b_th), float(ratio), _p(z), _p(pos), _p(cu_q),
          _p(row_of), _p(n_sel_total), _stream())
    return z, pos, cu_q, row_of, n_sel_total


def logo_local_attn_fwd(q, k, v, window: int, scale: float = 0.0, o=None, lse=None):
    """Eq. 6 local branch.  Returns (o [B,T,Hq,D] bf16, lse [B,Hq,T] fp32)."""
    for t, n in ((q, "q"), (k, "k"), (v, "v")):
        _need(t, torch.bfloat16, n)
    d = dims_of(q, k)
    o = o if o is not None else torch.empty_like(q)
    lse = lse if lse is not None else torch.empty((d.B, d.Hq, d.T), dtype=torch.float32, device=q.device)
    _call("logo_local_attn_fwd", _p(q), _p(k), _p(v), _p(o), _p(lse), d, int(window), float(scale), _stream())
    return o, lse


def logo_local_attn_bwd(q, k, v, o, lse, dO, window: int, scale: float = 0.0, dq=None, dk=None, dv=None,
                        workspace=None):
    """Gradients of the local branch.  Returns (dq, dk, dv)."""
    d = dims_of(q, k)
    for t, n in ((q, "q"), (k, "k"), (v, "v"), (o, "o"), (dO, "dO")):
        _need(t, torch.bfloat16, n)
    _need(lse, torch.float32, "lse", (d.B, d.Hq, d.T))
    dq = dq if dq is not None else torch.empty_like(q)
    dk = dk if dk is not None else torch.empty_like(k)
    dv = dv if dv is not None else torch.empty_like(v)
    nbytes = workspace_bytes("local_bwd", d)
    ws = _workspace(nbytes, q.device, workspace)
    _call("logo_local_attn_bwd", _p(q), _p(k), _p(v), _p(o), _p(lse), _p(dO), _p(dq), _p(dk), _p(dv), d,
          int(window), float(scale), _p(ws), nbytes, _stream())
    return dq, dk, dv


def logo_global_sparse_attn_fwd(q, k, v, pos, cu_q, n_sel_total, scale: float = 0.0, o_c=None, lse_c=None,
                                workspace=None):
    """Eq. 8 query-sparse global branch.  Returns (o_c [B*T,Hq,D], lse_c [Hq,B*T])."""
    for t, n in ((q, "q"), (k, "k"), (v, "v")):
        _need(t, torch.bfloat16, n)
    for t, n in ((pos, "pos"), (cu_q, "cu_q"), (n_sel_total, "n_sel_total")):
        _need(t, torch.int32, n)
    d = dims_of(q, k)
    cap = d.B * d.T
    o_c = o_c if o_c is not None else torch.empty((cap, d.Hq, d.D), dtype=torch.bfloat16, device=q.device)
    lse_c = lse_c if lse_c is not None else torch.empty((d.Hq, cap), dtype=torch.float32, device=q.device)
    nbytes = workspace_bytes("global_fwd", d)
    ws = _workspace(nbytes, q.device, workspace)
    _call("logo_global_sparse_attn_fwd", _p(q), _p(k), _p(v), _p(pos), _p(cu_q), _p(n_sel_total), _p(o_c),
          _p(lse_c), d, float(scale), _p(ws), nbytes, _stream())
    return o_c, lse_c


def logo_global_sparse_attn_bwd(q, k, v, pos, cu_q, n_sel_total, o_c, lse_c, dO_c, scale: float = 0.0, dq=None,
                                dk=None, dv=None, workspace=None):
    """Row-sparse gradients of the global branch.  Returns (dq dense, dk, dv)."""
    d = dims_of(q, k)
    for t, n in ((q, "q"), (k, "k"), (v, "v"), (o_c, "o_c"), (dO_c, "dO_c")):
        _need(t, torch.bfloat16, n)
    _need(lse_c, torch.float32, "lse_c")
    dq = dq if dq is not None else torch.empty_like(q)
    dk = dk if dk is not None else torch.empty_like(k)
    dv = dv if dv is not None else torch.empty_like(v)
    nbytes = workspace_bytes("global_bwd", d)
    ws = _workspace(nbytes, q.device, workspace)
    _call("logo_global_sparse_attn_bwd", _p(q), _p(k), _p(v), _p(pos), _p(cu_q), _p(n_sel_total), _p(o_c),
          _p(lse_c), _p(dO_c), _p(dq), _p(dk), _p(dv), d, float(scale), _p(ws), nbytes, _stream())
    return dq, dk, dv


def logo_combine(o_l, o_c, gate_p, z, row_of, gain_l=None, gain_g=None, eps: float = 1e-6, o=None, rstd_l=None,
                 rstd_g=None):
    """Eq. 9 ContextNorm + Eq. 10 fusion.  Returns (o, rstd_l, rstd_g)."""
    _need(o_l, torch.bfloat16, "o_l")
    _need(o_c, torch.bfloat16, "o_c")
    B, T, H, D = o_l.shape
    d = Dims(B, T, H, H, D)
    o = o if o is not None else torch.empty_like(o_l)
    rstd_l = rstd_l if rstd_l is not None else torch.empty((B, T, H), dtype=torch.float32, device=o_l.device)
    rstd_g = rstd_g if rstd_g is not None else torch.empty((B * T, H), dtype=torch.float32, device=o_l.device)
    _call("logo_combine", _p(o_l), _p(o_c), _p(gate_p), _p(z), _p(row_of), _p(gain_l), _p(gain_g), float(eps),
          _p(o), _p(rstd_l), _p(rstd_g), d, _stream())
    return o, rstd_l, rstd_g


def logo_combine_bwd(dO, o_l, o_c, gate_p, z, row_of, gain_l=None, gain_g=None, eps: float = 1e-6, dO_l=None,
                     dO_c=None, dgate_p=None):
    """Backward of logo_combine with z fixed.  Returns (dO_l, dO_c, dgate_p)."""
    _need(dO, torch.bfloat16, "dO")
    B, T, H, D = o_l.shape
    d = Dims(B, T, H, H, D)
    dO_l = dO_l if dO_l is not None else torch.empty_like(o_l)
    dO_c = dO_c if dO_c is not None else torch.empty((B * T, H, D), dtype=torch.bfloat16, device=o_l.device)
    dgate_p = dgate_p if dgate_p is not None else torch.empty((B, T), dtype=torch.float32, device=o_l.device)
    _call("logo_combine_bwd", _p(dO), _p(o_l), _p(o_c), _p(gate_p), _p(z), _p(row_of), _p(gain_l), _p(gain_g),
          float(eps), _p(dO_l), _p(dO_c), _p(dgate_p), d, _stream())
    return dO_l, dO_c, dgate_p


def logo_combine_bwd_gains(dO, o_l, o_c, gate_p, z, row_of, gain_l=None, gain_g=None, eps: float = 1e-6,
                           dO_l=None, dO_c=None, dgate_p=None, dgain_l=None, dgain_g=None, workspace=None):
    """logo_combine_bwd plus the ContextNorm gain gradients (Eq. 9).
    Returns (dO_l, dO_c, dgate_p, dgain_l, dgain_g); the gain gradients are
    [Hq, D] float32."""
    _need(dO, torch.bfloat16, "dO")
    B, T, H, D = o_l.shape
    d = Dims(B, T, H, H, D)
    dev = o_l.device
    dO_l = dO_l if dO_l is not None else torch.empty_like(o_l)
    dO_c = dO_c if dO_c is not None else torch.empty((B * T, H, D), dtype=torch.bfloat16, device=dev)
    dgate_p = dgate_p if dgate_p is not None else torch.empty((B, T), dtype=torch.float32, device=dev)
    dgain_l = dgain_l if dgain_l is not None else torch.empty((H, D), dtype=torch.float32, device=dev)
    dgain_g = dgain_g if dgain_g is not None else torch.empty((H, D), dtype=torch.float32, device=dev)
    nbytes = int(lib().logo_combine_bwd_workspace_size(d))
    ws = _workspace(nbytes, dev, workspace)
    _call("logo_combine_bwd_gains", _p(dO), _p(o_l), _p(o_c), _p(gate_p), _p(z), _p(row_of), _p(gain_l),
          _p(gain_g), float(eps), _p(dO_l), _p(dO_c), _p(dgate_p), _p(dgain_l), _p(dgain_g), d, _p(ws),
          ws.numel(), _stream())
    return dO_l, dO_c, dgate_p, dgain_l, dgain_g
