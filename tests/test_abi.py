"""The C-ABI library builds, loads and exports every entry point that
include/logo.h declares; host-side argument checks reject bad calls before any
CUDA work.  CPU only: nothing here launches a kernel."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2608_29539_gb300 import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "logo.h")


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^LOGO_API\s+\w+\s+(logo_\w+)\s*\(", text, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_hot_path():
    syms = declared_symbols()
    for name in ("logo_select", "logo_local_attn_fwd", "logo_local_attn_bwd", "logo_global_sparse_attn_fwd",
                 "logo_global_sparse_attn_bwd", "logo_combine", "logo_combine_bwd", "logo_get_device_status"):
        assert name in syms


def test_every_declared_symbol_is_exported(lib):
    missing = [s for s in declared_symbols() if not hasattr(lib, s)]
    assert not missing, missing


def test_binding_covers_every_symbol():
    from paper_2608_29539_gb300 import logo
    assert set(declared_symbols()) == set(logo._SIGS)


def test_host_side_argument_checks(lib):
    from paper_2608_29539_gb300 import logo
    L = logo.lib()
    d = logo.Dims(1, 128, 2, 2, 128)
    null = None
    # null pointers
    assert L.logo_select(null, d, 0, 0.5, 0.0, null, null, null, null, null, null, 0, null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_local_attn_fwd(null, null, null, null, null, d, 64, 0.0, null) == logo.LOGO_ERR_INVALID_ARG
    # unsupported head dim / grouping, invalid sizes
    fake = ctypes.c_void_p(1 << 20)  # aligned, never dereferenced: rejected before use
    for bad in (logo.Dims(1, 128, 2, 2, 96), logo.Dims(1, 128, 3, 2, 128)):
        assert L.logo_local_attn_fwd(fake, fake, fake, fake, fake, bad, 64, 0.0, null) == logo.LOGO_ERR_UNSUPPORTED
    assert L.logo_local_attn_fwd(fake, fake, fake, fake, fake, logo.Dims(0, 128, 2, 2, 128), 64, 0.0,
                                 null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_local_attn_fwd(fake, fake, fake, fake, fake, d, 0, 0.0, null) == logo.LOGO_ERR_INVALID_ARG
    # misaligned pointers
    odd = ctypes.c_void_p((1 << 20) + 2)
    assert L.logo_local_attn_fwd(odd, fake, fake, fake, fake, d, 64, 0.0, null) == logo.LOGO_ERR_UNSUPPORTED
    # workspace too small
    assert L.logo_global_sparse_attn_fwd(fake, fake, fake, fake, fake, fake, fake, fake, d, 0.0, fake, 16,
                                         null) == logo.LOGO_ERR_WORKSPACE
    assert L.logo_select(fake, d, 0, 0.5, 0.0, fake, fake, fake, fake, fake, fake, 0, null) == logo.LOGO_ERR_WORKSPACE
    # bad mode / ratio
    ws = L.logo_select_workspace_size(d)
    assert L.logo_select(fake, d, 7, 0.5, 0.0, fake, fake, fake, fake, fake, fake, ws, null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_select(fake, d, 1, 0.5, 1.5, fake, fake, fake, fake, fake, fake, ws, null) == logo.LOGO_ERR_INVALID_ARG
    # combine: eps must be positive
    assert L.logo_combine(fake, fake, fake, fake, fake, null, null, ctypes.c_float(0.0), fake, null, null, d,
                          null) == logo.LOGO_ERR_INVALID_ARG


def test_budget_controller_host_checks(lib):
    from paper_2608_29539_gb300 import logo
    import oracle
    L = logo.lib()
    d = logo.Dims(2, 300, 1, 1, 64)
    null = None
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: rejected before use
    f = ctypes.c_float
    assert L.logo_budget_update(null, d, f(0.5), f(0.01), fake, null, null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_budget_update(fake, d, f(0.5), f(0.01), null, null, null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_budget_update(fake, d, f(1.5), f(0.01), fake, null, null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_budget_update(fake, d, f(0.5), f(-0.01), fake, null, null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_budget_update(fake, d, f(0.5), f(float("inf")), fake, null, null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_budget_update(fake, logo.Dims(0, 300, 1, 1, 64), f(0.5), f(0.01), fake, null,
                                null) == logo.LOGO_ERR_INVALID_ARG
    ws = L.logo_select_workspace_size(d)
    assert L.logo_select_device_threshold(fake, d, null, fake, fake, fake, fake, fake, fake, ws,
                                          null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_select_device_threshold(fake, d, fake, fake, fake, fake, fake, fake, fake, 16,
                                          null) == logo.LOGO_ERR_WORKSPACE
    # the P-mask start is a host function: against the oracle and App. C.1's value
    for gamma, steps in ((0.0005, 5000), (2.0 ** -11, 4096), (0.01, 0), (0.003, 1234)):
        got = logo.logo_pmask_initial_threshold(gamma, steps)
        assert got == float(np.float32(oracle.pmask_threshold(float(np.float32(gamma)), steps)))
    assert logo.logo_pmask_initial_threshold(0.0005, 5000) == -2.0


def test_decode_host_checks(lib):
    from paper_2608_29539_gb300 import logo
    L = logo.lib()
    d = logo.Dims(4, 2048, 8, 2, 128)
    null = None
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: rejected before use
    f = ctypes.c_float
    ws = L.logo_decode_workspace_size(d)
    assert ws >= 4 * 8 * 16 * 130 * 4
    assert L.logo_decode_workspace_size(logo.Dims(4, 2048, 64, 2, 128)) == 0  # group of 32 > 16
    assert L.logo_decode_local_attn(null, fake, fake, fake, fake, d, 1024, f(0.0), fake, ws,
                                    null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_decode_local_attn(fake, fake, fake, fake, fake, d, 0, f(0.0), fake, ws,
                                    null) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_decode_local_attn(fake, fake, fake, fake, fake, d, 1024, f(0.0), fake, 16,
                                    null) == logo.LOGO_ERR_WORKSPACE
    assert L.logo_decode_local_attn(fake, fake, fake, fake, fake, logo.Dims(4, 2048, 8, 2, 96), 1024, f(0.0), fake,
                                    ws, null) == logo.LOGO_ERR_UNSUPPORTED
    assert L.logo_decode_global_sparse_attn(fake, fake, fake, fake, null, fake, fake, d, f(0.0), fake, ws,
                                            null) == logo.LOGO_ERR_INVALID_ARG
    odd = ctypes.c_void_p((1 << 20) + 2)
    assert L.logo_decode_global_sparse_attn(odd, fake, fake, fake, fake, fake, fake, d, f(0.0), fake, ws,
                                            null) == logo.LOGO_ERR_UNSUPPORTED


def test_combine_gains_host_checks(lib):
    from paper_2608_29539_gb300 import logo
    L = logo.lib()
    d = logo.Dims(2, 300, 4, 4, 128)
    null = None
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: rejected before use
    f = ctypes.c_float
    ws = L.logo_combine_bwd_workspace_size(d)
    assert ws >= 2 * 4 * 128 * 4  # at least one block's two [H, D] partial sums
    assert L.logo_combine_bwd_workspace_size(logo.Dims(2, 300, 72, 72, 128)) == 0  # Hq*D > 8192
    args = lambda dgl, dgg, dims, w, wb: (fake, fake, fake, fake, fake, fake, null, null, f(1e-6), fake, fake,  # noqa: E731
                                          fake, dgl, dgg, dims, w, wb, null)
    assert L.logo_combine_bwd_gains(*args(null, null, d, fake, ws)) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_combine_bwd_gains(*args(fake, fake, d, null, ws)) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_combine_bwd_gains(*args(fake, fake, d, fake, 16)) == logo.LOGO_ERR_WORKSPACE
    assert L.logo_combine_bwd_gains(*args(fake, null, logo.Dims(2, 300, 72, 72, 128), fake,
                                          1 << 30)) == logo.LOGO_ERR_UNSUPPORTED
    assert L.logo_combine_bwd_gains(*args(fake, fake, logo.Dims(2, 300, 4, 4, 96), fake,
                                          ws)) == logo.LOGO_ERR_UNSUPPORTED
    # the plain combine calls reject Hq*D > 16384
    assert L.logo_combine(fake, fake, fake, fake, fake, null, null, f(1e-6), fake, null, null,
                          logo.Dims(1, 8, 130, 130, 128), null) == logo.LOGO_ERR_UNSUPPORTED


def test_gate_host_checks(lib):
    from paper_2608_29539_gb300 import logo
    L = logo.lib()
    d = logo.Dims(2, 300, 1, 1, 64)
    null = None
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: rejected before use
    odd = ctypes.c_void_p((1 << 20) + 2)
    f = ctypes.c_float
    ws = L.logo_select_workspace_size(d)
    sel = lambda x, w, dm, mode, ratio, wsz: L.logo_gate_select(x, w, dm, d, mode, f(0.5), f(ratio), fake, fake,  # noqa: E731
                                                                  fake, fake, fake, fake, fake, wsz, null)
    assert sel(fake, fake, 4096, 1, 0.125, ws - 1) == logo.LOGO_ERR_WORKSPACE
    for dm in (0, 4, 100, 8200):
        assert sel(fake, fake, dm, 1, 0.125, ws) == logo.LOGO_ERR_UNSUPPORTED
    assert sel(null, fake, 4096, 1, 0.125, ws) == logo.LOGO_ERR_INVALID_ARG
    assert sel(fake, fake, 4096, 3, 0.125, ws) == logo.LOGO_ERR_INVALID_ARG
    assert sel(fake, fake, 4096, 1, 1.5, ws) == logo.LOGO_ERR_INVALID_ARG
    assert sel(odd, fake, 4096, 1, 0.125, ws) == logo.LOGO_ERR_UNSUPPORTED
    wb = L.logo_gate_bwd_workspace_size(d, 4096)
    assert wb >= 4096 * 4 and L.logo_gate_bwd_workspace_size(d, 8200) == 0
    bwd = lambda dx, acc, dw, w, wsz: L.logo_gate_bwd(fake, fake, fake, fake, 4096, d, dx, acc, dw, w, wsz,  # noqa: E731
                                                     null)
    assert bwd(null, 0, null, fake, wb) == logo.LOGO_ERR_INVALID_ARG
    assert bwd(fake, 2, fake, fake, wb) == logo.LOGO_ERR_INVALID_ARG
    assert bwd(fake, 0, fake, null, wb) == logo.LOGO_ERR_WORKSPACE
    assert bwd(fake, 0, fake, fake, wb - 4) == logo.LOGO_ERR_WORKSPACE
    assert bwd(odd, 0, null, null, 0) == logo.LOGO_ERR_UNSUPPORTED


def test_branch_transform_host_checks(lib):
    from paper_2608_29539_gb300 import logo
    L = logo.lib()
    d = logo.Dims(2, 300, 4, 4, 128)
    null = None
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: rejected before use
    odd = ctypes.c_void_p((1 << 20) + 2)
    fwd = lambda u, a, s_, b, pos, cu, n, out, dims: L.logo_branch_transform(u, a, s_, b, pos, cu, n, out, dims,  # noqa: E731
                                                                              null)
    assert fwd(fake, null, null, null, null, null, null, fake, d) == logo.LOGO_ERR_INVALID_ARG       # no form
    assert fwd(fake, fake, fake, fake, null, null, null, fake, d) == logo.LOGO_ERR_INVALID_ARG       # both forms
    assert fwd(fake, null, fake, null, null, null, null, fake, d) == logo.LOGO_ERR_INVALID_ARG       # SO without b
    assert fwd(fake, fake, null, null, fake, null, fake, fake, d) == logo.LOGO_ERR_INVALID_ARG       # rows without cu_q
    assert fwd(fake, fake, null, null, null, null, null, fake, logo.Dims(2, 300, 4, 4, 96)) == logo.LOGO_ERR_UNSUPPORTED
    assert fwd(fake, fake, null, null, null, null, null, fake, logo.Dims(2, 300, 72, 72, 128)) == logo.LOGO_ERR_UNSUPPORTED
    assert fwd(odd, fake, null, null, null, null, null, fake, d) == logo.LOGO_ERR_UNSUPPORTED
    ws = L.logo_branch_transform_bwd_workspace_size(d)
    assert ws >= 4 * 128 * 128 * 4
    bwd = lambda a, s_, acc, da, w, wb: L.logo_branch_transform_bwd(fake, a, s_, null, null, null, fake, fake, acc,  # noqa: E731
                                                                    da, null, null, d, w, wb, null)
    assert bwd(fake, fake, 0, fake, fake, ws) == logo.LOGO_ERR_INVALID_ARG   # both forms
    assert bwd(fake, null, 0, null, fake, ws) == logo.LOGO_ERR_INVALID_ARG   # LP without da
    assert bwd(fake, null, 3, fake, fake, ws) == logo.LOGO_ERR_INVALID_ARG   # accumulate flag
    assert bwd(fake, null, 0, fake, fake, ws - 4) == logo.LOGO_ERR_WORKSPACE
    assert bwd(fake, null, 0, fake, null, ws) == logo.LOGO_ERR_WORKSPACE


def test_workspace_sizes_grow_with_shape(lib):
    from paper_2608_29539_gb300 import logo
    L = logo.lib()
    small, big = logo.Dims(1, 1024, 4, 4, 128), logo.Dims(2, 4096, 16, 16, 128)
    for fn in ("logo_select_workspace_size", "logo_local_attn_bwd_workspace_size",
               "logo_global_attn_fwd_workspace_size", "logo_global_attn_bwd_workspace_size"):
        a, b = getattr(L, fn)(small), getattr(L, fn)(big)
        assert 0 < a <= b, fn
        if fn != "logo_select_workspace_size":
            assert a < b, fn
    assert L.logo_global_attn_fwd_workspace_size(logo.Dims(1, 128, 2, 2, 96)) == 0


def test_wait_expiry_selftest_host_checks(lib):
    from paper_2608_29539_gb300 import logo
    L = lib
    L.logo_selftest_wait_expiry.restype = ctypes.c_int
    L.logo_selftest_wait_expiry.argtypes = [ctypes.c_uint64, ctypes.c_void_p]
    assert L.logo_selftest_wait_expiry(0, None) == logo.LOGO_ERR_INVALID_ARG
    assert L.logo_selftest_wait_expiry(2_000_000_001, None) == logo.LOGO_ERR_INVALID_ARG
