"""logo_select_noalloc: the selection entry point for callers that cannot
allocate (a runtime whose device memory is fixed at start-up, or a host that
reaches the library through a plain C FFI with no device allocator).  It keeps
its scratch in a static device array inside the library, so it must give the
same results as logo_select, call after call, even though the array still
holds the previous call's data.

This file is collected last on purpose: it runs after every other test when
the suite runs, and also passes on its own in a fresh process."""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    from paper_2608_29539_gb300 import build, logo
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return logo


def _call_abi(logo, fn, p, mode, b_th, ratio, with_ws):
    """Call the C entry point directly through ctypes; returns host copies."""
    B, T = p.shape
    dev = p.device
    z = torch.full((B, T), 7, dtype=torch.uint8, device=dev)
    pos = torch.full((B * T,), -7, dtype=torch.int32, device=dev)
    cu_q = torch.full((B + 1,), -7, dtype=torch.int32, device=dev)
    row_of = torch.full((B, T), -7, dtype=torch.int32, device=dev)
    n = torch.full((1,), -7, dtype=torch.int32, device=dev)
    dims = logo.Dims(B, T, 1, 1, 64)
    L = logo.lib()
    vp = lambda t: ctypes.c_void_p(t.data_ptr())  # noqa: E731
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if with_ws:
        nbytes = L.logo_select_workspace_size(dims)
        ws = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=dev)
        rc = L.logo_select(vp(p), dims, mode, b_th, ratio, vp(z), vp(pos), vp(cu_q), vp(row_of), vp(n), vp(ws),
                           nbytes, stream)
    else:
        rc = L.logo_select_noalloc(vp(p), dims, mode, b_th, ratio, vp(z), vp(pos), vp(cu_q), vp(row_of), vp(n),
                                   stream)
    assert rc == logo.LOGO_OK, rc
    torch.cuda.synchronize()
    k = int(n.item())
    return z.cpu().numpy(), pos[:k].cpu().numpy(), cu_q.cpu().numpy(), row_of.cpu().numpy(), k


def _gates(B, T, seed, ties=False):
    g = torch.Generator().manual_seed(seed)
    if ties:
        return (torch.randint(0, 5, (B, T), generator=g).float() / 8.0).cuda()
    return torch.sigmoid(torch.randn((B, T), generator=g)).cuda()


@pytest.mark.parametrize("case", [
    # two calls in a row on the shared scratch: a large call then a small one,
    # then threshold mode after ratio mode
    [(3, 70000, 1, 0.0, 0.125, False), (2, 3000, 1, 0.0, 0.3, True)],
    [(1, 16384, 1, 0.0, 0.125, False), (4, 5000, 0, 0.55, 0.0, False)],
])
def test_noalloc_matches_select_on_consecutive_calls(lib, case):
    for i, (B, T, mode, b_th, ratio, ties) in enumerate(case):
        p = _gates(B, T, seed=100 + i, ties=ties)
        ref = _call_abi(lib, "select", p, mode, b_th, ratio, with_ws=True)
        got = _call_abi(lib, "noalloc", p, mode, b_th, ratio, with_ws=False)
        assert got[4] == ref[4]
        for a, b in zip(got[:4], ref[:4]):
            np.testing.assert_array_equal(a, b)  # integer outputs: bit-exact


def test_noalloc_rejects_shapes_beyond_its_scratch(lib):
    L = lib.lib()
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: rejected on the host
    too_many_tokens = lib.Dims(1, 16384 * 1024 + 1, 1, 1, 64)
    too_many_seqs = lib.Dims(4097, 8, 1, 1, 64)
    for d in (too_many_tokens, too_many_seqs):
        rc = L.logo_select_noalloc(fake, d, 1, 0.0, 0.5, fake, fake, fake, fake, fake, None)
        assert rc == lib.LOGO_ERR_SCRATCH_LIMIT
    assert lib.logo_get_device_status() == 0
