"""The bounded device waits, exercised without a fault: a warp waits on an
mbarrier that nothing arrives at (logo_selftest_wait_expiry).  The wait must
give up after its budget, the device status must read LOGO_ERR_TIMEOUT (then
LOGO_OK once read), and the context must stay usable: a normal call afterwards
matches the oracle."""
import time

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def test_bounded_wait_expires_and_reports_timeout():
    from paper_2608_29539_gb300 import logo as L
    torch.cuda.synchronize()
    assert L.logo_get_device_status() == L.LOGO_OK
    budget_ns = 50_000_000  # 50 ms
    t0 = time.perf_counter()
    L.logo_selftest_wait_expiry(budget_ns)
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert 0.045 <= dt < 1.5, dt  # it waited out its budget, and no longer
    assert L.logo_get_device_status() == L.LOGO_ERR_TIMEOUT
    assert L.logo_get_device_status() == L.LOGO_OK  # reading clears the word
    # the context is intact: a selection runs and is bit-exact
    g = torch.Generator().manual_seed(11)
    p = torch.rand(2, 300, generator=g)
    z, pos, cu_q, row_of, n = L.logo_select(p.cuda(), L.LOGO_SELECT_RATIO, 0.5, 0.25)
    torch.cuda.synchronize()
    zr = oracle.select_ratio(p.numpy(), oracle.k_from_ratio(0.25, 300))
    assert np.array_equal(z.cpu().numpy(), zr)
    assert L.logo_get_device_status() == L.LOGO_OK
