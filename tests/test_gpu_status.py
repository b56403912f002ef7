"""The device failure path without a GPU fault: a bounded mbarrier wait for a
phase that nothing completes (a producer that never arrives) gives up after
its limit, reports ZSAA_ERR_TIMEOUT through the status word, and leaves the
context usable -- the next GEMM still matches its float64 reference."""

import time

import pytest
import torch

from tests.helpers import check_linear, linear_case, need_gpu

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout_and_context_survives(zlib):
    need_gpu()
    z = zlib
    z.zsaa_device_status()  # nothing pending
    t0 = time.perf_counter()
    st = z.zsaa_selftest_wait_timeout()
    dt = time.perf_counter() - t0
    assert st == z.ZSAA_ERR_TIMEOUT, (st, z.zsaa_last_error())
    assert "bounded wait" in z.zsaa_last_error()
    assert 1.5 < dt < 60.0, dt  # the 2 s limit, not an endless spin
    z.zsaa_device_status()  # the report cleared the word
    out, ref, tol = linear_case(z, "store", 300, 1040, 1024, 77)
    check_linear(out, ref, tol, "store", "GEMM after the timeout")
    torch.cuda.synchronize()
