"""Failure detection without a GPU fault: bounded device waits report through the status word.

A self-test kernel waits on an mbarrier that nothing ever arrives at.  Its bounded wait must
give up after the requested limit, record PACE_ERR_TIMEOUT with the kernel's id in the
device status word, and leave the CUDA context usable for the next launch.
"""
import time

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pace():
    from paper_2608_27206_gb300 import build
    build.build()
    from paper_2608_27206_gb300 import pace as P
    P.pace_init(0)
    P.pace_device_status(clear=True)
    return P


def test_bounded_wait_reports_timeout_and_context_survives(pace):
    t0 = time.perf_counter()
    pace.pace_selftest_wait_timeout(20000)            # 20 ms
    code, where = pace.pace_device_status(clear=True)
    dt = time.perf_counter() - t0
    assert code == pace.PACE_ERR_TIMEOUT and where == 11
    assert 0.015 < dt < 5.0
    assert pace.pace_device_status(clear=True) == (0, 0)   # cleared
    E = torch.arange(32 * 8, dtype=torch.int16, device="cuda").view(32, 8)
    idx = torch.tensor([5, 1], dtype=torch.int32, device="cuda")
    out = pace.pace_gather(E, idx).cpu().numpy()            # the context still works
    np.testing.assert_array_equal(out, E.cpu().numpy()[[5, 1]])


def test_selftest_rejects_bad_limits(pace):
    with pytest.raises(pace.PaceError):
        pace.pace_selftest_wait_timeout(0)
    with pytest.raises(pace.PaceError):
        pace.pace_selftest_wait_timeout(2_000_000)
