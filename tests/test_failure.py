"""Failure detection without a GPU fault.

Every wait inside the kernels is bounded.  A wait that runs out records
GLIDE_ERR_DEVICE_TIMEOUT in the workspace and releases the CTA's other waiters;
the host reads it with glide_read_device_status.  The self-test kernel waits on
a barrier that nothing ever completes (short limit, no trap, no hang) and the
context must stay usable afterwards."""
import time

import numpy as np
import pytest
import torch

from paper_2402_02082_gb300 import binding as gb
from paper_2402_02082_gb300 import build

FAKE = 0x10000


@pytest.fixture(scope="module")
def L():
    build.build()
    return gb.lib()


def test_selftest_rejects_bad_arguments(L):
    # host-side checks only: nothing is launched
    assert L.glide_selftest_wait_timeout(None, 1000, None) == gb.GLIDE_ERR_INVALID
    assert L.glide_selftest_wait_timeout(FAKE + 4, 1000, None) == gb.GLIDE_ERR_INVALID
    assert L.glide_selftest_wait_timeout(FAKE, 0, None) == gb.GLIDE_ERR_INVALID
    assert L.glide_selftest_wait_timeout(FAKE, 3000000, None) == gb.GLIDE_ERR_INVALID


@pytest.mark.gpu
def test_bounded_wait_reports_timeout_and_context_survives(L):
    ws = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    assert gb.glide_selftest_wait_timeout(ws, 20000) == gb.GLIDE_OK      # 20 ms limit
    assert gb.glide_read_device_status(ws) == gb.GLIDE_ERR_DEVICE_TIMEOUT
    elapsed = time.perf_counter() - t0
    # the second waiter (10x the limit) was released by the abort flag
    assert elapsed < 0.15, elapsed
    assert gb.glide_read_device_status(ws) == gb.GLIDE_OK                # read clears it
    # the context is still usable: a normal call succeeds afterwards
    x = torch.arange(1000, dtype=torch.float32, device="cuda")
    assert float(x.sum().item()) == 499500.0
