"""Failure detection on the GPU without a fault.

Every device-side wait of the library's kernels is bounded: when a wait runs
out it sets the timeout bit of a device status word and the kernel returns, so
the CUDA context stays usable and the host learns of it through
bcmt_device_status().  Here a test-only kernel waits on an mbarrier that
nothing arrives at, with the bound cut to a few milliseconds, and the test
checks the status the host reads, that reading it clears it, and that the
layer runs normally afterwards.  No TMA copy, tcgen05 operation or TMEM is
involved, and nothing faults or hangs.
"""

import pytest
import torch

from paper_2608_13578_gb300.inputs import make_inputs
from tests.helpers import gpu_run, to_device
from tests.test_gpu_parity import W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def C(cuda_ok):
    from paper_2608_13578_gb300 import bcmt
    return bcmt


def test_expired_wait_reports_timeout_and_clears(C):
    s = torch.cuda.current_stream()
    C.bcmt_device_status(s)  # clean start (and clears anything left over)
    C.bcmt_test_wait_expiry(1 << 24, s)  # about 8 ms of SM clock
    with pytest.raises(C.BCMTError) as e:
        C.bcmt_device_status(s)
    assert e.value.code == C.BCMT_ERR_TIMEOUT
    assert "bounded" in C.bcmt_last_error()
    # reading the status cleared it
    C.bcmt_device_status(s)


def test_layer_runs_normally_after_an_expired_wait(C):
    w = W(2, 256, 128, 2, 64, "bf16")
    t = to_device(make_inputs(w))
    y0, g0 = gpu_run(w, t)  # BCMT_FLAG_CHECK: each call reads the status word
    s = torch.cuda.current_stream()
    C.bcmt_test_wait_expiry(1 << 20, s)
    with pytest.raises(C.BCMTError) as e:
        C.bcmt_device_status(s)
    assert e.value.code == C.BCMT_ERR_TIMEOUT
    y1, g1 = gpu_run(w, t)
    assert torch.equal(y0, y1)
    for n in g0:
        assert torch.equal(g0[n], g1[n]), n


def test_wait_expiry_rejects_bad_bounds(C):
    for cycles in (0, -5, (1 << 31) + 1):
        with pytest.raises(C.BCMTError):
            C.bcmt_test_wait_expiry(cycles)
