"""Failure detection on the GPU without a fault: the bounded wait that guards
every pipeline hand-off of the tensor-core GEMM gives up on a barrier that
nothing completes, reports CURVEFP_DEV_TIMEOUT through the device status
word, and returns, leaving the context usable (a GEMM right after it is
still correct)."""
import time

import numpy as np
import pytest

from paper_2608_10010_gb300 import inputs
from tests.gpu_util import new_status, status_bits, to_dev, torch_cuda

pytestmark = pytest.mark.gpu
TIMEOUT = 4


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


def test_completed_barrier_does_not_time_out(torch):
    import paper_2608_10010_gb300 as cfp

    st = new_status(torch)
    cfp.selftest_bounded_wait(True, 2_000_000, st)
    torch.cuda.synchronize()
    assert status_bits(st) == 0


@pytest.mark.parametrize("limit", [1, 2_000_000, 40_000_000])
def test_wait_that_nothing_completes_reports_timeout(torch, limit):
    """2e6 / 4e7 SM cycles: about 1 ms / 20 ms at 2 GHz; the wait parks in
    hardware for at most 0.1 ms per try, so it ends within a few ms of the
    limit."""
    import paper_2608_10010_gb300 as cfp

    st = new_status(torch)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    cfp.selftest_bounded_wait(False, limit, st)
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert status_bits(st) == TIMEOUT
    assert dt < 1.0, dt


def test_context_usable_after_timeout(torch):
    import paper_2608_10010_gb300 as cfp

    st = new_status(torch)
    cfp.selftest_bounded_wait(False, 2_000_000, st)
    x = to_dev(torch, inputs.outlier_channels((130, 256), 5))
    w = to_dev(torch, inputs.normal((200, 256), 6, 0.02))
    a, sa = cfp.quantize(x, "E4C3", 32, 0)
    b, sb = cfp.quantize(w, "E4C3", 32, 0)
    st2 = new_status(torch)
    c_tc = cfp.gemm(a, sa, b, sb, "E4C3", "E4C3", 32, "tensor", status=st2)
    c_ex = cfp.gemm(a, sa, b, sb, "E4C3", "E4C3", 32, "exact", status=st2)
    torch.cuda.synchronize()
    assert status_bits(st) == TIMEOUT and status_bits(st2) == 0
    # within 1e-5 of the exact kernel, normalised by the dequantized rows' norms
    na = cfp.dequantize(a, sa, "E4C3", 32).double().norm(dim=1).cpu().numpy()
    nb = cfp.dequantize(b, sb, "E4C3", 32).double().norm(dim=1).cpu().numpy()
    err = np.abs(c_tc.cpu().numpy().astype(np.float64) - c_ex.cpu().numpy()) / np.outer(na, nb)
    assert float(err.max()) <= 1e-5


def test_status_is_required(torch):
    import paper_2608_10010_gb300 as cfp

    with pytest.raises(cfp.CurveFPError):
        cfp.selftest_bounded_wait(False, 1000, None)
