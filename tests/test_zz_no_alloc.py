"""The static quantizer's entry point that allocates nothing.

Some callers cannot allocate device memory: code where cudaMalloc is not
allowed or would stall other work (it can synchronize the device), code whose
device memory belongs to a host framework's own pool, and hosts that reserve a
fixed memory budget up front.  For them the library keeps the static
quantizer's scratch in a fixed device array of its own.  This file checks that
entry point against the workspace entry point on two calls in a row (the
array keeps the previous call's contents, so each call must clear what it
needs) and that oversize requests are rejected before any device work.  It is
collected last so that it also runs after every other GPU test."""
import ctypes

import numpy as np
import pytest

from paper_2608_10010_gb300 import inputs

UNSUPPORTED = 2


def test_oversize_is_rejected_on_the_host():
    """Row groups of 200,000 rows need more scratch than the array holds."""
    import paper_2608_10010_gb300 as cfp

    lib = cfp.load()
    dummy = ctypes.c_void_p(4096)
    assert lib.curvefp_quantize_static_noalloc(1, 32, 1, 1, dummy, 0, 200000, 64, dummy, dummy, None, None) == UNSUPPORTED
    # block groups need no scratch at all, tensor groups a few bytes: accepted sizes are not rejected
    assert lib.curvefp_quantize_static_workspace(200000, 64, 32, 0) == 0


@pytest.mark.gpu
@pytest.mark.parametrize("group", ["row", "tensor", "block"])
@pytest.mark.parametrize("fmt", ["E3C3", "E5C2"])
def test_matches_workspace_entry_point_twice(group, fmt):
    from tests.gpu_util import torch_cuda

    torch = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    rng = np.random.default_rng(21)
    x1 = torch.from_numpy((rng.standard_normal((300, 512)) * np.exp(rng.standard_normal((300, 512)) * 2)).astype(np.float32)).cuda()
    x2 = torch.from_numpy(inputs.normal((257, 256), 5, 0.02)).cuda()
    for x in (x1, x2):  # two calls in a row: the scratch is cleared by each call
        c0, s0 = cfp.quantize_static(x, fmt, 32, group, "mse")
        c1, s1 = cfp.quantize_static_noalloc(x, fmt, 32, group, "mse")
        torch.cuda.synchronize()
        assert torch.equal(c0, c1) and torch.equal(s0, s1)
