"""GPU parity of the histogram accumulation layout (Eq. 5, App. A.1: equal
addresses merged with signed popcounts): its phase sums are bit-identical
to the oracle's wide per-phase accumulators and to the GPU's exact kernel,
through the C ABI (curvefp_gemm_phases_histogram)."""
import numpy as np
import pytest

import oracle
from paper_2608_10010_gb300 import inputs
from tests.gpu_util import new_status, status_bits, to_dev, torch_cuda

pytestmark = pytest.mark.gpu
FORMATS = ["E3C3", "E4C3", "E5C2"]
PAIRS = [(a, b) for a in FORMATS for b in FORMATS] + [("E4C3_R8_9", "E4C3_R8_9"), ("E4C3_R3_4", "E4C3_R3_4")]


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


@pytest.mark.parametrize("fa,fb", PAIRS)
def test_histogram_layout_phase_sums(torch, fa, fb):
    import paper_2608_10010_gb300 as cfp

    M, N, K, G = 40, 24, 512, 32
    a, sa, _ = oracle.quantize(inputs.outlier_channels((M, K), 13), fa, G, 0)
    b, sb, _ = oracle.quantize(inputs.heavy_tailed_grad((N, K), 14), fb, G, 0)
    args = [to_dev(torch, v) for v in (a, sa, b, sb)]
    st = new_status(torch)
    c, ps, pl = cfp.gemm_phases_histogram(*args, fa, fb, G, status=st)
    c2, ps2, pl2 = cfp.gemm_phases(*args, fa, fb, G)
    torch.cuda.synchronize()
    ref = oracle.gemm(a, sa, b, sb, fa, fb, G)
    assert status_bits(st) == 0
    assert np.array_equal(ps.cpu().numpy(), ref["S_raw"]) and np.array_equal(pl.cpu().numpy(), ref["lsb"])
    assert np.array_equal(ps.cpu().numpy(), ps2.cpu().numpy())
    assert np.array_equal(c.cpu().numpy().view(np.uint32), c2.cpu().numpy().view(np.uint32))


def test_histogram_counts_match_oracle_histogram(torch):
    """The phase sums of single outputs against the oracle's own histogram
    layout (counts n_{h,t} summed with their binary weights)."""
    import paper_2608_10010_gb300 as cfp

    K, G = 256, 32
    a, sa, _ = oracle.quantize(inputs.normal((3, K), 15), "E4C3", G, 0)
    b, sb, _ = oracle.quantize(inputs.normal((2, K), 16, 0.02), "E4C3", G, 0)
    _, ps, pl = cfp.gemm_phases_histogram(*[to_dev(torch, v) for v in (a, sa, b, sb)], "E4C3", "E4C3", G)
    torch.cuda.synchronize()
    S = oracle.int128_to_int(ps.cpu().numpy())
    for i in range(3):
        for j in range(2):
            lam = int(pl.cpu().numpy()[i, j])
            counts = oracle.histogram(a[i], sa[i], b[j], sb[j], "E4C3", "E4C3", G, lam, 160)
            for h in range(8):
                assert int(S[i, j, h]) == sum(int(counts[h, t]) << t for t in range(160))


def test_histogram_range_flag(torch):
    """An output whose scale spread leaves the int128 window is flagged
    (CURVEFP_DEV_RANGE) and its C is NaN, as in the exact kernel."""
    import paper_2608_10010_gb300 as cfp

    K, G = 64, 32
    a = np.full((1, K), 0x7F, np.uint8)
    s = np.array([[-128, 127]], np.int8)
    st = new_status(torch)
    c, _, _ = cfp.gemm_phases_histogram(*[to_dev(torch, v) for v in (a, s, a, s)], "E5C2", "E5C2", G, status=st)
    torch.cuda.synchronize()
    assert status_bits(st) & 2 and np.isnan(c.cpu().numpy()[0, 0])
