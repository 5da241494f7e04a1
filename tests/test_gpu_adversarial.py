"""Inputs built to break a tensor-core path that loses small products: FP32
output within 1e-5 of the oracle's fp64 phase combine (normalised by
||a_i|| ||b_j||) on

* aligned outlier rows: one element per row in a block of its own, every
  other block of the row 14-20 binades lower, all of B positive, so that
  nothing the small blocks contribute cancels (Sec. 3.2, Eq. 5: every
  nonzero product is routed into its phase sum, however small);
* rows with an all-zero block (scale 0, as the quantizer writes it) beside
  small-magnitude data: E5C2 gradients of size 1e-3 t_3 and E4C3 weights of
  size 0.02, the training GEMMs' operands;
* block scales spread over 30 binades along a row.

Codes are built (or quantized by the oracle) on the CPU; every tensor-core
algorithm and AUTO run on the same inputs."""
import numpy as np
import pytest

import oracle
from tests.gpu_util import new_status, normalised_error, status_bits, to_dev, torch_cuda

pytestmark = pytest.mark.gpu
TC_PAIRS = [("E3C3", "E3C3"), ("E4C3", "E4C3"), ("E5C2", "E4C3"), ("E4C3", "E5C2"), ("E5C2", "E5C2")]
TOL = 1e-5
FMT = {"E3C3": (3, 3), "E4C3": (4, 3), "E5C2": (5, 2)}


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


def gemm(torch, a, sa, b, sb, fa, fb, algo):
    import paper_2608_10010_gb300 as cfp

    st = new_status(torch)
    c = cfp.gemm(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fa, fb, 32, algo,
                 status=st)
    torch.cuda.synchronize()
    return c.cpu().numpy(), status_bits(st)


def check_all(torch, a, sa, b, sb, fa, fb, algos):
    ref = oracle.gemm(a, sa, b, sb, fa, fb, 32, phases=False)
    assert not ref["range"].any()
    na, nb = oracle.row_norms(a, sa, fa, 32), oracle.row_norms(b, sb, fb, 32)
    for algo in algos:
        c, st = gemm(torch, a, sa, b, sb, fa, fb, algo)
        assert st == 0, algo
        err = normalised_error(c, ref["C"], na, nb)
        assert err <= TOL, (algo, err)


def top_codes(rng, fmt, shape):
    """Positive codes of the two top binades of a format (the ranks a
    ceil-absmax block holds near its maximum)."""
    E, C = FMT[fmt]
    K, B = 1 << C, 1 << (E + C - 1)
    nmax = B - 1
    return (B + rng.integers(nmax - 2 * K + 1, nmax + 1, size=shape)).astype(np.uint8)


def outlier_rows(rng, fmt, M, K, s):
    """Each row: one top-binade element alone in its block (scale 0), every
    other block of top-binade elements at scale -s."""
    codes = top_codes(rng, fmt, (M, K))
    scales = np.full((M, K // 32), -s, np.int8)
    for i in range(M):
        blk = rng.integers(0, K // 32)
        pos = blk * 32 + rng.integers(0, 32)
        keep = codes[i, pos]
        codes[i, blk * 32:(blk + 1) * 32] = 0
        codes[i, pos] = keep
        scales[i, blk] = 0
    return codes, scales


@pytest.mark.parametrize("fa,fb", TC_PAIRS)
@pytest.mark.parametrize("K,s", [(4096, 14), (4096, 18), (4096, 20), (11008, 18)])
def test_aligned_outlier_rows(torch, fa, fb, K, s):
    rng = np.random.default_rng(K + s + 10 * len(fa + fb))
    a, sa = outlier_rows(rng, fa, 16, K, s)
    b = top_codes(rng, fb, (256, K))
    sb = np.zeros((256, K // 32), np.int8)
    check_all(torch, a, sa, b, sb, fa, fb, ["tensor", "tensor_narrow", "auto"])


@pytest.mark.parametrize("fa,fb", TC_PAIRS)
def test_aligned_outlier_weights(torch, fa, fb):
    """The same construction on the B (weight) side, A positive."""
    rng = np.random.default_rng(5 + len(fa + fb))
    K = 4096
    b, sb = outlier_rows(rng, fb, 136, K, 18)
    a = top_codes(rng, fa, (24, K))
    sa = np.zeros((24, K // 32), np.int8)
    check_all(torch, a, sa, b, sb, fa, fb, ["tensor", "tensor_narrow", "auto"])


def zero_block(x, rng):
    x = x.copy()
    for i in range(x.shape[0]):
        j = rng.integers(0, x.shape[1] // 32)
        x[i, j * 32:(j + 1) * 32] = 0
    return x


@pytest.mark.parametrize("M", [1, 8, 40, 130])
def test_zero_blocks_beside_small_gradients(torch, M):
    """E5C2 gradients 1e-3 t_3 with an all-zero block per row (the quantizer
    gives it scale 0, about 26 binades above the data's blocks) times E4C3
    weights, in both operand orders; and E4C3 weights with zero blocks."""
    rng = np.random.default_rng(M)
    K = 1024
    g = zero_block(1e-3 * rng.standard_t(3, size=(M, K)).astype(np.float32), rng)
    w = (0.02 * rng.standard_normal((264, K))).astype(np.float32)
    a, sa, _ = oracle.quantize(g, "E5C2", 32, 0)
    b, sb, _ = oracle.quantize(w, "E4C3", 32, 0)
    check_all(torch, a, sa, b, sb, "E5C2", "E4C3", ["tensor", "tensor_narrow", "auto"])
    wz = zero_block(w, rng)
    bz, sbz, _ = oracle.quantize(wz, "E4C3", 32, 0)
    x = rng.standard_normal((M, K)).astype(np.float32)
    ax, sax, _ = oracle.quantize(x, "E4C3", 32, 0)
    check_all(torch, ax, sax, bz, sbz, "E4C3", "E4C3", ["tensor", "tensor_narrow", "auto"])
    check_all(torch, bz[:8], sbz[:8], a, sa, "E4C3", "E5C2", ["tensor", "tensor_narrow", "auto"])


@pytest.mark.parametrize("fa,fb", TC_PAIRS)
def test_scale_spread_of_30_binades(torch, fa, fb):
    """Random codes (every byte) under block scales uniform in [-15, 15]
    ([-12, 12] for E5C2 x E5C2, whose 63 bins leave the oracle's exact int128
    window less room)."""
    rng = np.random.default_rng(77 + len(fa + fb))
    K = 2048
    a = rng.integers(0, 256, size=(40, K), dtype=np.uint8)
    b = rng.integers(0, 256, size=(200, K), dtype=np.uint8)
    if fa == "E3C3":
        a &= 0xBF
    if fb == "E3C3":
        b &= 0xBF
    sp = 12 if fa == fb == "E5C2" else 15
    sa = rng.integers(-sp, sp + 1, size=(40, K // 32)).astype(np.int8)
    sb = rng.integers(-sp, sp + 1, size=(200, K // 32)).astype(np.int8)
    check_all(torch, a, sa, b, sb, fa, fb, ["tensor", "tensor_narrow"])
