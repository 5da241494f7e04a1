"""TENSOR_NARROW (phases along the MMA's N dimension, weight rows as the
128-row operand): FP32 output within 1e-5 of the oracle's fp64 phase combine,
normalised by ||a_i|| ||b_j|| of the dequantized operands, for every format
pair of the tensor path; ragged weight tiles, several token groups, split-K
pieces (every tile split when the tiles do not fill the SMs) and their
order-independent sum (two runs bit-identical)."""
import numpy as np
import pytest

import oracle
from paper_2608_10010_gb300 import inputs
from tests.gpu_util import new_status, normalised_error, status_bits, to_dev, torch_cuda

pytestmark = pytest.mark.gpu
TC_PAIRS = [("E3C3", "E3C3"), ("E4C3", "E4C3"), ("E5C2", "E4C3"), ("E4C3", "E5C2"), ("E5C2", "E5C2")]
TOL = 1e-5


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


def rand_operand(rng, fmt, rows, K, block, spread=4):
    """Every code byte (zero codes, both signs, all ranks) under random block scales."""
    codes = rng.integers(0, 256, size=(rows, K), dtype=np.uint8)
    if fmt == "E3C3":
        codes &= 0xBF
    scales = rng.integers(-spread, spread + 1, size=(rows, K // block)).astype(np.int8)
    return codes, scales


def run(torch, a, sa, b, sb, fa, fb, G, algo="tensor_narrow"):
    import paper_2608_10010_gb300 as cfp

    st = new_status(torch)
    c = cfp.gemm(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fa, fb, G, algo,
                 status=st)
    torch.cuda.synchronize()
    return c.cpu().numpy(), status_bits(st)


def check(torch, a, sa, b, sb, fa, fb, G):
    c, st = run(torch, a, sa, b, sb, fa, fb, G)
    assert st == 0
    ref = oracle.gemm(a, sa, b, sb, fa, fb, G, phases=False)
    na, nb = oracle.row_norms(a, sa, fa, G), oracle.row_norms(b, sb, fb, G)
    assert normalised_error(c, ref["C"], na, nb) <= TOL
    return c


@pytest.mark.parametrize("fa,fb", TC_PAIRS)
@pytest.mark.parametrize("M", [1, 8, 13, 40])
def test_random_codes_within_tolerance(torch, fa, fb, M):
    """N = 300: two whole weight tiles and a ragged one (44 rows); K = 512
    (16 steps); M = 40 runs two token groups of 24 (one of 16 tokens)."""
    rng = np.random.default_rng(100 + M)
    a, sa = rand_operand(rng, fa, M, 512, 32)
    b, sb = rand_operand(rng, fb, 300, 512, 32)
    check(torch, a, sa, b, sb, fa, fb, 32)


@pytest.mark.parametrize("fa,fb", [("E3C3", "E3C3"), ("E4C3", "E4C3"), ("E5C2", "E5C2"), ("E5C2", "E4C3")])
@pytest.mark.parametrize("M", [512, 601])
def test_two_token_groups_per_cta(torch, fa, fb, M):
    """Many token groups of 32 (16 for M = 512; 19 for M = 601, the last
    with 25 real tokens and 7 padding columns), N = 260 a ragged weight
    tile, K = 256 (8 scale bytes per row: the 8-byte chunks of the
    cooperative row references)."""
    rng = np.random.default_rng(M)
    a, sa = rand_operand(rng, fa, M, 256, 32)
    b, sb = rand_operand(rng, fb, 260, 256, 32)
    check(torch, a, sa, b, sb, fa, fb, 32)


@pytest.mark.parametrize("fa,fb", [("E3C3", "E3C3"), ("E5C2", "E4C3")])
@pytest.mark.parametrize("G", [64, 128, 512])
def test_larger_blocks(torch, fa, fb, G):
    """Block scales that span several 32-code steps (the step's scale is
    step >> log2(G/32))."""
    rng = np.random.default_rng(G)
    a, sa = rand_operand(rng, fa, 16, 1024, G)
    b, sb = rand_operand(rng, fb, 200, 1024, G)
    check(torch, a, sa, b, sb, fa, fb, G)


@pytest.mark.parametrize("fa,fb", [("E3C3", "E3C3"), ("E5C2", "E5C2")])
def test_quantized_activations_and_weights(torch, fa, fb):
    """Quantized lognormal-channel activations against N(0, 0.02) weights, the
    FFN decode inputs at a reduced size."""
    G = 32
    a, sa, _ = oracle.quantize(inputs.lognormal_channels((24, 768), 5), fa, G, 0)
    b, sb, _ = oracle.quantize(inputs.normal((520, 768), 6, 0.02), fb, G, 0)
    check(torch, a, sa, b, sb, fa, fb, G)


def test_wide_scale_spread_in_the_factors(torch):
    """Block scales 40 binades apart: both tensor paths carry them in the
    MMAs' scale factors, within tolerance of the oracle and of each other."""
    rng = np.random.default_rng(7)
    a, sa = rand_operand(rng, "E4C3", 8, 512, 32, spread=20)
    b, sb = rand_operand(rng, "E4C3", 256, 512, 32, spread=20)
    c = check(torch, a, sa, b, sb, "E4C3", "E4C3", 32)
    c2, _ = run(torch, a, sa, b, sb, "E4C3", "E4C3", 32, "tensor")
    na, nb = oracle.row_norms(a, sa, "E4C3"), oracle.row_norms(b, sb, "E4C3")
    assert normalised_error(c, c2.astype(np.float64), na, nb) <= 2 * TOL


def test_split_pieces_are_order_independent(torch):
    """With fewer weight tiles than SMs every tile is split in K and both
    pieces add to zeroed C: two runs give the same bits."""
    rng = np.random.default_rng(11)
    a, sa = rand_operand(rng, "E3C3", 4, 2048, 32)
    b, sb = rand_operand(rng, "E3C3", 1000, 2048, 32)
    c1 = check(torch, a, sa, b, sb, "E3C3", "E3C3", 32)
    c2, _ = run(torch, a, sa, b, sb, "E3C3", "E3C3", 32)
    assert np.array_equal(c1.view(np.int32), c2.view(np.int32))


@pytest.mark.parametrize("M", [1, 16, 64, 128])
def test_ffn_full_size_sampled(torch, M):
    """The FFN sweep's shapes (E3C3, W[14336 x 4096], lognormal activation
    channels): 256 sampled weight rows against the oracle at the launch
    configuration the benchmark times (M = 64: 224 tiles, a split tail;
    M = 128: 448 whole tiles)."""
    import paper_2608_10010_gb300 as cfp

    G = 32
    Xf, Wf = inputs.ffn_cuda(M, 4096)
    a, sa = cfp.quantize(Xf, "E3C3", G, 0)
    b, sb = cfp.quantize(Wf, "E3C3", G, 1)
    st = new_status(torch)
    c = cfp.gemm(a, sa, b, sb, "E3C3", "E3C3", G, "tensor_narrow", status=st)
    torch.cuda.synchronize()
    assert status_bits(st) == 0
    jj = np.sort(np.random.default_rng(5).choice(b.shape[0], 256, replace=False))
    ah, sah = a.cpu().numpy(), sa.cpu().numpy()
    bh, sbh = b.cpu().numpy()[jj], sb.cpu().numpy()[jj]
    ref = oracle.gemm(ah, sah, bh, sbh, "E3C3", "E3C3", G, phases=False)
    na, nb = oracle.row_norms(ah, sah, "E3C3", G), oracle.row_norms(bh, sbh, "E3C3", G)
    assert normalised_error(c.cpu().numpy()[:, jj], ref["C"], na, nb) <= TOL


def test_radix_and_unsupported_pairs_are_rejected(torch):
    import paper_2608_10010_gb300 as cfp

    rng = np.random.default_rng(1)
    a, sa = rand_operand(rng, "E4C3", 8, 64, 32)
    lib = cfp.load()
    args = [to_dev(torch, t) for t in (a, sa, a, sa)]
    c = torch.empty((8, 8), dtype=torch.float32, device="cuda")
    import ctypes

    P = ctypes.c_void_p
    for fa, fb in [(3, 3), (0, 1), (1, 0)]:  # E4C3_R8_9, E3C3 x E4C3, E4C3 x E3C3
        rc = lib.curvefp_gemm(5, fa, fb, 32, *[P(t.data_ptr()) for t in args], 8, 8, 64, P(c.data_ptr()), None, None)
        assert rc == 2
