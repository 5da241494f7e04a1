"""GPU closed-product GEMM parity through the C ABI.

EXACT kernel: per-phase int128 sums and their LSBs bit-identical to the
oracle; FP32 output within 1e-5 of the oracle's fp64 phase combine,
normalised by ||a_i|| ||b_j|| of the dequantized operands.
TENSOR kernel: FP32 output within the same 1e-5 normalised bound.
"""
import numpy as np
import pytest

import oracle
from paper_2608_10010_gb300 import inputs
from tests.gpu_util import new_status, normalised_error, status_bits, to_dev, torch_cuda

pytestmark = pytest.mark.gpu
FORMATS = ["E3C3", "E4C3", "E5C2"]
PAIRS = [(a, b) for a in FORMATS for b in FORMATS]
TC_PAIRS = [("E3C3", "E3C3"), ("E4C3", "E4C3"), ("E5C2", "E4C3"), ("E4C3", "E5C2"), ("E5C2", "E5C2")]
TOL = 1e-5


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


def rand_operand(rng, fmt, rows, K, block, spread=4):
    codes = rng.integers(0, 256, size=(rows, K), dtype=np.uint8)
    if fmt == "E3C3":
        codes &= 0xBF
    scales = rng.integers(-spread, spread + 1, size=(rows, K // block)).astype(np.int8)
    return codes, scales


def quantized(x, fmt, block=32, axis=0):
    c, s, _ = oracle.quantize(x, fmt, block, axis)
    return c, s


def gpu_exact(torch, a, sa, b, sb, fa, fb, block):
    import paper_2608_10010_gb300 as cfp

    st = new_status(torch)
    c, ps, pl = cfp.gemm_phases(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fa, fb,
                                block, status=st)
    torch.cuda.synchronize()
    return c.cpu().numpy(), ps.cpu().numpy(), pl.cpu().numpy(), status_bits(st)


def gpu_gemm(torch, a, sa, b, sb, fa, fb, block, algo):
    import paper_2608_10010_gb300 as cfp

    st = new_status(torch)
    c = cfp.gemm(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fa, fb, block, algo,
                 status=st)
    torch.cuda.synchronize()
    return c.cpu().numpy(), status_bits(st)


def check_exact(torch, a, sa, b, sb, fa, fb, block, rows=None):
    c, ps, pl, st = gpu_exact(torch, a, sa, b, sb, fa, fb, block)
    ra = a if rows is None else a[rows]
    rsa = sa if rows is None else sa[rows]
    ref = oracle.gemm(ra, rsa, b, sb, fa, fb, block)
    if rows is not None:
        c, ps, pl = c[rows], ps[rows], pl[rows]
    ok = ~ref["range"]
    assert np.array_equal(ps[ok], ref["S_raw"][ok])
    assert np.array_equal(pl[ok], ref["lsb"][ok])
    assert bool(st & 2) == bool(ref["range"].any()) or rows is not None
    na = oracle.row_norms(ra, rsa, fa, block)
    nb = oracle.row_norms(b, sb, fb, block)
    assert normalised_error(np.where(ok, c, 0), np.where(ok, ref["C"], 0), na, nb) <= TOL
    return c, ref


def check_tensor(torch, a, sa, b, sb, fa, fb, block, rows=None, algo="tensor"):
    c, st = gpu_gemm(torch, a, sa, b, sb, fa, fb, block, algo)
    assert st == 0
    ra = a if rows is None else a[rows]
    rsa = sa if rows is None else sa[rows]
    ref = oracle.gemm(ra, rsa, b, sb, fa, fb, block, phases=False)
    if rows is not None:
        c = c[rows]
    na = oracle.row_norms(ra, rsa, fa, block)
    nb = oracle.row_norms(b, sb, fb, block)
    err = normalised_error(c, ref["C"], na, nb)
    assert err <= TOL, err
    return err


# ---- the small E4C3 workload, in full ------------------------------------------

def test_small_e4c3_workload_exact_and_tensor(torch):
    A, B = inputs.small_e4c3()
    a, sa = quantized(A, "E4C3", 32, 0)
    b, sb = quantized(B, "E4C3", 32, 1)  # B[K x N] -> [N x K] operand
    check_exact(torch, a, sa, b, sb, "E4C3", "E4C3", 32)
    check_tensor(torch, a, sa, b, sb, "E4C3", "E4C3", 32)


# ---- exact kernel: all format pairs, full code space, ragged shapes -------------

@pytest.mark.parametrize("fa,fb", PAIRS)
def test_exact_all_pairs_random_codes(torch, fa, fb):
    rng = np.random.default_rng(hash((fa, fb)) % 2**32)
    for (M, N, K, block) in [(1, 1, 32, 32), (3, 17, 96, 32), (17, 33, 128, 64), (130, 37, 512, 128), (5, 3, 512, 512)]:
        a, sa = rand_operand(rng, fa, M, K, block)
        b, sb = rand_operand(rng, fb, N, K, block)
        check_exact(torch, a, sa, b, sb, fa, fb, block)


def test_exact_range_flag(torch):
    K = 64
    a = np.full((2, K), 0x7F, np.uint8)
    b = np.full((3, K), 0x7F, np.uint8)
    sa = np.array([[-128, 127], [0, 1]], np.int8)
    sb = np.array([[-128, 127], [0, 1], [2, 2]], np.int8)
    c, ps, pl, st = gpu_exact(torch, a, sa, b, sb, "E5C2", "E5C2", 32)
    ref = oracle.gemm(a, sa, b, sb, "E5C2", "E5C2", 32)
    assert ref["range"][0, 0] and st & 2
    assert np.isnan(c[0, 0])
    ok = ~ref["range"]
    assert np.array_equal(ps[ok], ref["S_raw"][ok])


def test_exact_zero_and_extreme_operands(torch):
    """All-zero rows, all-maximum codes, scales at both int8 extremes within
    the window, alternating signs."""
    K = 256
    a = np.zeros((4, K), np.uint8)
    a[1] = 0x7F
    a[2] = np.where(np.arange(K) % 2, 0xFF, 0x7F)
    a[3] = 0x01
    b = np.zeros((3, K), np.uint8)
    b[0] = 0x7F
    b[1] = 0x81
    b[2] = np.arange(K) % 256
    sa = np.full((4, K // 32), 100, np.int8)
    sb = np.full((3, K // 32), -120, np.int8)
    sa[3] = -128
    sb[2] = 127
    check_exact(torch, a, sa, b, sb, "E4C3", "E4C3", 32)


# ---- tensor kernel ------------------------------------------------------------------

@pytest.mark.parametrize("algo", ["tensor", "tensor_narrow"])
@pytest.mark.parametrize("fa,fb", TC_PAIRS)
def test_tensor_pairs_ragged(torch, fa, fb, algo):
    rng = np.random.default_rng(99 + hash((fa, fb)) % 1000)
    for (M, N, K, block) in [(1, 1, 32, 32), (3, 17, 64, 32), (130, 33, 160, 32), (257, 70, 1024, 64), (128, 32, 512, 512)]:
        x = inputs.normal((M, K), int(rng.integers(1 << 30)))
        w = inputs.normal((N, K), int(rng.integers(1 << 30)), 0.02)
        a, sa = quantized(x, fa, block)
        b, sb = quantized(w, fb, block)
        check_tensor(torch, a, sa, b, sb, fa, fb, block, algo=algo)


@pytest.mark.parametrize("algo", ["tensor", "tensor_narrow"])
@pytest.mark.parametrize("fa,fb", TC_PAIRS)
def test_tensor_full_code_space(torch, fa, fb, algo):
    """Uniformly random codes (every level, both signs, zeros) and scale spread."""
    rng = np.random.default_rng(5)
    a, sa = rand_operand(rng, fa, 200, 256, 32, spread=6)
    b, sb = rand_operand(rng, fb, 100, 256, 32, spread=6)
    check_tensor(torch, a, sa, b, sb, fa, fb, 32, algo=algo)


@pytest.mark.parametrize("fa,fb", TC_PAIRS)
def test_narrow_matches_tile(torch, fa, fb):
    """The two tensor-core kernels (2:4-sparse pair planes along N against
    dense plane pairs of a tile): the same exact products, summed in a
    different order in FP32."""
    rng = np.random.default_rng(11)
    a, sa = rand_operand(rng, fa, 300, 1024, 32, spread=4)
    b, sb = rand_operand(rng, fb, 200, 1024, 32, spread=4)
    cs, st = gpu_gemm(torch, a, sa, b, sb, fa, fb, 32, "tensor_narrow")
    cd, st2 = gpu_gemm(torch, a, sa, b, sb, fa, fb, 32, "tensor")
    assert st == 0 and st2 == 0
    na = oracle.row_norms(a, sa, fa)
    nb = oracle.row_norms(b, sb, fb)
    assert normalised_error(cs, cd.astype(np.float64), na, nb) <= TOL


def test_tensor_matches_exact_kernel(torch):
    """The tensor path against the exact kernel on a mid-size problem."""
    x = inputs.outlier_channels((512, 1024), 3)
    w = inputs.normal((384, 1024), 4, 0.02)
    a, sa = quantized(x, "E3C3")
    b, sb = quantized(w, "E3C3")
    ce, st = gpu_gemm(torch, a, sa, b, sb, "E3C3", "E3C3", 32, "exact")
    ct, st2 = gpu_gemm(torch, a, sa, b, sb, "E3C3", "E3C3", 32, "tensor")
    assert st == 0 and st2 == 0
    na = oracle.row_norms(a, sa, "E3C3")
    nb = oracle.row_norms(b, sb, "E3C3")
    assert normalised_error(ct, ce.astype(np.float64), na, nb) <= TOL


@pytest.mark.parametrize("M,N,K", [(1024, 4096, 256), (2048, 4096, 96), (2048, 4096, 32), (1280, 9120, 128)])
def test_tensor_tail_pieces_every_output(torch, M, N, K):
    """Tile counts whose tail is split in K (1024 x 4096: 344 tiles, 192 of
    them split; 2048 x 4096: 688 tiles, 80 split 2/3 + 1/3; 1280 x 9120:
    950 tiles, split 3/4 + 1/4; K = 32 is one step, too short to split):
    every output of the tensor path against the exact kernel, and two runs
    bit-identical (the pieces' atomic additions onto zero do not depend on
    their order)."""
    import paper_2608_10010_gb300 as cfp

    x = inputs.outlier_channels((M, K), 23)
    w = inputs.normal((N, K), 24, 0.02)
    a, sa = quantized(x, "E3C3")
    b, sb = quantized(w, "E3C3")
    args = [to_dev(torch, v) for v in (a, sa, b, sb)]
    st = new_status(torch)
    ce = cfp.gemm(*args, "E3C3", "E3C3", 32, "exact", status=st)
    ct = cfp.gemm(*args, "E3C3", "E3C3", 32, "tensor", status=st)
    ct2 = cfp.gemm(*args, "E3C3", "E3C3", 32, "tensor", status=st)
    torch.cuda.synchronize()
    assert status_bits(st) == 0
    assert torch.equal(ct.view(torch.int32), ct2.view(torch.int32))
    na = oracle.row_norms(a, sa, "E3C3")
    nb = oracle.row_norms(b, sb, "E3C3")
    assert normalised_error(ct.cpu().numpy(), ce.cpu().numpy().astype(np.float64), na, nb) <= TOL


# ---- full-size workloads, sampled rows ---------------------------------------------

SAMPLE_ROWS = 16


def _sample(M, seed=0):
    return np.sort(np.random.default_rng(seed).choice(M, min(SAMPLE_ROWS, M), replace=False))


def test_llama7b_linear_full_size(torch):
    """The benchmark workload: E3C3 W[4096x4096] ~ N(0, 0.02^2), X[2048x4096]
    with 1% x20 outlier channels; quantized on the GPU in the benchmark's launch
    configuration, both GEMM kernels on the full problem, parity on sampled
    rows (exact kernel bit-exact per phase)."""
    import paper_2608_10010_gb300 as cfp

    X, W = inputs.llama7b_linear()
    xd, wd = to_dev(torch, X), to_dev(torch, W)
    a, sa = cfp.quantize(xd, "E3C3", 32, 0)
    b, sb = cfp.quantize(wd, "E3C3", 32, 0)
    ra, rsa = quantized(X, "E3C3")
    rb, rsb = quantized(W, "E3C3")
    assert np.array_equal(a.cpu().numpy(), ra) and np.array_equal(sa.cpu().numpy(), rsa)
    assert np.array_equal(b.cpu().numpy(), rb) and np.array_equal(sb.cpu().numpy(), rsb)
    rows = _sample(2048)
    check_exact(torch, ra, rsa, rb, rsb, "E3C3", "E3C3", 32, rows=rows)
    check_tensor(torch, ra, rsa, rb, rsb, "E3C3", "E3C3", 32, rows=rows)
    # the benchmark's GEMM: phases along N, 2:4-sparse pair planes (64 token groups x 32 weight tiles)
    check_tensor(torch, ra, rsa, rb, rsb, "E3C3", "E3C3", 32, rows=rows, algo="tensor_narrow")


@pytest.mark.parametrize("which", ["fwd", "dgrad", "wgrad"])
def test_training_triplet_full_size(torch, which):
    """CurveFP8 training GEMMs (E4C3 X, W; E5C2 dY = 1e-3 t_3), each operand
    quantized along its own GEMM's reduction axis; the tile and the narrow
    tensor-core kernels on the full problem, parity on sampled rows."""
    X, W, dY = inputs.training_triplet()
    if which == "fwd":  # Y = X W: M = tokens, N = out, K = in
        a, sa = quantized(X, "E4C3", 32, 0)
        b, sb = quantized(W, "E4C3", 32, 1)
        fa, fb = "E4C3", "E4C3"
    elif which == "dgrad":  # dX = dY W^T: M = tokens, N = in, K = out
        a, sa = quantized(dY, "E5C2", 32, 0)
        b, sb = quantized(W, "E4C3", 32, 0)
        fa, fb = "E5C2", "E4C3"
    else:  # dW^T = dY^T X: M = out, N = in, K = tokens
        a, sa = quantized(dY, "E5C2", 32, 1)
        b, sb = quantized(X, "E4C3", 32, 1)
        fa, fb = "E5C2", "E4C3"
    check_tensor(torch, a, sa, b, sb, fa, fb, 32, rows=_sample(a.shape[0], 1))
    check_tensor(torch, a, sa, b, sb, fa, fb, 32, rows=_sample(a.shape[0], 1), algo="tensor_narrow")


@pytest.mark.parametrize("M", [1, 16, 128])
def test_ffn_sweep_small_m(torch, M):
    """CurveFP7 E3C3 FFN: W[4096 x 14336] (blocks along K = rows), X[M x 4096]
    with LogNormal(0, 1.5)-scaled channels; both kernels, all rows."""
    X, W = inputs.ffn_sweep(M)
    a, sa = quantized(X, "E3C3", 32, 0)
    b, sb = quantized(W, "E3C3", 32, 1)
    cols = np.sort(np.random.default_rng(2).choice(b.shape[0], 512, replace=False))
    bs, sbs = b[cols], sb[cols]
    check_exact(torch, a, sa, bs, sbs, "E3C3", "E3C3", 32)
    check_tensor(torch, a, sa, bs, sbs, "E3C3", "E3C3", 32)


# ---- output requantization ------------------------------------------------------

@pytest.mark.parametrize("algo", ["tensor", "exact"])
@pytest.mark.parametrize("fa,fb,fc", [("E3C3", "E3C3", "E3C3"), ("E4C3", "E4C3", "E4C3"), ("E5C2", "E4C3", "E5C2")])
def test_gemm_requant(torch, algo, fa, fb, fc):
    """C within tolerance of the oracle, and its requantized codes/scales
    bit-exact with the oracle's quantization of that same FP32 C."""
    import paper_2608_10010_gb300 as cfp

    x = inputs.outlier_channels((200, 512), 3)
    w = inputs.normal((96 * 3, 512), 4, 0.02)
    a, sa = quantized(x, fa)
    b, sb = quantized(w, fb)
    st = new_status(torch)
    c, codes, scales = cfp.gemm_requant(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb),
                                        fa, fb, fc, 32, 32, algo, status=st)
    torch.cuda.synchronize()
    assert status_bits(st) == 0
    c = c.cpu().numpy()
    ref = oracle.gemm(a, sa, b, sb, fa, fb, 32, phases=False)
    na, nb = oracle.row_norms(a, sa, fa), oracle.row_norms(b, sb, fb)
    assert normalised_error(c, ref["C"], na, nb) <= TOL
    rc, rs, _ = oracle.quantize(c, fc, 32, 0)
    assert np.array_equal(codes.cpu().numpy(), rc) and np.array_equal(scales.cpu().numpy(), rs)


# ---- decode-sized GEMMs on the CUDA cores ------------------------------------

@pytest.mark.parametrize("fa,fb", [(a, b) for a in ("E3C3", "E4C3", "E5C2") for b in ("E3C3", "E4C3", "E5C2")])
@pytest.mark.parametrize("M", [1, 3, 8])
def test_skinny_within_tolerance(torch, fa, fb, M):
    """SKINNY (FP32 per-phase accumulation of exact powers of two, M <= 8):
    within 1e-5 of the oracle; N = 300 leaves a partial CTA of rows."""
    import paper_2608_10010_gb300 as cfp

    N, K, G = 300, 1024, 32
    a, sa = quantized(inputs.lognormal_channels((M, K), 20 + M), fa, G)
    b, sb = quantized(inputs.normal((N, K), 21, 0.02), fb, G)
    st = new_status(torch)
    c = cfp.gemm(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fa, fb, G, "skinny",
                 status=st)
    torch.cuda.synchronize()
    ref = oracle.gemm(a, sa, b, sb, fa, fb, G, phases=False)
    na, nb = oracle.row_norms(a, sa, fa, G), oracle.row_norms(b, sb, fb, G)
    assert status_bits(st) == 0
    assert normalised_error(c.cpu().numpy(), ref["C"], na, nb) <= TOL


@pytest.mark.parametrize("M", [1, 8])
def test_skinny_ffn_full_size_sampled(torch, M):
    """The decode shapes of the FFN sweep (E3C3, W[14336 x 4096]) through
    SKINNY: 256 sampled columns against the oracle; AUTO (SKINNY for M = 1,
    TENSOR_NARROW up to M = 96) equal to the kernel it picks, bit for bit."""
    import paper_2608_10010_gb300 as cfp

    G = 32
    Xf, Wf = inputs.ffn_cuda(M, 4096)
    a, sa = cfp.quantize(Xf, "E3C3", G, 0)
    b, sb = cfp.quantize(Wf, "E3C3", G, 1)
    c = cfp.gemm(a, sa, b, sb, "E3C3", "E3C3", G, "skinny")
    c2 = cfp.gemm(a, sa, b, sb, "E3C3", "E3C3", G, "auto")
    c3 = cfp.gemm(a, sa, b, sb, "E3C3", "E3C3", G, "skinny" if M <= 1 else "tensor_narrow")
    torch.cuda.synchronize()
    assert torch.equal(c2.view(torch.int32), c3.view(torch.int32))
    jj = np.sort(np.random.default_rng(3).choice(b.shape[0], 256, replace=False))
    ah, sah = a.cpu().numpy(), sa.cpu().numpy()
    bh, sbh = b.cpu().numpy()[jj], sb.cpu().numpy()[jj]
    ref = oracle.gemm(ah, sah, bh, sbh, "E3C3", "E3C3", G, phases=False)
    na, nb = oracle.row_norms(ah, sah, "E3C3", G), oracle.row_norms(bh, sbh, "E3C3", G)
    assert normalised_error(c.cpu().numpy()[:, jj], ref["C"], na, nb) <= TOL
