"""GPU parity of the rational-radix E4C3 formats (r = 2^{8/9}, 9 phases;
r = 2^{3/4}, 32 phases; Sec. 3.1 Eq. 1, Eq. 4, Table 2): codes, scales,
dequantized values and exact per-phase int128 sums bit-identical to the
oracle, through the C ABI."""
import numpy as np
import pytest

import oracle
from paper_2608_10010_gb300 import inputs
from tests.gpu_util import new_status, status_bits, to_dev, torch_cuda, widen

pytestmark = pytest.mark.gpu
RADIX = ["E4C3_R8_9", "E4C3_R3_4"]


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


def check_q(torch, x, fmt, block, dtype="f32", axis=0):
    import paper_2608_10010_gb300 as cfp

    xd = to_dev(torch, x, dtype)
    st = new_status(torch)
    codes, scales = cfp.quantize(xd, fmt, block, axis, status=st)
    torch.cuda.synchronize()
    rc, rs, nan = oracle.quantize(widen(torch, xd), fmt, block, axis)
    assert np.array_equal(scales.cpu().numpy(), rs), (fmt, block, dtype)
    assert np.array_equal(codes.cpu().numpy(), rc), (fmt, block, dtype)
    assert bool(status_bits(st) & 1) == nan
    return rc, rs


def midpoint_probes(fmt, block):
    """Blocks of FP32 neighbours of every level midpoint and of the zero
    boundary, each block anchored at L_nmax so that its scale is 0."""
    lv = oracle.levels(fmt)
    mids = np.concatenate([[lv[0] / 2], (lv[1:] + lv[:-1]) / 2]).astype(np.float32)
    pr = np.concatenate([np.nextafter(mids, np.float32(0)), mids, np.nextafter(mids, np.float32(np.inf))])
    pr = pr[pr <= np.float32(lv[-1])].astype(np.float32)
    pr = pr * np.where(np.arange(len(pr)) % 2 == 0, 1, -1).astype(np.float32)
    per = block - 1
    nblk = -(-len(pr) // per)
    x = np.zeros((nblk, block), np.float32)
    x[:, 0] = np.float32(lv[-1])
    flat = x[:, 1:].reshape(-1)
    flat[: len(pr)] = pr
    x[:, 1:] = flat.reshape(nblk, per)
    return x


@pytest.mark.parametrize("fmt", RADIX)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("block", [32, 128, 512])
def test_quantize_distributions(torch, fmt, dtype, block):
    """Outlier activations, heavy-tailed gradients, N(0, 0.02^2) weights and a
    wide log-uniform magnitude sweep (2^-140 .. 2^120, subnormals included)."""
    rng = np.random.default_rng(block)
    check_q(torch, inputs.outlier_channels((40, 1024), 1), fmt, block, dtype)
    check_q(torch, inputs.heavy_tailed_grad((40, 1024), 2), fmt, block, dtype)
    check_q(torch, inputs.normal((40, 1024), 3, 0.02), fmt, block, dtype)
    wide = (2.0 ** rng.uniform(-140, 120, (40, 1024))).astype(np.float32)
    wide *= np.where(rng.random((40, 1024)) < 0.5, -1, 1).astype(np.float32)
    check_q(torch, wide, fmt, block, dtype)


@pytest.mark.parametrize("fmt", RADIX)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_quantize_shapes_and_paths(torch, fmt, dtype):
    """Every kernel path of the shared quantizer: dense G32 rows (bulk-fed),
    strided rows (register-fed), G 64..512, and block axis 1 (transposed
    output)."""
    x = inputs.elementwise_outliers((37, 1024), 8)
    for block in (32, 64, 128, 256, 512):
        check_q(torch, x, fmt, block, dtype)
    y = inputs.elementwise_outliers((1024, 40), 9)
    for block in (32, 64, 512):
        check_q(torch, y, fmt, block, dtype, axis=1)
    # a strided view (ld > cols): the register-fed kernel
    import paper_2608_10010_gb300 as cfp

    big = to_dev(torch, inputs.outlier_channels((64, 1536), 10), dtype)
    view = big[:, :1024]
    st = new_status(torch)
    codes, scales = cfp.quantize(view, fmt, 32, 0, status=st)
    torch.cuda.synchronize()
    rc, rs, _ = oracle.quantize(np.ascontiguousarray(widen(torch, view)), fmt, 32, 0)
    assert np.array_equal(codes.cpu().numpy(), rc) and np.array_equal(scales.cpu().numpy(), rs)


@pytest.mark.parametrize("fmt", RADIX)
@pytest.mark.parametrize("group,rule", [("block", "mse"), ("row", "mse"), ("tensor", "ceil")])
def test_quantize_static(torch, fmt, group, rule):
    """Static-operand scales (block / row / tensor groups, MSE search) with
    the rational levels, bit-exact against the oracle."""
    import paper_2608_10010_gb300 as cfp

    x = inputs.normal((48, 1024), 11, 0.02)
    xd = to_dev(torch, x)
    codes, scales = cfp.quantize_static(xd, fmt, 512, group, rule)
    torch.cuda.synchronize()
    rc, rs, _ = oracle.quantize_static(x, fmt, 512, group, rule)
    assert np.array_equal(scales.cpu().numpy(), rs) and np.array_equal(codes.cpu().numpy(), rc)


@pytest.mark.parametrize("fmt", RADIX)
@pytest.mark.parametrize("block", [32, 512])
def test_quantize_midpoints_and_specials(torch, fmt, block):
    """Every level midpoint and the zero boundary L_nmin/2 (for r = 2^{8/9}
    exactly 2^-8: the tie goes to zero) with their FP32 neighbours; zero,
    signed-zero, subnormal-only, Inf and NaN blocks."""
    check_q(torch, midpoint_probes(fmt, block), fmt, block)
    x = np.zeros((6, block), np.float32)
    x[1, :] = -0.0
    x[2, 0], x[2, 1], x[2, 2] = np.inf, 1.0, -np.inf
    x[3, :] = np.float32(2.0) ** -135
    x[3, 1] = -x[3, 1]
    x[4, :] = 1.0
    x[4, 3] = np.nan
    x[5, :] = np.float32(2.0 ** -8)
    x[5, 0] = np.float32(oracle.levels(fmt)[-1])
    rc, _ = check_q(torch, x, fmt, block)
    if fmt == "E4C3_R8_9":
        assert np.all(rc[5, 1:] == 0)  # y = L_nmin / 2 exactly: the tie goes to zero


@pytest.mark.parametrize("fmt", RADIX)
def test_dequantize_every_code_and_scale(torch, fmt):
    import paper_2608_10010_gb300 as cfp

    svals = np.array([-128, -127, -40, -8, 0, 3, 60, 120, 127], np.int8)
    codes = np.tile(np.arange(256, dtype=np.uint8), len(svals))[None, :]
    scales = np.repeat(svals, 256 // 32)[None, :]
    out = cfp.dequantize(to_dev(torch, codes), to_dev(torch, scales), fmt, 32)
    torch.cuda.synchronize()
    ref = oracle.dequantize(codes, scales, fmt, 32)
    assert np.array_equal(out.cpu().numpy().view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("fmt", RADIX)
@pytest.mark.parametrize("block", [32, 512])
def test_exact_gemm_phase_sums(torch, fmt, block):
    """9- and 32-phase int128 sums, LSBs and the combine bit-identical to the
    oracle; M, N ragged against the 16 x 16 tiles."""
    import paper_2608_10010_gb300 as cfp

    M, N, K = 40, 24, 1024
    a, sa, _ = oracle.quantize(inputs.outlier_channels((M, K), 5), fmt, block, 0)
    b, sb, _ = oracle.quantize(inputs.normal((N, K), 6, 0.02), fmt, block, 0)
    st = new_status(torch)
    c, ps, pl = cfp.gemm_phases(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fmt, fmt,
                                block, status=st)
    torch.cuda.synchronize()
    ref = oracle.gemm(a, sa, b, sb, fmt, fmt, block)
    assert status_bits(st) == 0
    assert ps.shape[2] == (9 if fmt == "E4C3_R8_9" else 32)
    assert np.array_equal(ps.cpu().numpy(), ref["S_raw"])
    assert np.array_equal(pl.cpu().numpy(), ref["lsb"])
    assert np.array_equal(c.cpu().numpy(), ref["C"].astype(np.float32))
    c2 = cfp.gemm(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fmt, fmt, block, "exact")
    assert np.array_equal(c2.cpu().numpy(), ref["C"].astype(np.float32))


@pytest.mark.parametrize("fmt", RADIX)
def test_llama_linear_g512_sampled(torch, fmt):
    """The radix-frontier setting (E4C3, G512) on the Llama-7B-like linear:
    X[2048 x 4096] with 1% outlier channels and W[4096 x 4096] ~ N(0, 0.02^2)
    quantized on the GPU (sampled rows bit-exact), then the exact GEMM of 64
    sampled rows of each against the oracle."""
    import paper_2608_10010_gb300 as cfp

    G = 512
    X, W = inputs.llama7b_linear(2048, 4096, 4096)
    Xd, Wd = to_dev(torch, X), to_dev(torch, W)  # W [d_out x d_in]: rows are GEMM rows
    qx, sx = cfp.quantize(Xd, fmt, G, 0)
    qw, sw = cfp.quantize(Wd, fmt, G, 0)
    torch.cuda.synchronize()
    rng = np.random.default_rng(12)
    ii = np.sort(rng.choice(2048, 64, replace=False))
    jj = np.sort(rng.choice(4096, 64, replace=False))
    rx, rsx, _ = oracle.quantize(X[ii], fmt, G, 0)
    rw, rsw, _ = oracle.quantize(W[jj], fmt, G, 0)
    assert np.array_equal(qx.cpu().numpy()[ii], rx) and np.array_equal(sx.cpu().numpy()[ii], rsx)
    assert np.array_equal(qw.cpu().numpy()[jj], rw) and np.array_equal(sw.cpu().numpy()[jj], rsw)
    st = new_status(torch)
    c, ps, pl = cfp.gemm_phases(qx[torch.from_numpy(ii).cuda()].contiguous(), sx[torch.from_numpy(ii).cuda()].contiguous(),
                                qw[torch.from_numpy(jj).cuda()].contiguous(), sw[torch.from_numpy(jj).cuda()].contiguous(),
                                fmt, fmt, G, status=st)
    torch.cuda.synchronize()
    ref = oracle.gemm(rx, rsx, rw, rsw, fmt, fmt, G)
    assert status_bits(st) == 0
    assert np.array_equal(ps.cpu().numpy(), ref["S_raw"]) and np.array_equal(pl.cpu().numpy(), ref["lsb"])


@pytest.mark.parametrize("block", [32, 512])
def test_tensor_gemm_r89_within_tolerance(torch, block):
    """Tensor-core GEMM for r = 2^{8/9} (nine planes per operand, 81 plane
    pairs, nine phases in three passes): within 1e-5 of the oracle's fp64
    combine, normalised by the row norms; M, N ragged against the tiles."""
    import paper_2608_10010_gb300 as cfp
    from tests.gpu_util import normalised_error

    fmt = "E4C3_R8_9"
    M, N, K = 200, 320, 1024
    a, sa, _ = oracle.quantize(inputs.outlier_channels((M, K), 17), fmt, block, 0)
    b, sb, _ = oracle.quantize(inputs.normal((N, K), 18, 0.02), fmt, block, 0)
    st = new_status(torch)
    c = cfp.gemm(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fmt, fmt, block, "tensor",
                 status=st)
    torch.cuda.synchronize()
    ref = oracle.gemm(a, sa, b, sb, fmt, fmt, block, phases=False)
    assert status_bits(st) == 0
    err = normalised_error(c.cpu().numpy(), ref["C"], oracle.row_norms(a, sa, fmt, block),
                           oracle.row_norms(b, sb, fmt, block))
    assert err <= 1e-5, err


def test_tensor_gemm_r89_llama_g512_sampled(torch):
    """The radix-frontier setting at full size (Llama-7B-like linear, G512)
    on the tensor cores: 64 x 64 sampled outputs against the oracle."""
    import paper_2608_10010_gb300 as cfp
    from tests.gpu_util import normalised_error

    fmt, G = "E4C3_R8_9", 512
    X, W = inputs.llama7b_linear(2048, 4096, 4096)
    qx, sx = cfp.quantize(to_dev(torch, X), fmt, G, 0)
    qw, sw = cfp.quantize(to_dev(torch, W), fmt, G, 0)
    st = new_status(torch)
    c = cfp.gemm(qx, sx, qw, sw, fmt, fmt, G, "tensor", status=st)
    torch.cuda.synchronize()
    assert status_bits(st) == 0
    rng = np.random.default_rng(19)
    ii = np.sort(rng.choice(2048, 64, replace=False))
    jj = np.sort(rng.choice(4096, 64, replace=False))
    ah, sah = qx.cpu().numpy()[ii], sx.cpu().numpy()[ii]
    bh, sbh = qw.cpu().numpy()[jj], sw.cpu().numpy()[jj]
    ref = oracle.gemm(ah, sah, bh, sbh, fmt, fmt, G, phases=False)
    err = normalised_error(c.cpu().numpy()[np.ix_(ii, jj)], ref["C"], oracle.row_norms(ah, sah, fmt, G),
                           oracle.row_norms(bh, sbh, fmt, G))
    assert err <= 1e-5, err


@pytest.mark.parametrize("block", [32, 512])
@pytest.mark.parametrize("algo", ["tensor_narrow", "auto"])
def test_narrow_gemm_r34_within_tolerance(torch, block, algo):
    """Tensor-core GEMM for r = 2^{3/4} (32 planes per operand, pair planes j
    and j + 16 in 2:4-sparse MMAs, the 32 phases along N): within 1e-5 of the
    oracle's fp64 combine, normalised by the row norms; M ragged against the
    8-token tiles, N against the 128-row tiles; AUTO takes the same kernel."""
    import paper_2608_10010_gb300 as cfp
    from tests.gpu_util import normalised_error

    fmt = "E4C3_R3_4"
    M, N, K = 37, 320, 1024
    a, sa, _ = oracle.quantize(inputs.outlier_channels((M, K), 21), fmt, block, 0)
    b, sb, _ = oracle.quantize(inputs.normal((N, K), 22, 0.02), fmt, block, 0)
    st = new_status(torch)
    c = cfp.gemm(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fmt, fmt, block, algo,
                 status=st)
    torch.cuda.synchronize()
    ref = oracle.gemm(a, sa, b, sb, fmt, fmt, block, phases=False)
    assert status_bits(st) == 0
    err = normalised_error(c.cpu().numpy(), ref["C"], oracle.row_norms(a, sa, fmt, block),
                           oracle.row_norms(b, sb, fmt, block))
    assert err <= 1e-5, err


def test_narrow_gemm_r34_every_code(torch):
    """Every code byte (both signs, the zero code, all 32 curve planes and
    both halves of each pair) on both operands with block scales spread over
    24 binades: within 1e-5 of the oracle."""
    import paper_2608_10010_gb300 as cfp
    from tests.gpu_util import normalised_error

    fmt, G = "E4C3_R3_4", 32
    rng = np.random.default_rng(23)
    M, N, K = 24, 256, 512
    a = rng.integers(0, 256, size=(M, K)).astype(np.uint8)
    b = rng.integers(0, 256, size=(N, K)).astype(np.uint8)
    a[0, :256] = np.arange(256, dtype=np.uint8)
    b[:, :256] = np.arange(256, dtype=np.uint8)[None, :]
    sa = rng.integers(-12, 12, size=(M, K // G)).astype(np.int8)
    sb = rng.integers(-12, 12, size=(N, K // G)).astype(np.int8)
    st = new_status(torch)
    c = cfp.gemm(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b), to_dev(torch, sb), fmt, fmt, G,
                 "tensor_narrow", status=st)
    torch.cuda.synchronize()
    ref = oracle.gemm(a, sa, b, sb, fmt, fmt, G, phases=False)
    assert status_bits(st) == 0
    err = normalised_error(c.cpu().numpy(), ref["C"], oracle.row_norms(a, sa, fmt, G),
                           oracle.row_norms(b, sb, fmt, G))
    assert err <= 1e-5, err


def test_narrow_gemm_r34_llama_g512_sampled(torch):
    """r = 2^{3/4} at full size (Llama-7B-like linear, G512) on the tensor
    cores, with the split tail of the last wave: 64 x 64 sampled outputs
    against the oracle."""
    import paper_2608_10010_gb300 as cfp
    from tests.gpu_util import normalised_error

    fmt, G = "E4C3_R3_4", 512
    X, W = inputs.llama7b_linear(2048, 4096, 4096)
    qx, sx = cfp.quantize(to_dev(torch, X), fmt, G, 0)
    qw, sw = cfp.quantize(to_dev(torch, W), fmt, G, 0)
    st = new_status(torch)
    c = cfp.gemm(qx, sx, qw, sw, fmt, fmt, G, "tensor_narrow", status=st)
    torch.cuda.synchronize()
    assert status_bits(st) == 0
    rng = np.random.default_rng(29)
    ii = np.sort(rng.choice(2048, 64, replace=False))
    jj = np.sort(rng.choice(4096, 64, replace=False))
    ah, sah = qx.cpu().numpy()[ii], sx.cpu().numpy()[ii]
    bh, sbh = qw.cpu().numpy()[jj], sw.cpu().numpy()[jj]
    ref = oracle.gemm(ah, sah, bh, sbh, fmt, fmt, G, phases=False)
    err = normalised_error(c.cpu().numpy()[np.ix_(ii, jj)], ref["C"], oracle.row_norms(ah, sah, fmt, G),
                           oracle.row_norms(bh, sbh, fmt, G))
    assert err <= 1e-5, err
