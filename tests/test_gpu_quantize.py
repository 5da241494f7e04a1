"""GPU quantizer / dequantizer parity: bit-exact codes and scales against the
oracle, through the C ABI."""
import numpy as np
import pytest

import oracle
from paper_2608_10010_gb300 import inputs
from tests.gpu_util import new_status, status_bits, to_dev, torch_cuda, widen

pytestmark = pytest.mark.gpu
FORMATS = ["E3C3", "E4C3", "E5C2"]


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


def run_q(torch, x, fmt, block=32, axis=0, dtype="f32"):
    import paper_2608_10010_gb300 as cfp

    xd = to_dev(torch, x, dtype)
    st = new_status(torch)
    codes, scales = cfp.quantize(xd, fmt, block, axis, status=st)
    torch.cuda.synchronize()
    return codes.cpu().numpy(), scales.cpu().numpy(), status_bits(st), widen(torch, xd)


def check_q(torch, x, fmt, block=32, axis=0, dtype="f32"):
    c, s, st, xw = run_q(torch, x, fmt, block, axis, dtype)
    rc, rs, nan = oracle.quantize(xw, fmt, block, axis)
    assert np.array_equal(s, rs), (fmt, block, axis, dtype)
    assert np.array_equal(c, rc), (fmt, block, axis, dtype)
    assert bool(st & 1) == nan
    return c, s


def test_small_e4c3_workload(torch):
    """CurveFP8 E4C3 block 32: A[128x256] (blocks along K = columns) and
    B[256x128] (blocks along K = rows, transposed output), N(0,1)."""
    A, B = inputs.small_e4c3()
    check_q(torch, A, "E4C3", 32, 0)
    check_q(torch, B, "E4C3", 32, 1)


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("block", [32, 64, 128, 256, 512])
def test_formats_blocks_dtypes(torch, fmt, dtype, block):
    x = inputs.elementwise_outliers((37, 1024), 40 + block)
    check_q(torch, x, fmt, block, 0, dtype)
    y = inputs.elementwise_outliers((1024, 37), 41 + block)
    check_q(torch, y, fmt, block, 1, dtype)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("shape", [(1, 32), (3, 96), (1000, 4160), (257, 8192)])
def test_chunk_boundaries(torch, dtype, shape):
    """Dense rows of 32-element blocks are streamed in 16 KB chunks (256 BF16 or
    128 FP32 blocks) by persistent CTAs: a single block, less than one chunk,
    a ragged last chunk, and more chunks than resident CTAs."""
    x = inputs.elementwise_outliers(shape, 70 + shape[0])
    for fmt in FORMATS:
        check_q(torch, x, fmt, 32, 0, dtype)


@pytest.mark.parametrize("fmt", FORMATS)
def test_binade_exhaustive(torch, fmt):
    """All 2^23 FP32 mantissas of the binade [1, 2) under a fixed block scale."""
    anchor = {"E3C3": 10.0, "E4C3": 200.0, "E5C2": 40000.0}[fmt]
    mant = np.arange(1 << 23, dtype=np.uint32)
    vals = ((np.uint32(127) << np.uint32(23)) | mant).view(np.float32)
    n = len(vals)
    x = np.zeros(((n + 30) // 31, 32), np.float32)
    x[:, 0] = anchor
    flat = x[:, 1:].reshape(-1)
    flat[:n] = vals
    x[:, 1:] = flat.reshape(x.shape[0], 31)
    x[1::2] *= -1
    check_q(torch, x, fmt)


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("axis", [0, 1])
def test_special_values(torch, fmt, axis):
    """Zero blocks, signed zeros, NaN (encoded 0 and flagged), +-Inf
    (saturate), subnormal-only blocks (scale clamps to -128), values near the
    FP32 maximum, tiny blocks, and random exponents over the whole FP32 range."""
    rng = np.random.default_rng(3)
    x = np.zeros((64, 64), np.float32)
    x[1] = -0.0
    x[2, 5] = np.nan
    x[2, 6] = 1.0
    x[3, 0] = np.inf
    x[3, 1] = -np.inf
    x[3, 2] = 7.0
    x[4] = np.float32(2.0) ** -140 * rng.integers(1, 200, 64)
    x[5] = np.float32(3.0e38) * rng.uniform(-1, 1, 64).astype(np.float32)
    x[6] = (np.float32(2.0) ** rng.integers(-149, 127, 64)).astype(np.float32) * rng.choice([-1, 1], 64)
    x[7] = np.float32(1e-39) * rng.uniform(-1, 1, 64).astype(np.float32)
    x[8:] = rng.standard_normal((56, 64)).astype(np.float32) * np.float32(2.0) ** rng.integers(-130, 120, (56, 1))
    x[20, 40] = np.nan
    check_q(torch, x, fmt, 32, axis)
    check_q(torch, x, fmt, 64, axis, "bf16")


def test_strided_rows(torch):
    """ld > cols: quantize a column slice of a wider tensor."""
    import paper_2608_10010_gb300 as cfp

    full = inputs.normal((64, 192), 12)
    xd = to_dev(torch, full)[:, 32:160]
    codes, scales = cfp.quantize(xd, "E4C3", 32, 0)
    rc, rs, _ = oracle.quantize(np.ascontiguousarray(full[:, 32:160]), "E4C3", 32, 0)
    assert np.array_equal(codes.cpu().numpy(), rc) and np.array_equal(scales.cpu().numpy(), rs)
    codes, scales = cfp.quantize(xd, "E4C3", 32, 1)
    rc, rs, _ = oracle.quantize(np.ascontiguousarray(full[:, 32:160]), "E4C3", 32, 1)
    assert np.array_equal(codes.cpu().numpy(), rc) and np.array_equal(scales.cpu().numpy(), rs)


def test_bandwidth_workload_sampled(torch):
    """The quantize-only sweep at its largest size, 2^30 BF16 elements (N(0,1),
    0.1% x100 outliers, block 32), all three formats, in the launch
    configuration the benchmark uses; parity on 4096 seeded sample rows of
    4096 elements (all of each row's blocks)."""
    import paper_2608_10010_gb300 as cfp

    n, cols = 1 << 30, 4096
    x = inputs.bandwidth_tensor_cuda(n, cols, seed=3)
    rows = np.sort(np.random.default_rng(0).choice(n // cols, 4096, replace=False))
    idx = torch.from_numpy(rows).cuda()
    xs = x[idx].float().cpu().numpy()
    for fmt in FORMATS:
        codes, scales = cfp.quantize(x, fmt, 32, 0)
        torch.cuda.synchronize()
        rc, rs, _ = oracle.quantize(xs, fmt, 32, 0)
        assert np.array_equal(codes[idx].cpu().numpy(), rc)
        assert np.array_equal(scales[idx].cpu().numpy(), rs)
        del codes, scales
    del x


@pytest.mark.parametrize("fmt", FORMATS)
def test_dequantize_all_codes_all_scales(torch, fmt):
    """Every code byte under every int8 scale, bit-exact FP32 (reading R4),
    including results that overflow to Inf or fall into the subnormal range."""
    import paper_2608_10010_gb300 as cfp

    codes = np.tile(np.arange(256, dtype=np.uint8), 256).reshape(256, 256)
    if fmt == "E3C3":
        codes &= 0xBF
    scales = np.repeat(np.arange(-128, 128, dtype=np.int16).astype(np.int8), 8).reshape(256, 8)
    out = cfp.dequantize(to_dev(torch, codes), to_dev(torch, scales), fmt, 32)
    ref = oracle.dequantize(codes, scales, fmt, 32)
    assert np.array_equal(out.cpu().numpy().view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("fmt", FORMATS)
def test_dequantize_large_grid(torch, fmt):
    """8.4M random codes (more words than one pass of the grid covers, so the
    grid-stride loop runs several times) under random scales, bit-exact."""
    import paper_2608_10010_gb300 as cfp

    rng = np.random.default_rng(404)
    codes = rng.integers(0, 256, size=(4096, 2048), dtype=np.uint8)
    if fmt == "E3C3":
        codes &= 0xBF
    scales = rng.integers(-40, 40, size=(4096, 2048 // 32), dtype=np.int8)
    out = cfp.dequantize(to_dev(torch, codes), to_dev(torch, scales), fmt, 32)
    ref = oracle.dequantize(codes, scales, fmt, 32)
    assert np.array_equal(out.cpu().numpy().view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("fmt", FORMATS)
def test_roundtrip_on_gpu(torch, fmt):
    """deq(Q(x)) on the GPU equals the oracle's, and re-quantizing it with the
    GPU gives the oracle's codes (the round-trip invariants are pinned on the
    oracle)."""
    import paper_2608_10010_gb300 as cfp

    x = inputs.elementwise_outliers((96, 512), 77)
    c, s = cfp.quantize(to_dev(torch, x), fmt, 32, 0)
    d = cfp.dequantize(c, s, fmt, 32)
    rc, rs, _ = oracle.quantize(x, fmt, 32, 0)
    rd = oracle.dequantize(rc, rs, fmt, 32)
    assert np.array_equal(d.cpu().numpy(), rd)
    c2, s2 = cfp.quantize(d, fmt, 32, 0)
    rc2, rs2, _ = oracle.quantize(rd, fmt, 32, 0)
    assert np.array_equal(c2.cpu().numpy(), rc2) and np.array_equal(s2.cpu().numpy(), rs2)


def test_empty_is_noop(torch):
    import paper_2608_10010_gb300 as cfp

    x = torch.empty((0, 64), device="cuda")
    codes, scales = cfp.quantize(x, "E4C3", 32, 0)
    assert codes.shape == (0, 64)
