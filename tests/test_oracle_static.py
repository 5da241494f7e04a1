"""Pins for the oracle's static-operand quantization (Sec. 3.1: MSE-search
power-of-two scales for static operands; Sec. 4.2: tensorwise, rowwise and
block scale granularity).  The MSE choice is checked against an exact
rational computation of the reconstruction error, not against the oracle's
own integer criterion."""
from fractions import Fraction

import numpy as np
import pytest

import oracle

FORMATS = ["E3C3", "E4C3", "E5C2"]


def exact_sse(x, xhat):
    """Sum of squared reconstruction errors, exactly (Fractions of the FP32 values)."""
    return sum((Fraction(float(a)) - Fraction(float(b))) ** 2 for a, b in zip(x, xhat))


def recon(x_row, a, fmt):
    """Codes of one group at scale a (oracle encode, R3) and their R4 reconstruction."""
    n = len(x_row)
    sc = np.full((1, 1), a, np.int8)
    codes, _ = oracle.encode(x_row.reshape(1, n), sc, fmt, n)
    return oracle.dequantize(codes, sc, fmt, n).reshape(-1)


@pytest.mark.parametrize("fmt", FORMATS)
def test_ceil_block_is_the_dynamic_quantizer(fmt):
    x = (np.random.default_rng(1).standard_normal((16, 256)) * 0.02).astype(np.float32)
    c0, s0, _ = oracle.quantize(x, fmt, 32, 0)
    c1, s1, _ = oracle.quantize_static(x, fmt, 32, "block", "ceil")
    assert np.array_equal(c0, c1) and np.array_equal(s0, s1)


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("gran", ["row", "tensor"])
def test_ceil_row_and_tensor_scales(fmt, gran):
    """Rowwise / tensorwise ceil-absmax: one scale = the ceil-absmax scale of
    the group's max (closed form of R2), stored in every block of the group,
    and every element encoded under it."""
    rng = np.random.default_rng(2)
    x = (rng.standard_normal((12, 192)) * np.exp(rng.standard_normal((12, 1)) * 2)).astype(np.float32)
    codes, scales, _ = oracle.quantize_static(x, fmt, 32, gran, "ceil")
    if gran == "row":
        want = np.array([oracle.block_scale(fmt, float(np.abs(r).max())) for r in x], np.int8)
        assert np.all(scales == want[:, None])
    else:
        assert np.all(scales == oracle.block_scale(fmt, float(np.abs(x).max())))
    ref, _ = oracle.encode(x, scales, fmt, 32)
    assert np.array_equal(codes, ref)


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("gran,shape", [("block", (24, 64)), ("row", (10, 96)), ("tensor", (4, 64))])
def test_mse_choice_minimises_exact_reconstruction_error(fmt, gran, shape):
    """The chosen scale's exact sum of squared FP32 reconstruction errors is
    the smallest over the candidates a_c - 3 .. a_c + 1 (up to the 2^-60
    grid of R12); equal minima go to the larger scale."""
    rng = np.random.default_rng(3)
    # heavy-tailed groups spanning more binades than the format covers, so
    # that lower scales (fewer flushes to zero) sometimes beat ceil-absmax
    spread = {"E3C3": 1.5, "E4C3": 3.5, "E5C2": 7.0}[fmt]
    x = (rng.standard_normal(shape) * np.exp(rng.standard_normal(shape) * spread)).astype(np.float32)
    codes, scales, _ = oracle.quantize_static(x, fmt, 32, gran, "mse")
    flat = x.reshape(-1)
    glen = {"block": 32, "row": shape[1], "tensor": flat.size}[gran]
    chosen_below_ceil = 0
    for g in range(flat.size // glen):
        grp = flat[g * glen:(g + 1) * glen]
        ac = oracle.block_scale(fmt, float(np.abs(grp).max()))
        a = int(scales.reshape(-1)[(g * glen) // 32])
        assert ac - 3 <= a <= ac + 1
        sse = {c: exact_sse(grp, recon(grp, c, fmt)) for c in range(ac - 3, ac + 2)}
        best = min(sse.values())
        tol = Fraction(2) ** (2 * ac - 60) * glen
        assert sse[a] <= best + tol
        # no larger candidate is strictly better, and no candidate beats it by more than the grid
        assert all(sse[c] >= sse[a] - tol for c in sse)
        chosen_below_ceil += a < ac
    if gran == "block":
        assert chosen_below_ceil > 0  # the search does move scales below ceil-absmax


@pytest.mark.parametrize("fmt", FORMATS)
def test_mse_tie_goes_to_the_larger_scale(fmt):
    """A block of exact levels in the middle of the range reconstructs exactly
    at a_c and at a_c + 1 (the codebook shifts by one binade), so D ties at 0
    and the larger scale is chosen."""
    levels = oracle.levels(fmt)
    mid = levels[len(levels) // 2: len(levels) // 2 + 8]  # around 2^0
    x = np.tile(np.concatenate([mid, -mid]), 2)[:32].astype(np.float32).reshape(1, 32)
    # block max just below the top level at scale -1 (RN32 of the top level
    # itself rounds up, which would move a_c to 0): a_c = -1 for every format
    x[0, 0] = np.nextafter(np.float32(levels[-1] * 0.5), np.float32(0))
    ac = oracle.block_scale(fmt, float(np.abs(x).max()))
    _, scales, _ = oracle.quantize_static(x, fmt, 32, "block", "mse")
    assert ac == -1 and int(scales[0, 0]) == ac + 1


@pytest.mark.parametrize("fmt", FORMATS)
def test_mse_special_groups(fmt):
    """All-zero groups keep scale 0 and codes 0; groups with Inf keep the
    ceil-absmax scale (127); NaN is encoded 0 and flagged."""
    x = np.zeros((3, 32), np.float32)
    x[1, 3] = np.inf
    x[2, 5] = np.nan
    x[2, 6] = 1.0
    codes, scales, nan = oracle.quantize_static(x, fmt, 32, "block", "mse")
    assert nan and scales[0, 0] == 0 and not codes[0].any()
    assert scales[1, 0] == 127 and codes[2, 5] == 0


@pytest.mark.parametrize("fmt", ["E3C3", "E4C3", "E5C2", "E4C3_R8_9"])
def test_block_ceil_is_the_quantizer(oracle, fmt):
    """R11: a block scale group with the ceil-absmax rule is Q(X) itself (the
    C ABI routes it to the streaming quantizer)."""
    from paper_2608_10010_gb300 import inputs

    x = inputs.elementwise_outliers((24, 256), 31)
    c0, s0, n0 = oracle.quantize(x, fmt, 32, 0)
    c1, s1, n1 = oracle.quantize_static(x, fmt, 32, "block", "ceil")
    assert np.array_equal(c0, c1) and np.array_equal(s0, s1) and n0 == n1
