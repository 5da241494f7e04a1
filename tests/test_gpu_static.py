"""Static-operand quantization on the GPU (block / row / tensor scale groups,
ceil-absmax or reconstruction-MSE scales): codes and scales bit-exact against
the oracle, through the C ABI."""
import numpy as np
import pytest

import oracle
from paper_2608_10010_gb300 import inputs
from tests.gpu_util import new_status, status_bits, to_dev, torch_cuda, widen

pytestmark = pytest.mark.gpu
FORMATS = ["E3C3", "E4C3", "E5C2"]
SPREAD = {"E3C3": 1.5, "E4C3": 3.5, "E5C2": 7.0}


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


def heavy(shape, fmt, seed):
    """N(0,1) times a per-element log-normal factor wider than the format's range."""
    rng = np.random.default_rng(seed)
    return (rng.standard_normal(shape) * np.exp(rng.standard_normal(shape) * SPREAD[fmt])).astype(np.float32)


def check(torch, x, fmt, block, group, rule, dtype="f32"):
    import paper_2608_10010_gb300 as cfp

    xd = to_dev(torch, x, dtype)
    st = new_status(torch)
    codes, scales = cfp.quantize_static(xd, fmt, block, group, rule, status=st)
    torch.cuda.synchronize()
    rc, rs, nan = oracle.quantize_static(widen(torch, xd), fmt, block, group, rule)
    assert np.array_equal(scales.cpu().numpy(), rs), (fmt, block, group, rule, dtype)
    assert np.array_equal(codes.cpu().numpy(), rc), (fmt, block, group, rule, dtype)
    assert bool(status_bits(st) & 1) == nan


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("group,shape", [("block", (48, 256)), ("row", (37, 512)), ("tensor", (16, 1024))])
@pytest.mark.parametrize("rule", ["ceil", "mse"])
def test_groups_rules_formats(torch, fmt, dtype, group, shape, rule):
    check(torch, heavy(shape, fmt, 7), fmt, 32, group, rule, dtype)


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("block", [64, 512])
def test_block_sizes(torch, fmt, block):
    x = heavy((8, 1024), fmt, 8)
    check(torch, x, fmt, block, "block", "mse")
    check(torch, x, fmt, block, "row", "mse")


@pytest.mark.parametrize("fmt", FORMATS)
def test_special_groups(torch, fmt):
    """All-zero groups, Inf groups, NaN elements (encoded 0, flagged), tiny
    and huge groups."""
    x = heavy((6, 96), fmt, 9)
    x[0] = 0.0
    x[1, 5] = np.inf
    x[2, 7] = np.nan
    x[3] *= np.float32(2.0 ** -120)
    x[4] *= np.float32(2.0 ** 100)
    for group in ("block", "row", "tensor"):
        check(torch, x, fmt, 32, group, "mse")


def test_llama_weight_rowwise_mse(torch):
    """A Llama-7B-like weight W[4096x4096] ~ N(0, 0.02^2) in E3C3 with rowwise
    MSE scales, checked on 32 sampled rows (rows are independent groups)."""
    import paper_2608_10010_gb300 as cfp

    W = inputs.normal((4096, 4096), 4, 0.02)
    codes, scales = cfp.quantize_static(to_dev(torch, W), "E3C3", 32, "row", "mse")
    rows = np.sort(np.random.default_rng(1).choice(4096, 32, replace=False))
    rc, rs, _ = oracle.quantize_static(W[rows], "E3C3", 32, "row", "mse")
    assert np.array_equal(codes.cpu().numpy()[rows], rc)
    assert np.array_equal(scales.cpu().numpy()[rows], rs)
