"""GPU parity of the GEMMs on reused operands (Sec. 4, training GEMMs: the
backward pass reuses the forward pass's quantized operands, one of them
transposed), through the C ABI (curvefp_gemm_oriented).

Integer work is bit-exact (the exact path's int128 phase sums and LSBs against
the oracle's per-element-scale GEMM); the tensor-core path's FP32 output is
within 1e-5 of the oracle's fp64 combine, normalised by the operand row norms.
"""
import numpy as np
import pytest

import oracle
from paper_2608_10010_gb300 import inputs
from tests.gpu_util import new_status, normalised_error, status_bits, to_dev, torch_cuda

pytestmark = pytest.mark.gpu
TOL = 1e-5
LAYOUTS = [("rows", "rows"), ("rows", "cols"), ("cols", "rows"), ("cols", "cols")]


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


def stored(x, fmt, block):
    """Quantize a stored matrix once along its rows' contiguous axis (blocks
    along columns), as the forward pass does."""
    c, s, _ = oracle.quantize(x, fmt, block, 0)
    return c, s


def operand(rng_seed, fmt, R, K, layout, block, dist="normal"):
    """Codes and scales of an operand with R GEMM rows in the given layout."""
    shape = (R, K) if layout == "rows" else (K, R)
    if dist == "outlier":
        x = inputs.outlier_channels(shape, rng_seed)
    elif dist == "grad":
        x = inputs.heavy_tailed_grad(shape, rng_seed)
    else:
        x = inputs.normal(shape, rng_seed)
    return stored(x, fmt, block)


def norms(codes, scales, layout, fmt, block):
    """||row||_2 of each GEMM row of an operand (fp64 of the FP32
    dequantization)."""
    v = oracle.dequantize(codes, scales, fmt, block).astype(np.float64)
    return np.sqrt((v * v).sum(axis=1 if layout == "rows" else 0))


def run(torch, a, sa, la, b, sb, lb, fa, fb, block, algo, phases=False):
    import paper_2608_10010_gb300 as cfp

    st = new_status(torch)
    out = cfp.gemm_oriented(to_dev(torch, a), to_dev(torch, sa), la, to_dev(torch, b), to_dev(torch, sb), lb, fa, fb,
                            block, algo, phases=phases, status=st)
    torch.cuda.synchronize()
    if phases:
        c, ps, pl = out
        return c.cpu().numpy(), ps.cpu().numpy(), pl.cpu().numpy(), status_bits(st)
    return out.cpu().numpy(), status_bits(st)


@pytest.mark.parametrize("la,lb", LAYOUTS)
@pytest.mark.parametrize("fa,fb,block", [("E4C3", "E4C3", 32), ("E5C2", "E4C3", 32), ("E3C3", "E5C2", 64)])
def test_exact_oriented_phase_sums(torch, la, lb, fa, fb, block):
    """Exact path: phase sums, LSBs and C bit-identical to the oracle, both
    layouts of both operands; M, N, K ragged against the 16 x 16 x 32 tiles."""
    # COLS row counts are multiples of the block; K is free when neither
    # operand is blocked along it
    M = 200 if la == "rows" else 192
    N = 136 if lb == "rows" else 128
    K = 200 if la == lb == "cols" else (160 if block == 32 else 192)
    a, sa = operand(1, fa, M, K, la, block, "outlier")
    b, sb = operand(2, fb, N, K, lb, block)
    c, ps, pl, bits = run(torch, a, sa, la, b, sb, lb, fa, fb, block, "exact", phases=True)
    ref = oracle.gemm_oriented(a, sa, la, b, sb, lb, fa, fb, block)
    assert bits == 0
    assert np.array_equal(ps, ref["S_raw"])
    assert np.array_equal(pl, ref["lsb"])
    assert np.array_equal(c, ref["C"].astype(np.float32))


@pytest.mark.parametrize("la,lb", LAYOUTS[1:])
@pytest.mark.parametrize("fa,fb", [("E3C3", "E3C3"), ("E4C3", "E4C3"), ("E5C2", "E4C3"), ("E4C3", "E5C2"),
                                   ("E5C2", "E5C2")])
def test_tensor_oriented_within_tolerance(torch, la, lb, fa, fb):
    """Tensor-core path with per-element scales: C within 1e-5 (normalised)
    of the oracle; M = 224 and N = 320 leave partial 128 x 96 tiles."""
    block = 32
    M, N, K = 224, 320, 512
    a, sa = operand(3, fa, M, K, la, block, "outlier")
    b, sb = operand(4, fb, N, K, lb, block, "grad" if fb == "E5C2" else "normal")
    c, bits = run(torch, a, sa, la, b, sb, lb, fa, fb, block, "tensor")
    ref = oracle.gemm_oriented(a, sa, la, b, sb, lb, fa, fb, block, phases=False)
    assert bits == 0
    err = normalised_error(c, ref["C"], norms(a, sa, la, fa, block), norms(b, sb, lb, fb, block))
    assert err <= TOL, err


@pytest.mark.parametrize("fa,fb", [("E4C3", "E4C3"), ("E5C2", "E4C3")])
def test_tensor_per_element_path_matches_block_path_bit_for_bit(torch, fa, fb):
    """A COLS operand whose scales do not change along its stored rows is the
    same operand as a ROWS one with those scales per block: the per-element
    tensor-core path then decodes the same planes as the block-scale path,
    so C is bit-identical."""
    import paper_2608_10010_gb300 as cfp

    block, M, N, K = 32, 256, 192, 256
    a, sa = operand(5, fa, M, K, "rows", block, "outlier")
    rng = np.random.default_rng(6)
    bt = rng.integers(0, 256, size=(K, N), dtype=np.uint8)  # stored [K x N]
    q = rng.integers(-3, 4, size=N // block).astype(np.int8)
    sbt = np.tile(q, (K, 1))                                 # [K x N/block], constant along K
    b_rows = np.ascontiguousarray(bt.T)
    sb_rows = np.tile(np.repeat(q, block)[:, None], (1, K // block))  # [N x K/block]
    assert sb_rows.shape == (N, K // block)
    c1, bits1 = run(torch, a, sa, "rows", bt, sbt, "cols", fa, fb, block, "tensor")
    st = new_status(torch)
    c0 = cfp.gemm(to_dev(torch, a), to_dev(torch, sa), to_dev(torch, b_rows), to_dev(torch, sb_rows), fa, fb, block,
                  "tensor", status=st).cpu().numpy()
    assert bits1 == 0 and status_bits(st) == 0
    assert np.array_equal(c0.view(np.uint32), c1.view(np.uint32))


def test_training_triplet_reused_operands(torch):
    """Forward, dgrad and wgrad on operands quantized once (X and W along the
    input features, dY along the output features; E4C3 / E5C2): exact phase
    sums bit-exact and tensor-core C within tolerance for all three GEMMs."""
    T, din, dout, G = 256, 512, 384, 32
    x = inputs.normal((T, din), 7)
    w = inputs.normal((dout, din), 8, 0.02)
    dy = inputs.heavy_tailed_grad((T, dout), 9)
    qx, sx = stored(x, "E4C3", G)
    qw, sw = stored(w, "E4C3", G)
    qg, sg = stored(dy, "E5C2", G)
    gemms = [
        ("fwd", qx, sx, "rows", "E4C3", qw, sw, "rows", "E4C3"),
        ("dgrad", qg, sg, "rows", "E5C2", qw, sw, "cols", "E4C3"),
        ("wgrad", qg, sg, "cols", "E5C2", qx, sx, "cols", "E4C3"),
    ]
    for name, a, sa, la, fa, b, sb, lb, fb in gemms:
        ref = oracle.gemm_oriented(a, sa, la, b, sb, lb, fa, fb, G)
        c, ps, pl, bits = run(torch, a, sa, la, b, sb, lb, fa, fb, G, "exact", phases=True)
        assert bits == 0, name
        assert np.array_equal(ps, ref["S_raw"]) and np.array_equal(pl, ref["lsb"]), name
        ct, bits = run(torch, a, sa, la, b, sb, lb, fa, fb, G, "tensor")
        assert bits == 0, name
        err = normalised_error(ct, ref["C"], norms(a, sa, la, fa, G), norms(b, sb, lb, fb, G))
        assert err <= TOL, (name, err)


def test_training_triplet_full_size_sampled(torch):
    """The training GEMMs at full size (4096 tokens, 4096 -> 11008 features),
    operands quantized once on the GPU, each backward GEMM in the launch
    configuration the benchmark times; 48 x 48 sampled outputs checked
    against the oracle."""
    import paper_2608_10010_gb300 as cfp

    G = 32
    X, Wt, dY = inputs.training_triplet_cuda()          # X [T x din], W [din x dout], dY [T x dout]
    W = Wt.t().contiguous()                             # [dout x din]
    qx, sx = cfp.quantize(X, "E4C3", G, 0)
    qw, sw = cfp.quantize(W, "E4C3", G, 0)
    qg, sg = cfp.quantize(dY, "E5C2", G, 0)
    del X, Wt, W, dY
    rng = np.random.default_rng(10)
    host = {k: v.cpu().numpy() for k, v in dict(qx=qx, sx=sx, qw=qw, sw=sw, qg=qg, sg=sg).items()}
    cases = [
        ("dgrad", "qg", "sg", "rows", "E5C2", "qw", "sw", "cols", "E4C3"),
        ("wgrad", "qg", "sg", "cols", "E5C2", "qx", "sx", "cols", "E4C3"),
    ]
    for name, ka, ksa, la, fa, kb, ksb, lb, fb in cases:
        st = new_status(torch)
        dev = dict(qx=qx, sx=sx, qw=qw, sw=sw, qg=qg, sg=sg)
        c = cfp.gemm_oriented(dev[ka], dev[ksa], la, dev[kb], dev[ksb], lb, fa, fb, G, "tensor", status=st)
        torch.cuda.synchronize()
        assert status_bits(st) == 0, name
        M, N = c.shape
        ii = np.sort(rng.choice(M, 48, replace=False))
        jj = np.sort(rng.choice(N, 48, replace=False))
        ca, ea = oracle.operand_view(host[ka], host[ksa], G, la)
        cb, eb = oracle.operand_view(host[kb], host[ksb], G, lb)
        ref = oracle.gemm_elem(ca[ii], ea[ii], cb[jj], eb[jj], fa, fb, phases=False)
        got = c.cpu().numpy()[np.ix_(ii, jj)]
        va = oracle.dequantize(host[ka], host[ksa], fa, G).astype(np.float64)
        vb = oracle.dequantize(host[kb], host[ksb], fb, G).astype(np.float64)
        na = np.sqrt((va * va).sum(axis=1 if la == "rows" else 0))[ii]
        nb = np.sqrt((vb * vb).sum(axis=1 if lb == "rows" else 0))[jj]
        err = normalised_error(got, ref["C"], na, nb)
        assert err <= TOL, (name, err)
