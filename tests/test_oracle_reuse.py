"""Pins for the oracle's per-element-scale GEMM (reused operands of the
training GEMMs, Sec. 4): the backward GEMMs take the forward pass's quantized
operands, one of them transposed, so the scale of an operand element follows
the element, not the GEMM's K.

Checked against real dot products of the decoded values (Eq. 1) computed to
80 digits, against the block-scale GEMM where the two definitions coincide,
and against the three training GEMMs written as plain loops over decoded
values (forward, dgrad, wgrad), so that a transposed operand or a scale read
from the wrong block fails.
"""
from decimal import Decimal

import numpy as np
import pytest

from tests import exact as X

FORMATS = ["E3C3", "E4C3", "E5C2"]


def _dec(fmt, code, a):
    f = X.FMT[fmt]
    m = int(code) & (0x3F if fmt == "E3C3" else 0x7F)
    if m == 0:
        return Decimal(0)
    v = X.level(fmt, m - f["B"]) * Decimal(2) ** int(a)
    return -v if int(code) >> 7 else v


def _codes(rng, fmt, shape):
    c = rng.integers(0, 256, size=shape, dtype=np.uint8)
    if fmt == "E3C3":
        c &= 0xBF
    return c


def _check_real(oracle, r, va, vb, L):
    S = oracle.int128_to_int(r["S_raw"])
    M, N = len(va), len(vb)
    for i in range(M):
        for j in range(N):
            ref = sum(x * y for x, y in zip(va[i], vb[j]))
            lam = int(r["lsb"][i, j])
            got = sum(X.pow2(h, L) * Decimal(int(S[i, j, h])) for h in range(L)) * Decimal(2) ** lam
            assert abs(got - ref) <= Decimal(10) ** -60 * (1 + abs(ref))
            assert not r["range"][i, j]
            assert abs(r["C"][i, j] - float(ref)) <= 1e-15 * max(1.0, abs(float(ref))) * 8


@pytest.mark.parametrize("fa,fb", [("E4C3", "E4C3"), ("E5C2", "E4C3"), ("E3C3", "E5C2")])
def test_elem_phase_sums_match_real_dot_products(oracle, fa, fb):
    """Per-element scales drawn independently for every element: the phase
    sums recombine to the 80-digit dot product of the decoded values, and the
    exported LSB is the smallest per-product scale sum plus t_min."""
    rng = np.random.default_rng(11)
    M, N, K = 3, 4, 40
    a, b = _codes(rng, fa, (M, K)), _codes(rng, fb, (N, K))
    ea = rng.integers(-4, 5, size=(M, K)).astype(np.int8)
    eb = rng.integers(-4, 5, size=(N, K)).astype(np.int8)
    r = oracle.gemm_elem(a, ea, b, eb, fa, fb)
    L, tmin, _ = oracle.pair_info(fa, fb)
    va = [[_dec(fa, a[i, d], ea[i, d]) for d in range(K)] for i in range(M)]
    vb = [[_dec(fb, b[j, d], eb[j, d]) for d in range(K)] for j in range(N)]
    _check_real(oracle, r, va, vb, L)
    for i in range(M):
        for j in range(N):
            assert r["lsb"][i, j] == int((ea[i].astype(int) + eb[j].astype(int)).min()) + tmin


@pytest.mark.parametrize("fmt", FORMATS)
def test_block_scales_broadcast_equal_block_gemm(oracle, fmt):
    """Block scales copied to every element of their block give the
    block-scale GEMM's phase sums, LSB and combine exactly."""
    rng = np.random.default_rng(5)
    M, N, K, G = 5, 7, 128, 32
    a, b = _codes(rng, fmt, (M, K)), _codes(rng, fmt, (N, K))
    sa = rng.integers(-6, 7, size=(M, K // G)).astype(np.int8)
    sb = rng.integers(-6, 7, size=(N, K // G)).astype(np.int8)
    r0 = oracle.gemm(a, sa, b, sb, fmt, fmt, G)
    r1 = oracle.gemm_oriented(a, sa, "rows", b, sb, "rows", fmt, fmt, G)
    assert np.array_equal(r0["S_raw"], r1["S_raw"])
    assert np.array_equal(r0["lsb"], r1["lsb"])
    assert np.array_equal(r0["C"], r1["C"])


def test_training_triplet_on_reused_operands(oracle):
    """Forward Y = Q(X) Q(W)^T, dgrad dX = Q(dY) Q(W) and wgrad
    dW = Q(dY)^T Q(X) on operands quantized once (X and W blocked along the
    input features, dY along the output features), each GEMM checked against
    plain loops over the decoded values with their own block scales."""
    from paper_2608_10010_gb300 import inputs

    T, din, dout, G = 3, 64, 96, 32
    x = inputs.normal((T, din), 1)
    w = inputs.normal((dout, din), 2, 0.02)
    dy = 1e-3 * inputs.normal((T, dout), 3)
    qx, sx, _ = oracle.quantize(x, "E4C3", G, 0)   # [T x din], blocks along din
    qw, sw, _ = oracle.quantize(w, "E4C3", G, 0)   # [dout x din], blocks along din
    qg, sg, _ = oracle.quantize(dy, "E5C2", G, 0)  # [T x dout], blocks along dout
    X_ = [[_dec("E4C3", qx[t, i], sx[t, i // G]) for i in range(din)] for t in range(T)]
    W_ = [[_dec("E4C3", qw[o, i], sw[o, i // G]) for i in range(din)] for o in range(dout)]
    D_ = [[_dec("E5C2", qg[t, o], sg[t, o // G]) for o in range(dout)] for t in range(T)]

    fwd = oracle.gemm_oriented(qx, sx, "rows", qw, sw, "rows", "E4C3", "E4C3", G)
    _check_real(oracle, fwd, X_, W_, 8)

    # dgrad: dX[t, i] = sum_o dY[t, o] W[o, i]; B row i = column i of W
    dg = oracle.gemm_oriented(qg, sg, "rows", qw, sw, "cols", "E5C2", "E4C3", G)
    assert dg["C"].shape == (T, din)
    Wt = [[W_[o][i] for o in range(dout)] for i in range(din)]
    _check_real(oracle, dg, D_, Wt, 8)

    # wgrad: dW[o, i] = sum_t dY[t, o] X[t, i]
    wg = oracle.gemm_oriented(qg, sg, "cols", qx, sx, "cols", "E5C2", "E4C3", G)
    assert wg["C"].shape == (dout, din)
    Dt = [[D_[t][o] for t in range(T)] for o in range(dout)]
    Xt = [[X_[t][i] for t in range(T)] for i in range(din)]
    _check_real(oracle, wg, Dt, Xt, 8)


def test_elem_range_flag(oracle):
    """The int128 window with per-element scales: a spread of scale sums that
    cannot fit is reported and the output is NaN."""
    K = 8
    a = np.full((1, K), 0x7F, np.uint8)
    ea = np.zeros((1, K), np.int8)
    ea[0, 0], ea[0, 1] = -128, 127
    r = oracle.gemm_elem(a, ea, a, ea, "E5C2", "E5C2")
    assert r["range"][0, 0] and np.isnan(r["C"][0, 0])
    ea[0, 0], ea[0, 1] = 0, 1
    r = oracle.gemm_elem(a, ea, a, ea, "E5C2", "E5C2")
    assert not r["range"][0, 0]
