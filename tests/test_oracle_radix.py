"""Pins for the oracle's rational-radix formats (Sec. 3.1 Eq. 1 with
r = 2^{p/q}, Eq. 4, App. A.1; Table 2's E4C3 points r = 2^{8/9} and
r = 2^{3/4}).  Every check is against 80-digit arithmetic, the exponent
identity of Eq. 1, or a value the paper prints.
"""
import json
import math
import os
from decimal import Decimal
from fractions import Fraction

import numpy as np
import pytest

from tests import exact as X

RADIX = {"E4C3_R8_9": (8, 9), "E4C3_R3_4": (3, 4)}
K, B, NMAX = 8, 64, 63
GOLD = os.path.join(os.path.dirname(__file__), "golden")
# a block whose maximum is this anchor has scale 0 (L_nmax = 128 and 2^{189/32})
ANCHOR = {"E4C3_R8_9": 100.0, "E4C3_R3_4": 50.0}


def lvl(fmt, n):
    p, q = RADIX[fmt]
    return X.pow2(p * n, q * K)


def nearest(fmt, v):
    """80-digit argmin over {0} U {levels}; ties to the smaller magnitude."""
    best, bestd = 0, abs(v)
    for n in range(-NMAX, NMAX + 1):
        d = abs(v - lvl(fmt, n))
        if d < bestd:
            best, bestd = n + B, d
    return best


def quant_one_block(oracle, fmt, vals):
    vals = np.asarray(vals, np.float32)
    per = 31
    nblk = -(-len(vals) // per)
    x = np.zeros((nblk, 32), np.float32)
    x[:, 0] = ANCHOR[fmt]
    flat = x[:, 1:].reshape(-1)
    flat[: len(vals)] = vals
    x[:, 1:] = flat.reshape(nblk, per)
    codes, scales, _ = oracle.quantize(x, fmt, 32)
    assert np.all(scales == 0)
    return codes[:, 1:].reshape(-1)[: len(vals)]


def test_table7_phase_counts(oracle):
    """Table 2 (radix frontier): E4C3 with r = 2^{8/9} needs 9 phases and
    r = 2^{3/4} needs 32; the oracle's lattice for each format has exactly
    that many phases, and every phase class is reached by some product (the
    subgroup argument of App. A.1)."""
    with open(os.path.join(GOLD, "radix_frontier_phases.json")) as fh:
        g = json.load(fh)
    want = {(c["p"], c["q"]): c["H"] for c in g["cases"]}
    for fmt, (p, q) in RADIX.items():
        H = oracle.pair_info(fmt, fmt)[0]
        assert H == want[(p, q)]
        seen = {oracle.closed_product(fmt, fmt, 64 + na, 64 + 1)[2] for na in range(-NMAX, NMAX + 1)}
        assert seen == set(range(H))
    with pytest.raises(ValueError):
        oracle.pair_info("E4C3_R8_9", "E4C3")


@pytest.mark.parametrize("fmt", list(RADIX))
def test_levels(oracle, fmt):
    """Eq. 1: level n is r^{n/K} = 2^{p n/(qK)} (fp64 within one ulp of the
    80-digit value); adjacent levels differ by r^{1/K}, adjacent exponents
    (n and n + K) by r."""
    lv = oracle.levels(fmt)
    assert len(lv) == 2 * NMAX + 1
    for i, v in enumerate(lv):
        assert abs(Decimal(float(v)) - lvl(fmt, i - NMAX)) <= Decimal(math.ulp(float(v)))
    p, q = RADIX[fmt]
    assert np.allclose(lv[1:] / lv[:-1], 2.0 ** (p / (q * K)), rtol=4e-16)
    assert np.allclose(lv[K:] / lv[:-K], 2.0 ** (p / q), rtol=4e-16)


@pytest.mark.parametrize("fmt", list(RADIX))
def test_closed_product_exponent_identity(oracle, fmt):
    """App. A.1: every nonzero product is delta 2^{t + h/H}, with
    t + h/H equal (as a rational number) to the product's exponent
    p (n_a + n_b)/(qK) from Eq. 1; zero codes give no update."""
    p, q = RADIX[fmt]
    H = oracle.pair_info(fmt, fmt)[0]
    for ca in range(0, 256, 3):
        for cb in range(256):
            nz, d, h, t = oracle.closed_product(fmt, fmt, ca, cb)
            ma, mb = ca & 0x7F, cb & 0x7F
            if ma == 0 or mb == 0:
                assert nz == 0
                continue
            assert 0 <= h < H
            assert Fraction(t) + Fraction(h, H) == Fraction(p * (ma - B + mb - B), q * K)
            assert d == (-1 if (ca ^ cb) & 0x80 else 1)


@pytest.mark.parametrize("fmt", list(RADIX))
def test_block_scale_is_ceil_absmax(oracle, fmt):
    top = lvl(fmt, NMAX)
    rng = np.random.default_rng(3)
    amaxes = list(rng.lognormal(0, 8, 1000).astype(np.float32))
    amaxes += list(np.float32(2.0) ** np.arange(-100, 100, dtype=np.float32))
    for F in (-20, 0, 9):  # straddle the switch point L_nmax 2^F
        s = np.float32(float(top * Decimal(2) ** F))
        amaxes += [np.nextafter(s, np.float32(0)), s, np.nextafter(s, np.float32(np.inf))]
    for am in amaxes:
        a = oracle.block_scale(fmt, float(am))
        A = Decimal(float(am))
        assert A <= top * Decimal(2) ** a
        if a > -128:
            assert A > top * Decimal(2) ** (a - 1)


@pytest.mark.parametrize("fmt", list(RADIX))
def test_nearest_level_adversarial(oracle, fmt):
    """FP32 neighbours of every midpoint, of the zero boundary L_nmin/2 and
    random values: oracle rank == 80-digit argmin (R3; for r = 2^{8/9} the
    zero boundary is the exact power of two 2^{-8}, a tie that R14 sends to
    zero)."""
    probes = []
    for n in range(-NMAX - 1, NMAX):
        mid = (lvl(fmt, n) + lvl(fmt, n + 1)) / 2 if n >= -NMAX else lvl(fmt, -NMAX) / 2
        m32 = np.float32(float(mid))
        probes += [np.nextafter(m32, np.float32(0)), m32, np.nextafter(m32, np.float32(np.inf))]
    rng = np.random.default_rng(5)
    top = float(lvl(fmt, NMAX))
    probes += list(rng.uniform(0, top, 300).astype(np.float32))
    probes += list((2.0 ** rng.uniform(-10, 0, 300)).astype(np.float32))
    probes = np.array(probes, np.float32)
    probes = probes[probes <= np.float32(top)]
    codes = quant_one_block(oracle, fmt, probes)
    for v, c in zip(probes, codes):
        assert int(c) == nearest(fmt, Decimal(float(v))), (fmt, float(v))
    if fmt == "E4C3_R8_9":
        c = quant_one_block(oracle, fmt, [np.float32(2.0 ** -8), np.nextafter(np.float32(2.0 ** -8), np.float32(1))])
        assert int(c[0]) == 0 and int(c[1]) == 1


def test_fp64_decisions_have_margin():
    """fp64 level arithmetic decides every FP32 input exactly: each midpoint
    of two adjacent rational-radix levels, each irrational zero boundary and
    scale switch point lies more than 2^-46 (relative) from every 25-bit
    dyadic, while fp64 errors stay below 2^-50."""
    worst = Decimal(1)
    for fmt in RADIX:
        for n in range(-NMAX, NMAX):
            mid = (lvl(fmt, n) + lvl(fmt, n + 1)) / 2
            e = int(math.floor(math.log2(float(mid))))
            worst = min(worst, X.dyadic_margin(mid / Decimal(2) ** e, 25))
    r34 = lvl("E4C3_R3_4", NMAX)
    worst = min(worst, X.dyadic_margin(r34 / Decimal(2) ** 5, 25))
    z34 = lvl("E4C3_R3_4", -NMAX) / 2
    worst = min(worst, X.dyadic_margin(z34 * Decimal(2) ** 7, 25))
    assert worst > Decimal(2) ** -46


@pytest.mark.parametrize("fmt", list(RADIX))
def test_dequantize_definition(oracle, fmt):
    """R4 with the rational exponent (R14): RN32(2^{j/(qK)}) 2^{a + floor(p n/(qK))},
    j = p n mod qK, compared with an 80-digit evaluation rounded once."""
    p, q = RADIX[fmt]
    codes = np.tile(np.arange(256, dtype=np.uint8), 5)[None, :]
    svals = [-128, -20, 0, 9, 120]
    scales = np.repeat(np.array(svals, np.int8), 8)[None, :]
    out = oracle.dequantize(codes, scales, fmt, 32)
    for c in range(codes.shape[1]):
        code = int(codes[0, c])
        a = svals[c // 256]
        m = code & 0x7F
        if m == 0:
            assert out[0, c] == 0.0
            continue
        n = m - B
        e, j = (p * n) // (q * K), (p * n) % (q * K)
        cj = X.rn32_mantissa(j, q * K) / float(1 << 23)
        with np.errstate(over="ignore"):
            want = np.float32(math.ldexp(cj, a + e) * (-1 if code >> 7 else 1))
        assert out[0, c] == want or (np.isinf(want) and np.isinf(out[0, c]))


@pytest.mark.parametrize("fmt", list(RADIX))
def test_phase_sums_match_real_dot_products(oracle, fmt):
    """Eq. 5 with H = 9 or 32 phases: sum_h 2^{h/H} S_h 2^lambda equals the
    80-digit dot product of the decoded values; 1, 2^{1/H}, ..., 2^{(H-1)/H}
    are linearly independent over the rationals, so a wrong phase, bin, sign
    or scale in any S_h shows up."""
    rng = np.random.default_rng(9)
    M, N, Kd, G = 3, 3, 64, 32
    a = rng.integers(0, 256, size=(M, Kd), dtype=np.uint8)
    b = rng.integers(0, 256, size=(N, Kd), dtype=np.uint8)
    sa = rng.integers(-3, 4, size=(M, Kd // G)).astype(np.int8)
    sb = rng.integers(-3, 4, size=(N, Kd // G)).astype(np.int8)
    r = oracle.gemm(a, sa, b, sb, fmt, fmt, G)
    S = oracle.int128_to_int(r["S_raw"])
    H = S.shape[2]

    def dec(code, s):
        m = int(code) & 0x7F
        if m == 0:
            return Decimal(0)
        v = lvl(fmt, m - B) * Decimal(2) ** int(s)
        return -v if int(code) >> 7 else v

    for i in range(M):
        for j in range(N):
            ref = sum(dec(a[i, d], sa[i, d // G]) * dec(b[j, d], sb[j, d // G]) for d in range(Kd))
            got = sum(X.pow2(h, H) * Decimal(int(S[i, j, h])) for h in range(H)) * Decimal(2) ** int(r["lsb"][i, j])
            assert abs(got - ref) <= Decimal(10) ** -60 * (1 + abs(ref))
            assert abs(r["C"][i, j] - float(ref)) <= 1e-15 * max(1.0, abs(float(ref))) * 8
