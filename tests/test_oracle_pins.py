"""Pins for the oracle: checks against what the paper prints and what the
mathematics fixes, never against the oracle's own formulas retyped.

Each test names the passage it pins.  A plausible mistake in the oracle (a
dropped term, a wrong sign or index, a transposed operand, an off-by-one
bias) fails at least one of them.
"""
import json
import math
import os
from decimal import Decimal
from fractions import Fraction

import numpy as np
import pytest

from tests import exact as X

GOLD = os.path.join(os.path.dirname(__file__), "golden")
FORMATS = ["E3C3", "E4C3", "E5C2"]
PAIRS = [(a, b) for a in FORMATS for b in FORMATS]


def _gold(name):
    with open(os.path.join(GOLD, name)) as fh:
        return json.load(fh)


# ---- Table 1: formats, level counts, phase counts ------------------------

def test_table1_formats(oracle):
    for row in _gold("formats_table1.json")["formats"]:
        p = oracle.format_params(row["name"])
        assert (p["E"], p["C"]) == (row["E"], row["C"])
        assert 1 + p["E"] + p["C"] == row["bits"]
        lv = oracle.levels(row["name"])
        assert len(lv) == row["positive_levels"]
        assert np.all(np.diff(lv) > 0) and np.all(lv > 0)
        # Eq. 4 with binary radix p = q = 1
        assert oracle.phase_count(1, 1, p["K"]) == row["H"]
        # the oracle's GEMM lattice for a same-format pair has H phases
        assert oracle.pair_info(row["name"], row["name"])[0] == row["H"]


def test_table2_radix_phase_counts(oracle):
    g = _gold("radix_frontier_phases.json")
    for c in g["cases"]:
        assert oracle.phase_count(c["p"], c["q"], g["K"]) == c["H"]


def test_eq6_effective_rates(oracle):
    g = _gold("effective_rates.json")
    p = oracle.format_params(g["format"])
    for c in g["cases"]:
        R = 1 + p["E"] + p["C"] + c["S"] / c["G"]
        assert round(R, g["printed_decimals"]) == pytest.approx(c["R"], abs=1e-9)


# ---- Eq. 1: levels --------------------------------------------------------

@pytest.mark.parametrize("fmt", FORMATS)
def test_levels_match_high_precision(oracle, fmt):
    lv = oracle.levels(fmt)
    nmax = X.FMT[fmt]["nmax"]
    for i, v in enumerate(lv):
        n = i - nmax
        true = X.level(fmt, n)
        # fp64 exp2 within one ulp of the true level
        assert abs(Decimal(float(v)) - true) <= Decimal(math.ulp(float(v)))
    # symmetric range: L_{-n} * L_{n} == 1 (Sec. 3.1: dropped smallest level)
    assert np.allclose(lv * lv[::-1], 1.0, rtol=4e-16)
    # adjacent levels differ by the fixed ratio 2^{1/K}
    assert np.allclose(lv[1:] / lv[:-1], 2.0 ** (1.0 / X.FMT[fmt]["K"]), rtol=4e-16)


def test_q16_tile_coefficients(oracle):
    """App. C.1: the tile selects round(2^{k/8} 2^16).  The oracle's E4C3 levels
    (n = k, e = 0) give the same eight coefficients."""
    lv = oracle.levels("E4C3")
    nmax = X.FMT["E4C3"]["nmax"]
    got = [int(round(lv[nmax + k] * 65536)) for k in range(8)]
    assert got == [X.q16(k) for k in range(8)]
    assert got == [65536, 71468, 77936, 84990, 92682, 101070, 110218, 120194]


# ---- App. C.1: rank packing and product coordinate -------------------------

def test_rank_packing_and_product_coordinate(oracle):
    """App. C.1: sign in bit 7, rank m in bits 6:0, m = 0 is zero, q = m - 64 and
    the product coordinate q_p = m_a + m_b - 128 = 8e + k for E4C3.  Checked
    over all 16,384 magnitude pairs (App. C.2 verification design)."""
    design = _gold("tile_verification_design.json")
    pairs = 0
    for ma in range(128):
        nz_a, sa, ea, ka, m_a = oracle.decode_fields("E4C3", ma)
        assert m_a == ma and nz_a == (ma != 0)
        if nz_a:
            assert 8 * ea + ka == ma - 64 and 0 <= ka < 8 and -8 <= ea <= 7
        for mb in range(128):
            pairs += 1
            nz, d, h, t = oracle.closed_product("E4C3", "E4C3", ma, mb | 0x80)
            if ma == 0 or mb == 0:
                assert nz == 0
                continue
            qp = ma + mb - 128
            assert nz == 1 and d == -1
            assert (t, h) == (qp // 8, qp % 8)
    assert pairs == design["magnitude_pairs"]


# ---- Eq. 2 / App. A.1: closed product, exhaustive --------------------------

@pytest.mark.parametrize("fa,fb", PAIRS)
def test_closed_product_exhaustive(oracle, fa, fb):
    """decode(a) * decode(b) == decode(a (x) b) over all code pairs: the
    widened product (delta, h, t) reproduces the real product of the two
    decoded values (Eq. 1 values, Eq. 2 mapping, App. A.1 addressing)."""
    L, tmin, tmax = oracle.pair_info(fa, fb)
    codes = np.arange(256, dtype=np.uint8)[:, None]
    zeros = np.zeros((256, 1), np.int8)
    va = oracle.decode(codes, zeros, fa, block=1)[:, 0]
    vb = oracle.decode(codes, zeros, fb, block=1)[:, 0]
    bad = 0
    for ca in range(256):
        for cb in range(256):
            nz, d, h, t = oracle.closed_product(fa, fb, ca, cb)
            if va[ca] == 0 or vb[cb] == 0:
                bad += nz != 0
                continue
            assert 0 <= h < L and tmin <= t <= tmax
            widened = d * math.ldexp(2.0 ** (h / L), t)
            bad += not math.isclose(widened, va[ca] * vb[cb], rel_tol=1e-15)
    assert bad == 0


# ---- Sec. 3.1: ceil-absmax block scale ------------------------------------

@pytest.mark.parametrize("fmt", FORMATS)
def test_block_scale_is_ceil_absmax(oracle, fmt):
    """a is the smallest integer with amax <= 2^a L_nmax (no saturation of the
    block maximum), checked in 80-digit arithmetic."""
    f = X.FMT[fmt]
    top = X.level(fmt, f["nmax"])
    rng = np.random.default_rng(11)
    amaxes = np.concatenate([
        rng.lognormal(0, 8, 2000).astype(np.float32),
        np.float32(2.0) ** np.arange(-120, 120, dtype=np.float32),
    ])
    # values that straddle the irrational switch point 2^{(K-1)/K} 2^F
    for F in (-20, 0, 7, 30):
        s = np.float32(math.ldexp(float(X.pow2(f["K"] - 1, f["K"])), F))
        amaxes = np.append(amaxes, [np.nextafter(s, np.float32(0)), s, np.nextafter(s, np.float32(np.inf))])
    for am in amaxes:
        a = oracle.block_scale(fmt, float(am))
        A = Decimal(float(am))
        assert A <= top * Decimal(2) ** a
        if a > -128:  # the int8 container clamps tiny blocks at -128
            assert A > top * Decimal(2) ** (a - 1)
    assert oracle.block_scale(fmt, 0.0) == 0
    assert oracle.block_scale(fmt, float("inf")) == 127
    assert oracle.block_scale(fmt, 1e-44) == -128


# ---- Sec. 3.1: nearest level, brute force ---------------------------------

def _quant_one_block(oracle, fmt, vals, anchor):
    """Quantize values in blocks whose first element is a fixed anchor, so
    every block has the anchor's scale."""
    vals = np.asarray(vals, np.float32)
    per = 31
    nblk = -(-len(vals) // per)
    x = np.zeros((nblk, 32), np.float32)
    x[:, 0] = anchor
    flat = x[:, 1:].reshape(-1)
    flat[: len(vals)] = vals
    x[:, 1:] = flat.reshape(nblk, per)
    codes, scales, _ = oracle.quantize(x, fmt, 32)
    return codes[:, 1:].reshape(-1)[: len(vals)], scales[:, 0]


ANCHOR = {"E3C3": 10.0, "E4C3": 200.0, "E5C2": 40000.0}  # all give a = 0


@pytest.mark.parametrize("fmt", FORMATS)
def test_nearest_level_binade_exhaustive(oracle, fmt):
    """All 2^23 FP32 mantissas of one binade: the oracle's codes switch
    exactly at the K midpoints (2^{k/K} + 2^{(k+1)/K})/2 computed in 80-digit
    arithmetic (thresholds depend only on the mantissa)."""
    f = X.FMT[fmt]
    mant = np.arange(1 << 23, dtype=np.uint32)
    vals = ((np.uint32(127) << np.uint32(23)) | mant).view(np.float32)  # [1, 2)
    codes, scales = _quant_one_block(oracle, fmt, vals, ANCHOR[fmt])
    assert np.all(scales == 0)
    thr = np.array([X.midpoint_mantissa_threshold(f["K"], k) for k in range(f["K"])])
    j = np.searchsorted(thr, mant, side="right")  # number of thresholds <= mant
    assert np.array_equal(codes.astype(np.int64), f["B"] + j)


@pytest.mark.parametrize("fmt", FORMATS)
def test_nearest_level_adversarial(oracle, fmt):
    """FP32 neighbours of every midpoint in many binades, the zero/L_nmin
    boundary L_nmin/2, and random values: oracle rank == 80-digit argmin."""
    f = X.FMT[fmt]
    K, B, nmax = f["K"], f["B"], f["nmax"]
    probes = []
    for n in range(-nmax - K, nmax):
        lo = X.level(fmt, n) if n >= -nmax else Decimal(0)
        mid = (X.level(fmt, n) + X.level(fmt, n + 1)) / 2 if n >= -nmax else X.level(fmt, -nmax) / 2
        m32 = np.float32(float(mid))
        probes += [np.nextafter(m32, np.float32(0)), m32, np.nextafter(m32, np.float32(np.inf))]
    rng = np.random.default_rng(5)
    probes += list(rng.uniform(0, float(X.level(fmt, nmax)), 300).astype(np.float32))
    probes += list((2.0 ** rng.uniform(-nmax / K - 3, 0, 300)).astype(np.float32))
    probes = np.array(probes, np.float32)
    probes = probes[probes <= np.float32(float(X.level(fmt, nmax)))]
    sign = np.where(np.arange(len(probes)) % 2 == 0, 1, -1).astype(np.float32)
    codes, _ = _quant_one_block(oracle, fmt, probes * sign, ANCHOR[fmt])
    for v, s, c in zip(probes, sign, codes):
        want = X.nearest_rank(fmt, Decimal(float(v)))
        got_m = int(c) & 0x7F
        assert got_m == want, (fmt, float(v))
        if want:
            assert (int(c) >> 7) == (1 if s < 0 else 0)
        else:
            assert int(c) == 0


@pytest.mark.parametrize("fmt", FORMATS)
def test_special_values(oracle, fmt):
    """Zero blocks, signed zeros, NaN (encoded 0, flagged), Inf (saturates),
    subnormal-only blocks (scale clamps to -128)."""
    f = X.FMT[fmt]
    x = np.zeros((4, 32), np.float32)
    x[1, :] = -0.0
    x[2, 0] = np.inf
    x[2, 1] = 1.0
    x[2, 2] = -np.inf
    x[3, :] = np.float32(2.0) ** np.float32(-135)  # subnormal
    x[3, 1] = -x[3, 1]
    codes, scales, nan = oracle.quantize(x, fmt, 32)
    assert not nan
    assert np.all(codes[0] == 0) and np.all(codes[1] == 0) and scales[0, 0] == 0 and scales[1, 0] == 0
    assert scales[2, 0] == 127 and codes[2, 0] == 2 * f["B"] - 1 and codes[2, 1] == 0
    assert codes[2, 2] == 0x80 | (2 * f["B"] - 1)
    assert scales[3, 0] == -128
    want = X.nearest_rank(fmt, Decimal(2) ** (-135 + 128))
    assert codes[3, 0] == want and codes[3, 1] == (0x80 | want if want else 0)
    y = np.ones((1, 32), np.float32)
    y[0, 3] = np.nan
    codes, scales, nan = oracle.quantize(y, fmt, 32)
    assert nan and codes[0, 3] == 0 and codes[0, 0] != 0


def test_fp64_decisions_have_margin():
    """The oracle decides nearest levels and scales with fp64 levels.  That is
    exact for every FP32 input because every decision threshold (midpoints,
    the zero boundary L_nmin/2 and the scale switch 2^{(K-1)/K}) lies more than
    2^-46 (relative) away from every 25-bit dyadic, while fp64 level and
    distance errors stay below 2^-50."""
    worst = Decimal(1)
    for K in (4, 8):
        for k in range(K):
            worst = min(worst, X.dyadic_margin((X.pow2(k, K) + X.pow2(k + 1, K)) / 2, 25))
            if k:
                worst = min(worst, X.dyadic_margin(X.pow2(k, K), 25))
    assert worst > Decimal(2) ** -46


# ---- R4: dequantization ----------------------------------------------------

@pytest.mark.parametrize("fmt", FORMATS)
def test_dequantize_definition(oracle, fmt):
    f = X.FMT[fmt]
    codes = np.tile(np.arange(256, dtype=np.uint8), 9)[None, :]
    svals = [-128, -127, -100, -20, 0, 5, 100, 110, 127]
    scales = np.repeat(np.array(svals, np.int8), 256 // 32 * 1)[None, :]
    scales = np.repeat(np.array(svals, np.int8), 8)[None, :]
    out = oracle.dequantize(codes, scales, fmt, 32)
    for c in range(codes.shape[1]):
        code = int(codes[0, c])
        a = int(scales[0, c // 32])
        m = code & (0x3F if fmt == "E3C3" else 0x7F)
        if m == 0:
            assert out[0, c] == 0.0
            continue
        n = m - f["B"]
        e, k = n // f["K"], n % f["K"]
        ck = X.rn32_mantissa(k, f["K"]) / float(1 << 23)
        with np.errstate(over="ignore"):
            want = np.float32(math.ldexp(ck, a + e) * (-1 if code >> 7 else 1))
        assert out[0, c] == want or (np.isinf(want) and np.isinf(out[0, c]))


@pytest.mark.parametrize("fmt", FORMATS)
def test_roundtrip_idempotence(oracle, fmt):
    """Round trip Q(deq(Q(x))).

    Fixed scale: encoding deq(Q(x)) with the original block scales gives back
    the original codes (every reconstructed value is within 2^-24 of its own
    level, and levels are 2^{1/K} apart).

    Recomputed scale: a' is a-1, a or a+1.  a' = a+1 happens exactly in blocks
    whose largest rank is n_max, because RN32(2^{n_max/K}) rounds up for all
    three formats (checked here in 80-digit arithmetic); in every block the
    elements whose shifted rank stays in range keep their reconstructed
    value."""
    from paper_2608_10010_gb300 import inputs

    f = X.FMT[fmt]
    K, B, nmax = f["K"], f["B"], f["nmax"]
    assert X.rn32_mantissa(nmax % K, K) > X.pow2(nmax % K, K) * (1 << 23)
    x = inputs.elementwise_outliers((64, 256), 9)
    c1, s1, _ = oracle.quantize(x, fmt, 32)
    d1 = oracle.dequantize(c1, s1, fmt, 32)
    c_fixed, _ = oracle.encode(d1, s1, fmt, 32)
    assert np.array_equal(c_fixed, c1)

    c2, s2, _ = oracle.quantize(d1, fmt, 32)
    d2 = oracle.dequantize(c2, s2, fmt, 32)
    mask = 0x3F if fmt == "E3C3" else 0x7F
    r1 = (c1 & mask).astype(np.int64).reshape(64, -1, 32)
    r2 = (c2 & mask).astype(np.int64).reshape(64, -1, 32)
    top = r1.max(axis=2)
    delta = (s2 - s1).astype(np.int64)
    assert np.all(np.isin(delta, (-1, 0, 1)))
    assert np.array_equal(delta == 1, top == 2 * B - 1)
    assert np.all(top[delta == -1] <= 2 * B - 1 - K)
    shifted = r1 - K * delta[:, :, None]
    keep = (r1 > 0) & (shifted >= 1)
    assert np.array_equal(r2[keep], shifted[keep])
    keep_el = keep.reshape(64, -1)
    assert np.array_equal(d1[keep_el], d2[keep_el])
    assert np.array_equal(d1[r1.reshape(64, -1) == 0], d2[r1.reshape(64, -1) == 0])


def test_block_axis_one_is_transpose(oracle):
    from paper_2608_10010_gb300 import inputs

    x = inputs.normal((96, 64), 21)
    c0, s0, _ = oracle.quantize(np.ascontiguousarray(x.T), "E4C3", 32, block_axis=0)
    c1, s1, _ = oracle.quantize(x, "E4C3", 32, block_axis=1)
    assert np.array_equal(c0, c1) and np.array_equal(s0, s1)


# ---- Eq. 5 / App. A.1: per-phase accumulation ------------------------------

def _random_operand(rng, fmt, rows, K, G, spread=3):
    codes = rng.integers(0, 256, size=(rows, K), dtype=np.uint8)
    if fmt == "E3C3":
        codes &= 0xBF
    scales = rng.integers(-spread, spread + 1, size=(rows, K // G)).astype(np.int8)
    return codes, scales


@pytest.mark.parametrize("fa,fb", PAIRS)
def test_phase_sums_match_real_dot_products(oracle, fa, fb):
    """S_h pinned individually: sum_h 2^{h/L} S_h 2^lambda equals the 80-digit
    real dot product of the decoded operands (Eq. 1 values multiplied
    directly, no phase bookkeeping).  Because 1, 2^{1/L}, ..., 2^{(L-1)/L}
    are linearly independent over the rationals (y^L - 2 is irreducible), a
    wrong phase address, bin, sign or scale in any S_h shows up."""
    rng = np.random.default_rng(7)
    M, N, K, G = 3, 4, 64, 32
    a, sa = _random_operand(rng, fa, M, K, G)
    b, sb = _random_operand(rng, fb, N, K, G)
    r = oracle.gemm(a, sa, b, sb, fa, fb, G)
    S = oracle.int128_to_int(r["S_raw"])
    L = S.shape[2]
    va = [[_dec(fa, a[i, d], sa[i, d // G]) for d in range(K)] for i in range(M)]
    vb = [[_dec(fb, b[j, d], sb[j, d // G]) for d in range(K)] for j in range(N)]
    for i in range(M):
        for j in range(N):
            ref = sum(va[i][d] * vb[j][d] for d in range(K))
            lam = int(r["lsb"][i, j])
            got = sum(X.pow2(h, L) * Decimal(int(S[i, j, h])) for h in range(L)) * Decimal(2) ** lam
            assert abs(got - ref) <= Decimal(10) ** -60 * (1 + abs(ref))
            assert not r["range"][i, j]
            assert abs(r["C"][i, j] - float(ref)) <= 1e-15 * max(1.0, abs(float(ref))) * 8


def _dec(fmt, code, a):
    f = X.FMT[fmt]
    m = int(code) & (0x3F if fmt == "E3C3" else 0x7F)
    if m == 0:
        return Decimal(0)
    v = X.level(fmt, m - f["B"]) * Decimal(2) ** int(a)
    return -v if int(code) >> 7 else v


@pytest.mark.parametrize("fmt", FORMATS)
def test_powers_of_two_reduce_to_integer_gemm(oracle, fmt):
    """Special case: with every curve index k = 0 the values are signed powers
    of two, only phase 0 is populated, and S_0 2^lambda equals a plain exact
    integer matrix product."""
    f = X.FMT[fmt]
    rng = np.random.default_rng(3)
    M, N, K, G = 5, 6, 96, 32

    def op(rows, seed_shift):
        e = rng.integers(-(f["emax"] + 1) + 1, f["emax"] + 1, size=(rows, K))
        m = (e + f["emax"] + 1) * f["K"]  # k = 0
        s = rng.integers(0, 2, size=(rows, K))
        z = rng.random((rows, K)) < 0.1
        codes = np.where(z, 0, (s << 7) | m).astype(np.uint8)
        scales = rng.integers(-2, 3, size=(rows, K // G)).astype(np.int8)
        return codes, scales, e, s, z

    a, sa, ea, sga, za = op(M, 0)
    b, sb, eb, sgb, zb = op(N, 1)
    r = oracle.gemm(a, sa, b, sb, fmt, fmt, G)
    S = oracle.int128_to_int(r["S_raw"])
    assert all(int(v) == 0 for v in S[:, :, 1:].reshape(-1))
    for i in range(M):
        for j in range(N):
            ref = Fraction(0)
            for d in range(K):
                if za[i, d] or zb[j, d]:
                    continue
                sgn = -1 if sga[i, d] ^ sgb[j, d] else 1
                ref += sgn * Fraction(2) ** int(ea[i, d] + eb[j, d] + sa[i, d // G] + sb[j, d // G])
            assert Fraction(int(S[i, j, 0])) * Fraction(2) ** int(r["lsb"][i, j]) == ref


@pytest.mark.parametrize("fa,fb", [("E4C3", "E4C3"), ("E5C2", "E4C3"), ("E3C3", "E3C3")])
def test_histogram_and_kulisch_layouts_agree(oracle, fa, fb):
    """Eq. 5 / App. A.1: merging equal (h, t) addresses with signed counts and
    shifting each update straight into a per-phase accumulator give the same
    phase sums; every count fits 1 + ceil(log2(D+1)) signed bits."""
    rng = np.random.default_rng(17)
    K, G = 512, 32
    a, sa = _random_operand(rng, fa, 1, K, G)
    b, sb = _random_operand(rng, fb, 1, K, G)
    r = oracle.gemm(a, sa, b, sb, fa, fb, G)
    S = oracle.int128_to_int(r["S_raw"])[0, 0]
    lam = int(r["lsb"][0, 0])
    L, tmin, tmax = oracle.pair_info(fa, fb)
    tlo, nt = tmin - 8, (tmax - tmin) + 17
    counts = oracle.histogram(a[0], sa[0], b[0], sb[0], fa, fb, G, tlo, nt)
    width = 1 + math.ceil(math.log2(K + 1))
    assert np.abs(counts).max() < 2 ** (width - 1)
    for h in range(L):
        via_hist = sum(int(counts[h, t]) * Fraction(2) ** (tlo + t) for t in range(nt))
        assert via_hist == Fraction(int(S[h])) * Fraction(2) ** lam


def test_tile_q32_semantics_variable_k(oracle):
    """App. C.1/C.2: the 4x4 E4C3 tile accumulates, per product, the Q16
    coefficient round(2^{k/8} 2^16) selected by q_p = m_a + m_b - 128 = 8e + k,
    shifted into a signed Q32 accumulator.  On the paper's verification design
    (64 seeded matrices, sum of K = 1,010, 1,024 outputs) the oracle's phase
    sums reproduce that accumulator exactly: sum_h Q16_h S_h 2^{lambda+16}."""
    design = _gold("tile_verification_design.json")
    rng = np.random.default_rng(2027)
    cuts = np.sort(rng.choice(np.arange(1, design["total_k"]), design["matrices"] - 1, replace=False))
    ks = np.diff(np.concatenate([[0], cuts, [design["total_k"]]]))
    assert len(ks) == design["matrices"] and ks.sum() == design["total_k"] and ks.min() >= 1
    q16 = [X.q16(k) for k in range(8)]
    outputs = 0
    for K in ks:
        a = rng.integers(0, 256, size=(4, K), dtype=np.uint8)
        b = rng.integers(0, 256, size=(4, K), dtype=np.uint8)  # B^T rows
        zs = np.zeros((4, 1), np.int8)
        r = oracle.gemm(a, zs, b, zs, "E4C3", "E4C3", int(K))
        S = oracle.int128_to_int(r["S_raw"])
        for i in range(4):
            for j in range(4):
                acc = 0
                for d in range(K):
                    ma, mb = int(a[i, d]) & 0x7F, int(b[j, d]) & 0x7F
                    if ma == 0 or mb == 0:
                        continue
                    qp = ma + mb - 128
                    e, k = qp >> 3, qp & 7
                    term = q16[k] << (16 + e)
                    acc += -term if (a[i, d] ^ b[j, d]) & 0x80 else term
                lam = int(r["lsb"][i, j])
                got = sum(q16[h] * Fraction(int(S[i, j, h])) for h in range(8)) * Fraction(2) ** (lam + 16)
                assert got == acc
                outputs += 1
    assert outputs == design["total_outputs"]


def test_range_flag(oracle):
    """The int128 window: a scale spread that cannot fit is reported."""
    K, G = 64, 32
    a = np.full((1, K), 0x7F, np.uint8)
    b = np.full((1, K), 0x7F, np.uint8)
    sa = np.array([[-128, 127]], np.int8)
    sb = np.array([[-128, 127]], np.int8)
    r = oracle.gemm(a, sa, b, sb, "E5C2", "E5C2", G)
    assert r["range"][0, 0] and np.isnan(r["C"][0, 0])
    sa = np.array([[0, 1]], np.int8)
    r = oracle.gemm(a, sa, b, sa, "E5C2", "E5C2", G)
    assert not r["range"][0, 0]
