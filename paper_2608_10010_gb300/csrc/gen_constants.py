"""Generate ``curvefp_constants.h`` for the CUDA kernels.

Every constant is computed here with exact integer arithmetic (integer K-th
roots of powers of two at 256 fractional bits), never with a floating-point
math library, so that bit parity of the kernels does not depend on any
library's exp2.  The header holds hex literals only.

Constants (binary radix, K in {4, 8}):
  * mantissa LUT for the nearest-level search: the FP32 mantissa (23 bits) of
    a scaled value v in [2^F, 2^{F+1}) passes the k-th midpoint
    (2^{k/K} + 2^{(k+1)/K})/2 * 2^F iff mant >= MU_k.  The LUT is indexed by
    the top 8 mantissa bits; entry = (thresholds passed by the whole bucket)
    << 24 | (the one threshold inside the bucket, or 2^23 if none).
  * MU_SAT: 1 + mant/2^23 > 2^{(K-1)/K} iff mant >= MU_SAT (block scale).
  * MU_Z:   1 + mant/2^23 > 2^{1/K}    iff mant >= MU_Z   (zero boundary).
  * C_K[k]: FP32 bits of RN32(2^{k/K}) (dequantization).
  * Q16_K[k]: round(2^{k/K} 2^16), the tile's integer coefficients (App. C.1).
  * phase constants 2^{h/L} for L in {4, 8, 9, 32}, as FP32 and FP64 bits.
  * rational radix r = 2^{p/q} (E4C3 with r = 2^{8/9}, 2^{3/4}): the
    nearest-level tables per binade class, the ceil-absmax and zero-boundary
    thresholds and the exact GEMM's address offsets (see radix_params).

Run:  python gen_constants.py > curvefp_constants.h
"""
from __future__ import annotations

import sys

P = 256  # fractional bits of the fixed-point reference values


def iroot(n: int, k: int) -> int:
    """floor(n ** (1/k)) for n >= 0 by integer Newton iteration."""
    if n < 2:
        return n
    x = 1 << ((n.bit_length() + k - 1) // k)  # >= true root
    while True:
        y = ((k - 1) * x + n // x ** (k - 1)) // k
        if y >= x:
            return x
        x = y


def fix_pow2(num: int, den: int) -> int:
    """floor(2^{num/den} * 2^P) for 0 <= num <= den."""
    return iroot(1 << (num + den * P), den)


def is_exact_power(num: int, den: int) -> bool:
    return num % den == 0


def mant_threshold_fix(x_fix: int, exact: bool) -> int:
    """Smallest 23-bit mu with 1 + mu/2^23 > x, x = x_fix / 2^P in [1, 2].

    x_fix is a floor (error < 2^-P).  For irrational x the answer is
    floor((x - 1) 2^23) + 1, provided x is not within 2^-P of a multiple of
    2^-23 (asserted)."""
    assert not exact
    shift = P - 23
    frac = x_fix - (1 << P)
    q, r = divmod(frac, 1 << shift)
    assert 2 < r < (1 << shift) - 2, "threshold too close to an FP32 mantissa"
    return q + 1


def q16_coeff(k: int, K: int) -> int:
    """App. C.1 tile coefficient round(2^{k/K} 2^16) (never a tie: irrational
    for 0 < k < K)."""
    x = fix_pow2(k, K)
    shift = P - 16
    q, r = divmod(x, 1 << shift)
    if k:
        assert 2 < abs(r - (1 << (shift - 1))), "coefficient too close to a half"
    return q + (1 if r >= (1 << (shift - 1)) else 0)


def midpoint_threshold(k: int, K: int) -> int:
    """Smallest mu with 1 + mu/2^23 > (2^{k/K} + 2^{(k+1)/K}) / 2."""
    s = fix_pow2(k, K) + fix_pow2(k + 1, K)  # floor sum, true sum in [s, s+2)
    shift = P - 23 + 1
    frac = s - (1 << (P + 1))
    q, r = divmod(frac, 1 << shift)
    assert 4 < r < (1 << shift) - 4, "midpoint too close to an FP32 mantissa"
    return q + 1


def rn_mantissa(num: int, den: int, bits: int) -> int:
    """round(2^{num/den} * 2^bits) with the true value irrational (num % den != 0)
    or exactly a power of two."""
    if num % den == 0:
        return 1 << (bits + num // den)
    x = fix_pow2(num, den)
    shift = P - bits
    q, r = divmod(x, 1 << shift)
    half = 1 << (shift - 1)
    assert abs(r - half) > 2, "rounding too close to a tie"
    return q + (1 if r > half else 0)


def f32_bits_pow2(num: int, den: int) -> int:
    m = rn_mantissa(num, den, 23)  # in [2^23, 2^24]
    if m == 1 << 24:
        return (128 << 23)
    return (127 << 23) | (m - (1 << 23))


def f64_bits_pow2(num: int, den: int) -> int:
    m = rn_mantissa(num, den, 52)
    if m == 1 << 53:
        return (1024 << 52)
    return (1023 << 52) | (m - (1 << 52))


def lut_for(K: int) -> list[int]:
    thr = [midpoint_threshold(k, K) for k in range(K)]
    assert thr == sorted(thr) and all(b - a > (1 << 15) for a, b in zip(thr, thr[1:]))
    out = []
    for idx in range(256):
        lo, hi = idx << 15, (idx + 1) << 15
        base = sum(1 for t in thr if t <= lo)
        inside = [t for t in thr if lo < t < hi]
        assert len(inside) <= 1
        out.append((base << 24) | (inside[0] if inside else (1 << 23)))
    return out


FORMATS = {"E3C3": (3, 3), "E4C3": (4, 3), "E5C2": (5, 2)}


def rank_table(E: int, C: int) -> tuple[int, list[int]]:
    """Rank lookup for the quantizer's fast path, indexed by (binade offset fo,
    top 7 mantissa bits m7) of the scaled value v = |x| 2^{-a}:
    binade F = F_z + fo, mantissa bucket [m7 2^16, m7 2^16 + 2^16).
    Entry = rank below the bucket's threshold | rank at/above it << 8 |
    threshold's low 16 mantissa bits << 16 (0 and equal ranks if none).
    Ranks follow the nearest-level rule: 0 below L_nmin/2, saturating at
    2^{E+C} - 1; at most one decision threshold falls in a bucket, and where
    one does the rank steps by exactly 1 at a threshold whose low 16 bits are
    nonzero (the FP32 kernels rely on both: rank = r_lo + [bits >= t16])."""
    K = 1 << C
    B = 1 << (E + C - 1)
    nmax = B - 1
    emax = (1 << (E - 1)) - 1
    fz = (-nmax - K - 1) // K
    mu_z = mant_threshold_fix(fix_pow2(1, K), False)
    thr = [midpoint_threshold(k, K) for k in range(K)]

    def rank(F: int, mant: int) -> int:
        if F < fz or (F == fz and mant < mu_z):
            return 0
        j = sum(1 for t in thr if mant >= t)
        n = K * F + j
        if n > nmax:
            return 2 * B - 1
        return max(n + B, 1)

    nbin = emax - fz + 1
    out = []
    for fo in range(nbin):
        F = fz + fo
        for m7 in range(128):
            lo, hi = m7 << 16, (m7 << 16) | 0xFFFF
            r_lo, r_hi = rank(F, lo), rank(F, hi)
            cuts = [t for t in thr + [mu_z] if lo < t <= hi and rank(F, t - 1) != rank(F, t)]
            assert len(cuts) <= 1
            t16 = (cuts[0] & 0xFFFF) if cuts else 0
            if not cuts:
                assert r_lo == r_hi
            else:
                assert r_hi == r_lo + 1 and t16 >= 1
            out.append(r_lo | (r_hi << 8) | (t16 << 16))
    return nbin, out


# ---- rational radix r = 2^{p/q}, K = 8 (E4C3 variants) ---------------------
# Level n has exponent lambda(n) = p n / (qK).  For a scaled value y with
# binade b and 23-bit mantissa mu, the nearest level of the unbounded lattice
# is n*(y) = N0[b mod PB] + floor(b / PB) NPER + #{i : mu >= THR[b mod PB][i]},
# N0[c] = n*(2^c) and THR[c] the mantissa thresholds of the level midpoints
# inside [2^c, 2^{c+1}); the pattern repeats every PB binades (NPER levels).
RADIX_FORMATS = {"R8_9": (8, 9), "R3_4": (3, 4)}
RADIX_K, RADIX_NMAX = 8, 63
RADIX_MAXTHR = 11  # largest number of midpoints in one binade


def fixp(num: int, den: int) -> int:
    """floor(2^{num/den} 2^P) for any integer num (den > 0)."""
    i, f = divmod(num, den)
    v = fix_pow2(f, den)
    return v << i if i >= 0 else v >> (-i)


def gcd(a: int, b: int) -> int:
    while b:
        a, b = b, a % b
    return a


def radix_params(p: int, q: int) -> dict:
    K, nmax = RADIX_K, RADIX_NMAX
    N = q * K
    g = gcd(p, N)
    H = N // g
    PB = p // g          # binades per period
    NPER = PB * N // p   # levels per period
    one = 1 << P

    def mid_rel(n: int, c: int) -> int:
        """floor-ish 2 (2^{lambda(n)-c} + 2^{lambda(n+1)-c}) 2^P / 2 (error < 2 units)."""
        return fixp(p * n - c * N, N) + fixp(p * (n + 1) - c * N, N)  # = 2 mid / 2^c, 2^P units

    n0, thr = [], []
    for c in range(PB):
        # nearest level at y = 2^c
        n = (c * N) // p  # lambda(n) <= c < lambda(n + 1)
        if p * n == c * N:
            nstar = n
        else:
            s2 = mid_rel(n, c)            # 2 mid / 2^c in 2^P units
            assert abs(s2 - 2 * one) > 4
            nstar = n if 2 * one < s2 else n + 1
        n0.append(nstar)
        ts = []
        for m in range(n - 2, n + NPER + 3):
            s2 = mid_rel(m, c)
            if not (2 * one <= s2 < 4 * one):
                assert abs(s2 - 2 * one) > 4 and abs(s2 - 4 * one) > 4
                continue
            frac = s2 - 2 * one           # 2 (mid/2^c - 1), 2^P units
            shift = P - 23 + 1
            qq, r = divmod(frac, 1 << shift)
            assert 4 < r < (1 << shift) - 4, "midpoint too close to an FP32 mantissa"
            ts.append(qq + 1)
        assert ts == sorted(ts) and len(ts) <= RADIX_MAXTHR
        thr.append(ts)
    for c in range(PB):  # the counts tile the period
        nxt = n0[c + 1] if c + 1 < PB else n0[0] + NPER
        assert n0[c] + len(thr[c]) == nxt
    # ceil-absmax: lambda(nmax) = F + f; MU_SAT = smallest mu with 1 + mu 2^-23 > 2^f
    F, fnum = divmod(p * nmax, N)
    mu_sat = 1 if fnum == 0 else mant_threshold_fix(fix_pow2(fnum, N), False)
    # zero boundary L_nmin / 2 = 2^{lambda(-nmax) - 1} = 2^{ZB} 2^{zf}
    ZB, zfnum = divmod(-p * nmax - N, N)
    zthr = 1 if zfnum == 0 else mant_threshold_fix(fix_pow2(zfnum, N), False)
    # exact GEMM addressing on biased ranks: V = p (m_a + m_b) - R0 + N >= 0,
    # h = (V mod N) / g, t - t_min = floor(V / N) - OFF
    B = 64
    Q, R0 = divmod(2 * p * B, N)
    us = [p * (na + nb) for na in range(-nmax, nmax + 1) for nb in range(-nmax, nmax + 1)]
    tmin, tmax = min(u // N for u in us), max(u // N for u in us)
    off = Q + 1 + tmin
    return dict(N=N, g=g, H=H, PB=PB, NPER=NPER, N0=n0, THR=thr, F=F, MU_SAT=mu_sat, ZB=ZB, ZTHR=zthr,
                R0=R0, OFF=off, TMIN=tmin, TMAX=tmax)


def radix_rank_table(r: dict) -> tuple[int, list[int]]:
    """rank_table for a rational radix: binades ZB - 1 .. F of the scaled
    value (nothing above F occurs under the block's own ceil-absmax scale;
    keys of smaller values clamp to the all-zero binade ZB - 1), same entry
    layout; ranks from the nearest-level rule of radix_params."""
    B, nmax = 64, RADIX_NMAX

    def rank(F: int, mant: int) -> int:
        if F < r["ZB"] or (F == r["ZB"] and mant < r["ZTHR"]):
            return 0
        k, c = divmod(F, r["PB"])
        n = r["N0"][c] + k * r["NPER"] + sum(1 for t in r["THR"][c] if mant >= t)
        return min(max(n, -nmax), nmax) + B

    nbin = r["F"] - r["ZB"] + 2
    out = []
    for fo in range(nbin):
        F = r["ZB"] - 1 + fo
        thr = r["THR"][F % r["PB"]] + ([r["ZTHR"]] if F == r["ZB"] else [])
        for m7 in range(128):
            lo, hi = m7 << 16, (m7 << 16) | 0xFFFF
            r_lo, r_hi = rank(F, lo), rank(F, hi)
            cuts = [t for t in thr if lo < t <= hi and rank(F, t - 1) != rank(F, t)]
            assert len(cuts) <= 1
            if not cuts:
                assert r_lo == r_hi
            else:
                assert r_hi == r_lo + 1 and (cuts[0] & 0xFFFF) >= 1
            out.append(r_lo | (r_hi << 8) | (((cuts[0] & 0xFFFF) if cuts else 0) << 16))
    return nbin, out


def main(out=sys.stdout):
    w = out.write
    w("/* Generated by gen_constants.py from exact integer arithmetic; do not edit. */\n")
    w("#pragma once\n#include <stdint.h>\n\n")
    for K in (4, 8):
        thr = [midpoint_threshold(k, K) for k in range(K)]
        w(f"/* K = {K}: midpoint mantissa thresholds {', '.join(hex(t) for t in thr)} */\n")
        w(f"#define CFP_MU_SAT_K{K} 0x{mant_threshold_fix(fix_pow2(K - 1, K), False):06x}u\n")
        w(f"#define CFP_MU_Z_K{K} 0x{mant_threshold_fix(fix_pow2(1, K), False):06x}u\n")
        lut = lut_for(K)
        w(f"#define CFP_LUT_K{K}_INIT {{ \\\n")
        for i in range(0, 256, 8):
            w("  " + ", ".join(f"0x{v:08x}u" for v in lut[i:i + 8]) + ", \\\n")
        w("}\n")
        w(f"#define CFP_CK_F32_K{K}_INIT {{" + ", ".join(f"0x{f32_bits_pow2(k, K):08x}u" for k in range(K)) + "}\n")
        w(f"#define CFP_Q16_K{K}_INIT {{" + ", ".join(f"{q16_coeff(k, K)}u" for k in range(K)) + "}\n\n")
    for name, (E, C) in FORMATS.items():
        nbin, tab = rank_table(E, C)
        w(f"#define CFP_RANK_{name}_NBIN {nbin}\n")
        w(f"#define CFP_RANK_{name}_INIT {{ \\\n")
        for i in range(0, len(tab), 8):
            w("  " + ", ".join(f"0x{v:08x}u" for v in tab[i:i + 8]) + ", \\\n")
        w("}\n")
    for L in (4, 8, 9, 32):
        w(f"#define CFP_PHASE_F32_L{L}_INIT {{" + ", ".join(f"0x{f32_bits_pow2(h, L):08x}u" for h in range(L)) + "}\n")
        w(f"#define CFP_PHASE_F64_L{L}_INIT {{" + ", ".join(f"0x{f64_bits_pow2(h, L):016x}ull" for h in range(L)) + "}\n")
    for name, (p, q) in RADIX_FORMATS.items():
        r = radix_params(p, q)
        w(f"/* E4C3, r = 2^({p}/{q}): N = qK = {r['N']}, H = {r['H']} phases, period {r['PB']} binade(s) / "
          f"{r['NPER']} levels */\n")
        for key in ("N", "g", "H", "PB", "NPER", "F", "ZB", "R0", "OFF", "TMIN", "TMAX"):
            w(f"#define CFP_{name}_{key} ({r[key]})\n")
        w(f"#define CFP_{name}_MU_SAT 0x{r['MU_SAT']:06x}u\n")
        w(f"#define CFP_{name}_ZTHR 0x{r['ZTHR']:06x}u\n")
        w(f"#define CFP_{name}_N0_INIT {{" + ", ".join(str(v) for v in r["N0"]) + "}\n")
        w(f"#define CFP_{name}_CNT_INIT {{" + ", ".join(str(len(t)) for t in r["THR"]) + "}\n")
        rows = []
        for t in r["THR"]:
            rows += t + [1 << 23] * (RADIX_MAXTHR - len(t))  # padding is never reached
        w(f"#define CFP_{name}_THR_INIT {{" + ", ".join(f"0x{v:06x}u" for v in rows) + "}\n")
        # bucket LUT per class (as lut_for): top 8 mantissa bits -> thresholds
        # passed by the whole bucket << 24 | the one threshold inside it
        lut = []
        for t in r["THR"]:
            assert all(b - a > (1 << 15) for a, b in zip(t, t[1:]))
            for idx in range(256):
                lo, hi = idx << 15, (idx + 1) << 15
                inside = [v for v in t if lo < v < hi]
                assert len(inside) <= 1
                lut.append((sum(1 for v in t if v <= lo) << 24) | (inside[0] if inside else (1 << 23)))
        nbin, tab = radix_rank_table(r)
        w(f"#define CFP_RANK_E4C3_{name}_NBIN {nbin}\n")
        w(f"#define CFP_RANK_E4C3_{name}_INIT {{ \\\n")
        for i in range(0, len(tab), 8):
            w("  " + ", ".join(f"0x{v:08x}u" for v in tab[i:i + 8]) + ", \\\n")
        w("}\n")
        w(f"#define CFP_{name}_LUT_INIT {{ \\\n")
        for i in range(0, len(lut), 8):
            w("  " + ", ".join(f"0x{v:08x}u" for v in lut[i:i + 8]) + ", \\\n")
        w("}\n")
    w(f"#define CFP_RADIX_MAXTHR {RADIX_MAXTHR}\n")


if __name__ == "__main__":
    main()
