"""Exact / high-precision arithmetic used by the oracle pins.

Nothing here is imported by the oracle or by the CUDA library: these are
independent restatements (Python ``decimal`` and integers) that the tests use
to check the oracle against what the paper and the mathematics fix.
"""
from __future__ import annotations

from decimal import Decimal, getcontext, ROUND_FLOOR, ROUND_HALF_EVEN

getcontext().prec = 80

FMT = {  # Table 1
    "E3C3": dict(E=3, C=3),
    "E4C3": dict(E=4, C=3),
    "E5C2": dict(E=5, C=2),
}
for _f in FMT.values():
    _f["K"] = 1 << _f["C"]
    _f["B"] = 1 << (_f["E"] + _f["C"] - 1)
    _f["nmax"] = _f["B"] - 1
    _f["emax"] = (1 << (_f["E"] - 1)) - 1


def pow2(num: int, den: int) -> Decimal:
    """2^(num/den) to 80 significant digits (decimal's power is correctly
    rounded)."""
    return Decimal(2) ** (Decimal(num) / Decimal(den))


def level(fmt: str, n: int) -> Decimal:
    return pow2(n, FMT[fmt]["K"])


def midpoint_mantissa_threshold(K: int, k: int) -> int:
    """Smallest 23-bit mantissa mu with 1 + mu/2^23 > (2^{k/K} + 2^{(k+1)/K})/2."""
    t = (pow2(k, K) + pow2(k + 1, K)) / 2
    return int(((t - 1) * (1 << 23)).to_integral_value(ROUND_FLOOR)) + 1


def mantissa_threshold(num: int, den: int) -> int:
    """Smallest 23-bit mantissa mu with 1 + mu/2^23 > 2^{num/den} (irrational)."""
    return int(((pow2(num, den) - 1) * (1 << 23)).to_integral_value(ROUND_FLOOR)) + 1


def dyadic_margin(x: Decimal, bits: int) -> Decimal:
    """Distance from x (in [1, 2)) to the nearest multiple of 2^-bits, relative."""
    s = x * (1 << bits)
    f = s - s.to_integral_value(ROUND_FLOOR)
    return min(f, 1 - f) / (1 << bits)


def nearest_rank(fmt: str, v: Decimal) -> int:
    """Brute-force nearest codebook entry for a non-negative scaled value v
    (rank 0 = zero, rank n + B = 2^{n/K})."""
    f = FMT[fmt]
    best, bestd = 0, abs(v)
    for n in range(-f["nmax"], f["nmax"] + 1):
        d = abs(v - level(fmt, n))
        if d < bestd:
            best, bestd = n + f["B"], d
    return best


def rn32_mantissa(num: int, den: int) -> int:
    """round(2^{num/den} * 2^23), ties impossible for irrational values."""
    return int((pow2(num, den) * (1 << 23)).to_integral_value(ROUND_HALF_EVEN))


def q16(k: int) -> int:
    """App. C.1 tile coefficient round(2^{k/8} 2^16)."""
    return int((pow2(k, 8) * (1 << 16)).to_integral_value(ROUND_HALF_EVEN))
