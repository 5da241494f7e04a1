"""CurveFP oracle — TEST INFRASTRUCTURE ONLY.

Plain, slow CPU reference for the CurveFP hot path (block-scaled quantization
into E3C3/E4C3/E5C2 codes, the closed product, per-phase accumulation and the
phase combine).  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it.
The CUDA library never imports, links or calls anything here, and this module
imports nothing from the CUDA side.

The arithmetic lives in ``curvefp_oracle.c`` (plain C, fp64 levels from libm
exp2, brute-force nearest-level search, exact ``__int128`` phase sums).  This
file only compiles it with gcc and marshals numpy arrays through ctypes.

Every function cites the passage of the paper it restates; the readings taken
where the paper is silent are listed at the top of ``curvefp_oracle.c``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "curvefp_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

# 3, 4: E4C3 with the rational radices r = 2^{8/9} and r = 2^{3/4} (R14)
FORMATS = {"E3C3": 0, "E4C3": 1, "E5C2": 2, "E4C3_R8_9": 3, "E4C3_R3_4": 4}


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP over independent rows only)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=gnu11", "-ffp-contract=off", "-fopenmp", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
        )
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i64 = ctypes.c_int64
            i32 = ctypes.c_int
            lib.oracle_format.argtypes = [i32] + [P] * 5
            lib.oracle_levels.argtypes = [i32, P]
            lib.oracle_phase_count.argtypes = [ctypes.c_long] * 3
            lib.oracle_phase_count.restype = ctypes.c_long
            lib.oracle_decode_fields.argtypes = [i32, ctypes.c_uint8, P, P, P, P]
            lib.oracle_block_scale.argtypes = [i32, ctypes.c_double]
            lib.oracle_quantize.argtypes = [i32, i32, P, i64, i64, i64, i32, P, P]
            lib.oracle_decode.argtypes = [i32, i32, P, P, i64, i64, P]
            lib.oracle_encode.argtypes = [i32, i32, P, i64, i64, P, P]
            lib.oracle_quantize_static.argtypes = [i32, i32, P, i64, i64, i32, i32, P, P]
            lib.oracle_dequantize.argtypes = [i32, i32, P, P, i64, i64, P]
            lib.oracle_closed_product.argtypes = [i32, i32, ctypes.c_uint8, ctypes.c_uint8, P, P, P]
            lib.oracle_pair_info.argtypes = [i32, i32, P, P, P]
            lib.oracle_gemm.argtypes = [i32, i32, i32, P, P, P, P, i64, i64, i64, P, P, P, P]
            lib.oracle_gemm.restype = i64
            lib.oracle_gemm_elem.argtypes = [i32, i32, P, P, P, P, i64, i64, i64, P, P, P, P]
            lib.oracle_gemm_elem.restype = i64
            lib.oracle_histogram.argtypes = [i32, i32, i32, P, P, P, P, i64, i32, i32, P]
            lib.oracle_row_norms.argtypes = [i32, i32, P, P, i64, i64, P]
            lib.oracle_num_threads.argtypes = []
            _lib = lib
    return _lib


def _fid(fmt) -> int:
    return FORMATS[fmt] if isinstance(fmt, str) else int(fmt)


def _ptr(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data)


def num_threads() -> int:
    return _load().oracle_num_threads()


def format_params(fmt) -> dict:
    """(E, C, K, B, nmax) of a format (Table 1; Sec. 3.1)."""
    out = [ctypes.c_int() for _ in range(5)]
    if _load().oracle_format(_fid(fmt), *[ctypes.byref(o) for o in out]):
        raise ValueError(fmt)
    E, C, K, B, nmax = (o.value for o in out)
    return {"E": E, "C": C, "K": K, "B": B, "nmax": nmax}


def levels(fmt) -> np.ndarray:
    """All positive levels r^{n/K} = 2^{p n/(qK)}, n = -nmax..nmax (Eq. 1)."""
    p = format_params(fmt)
    out = np.empty(2 * p["nmax"] + 1, np.float64)
    _load().oracle_levels(_fid(fmt), _ptr(out))
    return out


def phase_count(p: int, q: int, K: int) -> int:
    """Eq. 4: H = qK / gcd(p, qK)."""
    return int(_load().oracle_phase_count(p, q, K))


def decode_fields(fmt, code: int):
    """(nonzero, s, e, k, m) of one code byte (App. C.1 packing)."""
    s, e, k, m = (ctypes.c_int() for _ in range(4))
    nz = _load().oracle_decode_fields(_fid(fmt), code, *[ctypes.byref(v) for v in (s, e, k, m)])
    return nz, s.value, e.value, k.value, m.value


def block_scale(fmt, amax: float) -> int:
    """Ceil-absmax block scale (Sec. 3.1; reading R2)."""
    return int(_load().oracle_block_scale(_fid(fmt), float(amax)))


def quantize(x: np.ndarray, fmt, block: int = 32, block_axis: int = 0):
    """Block-scaled quantization Q(X) (Sec. 3.1).

    x: 2-D float32 array (BF16 inputs must be widened to float32 first).
    Returns (codes uint8, scales int8, nan_flag).  block_axis 0 blocks along
    columns; block_axis 1 blocks along rows and returns the transposed
    operand ([cols x rows] codes)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    rows, cols = x.shape
    R, Cc = (cols, rows) if block_axis else (rows, cols)
    if Cc % block:
        raise ValueError("blocked extent must be a multiple of the block size")
    codes = np.empty((R, Cc), np.uint8)
    scales = np.empty((R, Cc // block), np.int8)
    flags = _load().oracle_quantize(
        _fid(fmt), block, _ptr(x), rows, cols, cols, block_axis, _ptr(codes), _ptr(scales)
    )
    if flags < 0:
        raise ValueError(fmt)
    return codes, scales, bool(flags & 1)


GRANULARITY = {"block": 0, "row": 1, "tensor": 2}
SCALE_RULE = {"ceil": 0, "mse": 1}


def quantize_static(x: np.ndarray, fmt, block: int = 32, granularity: str = "block", rule: str = "mse"):
    """Q(X) with a scale per block / row / tensor (R11) chosen by ceil-absmax
    or by reconstruction-MSE search (R12).  x [rows x cols] FP32, blocks along
    columns.  Returns (codes, scales [rows x cols/block], nan_flag)."""
    x = np.ascontiguousarray(x, np.float32)
    rows, cols = x.shape
    codes = np.empty((rows, cols), np.uint8)
    scales = np.empty((rows, cols // block), np.int8)
    flags = _load().oracle_quantize_static(_fid(fmt), block, _ptr(x), rows, cols, GRANULARITY[granularity],
                                           SCALE_RULE[rule], _ptr(codes), _ptr(scales))
    if flags < 0:
        raise ValueError("bad arguments")
    return codes, scales, bool(flags & 1)


def encode(x: np.ndarray, scales: np.ndarray, fmt, block: int = 32):
    """Nearest-level encode with given block scales (Sec. 3.1).  x: [R x C]
    float32, scales [R x C/block].  Returns (codes, nan_flag)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    scales = np.ascontiguousarray(scales, np.int8)
    codes = np.empty(x.shape, np.uint8)
    flags = _load().oracle_encode(_fid(fmt), block, _ptr(x), x.shape[0], x.shape[1], _ptr(scales), _ptr(codes))
    return codes, bool(flags & 1)


def decode(codes: np.ndarray, scales: np.ndarray, fmt, block: int = 32) -> np.ndarray:
    """Real values (fp64) of codes under their block scales (Eq. 1)."""
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.int8)
    out = np.empty(codes.shape, np.float64)
    _load().oracle_decode(_fid(fmt), block, _ptr(codes), _ptr(scales), codes.shape[0], codes.shape[1], _ptr(out))
    return out


def dequantize(codes: np.ndarray, scales: np.ndarray, fmt, block: int = 32) -> np.ndarray:
    """FP32 dequantization, reading R4."""
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.int8)
    out = np.empty(codes.shape, np.float32)
    _load().oracle_dequantize(_fid(fmt), block, _ptr(codes), _ptr(scales), codes.shape[0], codes.shape[1], _ptr(out))
    return out


def closed_product(fmt_a, fmt_b, ca: int, cb: int):
    """Eq. 2 / App. A.1: (nonzero, delta, h, t) for one code pair."""
    d, h, t = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    nz = _load().oracle_closed_product(_fid(fmt_a), _fid(fmt_b), ca, cb, ctypes.byref(d), ctypes.byref(h), ctypes.byref(t))
    if nz < 0:
        raise ValueError((fmt_a, fmt_b))
    return nz, d.value, h.value, t.value


def pair_info(fmt_a, fmt_b):
    """(L, t_min, t_max): shared lattice size (= phase count H) and bin range."""
    L, lo, hi = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    if _load().oracle_pair_info(_fid(fmt_a), _fid(fmt_b), ctypes.byref(L), ctypes.byref(lo), ctypes.byref(hi)):
        raise ValueError("format pair not supported (rational radices pair only with themselves)")
    return L.value, lo.value, hi.value


def gemm(a, sa, b, sb, fmt_a, fmt_b, block: int = 32, phases: bool = True):
    """Closed-product GEMM with exact per-phase sums (Eq. 5, App. A.1).

    a: [M x K] codes, sa: [M x K/block]; b: [N x K] codes, sb: [N x K/block].
    Returns dict with C (fp64 [M x N], phase combine), S (object array of
    Python ints [M x N x L], if phases), lsb (int32 [M x N]), range (bool)."""
    a = np.ascontiguousarray(a, np.uint8)
    b = np.ascontiguousarray(b, np.uint8)
    sa = np.ascontiguousarray(sa, np.int8)
    sb = np.ascontiguousarray(sb, np.int8)
    M, K = a.shape
    N = b.shape[0]
    L = pair_info(fmt_a, fmt_b)[0]
    C = np.empty((M, N), np.float64)
    S = np.empty((M, N, L, 2), np.int64) if phases else None
    lsb = np.empty((M, N), np.int32)
    rng = np.empty((M, N), np.uint8)
    _load().oracle_gemm(
        _fid(fmt_a), _fid(fmt_b), block, _ptr(a), _ptr(sa), _ptr(b), _ptr(sb), M, N, K,
        _ptr(C), _ptr(S) if phases else None, _ptr(lsb), _ptr(rng),
    )
    out = {"C": C, "lsb": lsb, "range": rng.astype(bool)}
    if phases:
        out["S_raw"] = S  # int128 as (lo, hi) int64 pairs
    return out


def operand_view(codes, scales, block: int, layout: str = "rows"):
    """A GEMM operand with one scale per element (R13).

    layout "rows": codes [R x K], scales [R x K/block] (blocked along the
    GEMM's K).  layout "cols": codes [K x R], scales [K x R/block], a matrix
    quantized along R and used transposed (the reused operand of a backward
    GEMM).  Returns (codes [R x K], per-element scales [R x K])."""
    codes = np.asarray(codes, np.uint8)
    scales = np.asarray(scales, np.int8)
    if layout == "rows":
        return np.ascontiguousarray(codes), np.ascontiguousarray(np.repeat(scales, block, axis=1))
    if layout == "cols":
        return np.ascontiguousarray(codes.T), np.ascontiguousarray(np.repeat(scales, block, axis=1).T)
    raise ValueError(layout)


def gemm_elem(a, ea, b, eb, fmt_a, fmt_b, phases: bool = True):
    """Closed-product GEMM with per-element scales (Eq. 5, R13).

    a: [M x K] codes with scales ea [M x K]; b: [N x K] with eb [N x K].
    Returns the same dict as ``gemm``."""
    a = np.ascontiguousarray(a, np.uint8)
    b = np.ascontiguousarray(b, np.uint8)
    ea = np.ascontiguousarray(ea, np.int8)
    eb = np.ascontiguousarray(eb, np.int8)
    M, K = a.shape
    N = b.shape[0]
    if ea.shape != a.shape or eb.shape != b.shape or b.shape[1] != K:
        raise ValueError("shape mismatch")
    L = pair_info(fmt_a, fmt_b)[0]
    C = np.empty((M, N), np.float64)
    S = np.empty((M, N, L, 2), np.int64) if phases else None
    lsb = np.empty((M, N), np.int32)
    rng = np.empty((M, N), np.uint8)
    _load().oracle_gemm_elem(
        _fid(fmt_a), _fid(fmt_b), _ptr(a), _ptr(ea), _ptr(b), _ptr(eb), M, N, K,
        _ptr(C), _ptr(S) if phases else None, _ptr(lsb), _ptr(rng),
    )
    out = {"C": C, "lsb": lsb, "range": rng.astype(bool)}
    if phases:
        out["S_raw"] = S
    return out


def gemm_oriented(a, sa, layout_a, b, sb, layout_b, fmt_a, fmt_b, block: int = 32, phases: bool = True):
    """GEMM of two operands in either layout (see ``operand_view``)."""
    ca, ea = operand_view(a, sa, block, layout_a)
    cb, eb = operand_view(b, sb, block, layout_b)
    return gemm_elem(ca, ea, cb, eb, fmt_a, fmt_b, phases)


def int128_to_int(raw: np.ndarray) -> np.ndarray:
    """(lo, hi) int64 pairs -> object array of Python ints."""
    lo = raw[..., 0].astype(np.uint64).astype(object)
    hi = raw[..., 1].astype(object)
    return hi * (1 << 64) + lo


def histogram(a, sa, b, sb, fmt_a, fmt_b, block: int, tlo: int, nt: int) -> np.ndarray:
    """Signed counts n_{h,t} of one dot product (Eq. 5 histogram layout)."""
    a = np.ascontiguousarray(a, np.uint8)
    b = np.ascontiguousarray(b, np.uint8)
    sa = np.ascontiguousarray(sa, np.int8)
    sb = np.ascontiguousarray(sb, np.int8)
    L = pair_info(fmt_a, fmt_b)[0]
    counts = np.empty((L, nt), np.int64)
    rc = _load().oracle_histogram(
        _fid(fmt_a), _fid(fmt_b), block, _ptr(a), _ptr(sa), _ptr(b), _ptr(sb), a.shape[0], tlo, nt, _ptr(counts)
    )
    if rc:
        raise ValueError("bin outside the requested window")
    return counts


def row_norms(codes, scales, fmt, block: int = 32) -> np.ndarray:
    """||row||_2 of the dequantized operand, fp64."""
    codes = np.ascontiguousarray(codes, np.uint8)
    scales = np.ascontiguousarray(scales, np.int8)
    out = np.empty(codes.shape[0], np.float64)
    _load().oracle_row_norms(_fid(fmt), block, _ptr(codes), _ptr(scales), codes.shape[0], codes.shape[1], _ptr(out))
    return out
