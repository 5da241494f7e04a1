"""The C-ABI library loads, exports every entry point that include/curvefp.h
declares, and rejects bad arguments on the host (no GPU needed: argument
validation happens before any CUDA call)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "curvefp.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_10010_gb300 import _build, load

    _build.build()
    return load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(curvefp_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for f in ("curvefp_quantize", "curvefp_dequantize", "curvefp_gemm", "curvefp_gemm_phases"):
        assert f in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_static_queries(lib):
    assert lib.curvefp_phase_count(0, 0) == 8
    assert lib.curvefp_phase_count(1, 1) == 8
    assert lib.curvefp_phase_count(2, 2) == 4
    assert lib.curvefp_phase_count(2, 1) == 8
    assert lib.curvefp_phase_count(7, 1) == -1
    assert lib.curvefp_status_string(0) == b"ok"
    assert lib.curvefp_status_string(1) == b"invalid argument"
    assert b"sm_103a" in lib.curvefp_version()


def test_host_side_validation(lib):
    P = ctypes.c_void_p
    dummy = P(4096)  # never dereferenced: every call below fails validation first
    INVALID = 1
    # bad format, bad block, bad dtype, bad axis, ld < cols
    assert lib.curvefp_quantize(9, 32, dummy, 0, 4, 64, 64, 0, dummy, dummy, None, None) == INVALID
    assert lib.curvefp_quantize(1, 33, dummy, 0, 4, 64, 64, 0, dummy, dummy, None, None) == INVALID
    assert lib.curvefp_quantize(1, 32, dummy, 5, 4, 64, 64, 0, dummy, dummy, None, None) == INVALID
    assert lib.curvefp_quantize(1, 32, dummy, 0, 4, 64, 64, 2, dummy, dummy, None, None) == INVALID
    assert lib.curvefp_quantize(1, 32, dummy, 0, 4, 64, 32, 0, dummy, dummy, None, None) == INVALID
    # cols not a multiple of the block (axis 0), rows not (axis 1)
    assert lib.curvefp_quantize(1, 32, dummy, 0, 4, 48, 48, 0, dummy, dummy, None, None) == INVALID
    assert lib.curvefp_quantize(1, 32, dummy, 0, 48, 64, 64, 1, dummy, dummy, None, None) == INVALID
    # NULL and misaligned pointers
    assert lib.curvefp_quantize(1, 32, None, 0, 4, 64, 64, 0, dummy, dummy, None, None) == INVALID
    assert lib.curvefp_quantize(1, 32, P(4100), 0, 4, 64, 64, 0, dummy, dummy, None, None) == INVALID
    # empty input is a no-op
    assert lib.curvefp_quantize(1, 32, None, 0, 0, 64, 64, 0, None, None, None, None) == 0
    assert lib.curvefp_dequantize(1, 32, None, None, 0, 64, None, None) == 0
    assert lib.curvefp_dequantize(1, 32, dummy, dummy, 4, 48, dummy, None) == INVALID
    # GEMM: SKINNY takes at most CURVEFP_SKINNY_MAX_M (8) rows
    assert lib.curvefp_gemm(3, 1, 1, 32, dummy, dummy, dummy, dummy, 9, 4, 64, dummy, None, None) == 2
    # GEMM: K not a multiple of the block, non-positive sizes, bad algo
    assert lib.curvefp_gemm(0, 1, 1, 32, dummy, dummy, dummy, dummy, 4, 4, 48, dummy, None, None) == INVALID
    assert lib.curvefp_gemm(0, 1, 1, 32, dummy, dummy, dummy, dummy, 0, 4, 64, dummy, None, None) == INVALID
    assert lib.curvefp_gemm(7, 1, 1, 32, dummy, dummy, dummy, dummy, 4, 4, 64, dummy, None, None) == INVALID
    assert lib.curvefp_gemm_phases(1, 1, 32, dummy, dummy, dummy, dummy, 4, 4, 64, None, None, dummy, None, None) == INVALID
    # static quantization: bad group / rule, cols not a multiple of the block,
    # missing or short workspace for row groups; block groups need none
    ws = lib.curvefp_quantize_static_workspace
    assert ws(4, 64, 32, 0) == 0 and ws(4, 64, 32, 1) > 0 and ws(4, 64, 32, 2) > 0 and ws(4, 64, 32, 3) == 0
    qs = lib.curvefp_quantize_static
    assert qs(1, 32, 3, 1, dummy, 0, 4, 64, dummy, dummy, None, 0, None, None) == INVALID
    assert qs(1, 32, 0, 2, dummy, 0, 4, 64, dummy, dummy, None, 0, None, None) == INVALID
    assert qs(1, 32, 0, 1, dummy, 0, 4, 48, dummy, dummy, None, 0, None, None) == INVALID
    assert qs(1, 32, 1, 1, dummy, 0, 4, 64, dummy, dummy, None, 0, None, None) == INVALID
    assert qs(1, 32, 1, 1, dummy, 0, 4, 64, dummy, dummy, dummy, 8, None, None) == INVALID
    assert qs(1, 32, 2, 1, None, 0, 0, 64, None, None, None, 0, None, None) == 0
    # bounded-wait self-test: the status word is required, the limit in 1 .. 2^31
    sw = lib.curvefp_selftest_bounded_wait
    assert sw(0, 1000, None, None) == INVALID
    assert sw(0, 0, dummy, None) == INVALID
    assert sw(0, (1 << 31) + 1, dummy, None) == INVALID


def test_oriented_gemm_validation(lib):
    """Layouts, blocked extents, workspace and algorithm rules of the oriented
    GEMM, all decided on the host before any launch."""
    import ctypes as C

    P = C.c_void_p
    d = P(4096)
    INVALID, UNSUPPORTED = 1, 2
    lib.curvefp_gemm_oriented_workspace_bytes.restype = C.c_size_t
    lib.curvefp_gemm_oriented_workspace_bytes.argtypes = [C.c_int, C.c_int, C.c_int, C.c_int64, C.c_int64, C.c_int64]
    wsb = lib.curvefp_gemm_oriented_workspace_bytes
    al = lambda v: (v + 255) // 256 * 256  # noqa: E731
    assert wsb(1, 0, 0, 256, 96, 64) == 0 and wsb(0, 1, 1, 256, 96, 64) == 0
    # per operand: [R K codes (COLS)] + R K exponent bytes + R K / 16 step-scale bytes + 4 R
    op = lambda R, K, cols: (al(R * K) if cols else 0) + al(R * K) + al(R * K // 16) + al(4 * R)  # noqa: E731
    assert wsb(1, 0, 1, 256, 96, 64) == op(256, 64, False) + op(96, 64, True)
    assert wsb(1, 1, 1, 256, 96, 64) == op(256, 64, True) + op(96, 64, True)
    go = lib.curvefp_gemm_oriented
    go.argtypes = [C.c_int] * 4 + [P, P, C.c_int, P, P, C.c_int, C.c_int64, C.c_int64, C.c_int64, P, P, P, P,
                                   C.c_size_t, P, P]

    def call(algo=1, la=0, lb=1, M=64, N=64, K=64, c=d, ps=None, pl=None, ws=None, wsn=0, block=32):
        return go(algo, 1, 1, block, d, d, la, d, d, lb, M, N, K, c, ps, pl, ws, wsn, None, None)

    assert call(la=2) == INVALID                       # unknown layout
    assert call(la=1, M=48) == INVALID                 # COLS rows not a multiple of the block
    assert call(lb=0, K=48) == INVALID                 # ROWS K not a multiple of the block
    assert call(lb=1, N=80) == INVALID
    assert call() == INVALID                           # TENSOR with a COLS operand needs workspace
    assert call(ws=P(4096 + 16), wsn=1 << 30) == INVALID  # workspace not 256-byte aligned
    assert call(ws=d, wsn=16) == INVALID               # workspace too small
    assert call(ps=d, pl=d, ws=d, wsn=1 << 30) == INVALID  # phase sums only from EXACT
    assert call(algo=2, ws=d, wsn=1 << 30) == INVALID      # 2 is not an algorithm
    assert call(la=1, lb=1, K=48, ws=d, wsn=1 << 30) == INVALID  # tensor steps need K % 32
    assert call(algo=0, c=None) == INVALID             # exact: nothing to write
    assert call(algo=0, ps=d, pl=None) == INVALID      # exact: both phase arrays or neither


def test_rational_radix_host_rules(lib):
    """The rational-radix formats: phase counts (Table 2: 9 and 32), pairing
    only with themselves, and the entry points that do not take them."""
    P = ctypes.c_void_p
    d = P(4096)
    INVALID, UNSUPPORTED = 1, 2
    assert lib.curvefp_phase_count(3, 3) == 9 and lib.curvefp_phase_count(4, 4) == 32
    assert lib.curvefp_phase_count(3, 1) == -1 and lib.curvefp_phase_count(4, 3) == -1
    assert lib.curvefp_phase_count(5, 5) == -1
    # quantize: the same shape rules as the binary formats; unknown ids rejected
    assert lib.curvefp_quantize(3, 32, d, 0, 48, 64, 64, 1, d, d, None, None) == INVALID
    assert lib.curvefp_quantize(5, 32, d, 0, 4, 64, 64, 0, d, d, None, None) == INVALID
    # GEMM: mixed radix, and the tensor-core algorithms
    assert lib.curvefp_gemm(0, 3, 1, 32, d, d, d, d, 4, 4, 64, d, None, None) == UNSUPPORTED
    assert lib.curvefp_gemm(1, 4, 4, 32, d, d, d, d, 4, 4, 64, d, None, None) == UNSUPPORTED  # r = 2^{3/4}
    assert lib.curvefp_gemm(5, 3, 3, 32, d, d, d, d, 4, 4, 64, d, None, None) == UNSUPPORTED  # narrow, r = 2^{8/9}
    assert lib.curvefp_gemm(3, 3, 3, 32, d, d, d, d, 4, 4, 64, d, None, None) == UNSUPPORTED  # skinny
    assert lib.curvefp_gemm(2, 4, 4, 32, d, d, d, d, 4, 4, 64, d, None, None) == UNSUPPORTED
    assert lib.curvefp_gemm_q32(3, 3, 32, d, d, d, d, 4, 4, 64, d, None, None) == UNSUPPORTED
    assert lib.curvefp_quantize_static(3, 32, 1, 0, d, 0, 4, 64, d, d, None, 0, None, None) == INVALID  # no workspace


def test_product_path_does_not_touch_the_oracle():
    """The CUDA library and its binding neither import nor link the oracle."""
    pkg = os.path.join(ROOT, "paper_2608_10010_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b", text, flags=re.M), f
                assert "liboracle" not in text and "curvefp_oracle" not in text, f
