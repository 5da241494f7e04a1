"""CurveFP on GB300: Python binding of the C ABI in ``include/curvefp.h``.

This module only marshals arguments (torch tensors -> device pointers, the
current CUDA stream) into ``libcurvefp.so``; every step of the quantizer and
the GEMM runs in the library's CUDA kernels.  There is no CPU fallback: if the
library is missing or was not built for this machine, the calls raise.
"""
from __future__ import annotations

import ctypes
import os

from . import _build

# E4C3_R8_9 / E4C3_R3_4: E4C3 codes with the rational radices 2^{8/9}, 2^{3/4}
FORMATS = {"E3C3": 0, "E4C3": 1, "E5C2": 2, "E4C3_R8_9": 3, "E4C3_R3_4": 4}
DTYPES = {"f32": 0, "bf16": 1}
ALGOS = {"exact": 0, "tensor": 1, "skinny": 3, "auto": 4, "tensor_narrow": 5}
STATUS_BITS = {"nan": 1, "range": 2, "timeout": 4}

_lib = None


class CurveFPError(RuntimeError):
    pass


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = False):
    """Load libcurvefp.so (raises if it is absent, unless asked to build)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_build.LIB):
            if not build_if_missing:
                raise CurveFPError(f"libcurvefp.so not built ({_build.LIB}); run __graft_entry__.build()")
            _build.build()
        lib = ctypes.CDLL(_build.LIB)
        P, I, L = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64
        lib.curvefp_quantize.argtypes = [I, I, P, I, L, L, L, I, P, P, P, P]
        lib.curvefp_dequantize.argtypes = [I, I, P, P, L, L, P, P]
        lib.curvefp_gemm.argtypes = [I, I, I, I, P, P, P, P, L, L, L, P, P, P]
        lib.curvefp_gemm_phases.argtypes = [I, I, I, P, P, P, P, L, L, L, P, P, P, P, P]
        lib.curvefp_gemm_phases_histogram.argtypes = [I, I, I, P, P, P, P, L, L, L, P, P, P, P, P]
        lib.curvefp_phase_count.argtypes = [I, I]
        lib.curvefp_quantize_static_workspace.argtypes = [L, L, I, I]
        lib.curvefp_quantize_static_workspace.restype = ctypes.c_size_t
        lib.curvefp_quantize_static.argtypes = [I, I, I, I, P, I, L, L, P, P, P, ctypes.c_size_t, P, P]
        lib.curvefp_quantize_static_noalloc.argtypes = [I, I, I, I, P, I, L, L, P, P, P, P]
        lib.curvefp_gemm_q32.argtypes = [I, I, I, P, P, P, P, L, L, L, P, P, P]
        lib.curvefp_gemm_requant.argtypes = [I, I, I, I, P, P, P, P, L, L, L, P, I, I, P, P, P, P]
        lib.curvefp_gemm_oriented_workspace_bytes.argtypes = [I, I, I, L, L, L]
        lib.curvefp_gemm_oriented_workspace_bytes.restype = ctypes.c_size_t
        lib.curvefp_gemm_oriented.argtypes = [I, I, I, I, P, P, I, P, P, I, L, L, L, P, P, P, P, ctypes.c_size_t,
                                              P, P]
        lib.curvefp_selftest_bounded_wait.argtypes = [I, L, P, P]
        lib.curvefp_status_string.argtypes = [I]
        lib.curvefp_status_string.restype = ctypes.c_char_p
        lib.curvefp_version.restype = ctypes.c_char_p
        for f in ("curvefp_quantize", "curvefp_quantize_static", "curvefp_quantize_static_noalloc",
                  "curvefp_dequantize", "curvefp_gemm", "curvefp_gemm_phases", "curvefp_gemm_q32",
                  "curvefp_gemm_requant", "curvefp_gemm_oriented", "curvefp_gemm_phases_histogram",
                  "curvefp_selftest_bounded_wait"):
            getattr(lib, f).restype = I
        _lib = lib
    return _lib


def _fmt(f) -> int:
    return FORMATS[f] if isinstance(f, str) else int(f)


def _check(rc: int):
    if rc != 0:
        raise CurveFPError(load().curvefp_status_string(rc).decode())


def _stream(stream):
    import torch

    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def phase_count(fmt_a, fmt_b) -> int:
    return load().curvefp_phase_count(_fmt(fmt_a), _fmt(fmt_b))


def quantize(x, fmt, block: int = 32, block_axis: int = 0, codes=None, scales=None, status=None, stream=None):
    """Q(X) of a 2-D FP32/BF16 CUDA tensor.  Returns (codes, scales): codes
    [rows x cols] (block_axis 0) or the transposed [cols x rows] (block_axis 1)."""
    import torch

    assert x.dim() == 2 and x.is_cuda and x.stride(1) == 1
    rows, cols = x.shape
    R, Cc = (cols, rows) if block_axis else (rows, cols)
    if codes is None:
        codes = torch.empty((R, Cc), dtype=torch.uint8, device=x.device)
    if scales is None:
        scales = torch.empty((R, Cc // block), dtype=torch.int8, device=x.device)
    dt = {torch.float32: 0, torch.bfloat16: 1}[x.dtype]
    _check(load().curvefp_quantize(_fmt(fmt), block, _p(x), dt, rows, cols, x.stride(0), block_axis,
                                   _p(codes), _p(scales), _p(status), _stream(stream)))
    return codes, scales


SCALE_GROUPS = {"block": 0, "row": 1, "tensor": 2}
SCALE_RULES = {"ceil": 0, "mse": 1}


def quantize_static(x, fmt, block: int = 32, group: str = "block", rule: str = "mse", codes=None, scales=None,
                    status=None, stream=None):
    """Static-operand Q(X): one scale per block / row / tensor, chosen by
    ceil-absmax or reconstruction-MSE search.  x [rows x cols] dense FP32/BF16
    CUDA tensor; returns (codes [rows x cols], scales [rows x cols/block])."""
    import torch

    assert x.dim() == 2 and x.is_cuda and x.is_contiguous()
    rows, cols = x.shape
    if codes is None:
        codes = torch.empty((rows, cols), dtype=torch.uint8, device=x.device)
    if scales is None:
        scales = torch.empty((rows, cols // block), dtype=torch.int8, device=x.device)
    lib = load()
    nws = lib.curvefp_quantize_static_workspace(rows, cols, block, SCALE_GROUPS[group])
    ws = torch.empty(max(int(nws), 16), dtype=torch.uint8, device=x.device) if nws else None
    dt = {torch.float32: 0, torch.bfloat16: 1}[x.dtype]
    _check(lib.curvefp_quantize_static(_fmt(fmt), block, SCALE_GROUPS[group], SCALE_RULES[rule], _p(x), dt, rows, cols,
                                       _p(codes), _p(scales), _p(ws), int(nws), _p(status), _stream(stream)))
    return codes, scales


def quantize_static_noalloc(x, fmt, block: int = 32, group: str = "block", rule: str = "mse", codes=None,
                            scales=None, status=None, stream=None):
    """quantize_static through the entry point that allocates nothing, for
    callers that cannot allocate device memory: its scratch is a fixed device
    array inside the library (row groups up to ~100,000 rows), shared by every
    call on the device, so calls that overlap on the GPU race."""
    import torch

    assert x.dim() == 2 and x.is_cuda and x.is_contiguous()
    rows, cols = x.shape
    if codes is None:
        codes = torch.empty((rows, cols), dtype=torch.uint8, device=x.device)
    if scales is None:
        scales = torch.empty((rows, cols // block), dtype=torch.int8, device=x.device)
    dt = {torch.float32: 0, torch.bfloat16: 1}[x.dtype]
    _check(load().curvefp_quantize_static_noalloc(_fmt(fmt), block, SCALE_GROUPS[group], SCALE_RULES[rule], _p(x), dt,
                                                  rows, cols, _p(codes), _p(scales), _p(status), _stream(stream)))
    return codes, scales


def dequantize(codes, scales, fmt, block: int = 32, out=None, stream=None):
    import torch

    if out is None:
        out = torch.empty(codes.shape, dtype=torch.float32, device=codes.device)
    _check(load().curvefp_dequantize(_fmt(fmt), block, _p(codes), _p(scales), codes.shape[0], codes.shape[1],
                                     _p(out), _stream(stream)))
    return out


def gemm(a, sa, b, sb, fmt_a, fmt_b, block: int = 32, algo: str = "tensor", out=None, status=None, stream=None):
    """C = A_hat B_hat^T for a [M x K] and b [N x K] codes (K contiguous)."""
    import torch

    M, K = a.shape
    N = b.shape[0]
    if out is None:
        out = torch.empty((M, N), dtype=torch.float32, device=a.device)
    _check(load().curvefp_gemm(ALGOS[algo], _fmt(fmt_a), _fmt(fmt_b), block, _p(a), _p(sa), _p(b), _p(sb),
                               M, N, K, _p(out), _p(status), _stream(stream)))
    return out


LAYOUTS = {"rows": 0, "cols": 1}


def _rows_of(x, layout):
    """GEMM rows of an operand's code matrix, and its K."""
    return (x.shape[0], x.shape[1]) if layout == "rows" else (x.shape[1], x.shape[0])


def gemm_oriented_workspace_bytes(layout_a, layout_b, M, N, K, algo: str = "tensor") -> int:
    return int(load().curvefp_gemm_oriented_workspace_bytes(ALGOS[algo], LAYOUTS[layout_a], LAYOUTS[layout_b], M, N,
                                                            K))


def gemm_oriented(a, sa, layout_a, b, sb, layout_b, fmt_a, fmt_b, block: int = 32, algo: str = "tensor", out=None,
                  phases: bool = False, workspace=None, status=None, stream=None):
    """C = A_hat B_hat^T with operands in either layout ("rows": codes [R x K]
    blocked along K; "cols": codes [K x R] blocked along R, used transposed).
    Returns C, or (C, phase_sums, phase_lsb) with phases=True (exact only)."""
    import torch

    M, K = _rows_of(a, layout_a)
    N, Kb = _rows_of(b, layout_b)
    if Kb != K:
        raise CurveFPError("operand K mismatch")
    c = out if out is not None else torch.empty((M, N), dtype=torch.float32, device=a.device)
    ps = pl = None
    if phases:
        H = phase_count(fmt_a, fmt_b)
        ps = torch.empty((M, N, H, 2), dtype=torch.int64, device=a.device)
        pl = torch.empty((M, N), dtype=torch.int32, device=a.device)
    need = gemm_oriented_workspace_bytes(layout_a, layout_b, M, N, K, algo)
    if workspace is None and need:
        workspace = torch.empty(need, dtype=torch.uint8, device=a.device)
    wsb = workspace.numel() if workspace is not None else 0
    _check(load().curvefp_gemm_oriented(ALGOS[algo], _fmt(fmt_a), _fmt(fmt_b), block, _p(a), _p(sa),
                                        LAYOUTS[layout_a], _p(b), _p(sb), LAYOUTS[layout_b], M, N, K, _p(c), _p(ps),
                                        _p(pl), _p(workspace), wsb, _p(status), _stream(stream)))
    return (c, ps, pl) if phases else c


def gemm_requant(a, sa, b, sb, fmt_a, fmt_b, fmt_c, block: int = 32, block_c: int = 32, algo: str = "tensor",
                 c=None, codes_c=None, scales_c=None, status=None, stream=None):
    """C = A_hat B_hat^T and its requantization Q(C) (blocks along N).
    Returns (c [M x N] fp32, codes_c, scales_c)."""
    import torch

    M, K = a.shape
    N = b.shape[0]
    if c is None:
        c = torch.empty((M, N), dtype=torch.float32, device=a.device)
    if codes_c is None:
        codes_c = torch.empty((M, N), dtype=torch.uint8, device=a.device)
    if scales_c is None:
        scales_c = torch.empty((M, N // block_c), dtype=torch.int8, device=a.device)
    _check(load().curvefp_gemm_requant(ALGOS[algo], _fmt(fmt_a), _fmt(fmt_b), block, _p(a), _p(sa), _p(b), _p(sb), M,
                                       N, K, _p(c), _fmt(fmt_c), block_c, _p(codes_c), _p(scales_c), _p(status),
                                       _stream(stream)))
    return c, codes_c, scales_c


def gemm_q32(a, sa, b, sb, fmt_a, fmt_b, block: int = 32, out=None, status=None, stream=None):
    """The tile's Q32 integer accumulators [M x N] int64 (value = acc 2^-32)."""
    import torch

    M, K = a.shape
    N = b.shape[0]
    if out is None:
        out = torch.empty((M, N), dtype=torch.int64, device=a.device)
    _check(load().curvefp_gemm_q32(_fmt(fmt_a), _fmt(fmt_b), block, _p(a), _p(sa), _p(b), _p(sb), M, N, K, _p(out),
                                   _p(status), _stream(stream)))
    return out


def gemm_phases_histogram(a, sa, b, sb, fmt_a, fmt_b, block: int = 32, status=None, stream=None):
    """gemm_phases computed with the histogram layout (signed-popcount merged
    counts n_{h,t}); returns (C, phase sums, LSBs) like gemm_phases."""
    import torch

    M, K = a.shape
    N = b.shape[0]
    H = phase_count(fmt_a, fmt_b)
    c = torch.empty((M, N), dtype=torch.float32, device=a.device)
    ps = torch.empty((M, N, H, 2), dtype=torch.int64, device=a.device)
    pl = torch.empty((M, N), dtype=torch.int32, device=a.device)
    _check(load().curvefp_gemm_phases_histogram(_fmt(fmt_a), _fmt(fmt_b), block, _p(a), _p(sa), _p(b), _p(sb), M, N,
                                                K, _p(c), _p(ps), _p(pl), _p(status), _stream(stream)))
    return c, ps, pl


def gemm_phases(a, sa, b, sb, fmt_a, fmt_b, block: int = 32, status=None, stream=None):
    """Exact GEMM that also returns the per-phase int128 sums as (lo, hi)
    int64 pairs [M x N x H x 2] and their LSB exponents [M x N]."""
    import torch

    M, K = a.shape
    N = b.shape[0]
    H = phase_count(fmt_a, fmt_b)
    c = torch.empty((M, N), dtype=torch.float32, device=a.device)
    ps = torch.empty((M, N, H, 2), dtype=torch.int64, device=a.device)
    pl = torch.empty((M, N), dtype=torch.int32, device=a.device)
    _check(load().curvefp_gemm_phases(_fmt(fmt_a), _fmt(fmt_b), block, _p(a), _p(sa), _p(b), _p(sb), M, N, K,
                                      _p(c), _p(ps), _p(pl), _p(status), _stream(stream)))
    return c, ps, pl


def selftest_bounded_wait(arrive: bool, limit_cycles: int, status, stream=None):
    """Failure-detection self-test of the tensor-core pipeline's bounded wait
    (curvefp_selftest_bounded_wait): with arrive=False the wait gives up after
    limit_cycles SM cycles and ORs the TIMEOUT bit into `status` (a CUDA
    int32/uint32 tensor of one element)."""
    _check(load().curvefp_selftest_bounded_wait(1 if arrive else 0, int(limit_cycles), _p(status), _stream(stream)))
