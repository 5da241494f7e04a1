"""Guard bands around every output buffer (the substitute for a memory
sanitizer): each entry point writes into a view in the middle of a larger
buffer whose bands before and after hold a byte pattern; after the call, the
bands must be unchanged, on ragged shapes (M, N in {1, 3, 17, 130, 200}),
both block axes, every GEMM algorithm (the tensor kernel's split tail tiles
included: their rows of C are zeroed by a memset first) and the static,
requantizing, oriented, Q32 and exact-phase entry points."""
import ctypes

import numpy as np
import pytest

from paper_2608_10010_gb300 import inputs
from tests.gpu_util import new_status, status_bits, to_dev, torch_cuda

pytestmark = pytest.mark.gpu
BAND = 4096  # bytes of guard before and after (keeps the view 16-byte aligned)
PATTERN = 0xA5


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


class Guarded:
    """A [shape] tensor of `dtype` inside a buffer with guard bands."""

    def __init__(self, torch, shape, dtype):
        self.n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        self.buf = torch.full((BAND + self.n + BAND,), PATTERN, dtype=torch.uint8, device="cuda")
        self.t = self.buf[BAND:BAND + self.n].view(dtype).view(*shape)

    def intact(self):
        head = self.buf[:BAND].cpu().numpy()
        tail = self.buf[BAND + self.n:].cpu().numpy()
        return bool(np.all(head == PATTERN) and np.all(tail == PATTERN))


SHAPES = [(1, 1, 32), (3, 17, 64), (17, 3, 96), (130, 200, 256), (200, 130, 512)]
WIDE = [(530, 130, 64)]  # two token groups per CTA in the narrow kernel (M >= 512)


def _operands(torch, cfp, M, N, K, fa, fb, G=32):
    x = to_dev(torch, inputs.outlier_channels((M, K), M * 7 + K))
    w = to_dev(torch, inputs.normal((N, K), N * 11 + K, 0.02))
    a, sa = cfp.quantize(x, fa, G, 0)
    b, sb = cfp.quantize(w, fb, G, 0)
    return a, sa, b, sb


@pytest.mark.parametrize("fmt", ["E3C3", "E4C3", "E5C2", "E4C3_R8_9", "E4C3_R3_4"])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("axis", [0, 1])
def test_quantize_and_dequantize_stay_inside(torch, fmt, dtype, axis):
    import paper_2608_10010_gb300 as cfp

    for rows, cols in [(1, 32), (3, 96), (17, 64), (130, 256)]:
        if axis == 1:
            rows, cols = cols, rows  # blocks run down the columns: rows a multiple of 32
        x = to_dev(torch, inputs.elementwise_outliers((rows, cols), rows + cols), dtype)
        R, C = (cols, rows) if axis else (rows, cols)
        codes, scales = Guarded(torch, (R, C), torch.uint8), Guarded(torch, (R, C // 32), torch.int8)
        cfp.quantize(x, fmt, 32, axis, codes=codes.t, scales=scales.t)
        out = Guarded(torch, (R, C), torch.float32)
        cfp.dequantize(codes.t, scales.t, fmt, 32, out=out.t)
        torch.cuda.synchronize()
        assert codes.intact() and scales.intact() and out.intact(), (rows, cols)


@pytest.mark.parametrize("group", ["block", "row", "tensor"])
@pytest.mark.parametrize("rule", ["ceil", "mse"])
def test_static_quantize_stays_inside(torch, group, rule):
    import paper_2608_10010_gb300 as cfp

    for rows, cols in [(1, 32), (17, 64), (130, 256)]:
        x = to_dev(torch, inputs.lognormal_channels((rows, cols), rows * cols))
        for fn in (cfp.quantize_static, cfp.quantize_static_noalloc):
            codes, scales = Guarded(torch, (rows, cols), torch.uint8), Guarded(torch, (rows, cols // 32), torch.int8)
            fn(x, "E4C3", 32, group, rule, codes=codes.t, scales=scales.t)
            torch.cuda.synchronize()
            assert codes.intact() and scales.intact(), (fn.__name__, rows, cols)


@pytest.mark.parametrize("algo,fa,fb", [("exact", "E3C3", "E5C2"), ("tensor", "E3C3", "E3C3"),
                                        ("tensor", "E5C2", "E4C3"), ("tensor", "E4C3_R8_9", "E4C3_R8_9"),
                                        ("tensor_narrow", "E5C2", "E4C3"), ("skinny", "E4C3", "E5C2"),
                                        ("auto", "E4C3", "E4C3"), ("exact", "E4C3_R3_4", "E4C3_R3_4"),
                                        ("tensor_narrow", "E3C3", "E3C3"), ("tensor_narrow", "E5C2", "E5C2"),
                                        ("tensor_narrow", "E4C3", "E5C2"),
                                        ("tensor_narrow", "E4C3_R3_4", "E4C3_R3_4")])
def test_gemm_stays_inside(torch, algo, fa, fb):
    import paper_2608_10010_gb300 as cfp

    for M, N, K in SHAPES + (WIDE if algo == "tensor_narrow" else []):
        if algo == "skinny" and M > 8:
            continue
        a, sa, b, sb = _operands(torch, cfp, M, N, K, fa, fb)
        c = Guarded(torch, (M, N), torch.float32)
        st = new_status(torch)
        cfp.gemm(a, sa, b, sb, fa, fb, 32, algo, out=c.t, status=st)
        torch.cuda.synchronize()
        assert c.intact() and status_bits(st) == 0, (M, N, K)


def test_exact_phase_entry_points_stay_inside(torch):
    """curvefp_gemm_phases, its histogram layout and curvefp_gemm_q32 with
    every output guarded (called through the C ABI directly)."""
    import paper_2608_10010_gb300 as cfp

    lib = cfp.load()
    P = ctypes.c_void_p
    for M, N, K in SHAPES:
        a, sa, b, sb = _operands(torch, cfp, M, N, K, "E4C3", "E3C3")
        H = cfp.phase_count("E4C3", "E3C3")
        ops = [P(t.data_ptr()) for t in (a, sa, b, sb)]
        for fn in (lib.curvefp_gemm_phases, lib.curvefp_gemm_phases_histogram):
            c = Guarded(torch, (M, N), torch.float32)
            ps = Guarded(torch, (M, N, H, 2), torch.int64)
            pl = Guarded(torch, (M, N), torch.int32)
            rc = fn(1, 0, 32, *ops, M, N, K, P(c.t.data_ptr()), P(ps.t.data_ptr()), P(pl.t.data_ptr()), None,
                    P(torch.cuda.current_stream().cuda_stream))
            torch.cuda.synchronize()
            assert rc == 0 and c.intact() and ps.intact() and pl.intact(), (fn.__name__, M, N, K)
        # Q32 tiles take the tensor kernel's format pairs
        a, sa, b, sb = _operands(torch, cfp, M, N, K, "E5C2", "E4C3")
        acc = Guarded(torch, (M, N), torch.int64)
        cfp.gemm_q32(a, sa, b, sb, "E5C2", "E4C3", 32, out=acc.t)
        torch.cuda.synchronize()
        assert acc.intact(), (M, N, K)


@pytest.mark.parametrize("algo", ["tensor", "exact"])
def test_requant_and_oriented_stay_inside(torch, algo):
    import paper_2608_10010_gb300 as cfp

    for M, N, K in [(3, 64, 64), (130, 96, 256), (200, 160, 512)]:
        a, sa, b, sb = _operands(torch, cfp, M, N, K, "E4C3", "E4C3")
        c = Guarded(torch, (M, N), torch.float32)
        codes = Guarded(torch, (M, N), torch.uint8)
        scales = Guarded(torch, (M, N // 32), torch.int8)
        cfp.gemm_requant(a, sa, b, sb, "E4C3", "E4C3", "E5C2", 32, 32, algo, c=c.t, codes_c=codes.t,
                         scales_c=scales.t)
        torch.cuda.synchronize()
        assert c.intact() and codes.intact() and scales.intact(), (M, N, K)
        # B read transposed: its codes stored [K x N], blocked along N
        w = to_dev(torch, inputs.normal((K, N), K + N, 0.02))
        bt, sbt = cfp.quantize(w, "E4C3", 32, 0)
        c2 = Guarded(torch, (M, N), torch.float32)
        need = cfp.gemm_oriented_workspace_bytes("rows", "cols", M, N, K, algo)
        ws = Guarded(torch, (max(need, 16),), torch.uint8)
        cfp.gemm_oriented(a, sa, "rows", bt, sbt, "cols", "E4C3", "E4C3", 32, algo, out=c2.t, workspace=ws.t)
        torch.cuda.synchronize()
        assert c2.intact() and ws.intact(), (M, N, K)
