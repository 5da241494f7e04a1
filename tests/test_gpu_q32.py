"""The tile's Q32 integer semantics on the GPU (App. C.1, C.2), bit-exact:
against the oracle's exact phase sums (sum_h round(2^{h/L} 2^16) S_h
2^{lambda+16}) and, on the paper's verification design, against the tile's
own per-product coefficient-select-and-shift."""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from tests import exact as X
from tests.gpu_util import new_status, status_bits, torch_cuda

pytestmark = pytest.mark.gpu
PAIRS = [("E4C3", "E4C3"), ("E3C3", "E3C3"), ("E5C2", "E5C2"), ("E5C2", "E4C3"), ("E4C3", "E5C2")]
GOLD = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def torch():
    t = torch_cuda()
    import paper_2608_10010_gb300 as cfp

    cfp.load()
    return t


def q16(k, L):
    return int((X.pow2(k, L) * (1 << 16)).to_integral_value())


def gpu_q32(torch, a, sa, b, sb, fa, fb, block):
    import paper_2608_10010_gb300 as cfp

    d = lambda t: torch.from_numpy(np.ascontiguousarray(t)).cuda()
    st = new_status(torch)
    acc = cfp.gemm_q32(d(a), d(sa), d(b), d(sb), fa, fb, block, status=st)
    torch.cuda.synchronize()
    return acc.cpu().numpy(), status_bits(st)


BIAS = {"E3C3": 32, "E4C3": 64, "E5C2": 64}
# rank band keeping every product's Q32 shift 16 + e + sa + sb in [0, 45]:
# the tile's fixed point covers E4C3's product range, not all of E5C2's
BAND = {"E3C3": 31, "E4C3": 63, "E5C2": 30}


def band_codes(rng, fmt, shape):
    n = rng.integers(-BAND[fmt], BAND[fmt] + 1, shape)
    codes = ((n + BIAS[fmt]) | (rng.integers(0, 2, shape) << 7)).astype(np.uint8)
    codes[rng.random(shape) < 0.05] = 0  # zero sentinels
    return codes


@pytest.mark.parametrize("fa,fb", PAIRS)
def test_q32_matches_phase_sums(torch, fa, fb):
    rng = np.random.default_rng(31)
    M, N, K, G = 37, 21, 320, 32
    a = band_codes(rng, fa, (M, K))
    b = band_codes(rng, fb, (N, K))
    sa = rng.integers(0, 4, (M, K // G)).astype(np.int8)
    sb = rng.integers(0, 4, (N, K // G)).astype(np.int8)
    acc, st = gpu_q32(torch, a, sa, b, sb, fa, fb, G)
    assert st == 0
    r = oracle.gemm(a, sa, b, sb, fa, fb, G)
    S = oracle.int128_to_int(r["S_raw"])
    L = oracle.pair_info(fa, fb)[0]
    q = [q16(h, L) for h in range(L)]
    for i in range(M):
        for j in range(N):
            lam = int(r["lsb"][i, j])
            want = sum(q[h] * int(S[i, j, h]) for h in range(L)) * Fraction(2) ** (lam + 16)
            assert want.denominator == 1 and int(acc[i, j]) == int(want)


def test_q32_range_flag(torch):
    """Scales far below zero need negative shifts, and the full E5C2 product
    range does not fit the tile's fixed point: reported, not wrapped."""
    a = np.full((2, 64), 0x41, np.uint8)
    b = np.full((2, 64), 0x41, np.uint8)
    s = np.full((2, 2), -20, np.int8)
    _, st = gpu_q32(torch, a, s, b, s, "E4C3", "E4C3", 32)
    assert st & 2
    lo = np.full((2, 64), 0x01, np.uint8)  # n = -63: e = -32 for E5C2 x E5C2
    _, st = gpu_q32(torch, lo, np.zeros((2, 2), np.int8), lo, np.zeros((2, 2), np.int8), "E5C2", "E5C2", 32)
    assert st & 2


def test_q32_paper_verification_design(torch):
    """App. C.2: 64 seeded E4C3 matrix pairs (sum of K = 1,010; 1,024 outputs)
    through the GPU Q32 kernel, each output against the tile semantics written
    per product: coefficient round(2^{k/8} 2^16) for q_p = m_a + m_b - 128 =
    8e + k, shifted by 16 + e into Q32, signed by s_a xor s_b.  K is padded
    with zero codes to a multiple of 32 (zeros never update)."""
    with open(os.path.join(GOLD, "tile_verification_design.json")) as fh:
        design = json.load(fh)
    rng = np.random.default_rng(2027)
    cuts = np.sort(rng.choice(np.arange(1, design["total_k"]), design["matrices"] - 1, replace=False))
    ks = np.diff(np.concatenate([[0], cuts, [design["total_k"]]]))
    q = [q16(k, 8) for k in range(8)]
    outputs = 0
    for K in ks:
        a = rng.integers(0, 256, size=(4, K), dtype=np.uint8)
        b = rng.integers(0, 256, size=(4, K), dtype=np.uint8)
        Kp = (K + 31) // 32 * 32
        ap = np.zeros((4, Kp), np.uint8)
        bp = np.zeros((4, Kp), np.uint8)
        ap[:, :K], bp[:, :K] = a, b
        zs = np.zeros((4, Kp // 32), np.int8)
        acc, st = gpu_q32(torch, ap, zs, bp, zs, "E4C3", "E4C3", 32)
        assert st == 0
        for i in range(4):
            for j in range(4):
                want = 0
                for d in range(K):
                    ma, mb = int(a[i, d]) & 0x7F, int(b[j, d]) & 0x7F
                    if ma == 0 or mb == 0:
                        continue
                    qp = ma + mb - 128
                    term = q[qp & 7] << (16 + (qp >> 3))
                    want += -term if (a[i, d] ^ b[j, d]) & 0x80 else term
                assert int(acc[i, j]) == want
                outputs += 1
    assert outputs == design["total_outputs"]
