"""The operand algebra of the TENSOR_NARROW kernel, checked on the CPU against
the oracle's closed-product GEMM (Eq. 2, Eq. 5).

A numpy model of what the kernel's MMAs compute, at the level of plane values
and scale factors (not bytes): every element's plane value is the power of
two 2^e of its code (one binade low on an E5C2 token operand, whose carry
copies need the room), every 32-code step of a row carries the scale factor
2^{a_b - ref + 32}, and weight pair plane j (planes j and j + K_W/2 at
logical positions 2k, 2k + 1) meets the window of L column blocks from R
block L - j WW, with R_b[2k] = Q_b[k], R_b[2k + 1] = Q_{b - PO}[k],
PO = K_W/2 WW, and Q = [carry copies of the token planes on lattice
positions 0..L-1 | plain copies], token plane k on position k WX (WX = 2
for E5C2 tokens against E4C3 weights, the odd positions empty).
D[w][h Mt + m] = S_h, and the phase combine
sum_h 2^{h/L} S_h 2^{ref_w + ref_m - 64} has to reproduce the oracle's C for
every format pair (tokens = A's rows, weights = B's rows); a wrong window
start, a missing carry copy, a swapped interleave, a plane on the wrong
lattice position or a scale factor on the wrong block fails it.

The byte-level arithmetic that forms the E5M2 plane bytes four codes at a
time (tc_mx.cuh mx_word) is emulated on every code byte in every lane."""
import numpy as np
import pytest

import oracle

FMTS = {"E3C3": (3, 3), "E4C3": (4, 3), "E5C2": (5, 2)}
PAIRS = [("E3C3", "E3C3"), ("E4C3", "E4C3"), ("E5C2", "E4C3"), ("E4C3", "E5C2"), ("E5C2", "E5C2")]
MX_OFF = 32


def fields(codes, fmt):
    E, C = FMTS[fmt]
    K, B = 1 << C, 1 << (E + C - 1)
    m = (codes & (0x3F if fmt == "E3C3" else 0x7F)).astype(np.int64)
    n = m - B
    e = np.floor_divide(n, K)
    return m, e, n - e * K


def planes(codes, scales, fmt, G, bias):
    """Per element: curve index k, the plane value +-2^{e - bias} (0 for zero
    codes and, with bias 1, for the plain copy of e = -16, which E5M2 cannot
    hold), the carry value +-2^{e - bias + 1}, the per-element scale factor
    exponent a_b - ref + 32 + bias, and the row reference."""
    m, e, k = fields(codes, fmt)
    sgn = np.where(codes & 0x80, -1.0, 1.0)
    v = np.where((m != 0) & (e - bias >= -16), sgn * np.exp2((e - bias).astype(float)), 0.0)
    vc = np.where(m != 0, sgn * np.exp2((e - bias + 1).astype(float)), 0.0)
    ref = scales.max(axis=1).astype(np.int64)
    sf = np.repeat(scales.astype(np.int64), G, axis=1) - ref[:, None] + MX_OFF + bias
    return k, v, vc, sf, ref


def narrow_model(x, sx, w, sw, fx, fw, G, Mt):
    """C[m][n] = x_hat[m] . w_hat[n] as the kernel forms it (tokens x, weights w)."""
    M, Kd = x.shape
    KX, KW = 1 << FMTS[fx][1], 1 << FMTS[fw][1]
    L = max(KX, KW)
    WX, WW = L // KX, L // KW
    bx = 1 if fx == "E5C2" else 0
    kx, vx, cx, fxs, rx = planes(x, sx, fx, G, bx)
    kw, vw, _, fws, rw = planes(w, sw, fw, G, 0)
    hb = KW // 2
    po = hb * WW
    C = np.zeros((M, w.shape[0]))
    for x0 in range(0, M, Mt):  # one token group per CTA tile
        toks = np.arange(x0, min(x0 + Mt, M))
        D = np.zeros((w.shape[0], L * Mt))
        # Q[u] (u < L: carry copy of position u; u >= L: plain), [Mt x K],
        # with the tokens' scale factors applied (the B factors of a column)
        Q = np.zeros((2 * L, Mt, Kd))
        scale_x = np.exp2(fxs[toks].astype(float))
        for u in range(L):
            Q[u, : len(toks)] = np.where(kx[toks] * WX == u, cx[toks], 0.0) * scale_x
            Q[L + u, : len(toks)] = np.where(kx[toks] * WX == u, vx[toks], 0.0) * scale_x
        scale_w = np.exp2(fws.astype(float))
        for j in range(hb):
            # logical K 2 Kd: A[2k] = plane j, A[2k + 1] = plane j + hb (the A factors)
            A = np.zeros((w.shape[0], 2 * Kd))
            A[:, 0::2] = np.where(kw == j, vw, 0.0) * scale_w
            A[:, 1::2] = np.where(kw == j + hb, vw, 0.0) * scale_w
            R = np.zeros((L, Mt, 2 * Kd))
            for h in range(L):
                R[h, :, 0::2] = Q[L - j * WW + h]
                R[h, :, 1::2] = Q[L - j * WW + h - po]
            D += A @ R.reshape(L * Mt, 2 * Kd).T
        ph = np.exp2(np.arange(L) / L)
        S = D.reshape(-1, L, Mt)  # [w, h, m]
        Ct = np.einsum("h,whm->mw", ph, S)[: len(toks)]
        C[toks] = Ct * np.exp2((rx[toks][:, None] + rw[None, :] - 2 * MX_OFF).astype(float))
    return C


def _operand(rng, fmt, rows, K, G, spread=4):
    codes = rng.integers(0, 256, size=(rows, K), dtype=np.uint8)
    if fmt == "E3C3":
        codes &= 0xBF
    return codes, rng.integers(-spread, spread + 1, size=(rows, K // G)).astype(np.int8)


@pytest.mark.parametrize("fa,fb", PAIRS)
def test_windows_reproduce_the_oracle(fa, fb):
    rng = np.random.default_rng(len(fa) + 7 * len(fb))
    G = 32
    a, sa = _operand(rng, fa, 21, 128, G)  # 21 tokens: groups of 8, 8 and 5 (padding)
    b, sb = _operand(rng, fb, 40, 128, G)
    if fa == "E5C2":
        a[:, :] = np.where((fields(a, fa)[1] == -16) & (a & 0x7F != 0), a + 4, a)  # no lowest-binade tokens
    ref = oracle.gemm(a, sa, b, sb, fa, fb, G, phases=False)["C"]
    got = narrow_model(a, sa, b, sb, fa, fb, G, 8)
    assert np.abs(got - ref).max() <= 1e-12 * np.abs(ref).max()


@pytest.mark.parametrize("fa,fb", PAIRS)
def test_scale_spread_is_carried_by_the_factors(fa, fb):
    """Block scales up to 30 binades apart along a row (beyond any FP8 plane range):
    the factors carry them, and the model still matches the oracle."""
    rng = np.random.default_rng(11 + len(fa))
    G = 32
    a, sa = _operand(rng, fa, 9, 256, G, spread=15)
    b, sb = _operand(rng, fb, 24, 256, G, spread=15)
    if fa == "E5C2":
        a[:, :] = np.where((fields(a, fa)[1] == -16) & (a & 0x7F != 0), a + 4, a)
    ref = oracle.gemm(a, sa, b, sb, fa, fb, G, phases=False)["C"]
    got = narrow_model(a, sa, b, sb, fa, fb, G, 8)
    na, nb = oracle.row_norms(a, sa, fa, G), oracle.row_norms(b, sb, fb, G)
    assert (np.abs(got - ref) / np.outer(na, nb)).max() <= 1e-12


def test_a_wrong_window_start_is_caught():
    """The same model with each weight pair plane meeting the window one block
    off (a plausible indexing slip) no longer matches the oracle."""
    rng = np.random.default_rng(3)
    a, sa = _operand(rng, "E4C3", 8, 64, 32)
    b, sb = _operand(rng, "E4C3", 16, 64, 32)
    ref = oracle.gemm(a, sa, b, sb, "E4C3", "E4C3", 32, phases=False)["C"]
    kx, vx, cx, fxs, rx = planes(a, sa, "E4C3", 32, 0)
    kw, vw, _, fws, rw = planes(b, sb, "E4C3", 32, 0)
    L, Mt = 8, 8
    Q = np.zeros((2 * L, Mt, 64))
    for u in range(L):
        Q[u] = np.where(kx == u, cx, 0.0) * np.exp2(fxs)
        Q[L + u] = np.where(kx == u, vx, 0.0) * np.exp2(fxs)
    D = np.zeros((16, L * Mt))
    for j in range(4):
        A = np.zeros((16, 128))
        A[:, 0::2] = np.where(kw == j, vw, 0.0) * np.exp2(fws)
        A[:, 1::2] = np.where(kw == j + 4, vw, 0.0) * np.exp2(fws)
        R = np.zeros((L, Mt, 128))
        start = L - j + (1 if j else 0)  # one block off for every pair but the first
        for h in range(L):
            R[h, :, 0::2] = Q[(start + h) % (2 * L)]
            R[h, :, 1::2] = Q[start + h - 4]
        D += A @ R.reshape(L * Mt, 128).T
    S = D.reshape(-1, L, Mt)
    C = np.einsum("h,whm->mw", np.exp2(np.arange(L) / L), S) * np.exp2(
        (rx[:, None] + rw[None, :] - 2 * MX_OFF).astype(float))
    assert np.abs(C - ref).max() > 1e-3 * np.abs(ref).max()


# ---- byte-level emulation of the plane-byte arithmetic (tc_mx.cuh) ----------

M32 = 0xFFFFFFFF


def prmt_sign(v, sel):
    """prmt.b32 r, v, 0, sel with sign replication (selector nibbles 8..B)."""
    out = 0
    for i in range(4):
        nib = (sel >> (4 * i)) & 0xF
        byte = (v >> (8 * (nib & 3))) & 0xFF
        out |= (0xFF if byte & 0x80 else 0) << (8 * i)
    return out


def e5m2_pow2(x):
    ge2 = prmt_sign((x + 0x7E7E7E7E) & M32, 0xBA98)
    nrm = (((((x | 0x80808080) - 0x01010101) & 0x1F1F1F1F) << 2) & M32) & ge2
    return nrm | ((x + 0x01010101) & ~ge2 & M32)


def mx_word(w, fmt, bias):
    E, C = FMTS[fmt]
    mm = (0x3F if fmt == "E3C3" else 0x7F) * 0x01010101
    sgn = w & 0x80808080
    nz = prmt_sign(((w & mm) + 0x7F7F7F7F) & M32, 0xBA98)
    eb = (w >> C) & (((1 << E) - 1) * 0x01010101)
    if E < 5:
        v = (sgn | (((eb + (15 - (1 << (E - 1))) * 0x01010101) << 2) & M32)) & nz
        return v, (v + (nz & 0x04040404)) & M32
    if bias == 0:
        return (sgn | e5m2_pow2(eb)) & nz, 0
    ge1 = prmt_sign((eb + 0x7F7F7F7F) & M32, 0xBA98)
    x = ((eb | 0x80808080) - 0x01010101) & 0x1F1F1F1F
    return (sgn | e5m2_pow2(x)) & nz & ge1, (sgn | e5m2_pow2(eb)) & nz


def e5m2_value(byte):
    s = -1.0 if byte & 0x80 else 1.0
    ex, man = (byte >> 2) & 31, byte & 3
    assert ex != 31, "no Inf/NaN plane bytes"
    return s * (man * 2.0 ** -16 if ex == 0 else (1 + man / 4) * 2.0 ** (ex - 15))


@pytest.mark.parametrize("fmt,bias", [("E3C3", 0), ("E4C3", 0), ("E5C2", 0), ("E5C2", 1)])
def test_plane_bytes_of_every_code_in_every_lane(fmt, bias):
    """Every code byte in every lane of a word (random neighbours): the plane
    byte is exactly +-2^{e - bias} (0 for the zero codes and, with bias 1, for
    e = -16), its carry byte +-2^{e - bias + 1}, and no lane disturbs
    another."""
    rng = np.random.default_rng(17)
    valid = [c for c in range(256) if not (fmt == "E3C3" and c & 0x40)]
    for c in valid:
        m, e, _ = fields(np.array([c], np.uint8), fmt)
        m, e = int(m[0]), int(e[0])
        s = -1.0 if c & 0x80 else 1.0
        want_v = 0.0 if m == 0 or e - bias < -16 else s * 2.0 ** (e - bias)
        want_c = 0.0 if m == 0 else s * 2.0 ** (e - bias + 1)
        for lane in range(4):
            nb = rng.choice(valid, size=4)
            nb[lane] = c
            w = int(nb[0]) | int(nb[1]) << 8 | int(nb[2]) << 16 | int(nb[3]) << 24
            v, vc = mx_word(w, fmt, bias)
            assert e5m2_value((v >> (8 * lane)) & 0xFF) == want_v, (c, lane)
            if fmt != "E5C2" or bias == 1:
                assert e5m2_value((vc >> (8 * lane)) & 0xFF) == want_c, (c, lane)


# ---- byte-level emulation of the activation R blocks and the weight metadata

def byte_perm(x, y, s):
    """__byte_perm(x, y, s): result byte i = byte (nibble i of s) of y:x."""
    src = (x & M32) | (y & M32) << 32
    return sum(((src >> (8 * ((s >> (4 * i)) & 7))) & 0xFF) << (8 * i) for i in range(4))


def r_blocks_emulated(w2, fx, bias, L, PO, RB0):
    """The X producer's R blocks for one work item (8 codes in two words),
    as gemm_tcn.cu forms them: three byte-duplicated words placed by the top
    curve-index bit, masked per block to the codes of class b mod PO."""
    C = FMTS[fx][1]
    qcc, qpc, qpp, dm0, dm1 = [0] * 4, [0] * 4, [0] * 4, [0] * 4, [0] * 4
    for q in range(2):
        w = w2[q]
        v, vc = mx_word(w, fx, bias)
        wt, w0, w1 = (w << (8 - C)) & M32, (w << 7) & M32, (w << 6) & M32
        for hh in range(2):
            sdup, dup, ilv = (0xBBAA, 0x3322, 0x7362) if hh else (0x9988, 0x1100, 0x5140)
            i = 2 * q + hh
            dt = prmt_sign(wt, sdup)
            dm0[i] = prmt_sign(w0, sdup)
            dm1[i] = prmt_sign(w1, sdup)
            qcc[i] = byte_perm(vc, vc, dup) & (dt ^ 0xFF00FF00)
            qpp[i] = byte_perm(v, v, dup) & (dt ^ 0xFF00FF00)
            qpc[i] = byte_perm(v, vc, ilv) & (dt ^ 0x00FF00FF)
    out = {}
    for b in range(RB0, 2 * L):
        j = b % PO
        words = []
        for i in range(4):
            src = qcc[i] if b < L else (qpc[i] if b < L + PO else qpp[i])
            words.append(src & (dm0[i] if j & 1 else ~dm0[i] & M32) & (dm1[i] if j & 2 else ~dm1[i] & M32))
        out[b] = b"".join(x.to_bytes(4, "little") for x in words)
    return out


def r_blocks_emulated_c2(w2, fx, bias, L, PO, RB0, WX):
    """The X producer's R blocks for two curve-index bits: the four planes of
    each word and of its carry copy by the curve-index masks, Q block u the
    plane on lattice position u mod L (plane k on position k WX), blocks whose
    two halves are both empty left unwritten (zero)."""
    pv, pc = [], []
    for w in w2:
        v, vc = mx_word(w, fx, bias)
        mk0, mk1 = prmt_sign((w << 7) & M32, 0xBA98), prmt_sign((w << 6) & M32, 0xBA98)
        n0, n1 = ~mk0 & M32, ~mk1 & M32
        pv.append([v & n0 & n1, v & mk0 & n1, v & n0 & mk1, v & mk0 & mk1])
        pc.append([vc & n0 & n1, vc & mk0 & n1, vc & n0 & mk1, vc & mk0 & mk1])

    def qb(q, u):
        pos = u if u < L else u - L
        if pos % WX:
            return 0
        return (pc if u < L else pv)[q][pos // WX]

    out = {}
    for b in range(RB0, 2 * L):
        if b % WX and (b - PO) % WX:
            out[b] = bytes(16)
            continue
        words = []
        for q in range(2):
            x, y = qb(q, b), qb(q, b - PO)
            words += [byte_perm(x, y, 0x5140), byte_perm(x, y, 0x7362)]
        out[b] = b"".join(x.to_bytes(4, "little") for x in words)
    return out


def r_blocks_defined(w2, fx, bias, L, PO, RB0, WX=1):
    """R_b[2k] = Q_b[k], R_b[2k + 1] = Q_{b - PO}[k]; Q_u = the carry bytes
    of the codes on lattice position u (u < L), the plain bytes of those on
    position u - L (u >= L); a code's position is its curve index (low C
    bits) times WX."""
    C = FMTS[fx][1]
    codes, vb, cb = [], [], []
    for w in w2:
        v, vc = mx_word(w, fx, bias)
        for lane in range(4):
            codes.append((w >> (8 * lane)) & 0xFF)
            vb.append((v >> (8 * lane)) & 0xFF)
            cb.append((vc >> (8 * lane)) & 0xFF)

    def Q(u, k):
        pos = (codes[k] & ((1 << C) - 1)) * WX
        if u < L:
            return cb[k] if pos == u else 0
        return vb[k] if pos == u - L else 0

    return {b: bytes(x for k in range(8) for x in (Q(b, k), Q(b - PO, k))) for b in range(RB0, 2 * L)}


@pytest.mark.parametrize("fx,fw", [("E3C3", "E3C3"), ("E4C3", "E4C3"), ("E4C3", "E5C2")])
def test_r_blocks_are_the_interleaved_q_blocks(fx, fw):
    """The R blocks the activation producers store for three curve-index bits
    (16 bytes per block and work item) equal their definition byte for byte,
    for every such kernel orientation's lattice (L, PO, first block) and
    random codes (zeros, both signs, every curve index)."""
    KX, KW = 1 << FMTS[fx][1], 1 << FMTS[fw][1]
    L = max(KX, KW)
    WW, HB = L // KW, KW // 2
    PO, RB0 = HB * WW, L - (HB - 1) * WW
    bias = 1 if fx == "E5C2" else 0
    rng = np.random.default_rng(29)
    valid = np.array([c for c in range(256) if not (fx == "E3C3" and c & 0x40)], np.int64)
    for _ in range(3000):
        c = rng.choice(valid, size=8)
        if rng.random() < 0.2:
            c[rng.integers(0, 8)] = 0  # zero codes
        w2 = [int(c[0] | c[1] << 8 | c[2] << 16 | c[3] << 24), int(c[4] | c[5] << 8 | c[6] << 16 | c[7] << 24)]
        assert r_blocks_emulated(w2, fx, bias, L, PO, RB0) == r_blocks_defined(w2, fx, bias, L, PO, RB0), c


def pair_meta_emulated(w, mbit):
    """gemm_tcn.cu pair_meta: gather the selector bits of four code words,
    transpose the 4 x 4 matrix of 2-bit cells with two delta swaps."""
    a = 0
    for q in range(4):
        sh = mbit - 2 * q
        a |= ((w[q] >> sh) if sh >= 0 else (w[q] << -sh)) & (0x01010101 << (2 * q)) & M32
    t = (a ^ (a >> 12)) & 0x0000F0F0
    a ^= t ^ (t << 12)
    t = (a ^ (a >> 6)) & 0x00CC00CC
    a ^= t ^ (t << 6)
    return (a | 0x88888888) & M32


@pytest.mark.parametrize("mbit", [1, 2])
def test_pair_metadata_selects_the_partner_plane(mbit):
    """Metadata of 16 codes of a 2:4 operand with 8-bit elements: per chunk of
    two elements (codes 2c, 2c + 1) the positions bit(2c) and 2 + bit(2c + 1)
    of the curve-index bit that selects the partner plane (nibble c)."""
    rng = np.random.default_rng(31)
    for _ in range(20000):
        w = [int(x) for x in rng.integers(0, 1 << 32, size=4, dtype=np.uint64)]
        codes = [(w[k // 4] >> (8 * (k % 4))) & 0xFF for k in range(16)]
        want = 0
        for c in range(8):
            b0, b1 = (codes[2 * c] >> mbit) & 1, (codes[2 * c + 1] >> mbit) & 1
            want |= (b0 | (2 + b1) << 2) << (4 * c)
        assert pair_meta_emulated(w, mbit) == want, w


# ---- the plane bytes of r = 2^{3/4} (gemm_tcn_r34.cu) -----------------------

def r34_word_emulated(w):
    """gemm_tcn_r34.cu r34_word: the E5M2 byte of +-2^q, the nonzero mask and
    the curve plane j of four codes, from 3m in 16-bit lanes."""
    m4 = w & 0x7F7F7F7F
    nz = prmt_sign((m4 + 0x7F7F7F7F) & M32, 0xBA98)
    lo = ((m4 & 0x00FF00FF) * 3) & M32
    hi = (((m4 >> 8) & 0x00FF00FF) * 3) & M32
    j4 = (lo & 0x001F001F) | ((hi & 0x001F001F) << 8)
    q4 = ((lo >> 5) & 0x000F000F) | (((hi >> 5) & 0x000F000F) << 8)
    v = ((w & 0x80808080) | (((q4 + 0x09090909) << 2) & M32)) & nz
    return v, nz, j4


def test_r34_plane_bytes_of_every_code_in_every_lane():
    """Every code byte in every lane: the element 2^{3n/32} (n = m - 64) is
    2^q 2^{j/32} with the plane byte +-2^q and the curve plane j (3n = 32 q +
    j, 0 <= j < 32); the zero code gives 0; no lane disturbs another."""
    rng = np.random.default_rng(37)
    for c in range(256):
        m = c & 0x7F
        n = m - 64
        q, j = (3 * n) // 32, (3 * n) % 32
        s = -1.0 if c & 0x80 else 1.0
        for lane in range(4):
            nb = rng.integers(0, 256, size=4)
            nb[lane] = c
            w = int(nb[0]) | int(nb[1]) << 8 | int(nb[2]) << 16 | int(nb[3]) << 24
            v, nz, j4 = r34_word_emulated(w)
            vb = (v >> (8 * lane)) & 0xFF
            if m == 0:
                assert vb == 0 and (nz >> (8 * lane)) & 0xFF == 0, c
                continue
            assert e5m2_value(vb) == s * 2.0 ** q, (c, lane)
            assert (j4 >> (8 * lane)) & 0xFF == j, (c, lane)
            assert np.isclose(s * 2.0 ** q * 2.0 ** (j / 32), s * 2.0 ** (3 * n / 32), rtol=1e-15)


@pytest.mark.parametrize("fx,fw", [("E5C2", "E5C2"), ("E5C2", "E4C3")])
def test_two_bit_r_blocks_are_the_interleaved_q_blocks(fx, fw):
    """The same for two curve-index bits (E5C2 tokens, one binade low):
    against E5C2 weights every lattice position holds a plane; against E4C3
    weights the planes sit on the even positions of the 8-phase lattice and
    the blocks of odd b hold nothing."""
    KX, KW = 1 << FMTS[fx][1], 1 << FMTS[fw][1]
    L = max(KX, KW)
    WX, WW, HB = L // KX, L // KW, KW // 2
    PO, RB0 = HB * WW, L - (HB - 1) * WW
    rng = np.random.default_rng(31)
    for _ in range(3000):
        c = rng.integers(0, 256, size=8)
        if rng.random() < 0.2:
            c[rng.integers(0, 8)] = 0
        w2 = [int(c[0] | c[1] << 8 | c[2] << 16 | c[3] << 24), int(c[4] | c[5] << 8 | c[6] << 16 | c[7] << 24)]
        got = r_blocks_emulated_c2(w2, fx, 1, L, PO, RB0, WX)
        assert got == r_blocks_defined(w2, fx, 1, L, PO, RB0, WX), c
        if WX == 2:
            assert all(got[b] == bytes(16) for b in range(RB0, 2 * L) if b % 2)
