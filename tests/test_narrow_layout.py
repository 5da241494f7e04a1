"""The operand algebra of the TENSOR_NARROW kernel, checked on the CPU against
the oracle's closed-product GEMM (Eq. 2, Eq. 5).

A numpy model of what the kernel's MMAs compute, at the level of plane values
(not bytes): weight plane k_w (the 128-row operand) against the window of L
column blocks from block L - k_w WW of Q = [carry copies of the activation
planes on lattice positions 0..L-1 | plain copies], accumulating
D[w][h Mt + m] = S_h; for same-format pairs the 2:4-sparse form, where pair
plane j (planes j and j + K/2 at logical positions 2k, 2k + 1) meets the
window of R blocks from L - j with R_b[2k] = Q_b[k], R_b[2k + 1] = Q_{b-K/2}[k].
The phase combine sum_h 2^{h/L} S_h then has to reproduce the oracle's C for
every format pair; a wrong window start, a missing carry copy or a swapped
interleave fails it."""
import numpy as np
import pytest

import oracle

FMTS = {"E3C3": (3, 3), "E4C3": (4, 3), "E5C2": (5, 2)}
PAIRS = [("E3C3", "E3C3"), ("E4C3", "E4C3"), ("E5C2", "E4C3"), ("E4C3", "E5C2"), ("E5C2", "E5C2")]


def planes(codes, scales, fmt, G):
    """Per element: curve index k and the power-of-two plane value
    +-2^{e + a_b - ref} (ref = the row's largest block scale), the code
    layout of the oracle's reading R1; zero codes have value 0."""
    E, C = FMTS[fmt]
    K, B = 1 << C, 1 << (E + C - 1)
    m = (codes & (0x3F if fmt == "E3C3" else 0x7F)).astype(np.int64)
    n = m - B
    e = np.floor_divide(n, K)
    k = n - e * K
    a = np.repeat(scales.astype(np.int64), G, axis=1)
    ref = scales.max(axis=1).astype(np.int64)
    v = np.where(codes & 0x80, -1.0, 1.0) * np.exp2((e + a - ref[:, None]).astype(float))
    return k, np.where(m != 0, v, 0.0), ref


def narrow_model(a, sa, b, sb, fx, fw, G, Mt, sparse):
    M, Kd = a.shape
    KX, KW = 1 << FMTS[fx][1], 1 << FMTS[fw][1]
    L = max(KX, KW)
    WX, WW = L // KX, L // KW
    kx, vx, rx = planes(a, sa, fx, G)
    kw, vw, rw = planes(b, sb, fw, G)
    C = np.zeros((M, b.shape[0]))
    for x0 in range(0, M, Mt):  # one token group per CTA tile
        toks = np.arange(x0, min(x0 + Mt, M))
        D = np.zeros((b.shape[0], L * Mt))
        # Q[u] (u < L: carry copy of position u; u >= L: plain), [Mt x K]
        Q = np.zeros((2 * L, Mt, Kd))
        for u in range(L):
            if u % WX == 0:
                pl = np.where(kx[toks] == u // WX, vx[toks], 0.0)
                Q[u, : len(toks)] = 2 * pl
                Q[L + u, : len(toks)] = pl
        if not sparse:
            for k in range(KW):
                window = Q[L - k * WW: 2 * L - k * WW].reshape(L * Mt, Kd)
                D += np.where(kw == k, vw, 0.0) @ window.T
        else:
            hb = KW // 2
            for j in range(hb):
                # logical K 2 Kd: A[2k] = plane j, A[2k + 1] = plane j + hb
                A = np.zeros((b.shape[0], 2 * Kd))
                A[:, 0::2] = np.where(kw == j, vw, 0.0)
                A[:, 1::2] = np.where(kw == j + hb, vw, 0.0)
                R = np.zeros((L, Mt, 2 * Kd))
                for h in range(L):
                    R[h, :, 0::2] = Q[L - j + h]
                    R[h, :, 1::2] = Q[L - j + h - hb]
                D += A @ R.reshape(L * Mt, 2 * Kd).T
        ph = np.exp2(np.arange(L) / L)
        S = D.reshape(-1, L, Mt)  # [w, h, m]
        Ct = np.einsum("h,whm->mw", ph, S)[: len(toks)]
        C[toks] = Ct * np.exp2((rx[toks][:, None] + rw[None, :]).astype(float))
    return C


def _operand(rng, fmt, rows, K, G):
    codes = rng.integers(0, 256, size=(rows, K), dtype=np.uint8)
    if fmt == "E3C3":
        codes &= 0xBF
    return codes, rng.integers(-4, 5, size=(rows, K // G)).astype(np.int8)


@pytest.mark.parametrize("fx,fw", PAIRS)
@pytest.mark.parametrize("sparse", [False, True])
def test_windows_reproduce_the_oracle(fx, fw, sparse):
    if sparse and fx != fw:
        pytest.skip("the sparse form is for same-format pairs")
    rng = np.random.default_rng(len(fx) + 7 * len(fw) + sparse)
    G = 32
    a, sa = _operand(rng, fx, 21, 128, G)  # 21 tokens: groups of 8, 8 and 5 (padding)
    b, sb = _operand(rng, fw, 40, 128, G)
    ref = oracle.gemm(a, sa, b, sb, fx, fw, G, phases=False)["C"]
    got = narrow_model(a, sa, b, sb, fx, fw, G, 8, sparse)
    assert np.abs(got - ref).max() <= 1e-12 * np.abs(ref).max()


def test_a_wrong_window_start_is_caught():
    """The same model with each weight plane meeting the window one block off
    (a plausible indexing slip) no longer matches the oracle."""
    rng = np.random.default_rng(3)
    a, sa = _operand(rng, "E4C3", 8, 64, 32)
    b, sb = _operand(rng, "E4C3", 16, 64, 32)
    ref = oracle.gemm(a, sa, b, sb, "E4C3", "E4C3", 32, phases=False)["C"]
    kx, vx, rx = planes(a, sa, "E4C3", 32)
    kw, vw, rw = planes(b, sb, "E4C3", 32)
    L, Mt = 8, 8
    Q = np.zeros((2 * L, Mt, 64))
    for u in range(L):
        pl = np.where(kx == u, vx, 0.0)
        Q[u], Q[L + u] = 2 * pl, pl
    D = np.zeros((16, L * Mt))
    for k in range(L):
        start = L - k + (1 if k else 0)  # one block off for every plane but the first
        D += np.where(kw == k, vw, 0.0) @ Q[start: start + L].reshape(L * Mt, 64).T
    S = D.reshape(-1, L, Mt)
    C = np.einsum("h,whm->mw", np.exp2(np.arange(L) / L), S) * np.exp2((rx[:, None] + rw[None, :]).astype(float))
    assert np.abs(C - ref).max() > 1e-3 * np.abs(ref).max()
