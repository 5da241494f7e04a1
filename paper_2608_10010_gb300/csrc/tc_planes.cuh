// Producer-side arithmetic shared by the tensor-core GEMM kernels: code words
// -> curve-plane values (FP8 E5M2 or BF16), curve-index masks and planes, the
// shared-memory block of the pipeline, and the phase constants of the
// epilogue (Sec. 3.2, Eq. 2, Eq. 5).
#pragma once
#include "cfp_common.cuh"

namespace cfp {

enum PlaneType { PLANE_BF16 = 0, PLANE_E5M2 = 1 };

constexpr int TC_MAX_RING = 4;  // capacity of the barrier rings below (= NSB)

// Step g is handed over on full[g % NSB] (A and B producers arrive once per
// warp) and released on empty[g % NSB] (one MMA commit): one wait and one
// commit per step on the MMA warp's path.  A producers refill TMEM unit g % 2
// after empty[(g - 2) % NSB]; B producers refill stage g % NSB after
// empty[(g - NSB) % NSB].
struct TcShared {
  uint64_t full[TC_MAX_RING], empty[TC_MAX_RING], acc_full, drain;
  uint64_t code_full[8], code_empty[8];  // ring of bulk-copied code tiles (where used)
  uint32_t tmem_base;
  int abort_flag;
  int refB[128];  // >= BN
};

__device__ __forceinline__ void raise_flag(uint32_t* status, uint32_t bit) {
  if (status) atomicOr(status, bit);
}
__device__ __forceinline__ int read_abort(const int* f) { return *reinterpret_cast<const volatile int*>(f); }

// ---------------------------------------------------------------------------
// Producer arithmetic, four codes per 32-bit word (SIMD within a register).
//
// A code byte is s | m with m = e_b K + k (e_b = e + 2^{E-1}, App. C.1), so
//   k   = the low C bits,  e_b = the next E bits,  s = bit 7.
// Plane value +-2^{x}, x = e_b - 2^{E-1} + off (off = block scale - row
// reference - plane bias).  An element is kept when x >= -14 (E5M2 normal
// range; smaller elements sit 2^14 below the row's largest element and flush
// to zero) or x >= -126 (BF16); its carry-plane copy is 2^{x+1}, which still
// fits (x <= 2^{E-1} - 1 - bias, so x + 1 + 15 <= 30).
//   E5M2:  byte s | (x + 15) << 2;   BF16:  half s | (x + 127) << 7.
// "Kept" is a threshold on the rank: e_b >= T  <=>  m >= max(K T, 1) = mt
// (m != 0 excludes the zero code), so bit 7 of m + (128 - mt) is the keep bit
// of each lane (m <= 127 and 128 - mt <= 127: no carry into the next lane).

// prmt with sign replication: byte i of the result is 0xFF where bit 7 of
// byte sel_i of v is set (selector nibbles 8..B pick bytes 0..3 with the sign
// mode).
__device__ __forceinline__ uint32_t prmt_sign(uint32_t v, uint32_t sel) {
  uint32_t r;
  asm("prmt.b32 %0, %1, 0, %2;" : "=r"(r) : "r"(v), "r"(sel));
  return r;
}

template <int FMT>
struct CodeBits {
  using F = Fmt<FMT>;
  static constexpr uint32_t MM = F::MMASK * 0x01010101u;                    // rank bits
  static constexpr uint32_t EB2 = (((1u << F::E) - 1u) << 2) * 0x01010101u;  // e_b << 2 after >> (C - 2)
};

// Per-step constants of a producer thread's block for E5M2 planes.
struct E5Const {
  uint32_t kt;  // per lane 128 - mt
  uint32_t kp;  // per lane 4 max(c5, 0)
  uint32_t km;  // per lane 4 max(-c5, 0)
};

template <int FMT>
__device__ __forceinline__ E5Const e5_const(int off) {
  using F = Fmt<FMT>;
  const int t = (1 << (F::E - 1)) - 14 - off;  // smallest kept e_b
  int mt = t * F::K;
  mt = mt < 1 ? 1 : (mt > 128 ? 128 : mt);
  // exponent field e5 = x + 15 = e_b + c5; when nothing is kept (mt = 128)
  // c5 is clamped so that the lane arithmetic below stays inside its byte
  int c5 = 15 - (1 << (F::E - 1)) + off;
  c5 = c5 < -30 ? -30 : c5;
  E5Const k;
  k.kt = (uint32_t)(128 - mt) * 0x01010101u;
  k.kp = (uint32_t)(4 * (c5 > 0 ? c5 : 0)) * 0x01010101u;
  k.km = (uint32_t)(4 * (c5 < 0 ? -c5 : 0)) * 0x01010101u;
  return k;
}

// E5M2 plane bytes of four codes and the lane keep mask.  The exponent byte
// is formed as (e_b << 2 | 0x80) + 4 max(c5,0) - 4 max(-c5,0): the guard bit
// 0x80 absorbs the subtraction (4 max(-c5,0) <= 120) and the addition stays
// below 256 (e5 <= 31), so no lane borrows from or carries into a neighbour.
template <int FMT>
__device__ __forceinline__ uint32_t e5m2_word(uint32_t w, const E5Const& k, uint32_t& keep) {
  using F = Fmt<FMT>;
  const uint32_t m4 = w & CodeBits<FMT>::MM;
  keep = prmt_sign(m4 + k.kt, 0xBA98u);
  const uint32_t eb = ((w >> (F::C - 2)) & CodeBits<FMT>::EB2) | 0x80808080u;
  const uint32_t x = eb + k.kp - k.km;
  return ((w & 0x80808080u) | (x & 0x7F7F7F7Fu)) & keep;
}

// BF16 plane halves of two codes (bytes 0 and 1 of w2 = codes c0 | c1 << 16).
template <int FMT>
__device__ __forceinline__ uint32_t bf16_word(uint32_t w2, int off) {
  using F = Fmt<FMT>;
  const int c = 127 - (1 << (F::E - 1)) + off;               // biased exponent = e_b + c
  const uint32_t MM2 = (uint32_t)F::MMASK * 0x00010001u;
  const uint32_t EB2 = ((1u << F::E) - 1u) * 0x00010001u;
  const uint32_t m2 = w2 & MM2;
  const uint32_t eb2 = (w2 >> F::C) & EB2;
  const uint32_t u2 = eb2 + (uint32_t)(c - 1 + 0x8000) * 0x00010001u;  // bit 15 <=> e_b + c >= 1
  const uint32_t nz = m2 + 0x7FFF7FFFu;                                 // bit 15 <=> m != 0
  const uint32_t keep = prmt_sign(u2 & nz & 0x80008000u, 0xBB99u);
  const uint32_t t = ((u2 & 0x7FFF7FFFu) + 0x00010001u) & keep;       // biased exponent where kept
  return (t << 7) | ((w2 & 0x00800080u & keep) << 8);
}

// Masks of the curve-index bits (0xFF / 0xFFFF per lane where bit b of k is 1):
// shift bit b of every lane's low byte to bit 7, then replicate it.
template <int PT, int KBITS>
__device__ __forceinline__ void k_masks(uint32_t w, uint32_t (&mk)[4]) {
  mk[3] = 0u;
#pragma unroll
  for (int b = 0; b < 3; ++b) {
    if (b >= KBITS)
      mk[b] = 0u;
    else
      mk[b] = prmt_sign(w << (7 - b), PT == PLANE_E5M2 ? 0xBA98u : 0xAA88u);
  }
}

// All 2^KBITS planes of a value word: the four products of v with the two
// low-bit masks are shared, the third bit splits each of them in two.
template <int KBITS, int NOUT>
__device__ __forceinline__ void planes_of(uint32_t v, const uint32_t (&mk)[4], uint32_t (&out)[NOUT]) {
  static_assert(NOUT >= 8, "eight plane slots");
  const uint32_t p0 = v & ~mk[0] & ~mk[1], p1 = v & mk[0] & ~mk[1];
  const uint32_t p2 = v & ~mk[0] & mk[1], p3 = v & mk[0] & mk[1];
  if (KBITS > 2) {
    out[0] = p0 & ~mk[2]; out[1] = p1 & ~mk[2]; out[2] = p2 & ~mk[2]; out[3] = p3 & ~mk[2];
    out[4] = p0 & mk[2];  out[5] = p1 & mk[2];  out[6] = p2 & mk[2];  out[7] = p3 & mk[2];
  } else {
    out[0] = p0; out[1] = p1; out[2] = p2; out[3] = p3;
    out[4] = out[5] = out[6] = out[7] = 0u;
  }
}

// Decode a thread's share of a row's 32-byte plane run: NW value words in the
// order the MMA operands expect along K (word w holds elements 4w..4w+3 as
// E5M2 bytes, or 2w..2w+1 as BF16 halves), the x2 carry words if asked, and
// the curve-index masks of every word.
template <int FMT, int PT, int NW>
__device__ __forceinline__ void decode_words(const uint4& cw, int off, uint32_t (&v)[NW], uint32_t (&vc)[NW],
                                             uint32_t (&mk)[NW][4], bool want_carry) {
  constexpr int KBITS = Fmt<FMT>::C;
  const uint32_t w[4] = {cw.x, cw.y, cw.z, cw.w};
  if (PT == PLANE_E5M2) {
    const E5Const k = e5_const<FMT>(off);
#pragma unroll
    for (int i = 0; i < NW; ++i) {
      uint32_t keep;
      v[i] = e5m2_word<FMT>(w[i], k, keep);
      vc[i] = want_carry ? v[i] + (keep & 0x04040404u) : 0u;  // exponent + 1
      k_masks<PT, KBITS>(w[i], mk[i]);
    }
  } else {
#pragma unroll
    for (int i = 0; i < NW; ++i) {
      const uint32_t w2 = __byte_perm(w[i >> 1], 0u, (i & 1) ? 0x4342u : 0x4140u);
      v[i] = bf16_word<FMT>(w2, off);
      vc[i] = want_carry ? bf16_word<FMT>(w2, off + 1) : 0u;
      k_masks<PT, KBITS>(w2, mk[i]);
    }
  }
}

// E5M2 plane bytes of four codes whose scales differ per element (reused
// operands).  Byte i of dp holds d_i + 64, d_i = max(a_i - ref, -64) the
// element's scale relative to the row reference, so the exponent field is
//   e5_i = e_b + 15 - 2^{E-1} - bias + d_i
// and the element is kept where e5_i >= 1 and m != 0 (as e5m2_word, which is
// the case d_i = const).  Per lane u = e5 + 127 = e_b + dp + (78 - 2^{E-1} -
// bias): every term is non-negative and u <= 2^E - 1 + 64 + 74 < 256, so no
// lane carries into its neighbour; bit 7 of u is e5 >= 1, and where it is set
// (u & 0x7F) + 1 = e5 <= 2^{E-1} + 14 - bias <= 30.
template <int FMT>
__device__ __forceinline__ uint32_t e5m2_word_pes(uint32_t w, uint32_t dp, uint32_t kc, uint32_t& keep) {
  using F = Fmt<FMT>;
  const uint32_t m4 = w & CodeBits<FMT>::MM;
  const uint32_t eb = (w >> F::C) & (((1u << F::E) - 1u) * 0x01010101u);
  const uint32_t u = eb + dp + kc;
  keep = prmt_sign(u & (m4 + 0x7F7F7F7Fu) & 0x80808080u, 0xBA98u);
  const uint32_t e5 = ((u & 0x7F7F7F7Fu) + 0x01010101u) & keep;
  return (w & 0x80808080u & keep) | (e5 << 2);
}

// decode_words for E5M2 planes with per-element scales (dw: the d + 64 bytes
// of the sixteen codes of cw).
template <int FMT, int NW>
__device__ __forceinline__ void decode_words_pes(const uint4& cw, const uint4& dw, int bias, uint32_t (&v)[NW],
                                                 uint32_t (&vc)[NW], uint32_t (&mk)[NW][4], bool want_carry) {
  constexpr int KBITS = Fmt<FMT>::C;
  const uint32_t w[4] = {cw.x, cw.y, cw.z, cw.w};
  const uint32_t d[4] = {dw.x, dw.y, dw.z, dw.w};
  const uint32_t kc = (uint32_t)(78 - (1 << (Fmt<FMT>::E - 1)) - bias) * 0x01010101u;
#pragma unroll
  for (int i = 0; i < NW; ++i) {
    uint32_t keep;
    v[i] = e5m2_word_pes<FMT>(w[i], d[i], kc, keep);
    vc[i] = want_carry ? v[i] + (keep & 0x04040404u) : 0u;  // exponent + 1
    k_masks<PLANE_E5M2, KBITS>(w[i], mk[i]);
  }
}

// ---------------------------------------------------------------------------
// E4C3 codes with the rational radix r = 2^{8/9} (Sec. 3.1 Eq. 1, Eq. 4):
// level 2^{n/9}, n = m - 64.  With v = m - 1 = 9 q + j (q in [0, 14],
// j in [0, 8]) the element is 2^{q - 7} 2^{j/9}: it sits in plane j with the
// power-of-two value 2^{a_b - ref + q - 7}, and plane j1 times plane j2 lands
// on phase (j1 + j2) mod 9 with carry (j1 + j2) >= 9.  Nine planes per word:
// q and j per byte from a 16-bit-lane multiply (floor(v/9) = (57 v) >> 9 for
// v <= 127), the E5M2 exponent e5 = q + 8 + off kept where e5 >= 1 (as for
// the binary planes: 2^14 below the row reference flushes), and the bits of
// j as masks (mk[0..2] its low bits, mk[3] bit 3, which only j = 8 has).
template <int NW>
__device__ __forceinline__ void decode_words_r89(const uint4& cw, int off, uint32_t (&v)[NW], uint32_t (&vc)[NW],
                                                 uint32_t (&mk)[NW][4], bool want_carry) {
  const uint32_t w[4] = {cw.x, cw.y, cw.z, cw.w};
  int cu = 8 + off - 1 + 128;  // u = q + cu = e5 + 127 per lane; off <= 0, so cu <= 135 and u <= 149
  cu = cu < 0 ? 0 : cu;
  const uint32_t cu4 = (uint32_t)cu * 0x01010101u;
#pragma unroll
  for (int i = 0; i < NW; ++i) {
    const uint32_t m4 = w[i] & 0x7F7F7F7Fu;
    const uint32_t nz = (m4 + 0x7F7F7F7Fu) & 0x80808080u;                    // m != 0
    const uint32_t v4 = ((m4 | 0x80808080u) - 0x01010101u) & 0x7F7F7F7Fu;    // m - 1 (no borrow)
    const uint32_t ql = (((v4 & 0x00FF00FFu) * 57u) >> 9) & 0x001F001Fu;
    const uint32_t qh = ((((v4 >> 8) & 0x00FF00FFu) * 57u) >> 9) & 0x001F001Fu;
    const uint32_t q4 = ql | (qh << 8);
    const uint32_t j4 = v4 - q4 * 9u;                                        // per lane in [0, 8]
    const uint32_t u = q4 + cu4;
    const uint32_t keep = prmt_sign(u & nz, 0xBA98u);
    const uint32_t e5 = ((u & 0x7F7F7F7Fu) + 0x01010101u) & keep;           // q + 8 + off where kept
    v[i] = (w[i] & 0x80808080u & keep) | (e5 << 2);
    vc[i] = want_carry ? v[i] + (keep & 0x04040404u) : 0u;                  // exponent + 1
#pragma unroll
    for (int b = 0; b < 4; ++b) mk[i][b] = prmt_sign(j4 << (7 - b), 0xBA98u);
  }
}

// Plane split of a format: PlaneFmt<FMT>::KP planes of a value word.
template <int FMT>
struct PlaneFmt {
  static constexpr int KP = Fmt<FMT>::K;
  template <int PT, int NW>
  __device__ __forceinline__ static void decode(const uint4& cw, int off, uint32_t (&v)[NW], uint32_t (&vc)[NW],
                                                uint32_t (&mk)[NW][4], bool want_carry) {
    decode_words<FMT, PT, NW>(cw, off, v, vc, mk, want_carry);
  }
  template <int NOUT>
  __device__ __forceinline__ static void planes(uint32_t v, const uint32_t (&mk)[4], uint32_t (&out)[NOUT]) {
    planes_of<Fmt<FMT>::C>(v, mk, out);
  }
};
template <>
struct PlaneFmt<CURVEFP_E4C3_R8_9> {
  static constexpr int KP = 9;
  template <int PT, int NW>
  __device__ __forceinline__ static void decode(const uint4& cw, int off, uint32_t (&v)[NW], uint32_t (&vc)[NW],
                                                uint32_t (&mk)[NW][4], bool want_carry) {
    static_assert(PT == PLANE_E5M2, "E5M2 planes");
    decode_words_r89<NW>(cw, off, v, vc, mk, want_carry);
  }
  template <int NOUT>
  __device__ __forceinline__ static void planes(uint32_t v, const uint32_t (&mk)[4], uint32_t (&out)[NOUT]) {
    static_assert(NOUT >= 9, "nine plane slots");
    planes_of<3>(v & ~mk[3], mk, out);
    out[8] = v & mk[3];
  }
};

static __constant__ uint32_t CFP_PHASE_F32_L9_TC[9] = CFP_PHASE_F32_L9_INIT;

__device__ __forceinline__ float phase_const(int L, int h) {
  return __uint_as_float(L == 8 ? CFP_PHASE_F32_L8_DEV[h] : (L == 9 ? CFP_PHASE_F32_L9_TC[h] : CFP_PHASE_F32_L4_DEV[h]));
}


}  // namespace cfp
