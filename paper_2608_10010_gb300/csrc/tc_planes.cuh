// Producer-side arithmetic shared by the tensor-core GEMM kernels: curve-index
// masks and the split of a plane word into curve planes, the r = 2^{8/9}
// decode, the shared-memory block of the pipeline, and the phase constants of
// the epilogue (Sec. 3.2, Eq. 2, Eq. 5).  The plane bytes of the binary
// formats are formed in tc_mx.cuh.
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
  uint32_t tmem_base;
  int abort_flag;
  int refB[128];  // >= BN
  int wref[128];  // the narrow kernel's weight-row references
};

__device__ __forceinline__ void raise_flag(uint32_t* status, uint32_t bit) {
  if (status) atomicOr(status, bit);
}
__device__ __forceinline__ int read_abort(const int* f) { return *reinterpret_cast<const volatile int*>(f); }

// Largest of the four signed bytes of v.
__device__ __forceinline__ int max_s8x4(uint32_t v) {
  return max(max((int)(int8_t)(v & 0xFF), (int)(int8_t)((v >> 8) & 0xFF)),
             max((int)(int8_t)((v >> 16) & 0xFF), (int)(int8_t)(v >> 24)));
}

// Row references of `rows` consecutive rows of nb scale bytes (one run of
// rows x nb bytes from s), read by threads t = 0 .. nthr - 1 together in
// chunks of 16, 8 or 4 bytes (the largest that divides nb and the run's
// alignment, single bytes otherwise; a chunk never spans two rows) and
// folded into ref[row] by shared-memory atomics; ref[] holds -128 on entry.
// A warp's loads cover whole lines, where a thread reading its own row
// touches one line per lane and load.
__device__ __forceinline__ void rows_ref_coop(const int8_t* s, int rows, int nb, int* ref, int t, int nthr) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(s);
  const int64_t bytes = (int64_t)rows * nb;
  if ((a & 15) == 0 && (nb & 15) == 0) {
    const uint4* p = reinterpret_cast<const uint4*>(s);
    for (int64_t i = t; i < bytes / 16; i += nthr) {
      const uint4 q = __ldg(p + i);
      atomicMax(ref + (int)(i * 16 / nb), max_s8x4(__vmaxs4(__vmaxs4(q.x, q.y), __vmaxs4(q.z, q.w))));
    }
  } else if ((a & 7) == 0 && (nb & 7) == 0) {
    const uint2* p = reinterpret_cast<const uint2*>(s);
    for (int64_t i = t; i < bytes / 8; i += nthr) {
      const uint2 q = __ldg(p + i);
      atomicMax(ref + (int)(i * 8 / nb), max_s8x4(__vmaxs4(q.x, q.y)));
    }
  } else if ((a & 3) == 0 && (nb & 3) == 0) {
    const uint32_t* p = reinterpret_cast<const uint32_t*>(s);
    for (int64_t i = t; i < bytes / 4; i += nthr) atomicMax(ref + (int)(i * 4 / nb), max_s8x4(__ldg(p + i)));
  } else {
    for (int64_t i = t; i < bytes; i += nthr) atomicMax(ref + (int)(i / nb), (int)__ldg(s + i));
  }
}

// ---------------------------------------------------------------------------
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

// ---------------------------------------------------------------------------
// E4C3 codes with the rational radix r = 2^{8/9} (Sec. 3.1 Eq. 1, Eq. 4):
// level 2^{n/9}, n = m - 64.  With v = m - 1 = 9 q + j (q in [0, 14],
// j in [0, 8]) the element is 2^{q - 7} 2^{j/9}: it sits in plane j with the
// power-of-two value 2^{q - 7} (the block scale is the MMA's scale factor),
// and plane j1 times plane j2 lands on phase (j1 + j2) mod 9 with carry
// (j1 + j2) >= 9.  Per byte of a word: q and j from a 16-bit-lane multiply
// (floor(v/9) = (57 v) >> 9 for v <= 127), the E5M2 exponent e5 = q + 8 (a
// normal exponent for every q), and the bits of j as masks (mk[0..2] its low
// bits, mk[3] bit 3, which only j = 8 has).
__device__ __forceinline__ void r89_word(uint32_t w, uint32_t& v, uint32_t (&mk)[4]) {
  const uint32_t m4 = w & 0x7F7F7F7Fu;
  const uint32_t nz = prmt_sign(m4 + 0x7F7F7F7Fu, 0xBA98u);              // m != 0
  const uint32_t v4 = ((m4 | 0x80808080u) - 0x01010101u) & 0x7F7F7F7Fu;  // m - 1 (no borrow)
  const uint32_t ql = (((v4 & 0x00FF00FFu) * 57u) >> 9) & 0x001F001Fu;
  const uint32_t qh = ((((v4 >> 8) & 0x00FF00FFu) * 57u) >> 9) & 0x001F001Fu;
  const uint32_t q4 = ql | (qh << 8);
  const uint32_t j4 = v4 - q4 * 9u;  // per lane in [0, 8]
  v = ((w & 0x80808080u) | ((q4 + 0x08080808u) << 2)) & nz;
#pragma unroll
  for (int b = 0; b < 4; ++b) mk[b] = prmt_sign(j4 << (7 - b), 0xBA98u);
}

// Plane split of a format: PlaneFmt<FMT>::KP planes of a value word.
template <int FMT>
struct PlaneFmt {
  static constexpr int KP = Fmt<FMT>::K;
  template <int NOUT>
  __device__ __forceinline__ static void planes(uint32_t v, const uint32_t (&mk)[4], uint32_t (&out)[NOUT]) {
    planes_of<Fmt<FMT>::C>(v, mk, out);
  }
};
template <>
struct PlaneFmt<CURVEFP_E4C3_R8_9> {
  static constexpr int KP = 9;
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
