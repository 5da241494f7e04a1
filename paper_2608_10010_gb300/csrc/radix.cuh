// Element encode / reconstruction of the rational-radix E4C3 formats
// (Sec. 3.1 Eq. 1 with r = 2^{p/q}): shared by the quantizers' exact paths.
//
// Levels sit at exponents lambda(n) = p n/(8q).  A scaled value y = |x| 2^{-a}
// with binade b and 23-bit mantissa mu has, on the unbounded lattice, the
// nearest level
//   n*(y) = N0[b mod PB] + floor(b / PB) NPER + (midpoints of binade b below y)
// with the count read from a 256-bucket table of the top mantissa bits per
// binade class (at most one midpoint per bucket); the codebook clamps n* to
// [-63, 63], and y <= L_nmin / 2 encodes as zero (the tie at equality, which
// exists for r = 2^{8/9}, goes to zero).  All tables come from exact integer
// arithmetic in gen_constants.py.
#pragma once
#include "cfp_common.cuh"

namespace cfp {

// global (not __constant__) tables: lanes read different entries
static __device__ const uint32_t CFP_RX89_LUT_G[256] = CFP_R8_9_LUT_INIT;
static __device__ const uint32_t CFP_RX34_LUT_G[3 * 256] = CFP_R3_4_LUT_INIT;
static __device__ const int CFP_RX89_N0_G[1] = CFP_R8_9_N0_INIT;
static __device__ const int CFP_RX34_N0_G[3] = CFP_R3_4_N0_INIT;
static __constant__ uint32_t CFP_RX_C9_DEV[9] = CFP_PHASE_F32_L9_INIT;    // RN32(2^{h/9})
static __constant__ uint32_t CFP_RX_C32_DEV[32] = CFP_PHASE_F32_L32_INIT;  // RN32(2^{h/32})

template <int FMT>
struct IsRadix {
  static constexpr bool value = FMT == CURVEFP_E4C3_R8_9 || FMT == CURVEFP_E4C3_R3_4;
};

__device__ __forceinline__ int rx_floordiv(int a, int b) { return a >= 0 ? a / b : -((-a + b - 1) / b); }

// Exact encode of an FP32 bit pattern at block scale a.  Sets nan for NaN.
template <int FMT>
__device__ __forceinline__ uint32_t radix_encode(uint32_t bits, int a, bool& nan) {
  using R = Radix<FMT>;
  constexpr int B = Fmt<FMT>::B, NMAX = Fmt<FMT>::NMAX;
  const uint32_t absb = bits & 0x7FFFFFFFu;
  const uint32_t sign = (bits >> 24) & 0x80u;
  if (absb > 0x7F800000u) {
    nan = true;
    return 0u;
  }
  if (absb == 0x7F800000u) return sign | (2 * B - 1);
  if (absb == 0u) return 0u;
  int Fx;
  uint32_t mant;
  if (absb >= 0x00800000u) {
    Fx = (int)(absb >> 23) - 127;
    mant = absb & 0x7FFFFFu;
  } else {
    const int p = 31 - __clz(absb);
    Fx = p - 149;
    mant = (absb << (23 - p)) & 0x7FFFFFu;
  }
  const int b = Fx - a;
  if (b > R::F + 1) return sign | (2 * B - 1);
  if (b < R::ZB || (b == R::ZB && mant < R::ZTHR)) return 0u;
  const int k = rx_floordiv(b, R::PB), c = b - k * R::PB;
  const uint32_t* lut = FMT == CURVEFP_E4C3_R8_9 ? CFP_RX89_LUT_G : CFP_RX34_LUT_G;
  const int* n0 = FMT == CURVEFP_E4C3_R8_9 ? CFP_RX89_N0_G : CFP_RX34_N0_G;
  const uint32_t e = __ldg(lut + c * 256 + (mant >> 15));
  int n = __ldg(n0 + c) + k * R::NPER + (int)(e >> 24) + (mant >= (e & 0xFFFFFFu) ? 1 : 0);
  n = n < -NMAX ? -NMAX : (n > NMAX ? NMAX : n);
  return sign | (uint32_t)(n + B);
}

// R4 with the rational exponent: RN32(RN32(2^{j/N}) 2^{a + floor(p n/N)}),
// j = p n mod N (a multiple of g, so the constant is 2^{(j/g)/H}).
template <int FMT>
__device__ __forceinline__ float radix_recon_f32(uint32_t code, int a) {
  using R = Radix<FMT>;
  const uint32_t m = code & 0x7Fu;
  if (m == 0u) return 0.0f;
  const int u = R::P * ((int)m - Fmt<FMT>::B);
  const int e = rx_floordiv(u, R::N), j = u - e * R::N;
  const float cj = __uint_as_float(R::H == 9 ? CFP_RX_C9_DEV[j / R::G] : CFP_RX_C32_DEV[j / R::G]);
  const float v = __double2float_rn(ldexp((double)cj, a + e));
  return (code & 0x80u) ? -v : v;
}

}  // namespace cfp
