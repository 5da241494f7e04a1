// Shared definitions of the CurveFP CUDA kernels (sm_103a).
//
// Format traits restate Table 1 and Sec. 3.1 of the paper: E exponent bits,
// C curve-index bits, K = 2^C curves, rank bias B = 2^{E+C-1}, lattice index
// n = m - B in [-(B-1), B-1], exponent e = floor(n/K) in [-2^{E-1}, 2^{E-1}-1].
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/curvefp.h"
#include "curvefp_constants.h"

namespace cfp {

template <int FMT>
struct Fmt;
template <>
struct Fmt<CURVEFP_E3C3> {
  static constexpr int E = 3, C = 3, K = 8, B = 32, NMAX = 31, EMAX = 3, MMASK = 0x3F;
};
template <>
struct Fmt<CURVEFP_E4C3> {
  static constexpr int E = 4, C = 3, K = 8, B = 64, NMAX = 63, EMAX = 7, MMASK = 0x7F;
};
template <>
struct Fmt<CURVEFP_E5C2> {
  static constexpr int E = 5, C = 2, K = 4, B = 64, NMAX = 63, EMAX = 15, MMASK = 0x7F;
};

// E4C3 codes with a rational radix r = 2^{p/q} (Sec. 3.1 Eq. 1, Eq. 4): the
// field layout of E4C3, levels 2^{p n/(8q)}.
template <>
struct Fmt<CURVEFP_E4C3_R8_9> : Fmt<CURVEFP_E4C3> {};
template <>
struct Fmt<CURVEFP_E4C3_R3_4> : Fmt<CURVEFP_E4C3> {};

// Rational-radix tables (generated; see gen_constants.py radix_params).
template <int FMT>
struct Radix;
template <>
struct Radix<CURVEFP_E4C3_R8_9> {
  static constexpr int P = 8, N = CFP_R8_9_N, G = CFP_R8_9_g, H = CFP_R8_9_H, PB = CFP_R8_9_PB,
                       NPER = CFP_R8_9_NPER, F = CFP_R8_9_F, ZB = CFP_R8_9_ZB, R0 = CFP_R8_9_R0,
                       OFF = CFP_R8_9_OFF, TMIN = CFP_R8_9_TMIN, TMAX = CFP_R8_9_TMAX;
  static constexpr uint32_t MU_SAT = CFP_R8_9_MU_SAT, ZTHR = CFP_R8_9_ZTHR;
};
template <>
struct Radix<CURVEFP_E4C3_R3_4> {
  static constexpr int P = 3, N = CFP_R3_4_N, G = CFP_R3_4_g, H = CFP_R3_4_H, PB = CFP_R3_4_PB,
                       NPER = CFP_R3_4_NPER, F = CFP_R3_4_F, ZB = CFP_R3_4_ZB, R0 = CFP_R3_4_R0,
                       OFF = CFP_R3_4_OFF, TMIN = CFP_R3_4_TMIN, TMAX = CFP_R3_4_TMAX;
  static constexpr uint32_t MU_SAT = CFP_R3_4_MU_SAT, ZTHR = CFP_R3_4_ZTHR;
};

// Exponent F_z and 23-bit mantissa threshold of the zero/L_nmin boundary
// L_nmin / 2 = 2^{(nmin - K)/K} = 2^{F_z} 2^{1/K}  (nmin - K = K F_z + 1).
template <int FMT>
struct ZeroBoundary {
  static constexpr int FZ = (-Fmt<FMT>::NMAX - Fmt<FMT>::K - 1) / Fmt<FMT>::K;
};

template <int K>
struct RadixConst;
template <>
struct RadixConst<4> {
  static constexpr uint32_t MU_SAT = CFP_MU_SAT_K4, MU_Z = CFP_MU_Z_K4;
};
template <>
struct RadixConst<8> {
  static constexpr uint32_t MU_SAT = CFP_MU_SAT_K8, MU_Z = CFP_MU_Z_K8;
};

// Shared lattice of a format pair: L = max(K_a, K_b), weights L/K.
template <int FA, int FB>
struct Pair {
  static constexpr int KA = Fmt<FA>::K, KB = Fmt<FB>::K;
  static constexpr int L = KA > KB ? KA : KB;
  static constexpr int LOG2L = L == 8 ? 3 : 2;
  static constexpr int WA = L / KA, WB = L / KB;
  // u_n = n_a WA + n_b WB in [-UMAX, UMAX]; t = floor(u_n / L)
  static constexpr int UMAX = Fmt<FA>::NMAX * WA + Fmt<FB>::NMAX * WB;
  static constexpr int TMIN = -((UMAX + L - 1) / L);  // floor(-UMAX / L)
  static constexpr int TMAX = UMAX / L;
};

// Device copies of the generated constants (one per translation unit).
static __constant__ uint32_t CFP_LUT_K4_DEV[256] = CFP_LUT_K4_INIT;
static __constant__ uint32_t CFP_LUT_K8_DEV[256] = CFP_LUT_K8_INIT;
static __constant__ uint32_t CFP_CK_F32_K4_DEV[4] = CFP_CK_F32_K4_INIT;
static __constant__ uint32_t CFP_CK_F32_K8_DEV[8] = CFP_CK_F32_K8_INIT;
static __constant__ uint32_t CFP_PHASE_F32_L4_DEV[4] = CFP_PHASE_F32_L4_INIT;
static __constant__ uint32_t CFP_PHASE_F32_L8_DEV[8] = CFP_PHASE_F32_L8_INIT;
static __constant__ uint64_t CFP_PHASE_F64_L4_DEV[4] = CFP_PHASE_F64_L4_INIT;
static __constant__ uint64_t CFP_PHASE_F64_L8_DEV[8] = CFP_PHASE_F64_L8_INIT;
static __constant__ uint64_t CFP_PHASE_F64_L9_DEV[9] = CFP_PHASE_F64_L9_INIT;
static __constant__ uint64_t CFP_PHASE_F64_L32_DEV[32] = CFP_PHASE_F64_L32_INIT;

// Phase-address policies of the exact GEMM.  addr() maps the biased ranks of
// two nonzero codes to the phase h and the bin offset sh = t - TMIN >= 0;
// phase64(h) is 2^{h/L} as FP64 bits.
template <int FA, int FB>
struct BinLat {  // binary radix, shared lattice L = max(K_a, K_b) (Eq. 2)
  using P = Pair<FA, FB>;
  static constexpr int L = P::L, TMIN = P::TMIN, TMAX = P::TMAX;
  static constexpr uint32_t MA = Fmt<FA>::MMASK, MB = Fmt<FB>::MMASK;
  __device__ __forceinline__ static void addr(uint32_t ma, uint32_t mb, int& h, int& sh) {
    const uint32_t u = ma * P::WA + mb * P::WB;
    h = (int)(u & (L - 1));
    sh = (int)(u >> P::LOG2L);
  }
  __device__ __forceinline__ static uint64_t phase64(int h) {
    return L == 8 ? CFP_PHASE_F64_L8_DEV[h] : CFP_PHASE_F64_L4_DEV[h];
  }
};
template <int FMT>
struct RadLat {  // rational radix, same format on both sides (App. A.1)
  using R = Radix<FMT>;
  static constexpr int L = R::H, TMIN = R::TMIN, TMAX = R::TMAX;
  static constexpr uint32_t MA = Fmt<FMT>::MMASK, MB = Fmt<FMT>::MMASK;
  // u = p (n_a + n_b) = p (m_a + m_b) - 2pB; V = u + 2pB - R0 + N >= 0 with
  // V = u (mod N), so h = (V mod N)/g and t = floor(V/N) - (OFF + TMIN).
  __device__ __forceinline__ static void addr(uint32_t ma, uint32_t mb, int& h, int& sh) {
    const uint32_t V = R::P * (ma + mb) - R::R0 + R::N;
    h = (int)((V % R::N) / R::G);
    sh = (int)(V / R::N) - R::OFF;
  }
  __device__ __forceinline__ static uint64_t phase64(int h) {
    return L == 9 ? CFP_PHASE_F64_L9_DEV[h] : CFP_PHASE_F64_L32_DEV[h];
  }
};

__host__ __device__ inline int bitlen64(int64_t v) {
  int b = 0;
  while (v) {
    ++b;
    v >>= 1;
  }
  return b;
}

}  // namespace cfp
