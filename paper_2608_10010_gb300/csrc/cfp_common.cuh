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

__host__ __device__ inline int bitlen64(int64_t v) {
  int b = 0;
  while (v) {
    ++b;
    v >>= 1;
  }
  return b;
}

}  // namespace cfp
