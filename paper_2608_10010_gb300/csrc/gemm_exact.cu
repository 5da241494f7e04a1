// Exact closed-product GEMM on the integer ALUs (Sec. 3.2, Eq. 2, Eq. 5,
// App. A.1): the per-phase Kulisch layout of the paper, realized per output.
//
// For every nonzero product of codes a and b the kernel forms
//   u  = m_a WA + m_b WB           (ranks on the shared lattice L)
//   h  = u mod L                    (phase)
//   sh = floor(u / L) = t - t_min   (bin, relative to the smallest product)
//   delta = +-1 from the sign XOR
// and adds delta * 2^sh to the phase-h accumulator of the current scale block.
// Within a block the sums are kept in 16-bit-wide parts (int32 counters in
// shared memory, indexed by phase and part: no data-dependent register
// indexing); at the end of each scale block they are shifted by
// (sa + sb) - min_b(sa + sb) and added into exact int128 per-phase sums.
// The epilogue combines C = sum_h 2^{h/L} S_h 2^lambda in FP64 and rounds
// once to FP32; the validation form also writes the int128 sums and lambda.
#include "cfp_common.cuh"
#include "kernels.cuh"

namespace cfp {

namespace {
constexpr int TM = 16, TN = 16, NT = TM * TN, KC = 32;

__device__ __forceinline__ int i128_bitlen_ok(int spread, int dt, int64_t K) {
  return bitlen64(K) + spread + dt <= 127;
}

// int128 -> double without cancellation: split the magnitude, not the
// two's-complement words (error <= 2^-52 relative).
__device__ __forceinline__ double i128_to_double(__int128 v) {
  const int64_t hi = (int64_t)(v >> 64);
  const uint64_t lo = (uint64_t)v;
  if ((hi == 0 && (int64_t)lo >= 0) || (hi == -1 && (int64_t)lo < 0)) return (double)(int64_t)lo;
  const bool neg = hi < 0;
  const unsigned __int128 m = neg ? (unsigned __int128)0 - (unsigned __int128)v : (unsigned __int128)v;
  const double d = fma((double)(uint64_t)(m >> 64), 18446744073709551616.0, (double)(uint64_t)m);
  return neg ? -d : d;
}
}  // namespace

// Lat: the phase-address policy (BinLat for binary radix, RadLat for a
// rational radix).  The 16-bit-part counters (L PARTS x NT int32) and, for
// more than 8 phases, the int128 phase sums (L x NT) live in dynamic shared
// memory (exact_smem bytes).
template <class Lat>
__host__ __device__ constexpr int exact_parts() {
  return (Lat::TMAX - Lat::TMIN) / 16 + 1;
}
template <class Lat>
__host__ __device__ constexpr size_t exact_smem() {
  return (size_t)Lat::L * exact_parts<Lat>() * NT * 4 + (Lat::L > 8 ? (size_t)Lat::L * NT * 16 : 0);
}

template <class Lat>
__global__ void __launch_bounds__(NT) gemm_exact_kernel(const uint8_t* __restrict__ A, const int8_t* __restrict__ sA,
                                                        const uint8_t* __restrict__ B, const int8_t* __restrict__ sB,
                                                        int M, int N, int K, int G, float* __restrict__ C,
                                                        int64_t* __restrict__ phase_sums,
                                                        int32_t* __restrict__ phase_lsb, uint32_t* status) {
  constexpr int L = Lat::L;
  constexpr int DT = Lat::TMAX - Lat::TMIN;  // largest bin offset sh
  constexpr int PARTS = exact_parts<Lat>();   // 16-bit parts of a bin offset
  constexpr uint32_t MA = Lat::MA, MB = Lat::MB;
  constexpr bool SREG = L <= 8;               // int128 sums in registers

  __shared__ uint32_t As[TM][KC / 4];
  __shared__ uint32_t Bs[TN][KC / 4];
  extern __shared__ __align__(16) uint8_t exact_dyn[];
  int32_t(*acc)[NT] = reinterpret_cast<int32_t(*)[NT]>(exact_dyn);
  __int128(*Ssm)[NT] = reinterpret_cast<__int128(*)[NT]>(exact_dyn + (size_t)L * PARTS * NT * 4);

  const int tid = threadIdx.x;
  const int ty = tid / TN, tx = tid % TN;
  const int i = blockIdx.y * TM + ty, j = blockIdx.x * TN + tx;
  const bool live = i < M && j < N;
  const int nb = K / G;

  // lambda = min_b(sa + sb) + t_min; the int128 window check
  int smin = 1 << 20, smax = -(1 << 20);
  if (live)
    for (int b = 0; b < nb; ++b) {
      int s = (int)sA[(int64_t)i * nb + b] + (int)sB[(int64_t)j * nb + b];
      smin = min(smin, s);
      smax = max(smax, s);
    }
  const bool in_range = live && i128_bitlen_ok(smax - smin, DT, K);
  if (live && !in_range && status) atomicOr(status, CURVEFP_DEV_RANGE);

  __int128 S[SREG ? L : 1];
#pragma unroll
  for (int h = 0; h < L; ++h) {
    if constexpr (SREG)
      S[h] = 0;
    else
      Ssm[h][tid] = 0;
  }
#pragma unroll
  for (int q = 0; q < L * PARTS; ++q) acc[q][tid] = 0;

  for (int k0 = 0; k0 < K; k0 += KC) {
    // stage a 16x32 code tile of A and of B (one 32-bit word per lane)
    {
      const int r = (tid & 127) >> 3, w = tid & 7;
      if (tid < 128) {
        const int gi = blockIdx.y * TM + r;
        As[r][w] = gi < M ? __ldg(reinterpret_cast<const uint32_t*>(A + (int64_t)gi * K + k0) + w) : 0u;
      } else {
        const int gj = blockIdx.x * TN + r;
        Bs[r][w] = gj < N ? __ldg(reinterpret_cast<const uint32_t*>(B + (int64_t)gj * K + k0) + w) : 0u;
      }
    }
    __syncthreads();
    if (in_range) {
#pragma unroll
      for (int w = 0; w < KC / 4; ++w) {
        const uint32_t aw = As[ty][w], bw = Bs[tx][w];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint32_t ca = (aw >> (8 * q)) & 0xFFu, cb = (bw >> (8 * q)) & 0xFFu;
          const uint32_t ma = ca & MA, mb = cb & MB;
          if (ma != 0u && mb != 0u) {
            int h, sh;
            Lat::addr(ma, mb, h, sh);
            const int idx = h * PARTS + (sh >> 4);
            const int32_t v = (int32_t)(1u << (sh & 15));
            acc[idx][tid] += ((ca ^ cb) & 0x80u) ? -v : v;
          }
        }
      }
    }
    __syncthreads();
    // end of a scale block: fold the parts into the int128 phase sums
    if (((k0 + KC) % G) == 0) {
      if (in_range) {
        const int b = (k0 + KC) / G - 1;
        const int sb = (int)sA[(int64_t)i * nb + b] + (int)sB[(int64_t)j * nb + b] - smin;
#pragma unroll
        for (int h = 0; h < L; ++h)
#pragma unroll
          for (int p = 0; p < PARTS; ++p) {
            const int32_t part = acc[h * PARTS + p][tid];
            if (part != 0) {
              const __int128 v = (__int128)((unsigned __int128)(__int128)part << (16 * p + sb));
              if constexpr (SREG)
                S[h] += v;
              else
                Ssm[h][tid] += v;
            }
          }
      }
#pragma unroll
      for (int q = 0; q < L * PARTS; ++q) acc[q][tid] = 0;
    }
  }

  if (!live) return;
  const int lambda = smin + Lat::TMIN;
  const int64_t o = (int64_t)i * N + j;
  auto sum_of = [&](int h) -> __int128 {
    if constexpr (SREG)
      return S[h];
    else
      return Ssm[h][tid];
  };
  if (C) {
    float out;
    if (in_range) {
      double c = 0.0;
#pragma unroll
      for (int h = 0; h < L; ++h) {
        const double sd = i128_to_double(sum_of(h));
        c = fma(__longlong_as_double((long long)Lat::phase64(h)), sd, c);
      }
      out = (float)scalbn(c, lambda);
    } else {
      out = __int_as_float(0x7fc00000);
    }
    C[o] = out;
  }
  if (phase_sums) {
#pragma unroll
    for (int h = 0; h < L; ++h) {
      const __int128 v = sum_of(h);
      phase_sums[(o * L + h) * 2 + 0] = (int64_t)(uint64_t)v;
      phase_sums[(o * L + h) * 2 + 1] = (int64_t)(v >> 64);
    }
  }
  if (phase_lsb) phase_lsb[o] = lambda;
}

// ---------------------------------------------------------------------------
// Operands with a scale per element (reused operands of the training GEMMs):
// element (r, k) of an operand view is code c[r cr + k ck] with scale
// s[(r >> rsh) sr + (k >> ksh) sk]; ROWS and COLS layouts are two settings of
// the strides.  Every product adds delta 2^{t - lambda} (t includes both
// element scales) to an exact int128 phase sum in shared memory; lambda =
// min_k (a(i,k) + b(j,k)) + t_min as for block scales.
struct OpView {
  const uint8_t* c;
  int64_t cr, ck;
  const int8_t* s;
  int64_t sr, sk;
  int rsh, ksh;
  __device__ __forceinline__ uint8_t code(int64_t r, int64_t k) const { return __ldg(c + r * cr + k * ck); }
  __device__ __forceinline__ int scale(int64_t r, int64_t k) const {
    return (int)__ldg(s + (r >> rsh) * sr + (k >> ksh) * sk);
  }
};

template <int FA, int FB>
__global__ void __launch_bounds__(NT) gemm_exact_view_kernel(const OpView va, const OpView vb, int M, int N, int K,
                                                             float* __restrict__ C, int64_t* __restrict__ phase_sums,
                                                             int32_t* __restrict__ phase_lsb, uint32_t* status) {
  using P = Pair<FA, FB>;
  constexpr int L = P::L;
  constexpr int DT = P::TMAX - P::TMIN;
  constexpr uint32_t MA = Fmt<FA>::MMASK, MB = Fmt<FB>::MMASK;
  __shared__ uint8_t Ac[TM][KC], Bc[TN][KC];
  __shared__ int8_t As[TM][KC], Bs[TN][KC];
  __shared__ __int128 acc[L][NT];

  const int tid = threadIdx.x;
  const int ty = tid / TN, tx = tid % TN;
  const int i = blockIdx.y * TM + ty, j = blockIdx.x * TN + tx;
  const bool live = i < M && j < N;

  // stage a 16 x 32 tile of codes and scales of each operand; the index
  // order follows the contiguous direction of the layout
  auto stage = [&](int k0, bool codes) {
    for (int e = tid; e < 2 * TM * KC; e += NT) {
      const bool is_b = e >= TM * KC;
      const int f = e - (is_b ? TM * KC : 0);
      const OpView& v = is_b ? vb : va;
      const int rr = v.ck == 1 ? f / KC : f % TM, kk = v.ck == 1 ? f % KC : f / TM;
      const int64_t r = (int64_t)(is_b ? blockIdx.x * TN : blockIdx.y * TM) + rr;
      const bool in = r < (is_b ? N : M) && k0 + kk < K;
      if (codes) (is_b ? Bc : Ac)[rr][kk] = in ? v.code(r, k0 + kk) : (uint8_t)0;
      (is_b ? Bs : As)[rr][kk] = in ? (int8_t)v.scale(r, k0 + kk) : (int8_t)0;
    }
  };

  int smin = 1 << 20, smax = -(1 << 20);
  for (int k0 = 0; k0 < K; k0 += KC) {
    __syncthreads();
    stage(k0, false);
    __syncthreads();
    if (live)
      for (int kk = 0; kk < KC && k0 + kk < K; ++kk) {
        const int s = (int)As[ty][kk] + (int)Bs[tx][kk];
        smin = min(smin, s);
        smax = max(smax, s);
      }
  }
  const bool in_range = live && i128_bitlen_ok(smax - smin, DT, K);
  if (live && !in_range && status) atomicOr(status, CURVEFP_DEV_RANGE);
#pragma unroll
  for (int h = 0; h < L; ++h) acc[h][tid] = 0;

  for (int k0 = 0; k0 < K; k0 += KC) {
    __syncthreads();
    stage(k0, true);
    __syncthreads();
    if (!in_range) continue;
    for (int kk = 0; kk < KC && k0 + kk < K; ++kk) {
      const uint32_t ca = Ac[ty][kk], cb = Bc[tx][kk];
      const uint32_t ma = ca & MA, mb = cb & MB;
      if (ma == 0u || mb == 0u) continue;
      const uint32_t u = ma * P::WA + mb * P::WB;
      const int sh = (int)(u >> P::LOG2L) + (int)As[ty][kk] + (int)Bs[tx][kk] - smin;
      const __int128 term = (__int128)1 << sh;
      acc[u & (L - 1)][tid] += ((ca ^ cb) & 0x80u) ? -term : term;
    }
  }

  if (!live) return;
  const int lambda = smin + P::TMIN;
  const int64_t o = (int64_t)i * N + j;
  if (C) {
    float out;
    if (in_range) {
      double c = 0.0;
#pragma unroll
      for (int h = 0; h < L; ++h) {
        const double sd = i128_to_double(acc[h][tid]);
        const uint64_t cb = L == 8 ? CFP_PHASE_F64_L8_DEV[h] : CFP_PHASE_F64_L4_DEV[h];
        c = fma(__longlong_as_double((long long)cb), sd, c);
      }
      out = (float)scalbn(c, lambda);
    } else {
      out = __int_as_float(0x7fc00000);
    }
    C[o] = out;
  }
  if (phase_sums) {
#pragma unroll
    for (int h = 0; h < L; ++h) {
      const __int128 v = acc[h][tid];
      phase_sums[(o * L + h) * 2 + 0] = (int64_t)(uint64_t)v;
      phase_sums[(o * L + h) * 2 + 1] = (int64_t)(v >> 64);
    }
  }
  if (phase_lsb) phase_lsb[o] = lambda;
}

static OpView view_of(int layout, const uint8_t* c, const int8_t* s, int64_t R, int64_t K, int G) {
  int g = 0;
  while ((1 << g) < G) ++g;
  if (layout == CURVEFP_LAYOUT_ROWS) return OpView{c, K, 1, s, K >> g, 1, 0, g};
  return OpView{c, 1, R, s, 1, R >> g, g, 0};
}

cudaError_t launch_gemm_exact_oriented(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, int la,
                                       const uint8_t* b, const int8_t* sb, int lb, int64_t M, int64_t N, int64_t K,
                                       float* c, int64_t* ps, int32_t* pl, uint32_t* st, cudaStream_t s) {
  const OpView va = view_of(la, a, sa, M, K, G), vb = view_of(lb, b, sb, N, K, G);
  dim3 grid((unsigned)((N + TN - 1) / TN), (unsigned)((M + TM - 1) / TM));
#define CFP_V(X, Y)                                                                                        \
  if (fa == X && fb == Y) {                                                                                \
    gemm_exact_view_kernel<X, Y><<<grid, NT, 0, s>>>(va, vb, (int)M, (int)N, (int)K, c, ps, pl, st);       \
    return cudaGetLastError();                                                                             \
  }
  CFP_V(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_V(CURVEFP_E3C3, CURVEFP_E4C3)
  CFP_V(CURVEFP_E3C3, CURVEFP_E5C2)
  CFP_V(CURVEFP_E4C3, CURVEFP_E3C3)
  CFP_V(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_V(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_V(CURVEFP_E5C2, CURVEFP_E3C3)
  CFP_V(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_V(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_V
  return cudaErrorInvalidValue;
}

template <class Lat>
static cudaError_t launch_exact_t(int G, const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb,
                                  int64_t M, int64_t N, int64_t K, float* c, int64_t* ps, int32_t* pl, uint32_t* st,
                                  cudaStream_t s) {
  constexpr size_t smem = exact_smem<Lat>();
  static_assert(smem + 2 * TM * KC <= 227 * 1024, "shared memory");
  auto kern = gemm_exact_kernel<Lat>;
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  dim3 grid((unsigned)((N + TN - 1) / TN), (unsigned)((M + TM - 1) / TM));
  kern<<<grid, NT, smem, s>>>(a, sa, b, sb, (int)M, (int)N, (int)K, G, c, ps, pl, st);
  return cudaGetLastError();
}

cudaError_t launch_gemm_exact(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                              const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, int64_t* ps,
                              int32_t* pl, uint32_t* st, cudaStream_t s) {
#define CFP_E(X, Y) \
  if (fa == X && fb == Y) return launch_exact_t<BinLat<X, Y>>(G, a, sa, b, sb, M, N, K, c, ps, pl, st, s);
  CFP_E(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_E(CURVEFP_E3C3, CURVEFP_E4C3)
  CFP_E(CURVEFP_E3C3, CURVEFP_E5C2)
  CFP_E(CURVEFP_E4C3, CURVEFP_E3C3)
  CFP_E(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_E(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_E(CURVEFP_E5C2, CURVEFP_E3C3)
  CFP_E(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_E(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_E
  if (fa == CURVEFP_E4C3_R8_9 && fb == CURVEFP_E4C3_R8_9)
    return launch_exact_t<RadLat<CURVEFP_E4C3_R8_9>>(G, a, sa, b, sb, M, N, K, c, ps, pl, st, s);
  if (fa == CURVEFP_E4C3_R3_4 && fb == CURVEFP_E4C3_R3_4)
    return launch_exact_t<RadLat<CURVEFP_E4C3_R3_4>>(G, a, sa, b, sb, M, N, K, c, ps, pl, st, s);
  return cudaErrorInvalidValue;
}

}  // namespace cfp
