// The histogram accumulation layout as a bit-exact GEMM (Eq. 5, App. A.1:
// equal addresses (h, t) merge with signed popcounts; the counts n_{h,t}
// reduce to the same phase sums S_h = sum_t n_{h,t} 2^t as the wide per-phase
// accumulators of the exact kernel).
//
// One warp owns one output (i, j) at a time: each lane forms the closed
// product of one k of a 32-wide slice (delta, phase h, bin t - lambda);
// __match_any_sync groups the lanes with equal addresses, and the group's
// lowest lane adds the signed popcount (lanes with delta = +1 minus lanes with
// delta = -1) to the warp's shared-memory histogram n[h][t].  At the end each
// phase's counts are shifted into an exact int128 sum.  Validation kernel:
// it shows on the GPU that both layouts of the paper give identical S_h.
#include "cfp_common.cuh"
#include "kernels.cuh"

namespace cfp {

namespace {

constexpr int HW = 8;      // warps (outputs in flight) per CTA
constexpr int NBIN = 128;  // bins per phase: t - lambda < 127 inside the int128 window

template <class Lat>
__global__ void __launch_bounds__(HW * 32) gemm_hist_kernel(const uint8_t* __restrict__ A, const int8_t* __restrict__ sA,
                                                            const uint8_t* __restrict__ B, const int8_t* __restrict__ sB,
                                                            int M, int N, int K, int G, float* __restrict__ C,
                                                            int64_t* __restrict__ phase_sums,
                                                            int32_t* __restrict__ phase_lsb, uint32_t* status) {
  constexpr int L = Lat::L;
  constexpr int DT = Lat::TMAX - Lat::TMIN;
  extern __shared__ int32_t hist_dyn[];  // [HW][L][NBIN]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int32_t* hist = hist_dyn + (size_t)warp * L * NBIN;
  const int nb = K / G;
  const int64_t nout = (int64_t)M * N;
  for (int64_t o = (int64_t)blockIdx.x * HW + warp; o < nout; o += (int64_t)gridDim.x * HW) {
    const int i = (int)(o / N), j = (int)(o - (int64_t)i * N);
    // lambda = min_b (sa + sb) + t_min, and the int128 window check
    int smin = 1 << 20, smax = -(1 << 20);
    for (int b = lane; b < nb; b += 32) {
      const int s = (int)sA[(int64_t)i * nb + b] + (int)sB[(int64_t)j * nb + b];
      smin = min(smin, s);
      smax = max(smax, s);
    }
    smin = __reduce_min_sync(0xffffffffu, smin);
    smax = __reduce_max_sync(0xffffffffu, smax);
    const bool in_range = bitlen64(K) + (smax - smin) + DT <= 127;
    for (int q = lane; q < L * NBIN; q += 32) hist[q] = 0;
    __syncwarp();
    if (in_range) {
      const uint8_t* arow = A + (int64_t)i * K;
      const uint8_t* brow = B + (int64_t)j * K;
      for (int k0 = 0; k0 < K; k0 += 32) {
        const int k = k0 + lane;
        int addr = -1, delta = 0;
        if (k < K) {
          const uint32_t ca = __ldg(arow + k), cb = __ldg(brow + k);
          const uint32_t ma = ca & Lat::MA, mb = cb & Lat::MB;
          if (ma != 0u && mb != 0u) {
            int h, sh;
            Lat::addr(ma, mb, h, sh);
            const int blk = k / G;
            sh += (int)sA[(int64_t)i * nb + blk] + (int)sB[(int64_t)j * nb + blk] - smin;
            addr = h * NBIN + sh;
            delta = ((ca ^ cb) & 0x80u) ? -1 : 1;
          }
        }
        const unsigned peers = __match_any_sync(0xffffffffu, addr);
        const unsigned pos = __ballot_sync(0xffffffffu, delta > 0), neg = __ballot_sync(0xffffffffu, delta < 0);
        if (addr >= 0 && lane == __ffs(peers) - 1) hist[addr] += __popc(peers & pos) - __popc(peers & neg);
        __syncwarp();
      }
    }
    // S_h = sum_t n_{h,t} 2^t, one phase per lane
    __int128 S = 0;
    if (lane < L && in_range)
      for (int t = 0; t < NBIN; ++t) {
        const int32_t n = hist[lane * NBIN + t];
        if (n != 0) S += (__int128)((unsigned __int128)(__int128)n << t);
      }
    const int lambda = smin + Lat::TMIN;
    if (phase_sums && lane < L) {
      phase_sums[(o * L + lane) * 2 + 0] = (int64_t)(uint64_t)S;
      phase_sums[(o * L + lane) * 2 + 1] = (int64_t)(S >> 64);
    }
    if (lane == 0) {
      if (phase_lsb) phase_lsb[o] = lambda;
      if (!in_range && status) atomicOr(status, CURVEFP_DEV_RANGE);
    }
    if (C) {
      // combine in FP64 as the exact kernel does: c = fma(2^{h/L}, S_h, c) for
      // h = 0 .. L-1 (lane 0 runs the chain, the sums come by shuffle)
      double sd = 0.0;
      if (lane < L && in_range) {
        const int64_t hi = (int64_t)(S >> 64);
        const uint64_t lo = (uint64_t)S;
        if ((hi == 0 && (int64_t)lo >= 0) || (hi == -1 && (int64_t)lo < 0)) {
          sd = (double)(int64_t)lo;
        } else {
          const bool neg = hi < 0;
          const unsigned __int128 m = neg ? (unsigned __int128)0 - (unsigned __int128)S : (unsigned __int128)S;
          const double d = fma((double)(uint64_t)(m >> 64), 18446744073709551616.0, (double)(uint64_t)m);
          sd = neg ? -d : d;
        }
      }
      double c = 0.0;
      for (int h = 0; h < L; ++h) {
        const double sh = __shfl_sync(0xffffffffu, sd, h);
        c = fma(__longlong_as_double((long long)Lat::phase64(h)), sh, c);
      }
      if (lane == 0) C[o] = in_range ? (float)scalbn(c, lambda) : __int_as_float(0x7fc00000);
    }
    __syncwarp();
  }
}

template <class Lat>
cudaError_t launch_hist_t(int G, const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb, int64_t M,
                          int64_t N, int64_t K, float* c, int64_t* ps, int32_t* pl, uint32_t* st, cudaStream_t s,
                          int sms) {
  static_assert(Lat::L <= 32, "one phase per lane");
  constexpr size_t smem = (size_t)HW * Lat::L * NBIN * 4;
  auto kern = gemm_hist_kernel<Lat>;
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  const int64_t want = (M * N + HW - 1) / HW;
  const unsigned grid = (unsigned)(want < (int64_t)sms * 4 ? want : (int64_t)sms * 4);
  kern<<<grid, HW * 32, smem, s>>>(a, sa, b, sb, (int)M, (int)N, (int)K, G, c, ps, pl, st);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_hist(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                             const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, int64_t* ps, int32_t* pl,
                             uint32_t* st, cudaStream_t s, int sms) {
#define CFP_H(X, Y) \
  if (fa == X && fb == Y) return launch_hist_t<BinLat<X, Y>>(G, a, sa, b, sb, M, N, K, c, ps, pl, st, s, sms);
  CFP_H(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_H(CURVEFP_E3C3, CURVEFP_E4C3)
  CFP_H(CURVEFP_E3C3, CURVEFP_E5C2)
  CFP_H(CURVEFP_E4C3, CURVEFP_E3C3)
  CFP_H(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_H(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_H(CURVEFP_E5C2, CURVEFP_E3C3)
  CFP_H(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_H(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_H
  if (fa == CURVEFP_E4C3_R8_9 && fb == CURVEFP_E4C3_R8_9)
    return launch_hist_t<RadLat<CURVEFP_E4C3_R8_9>>(G, a, sa, b, sb, M, N, K, c, ps, pl, st, s, sms);
  if (fa == CURVEFP_E4C3_R3_4 && fb == CURVEFP_E4C3_R3_4)
    return launch_hist_t<RadLat<CURVEFP_E4C3_R3_4>>(G, a, sa, b, sb, M, N, K, c, ps, pl, st, s, sms);
  return cudaErrorInvalidValue;
}

}  // namespace cfp
