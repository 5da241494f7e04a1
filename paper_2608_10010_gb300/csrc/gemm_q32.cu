// The spatial tile's integer semantics as a second bit-exact GEMM (App. C.1,
// C.2): every nonzero product a (x) b has lattice exponent
// u = n_a L/K_a + n_b L/K_b = L e + k and adds
//   (-1)^{s_a xor s_b} round(2^{k/L} 2^16) 2^{16 + e + sa + sb}
// to a signed 64-bit Q32 accumulator (value = acc 2^-32); nothing is rounded
// along the way.  For E4C3 x E4C3 this is the tile's q_p = m_a + m_b - 128 =
// 8e + k coefficient select and shift.  A product that would need a negative
// shift, or a sum that leaves int64, raises CURVEFP_DEV_RANGE.
//
// One CTA owns 16 x 16 outputs (one thread each); 64-code slices of the A and
// B rows are staged in shared memory; accumulation in 128-bit integers.
#include "cfp_common.cuh"
#include "kernels.cuh"

namespace cfp {

namespace {

constexpr int QT = 16;   // outputs per CTA side
constexpr int QKC = 64;  // codes per staged slice

template <int FA, int FB>
__global__ void __launch_bounds__(QT* QT) gemm_q32_kernel(const uint8_t* __restrict__ A, const int8_t* __restrict__ sA,
                                                          const uint8_t* __restrict__ B, const int8_t* __restrict__ sB,
                                                          int M, int N, int K, int G, int64_t* __restrict__ out,
                                                          uint32_t* status) {
  using P = Pair<FA, FB>;
  constexpr int L = P::L, WA = P::WA, WB = P::WB, LOG2L = P::LOG2L;
  constexpr int BA = Fmt<FA>::B, BB = Fmt<FB>::B;
  __shared__ uint8_t as[QT][QKC], bs[QT][QKC];
  __shared__ uint32_t q16[8];
  const int tx = threadIdx.x % QT, ty = threadIdx.x / QT;
  const int i = blockIdx.y * QT + ty, j = blockIdx.x * QT + tx;
  if (threadIdx.x < L) {
    const uint32_t c8[8] = CFP_Q16_K8_INIT;
    const uint32_t c4[4] = CFP_Q16_K4_INIT;
    q16[threadIdx.x] = L == 8 ? c8[threadIdx.x] : c4[threadIdx.x & 3];
  }
  __int128 acc = 0;
  bool range = false;
  const int nb = K / G;
  for (int k0 = 0; k0 < K; k0 += QKC) {
    __syncthreads();
    for (int t = threadIdx.x; t < QT * QKC; t += QT * QT) {
      const int r = t / QKC, c = t % QKC;
      const int ra = blockIdx.y * QT + r, rb = blockIdx.x * QT + r;
      as[r][c] = (ra < M && k0 + c < K) ? A[(int64_t)ra * K + k0 + c] : 0;
      bs[r][c] = (rb < N && k0 + c < K) ? B[(int64_t)rb * K + k0 + c] : 0;
    }
    __syncthreads();
    if (i >= M || j >= N) continue;
    for (int c = 0; c < QKC && k0 + c < K; ++c) {
      const uint32_t ca = as[ty][c], cb = bs[tx][c];
      const int ma = (int)(ca & 0x7Fu), mb = (int)(cb & 0x7Fu);
      if (ma == 0 || mb == 0) continue;  // zero sentinel: no update
      const int u = (ma - BA) * WA + (mb - BB) * WB;
      const int e = u >> LOG2L, k = u & (L - 1);
      const int blk = (k0 + c) / G;
      const int sh = 16 + e + (int)sA[(int64_t)i * nb + blk] + (int)sB[(int64_t)j * nb + blk];
      if (sh < 0 || sh > 45) {  // |term| < 2^62 keeps every partial sum exact
        range = true;
        continue;
      }
      const __int128 term = (__int128)q16[k] << sh;
      acc += ((ca ^ cb) & 0x80u) ? -term : term;
    }
  }
  if (i < M && j < N) {
    if (acc > (__int128)INT64_MAX || acc < (__int128)INT64_MIN) range = true;
    out[(int64_t)i * N + j] = (int64_t)acc;
    if (range && status) atomicOr(status, CURVEFP_DEV_RANGE);
  }
}

}  // namespace

cudaError_t launch_gemm_q32(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                            const int8_t* sb, int64_t M, int64_t N, int64_t K, int64_t* out, uint32_t* status,
                            cudaStream_t s) {
  dim3 grid((unsigned)((N + QT - 1) / QT), (unsigned)((M + QT - 1) / QT));
#define CFP_Q(X, Y)                                                                                              \
  if (fa == X && fb == Y) {                                                                                      \
    gemm_q32_kernel<X, Y><<<grid, QT * QT, 0, s>>>(a, sa, b, sb, (int)M, (int)N, (int)K, G, out, status);        \
    return cudaGetLastError();                                                                                   \
  }
  CFP_Q(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_Q(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_Q(CURVEFP_E5C2, CURVEFP_E5C2)
  CFP_Q(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_Q(CURVEFP_E4C3, CURVEFP_E5C2)
#undef CFP_Q
  return cudaErrorInvalidValue;
}

}  // namespace cfp
