// GEMMs on reused operands (Sec. 4, training GEMMs: the backward GEMMs take
// the forward pass's quantized operands, one of them transposed).
//
// A COLS operand is a [K x R] code matrix quantized along R (scales [K x R/G])
// that the GEMM reads as R rows of K codes: the scale of an element follows
// the element, so along a GEMM row it changes with k.  The tensor-core path
// handles that with per-element exponents (gemm_tc.cuh, PES): for every
// 32-code step of a GEMM row the preparation kernels below find the largest
// element exponent x = a + e over the step's nonzero codes, store
// f = that maximum - 15 as the step's scale (it becomes the step's UE8M0
// factor 2^{f - ref + 32}, ref = max over the row's steps) and, per element,
// the plane exponent x - f + 16 in [0, 31] (0x80 for zero codes and for the
// elements more than 31 binades below the step's largest one, whose plane
// value 2^{x - f} would leave E5M2).  A COLS operand's codes are transposed
// once into K-contiguous rows.  Everything goes into the caller's workspace;
// the kernels stream the operand once (HBM-bound: R K bytes read, 2 R K
// written for a COLS operand, R K for a ROWS operand, plus 2 R K / 32 bytes
// of step scales).
#include "gemm_tc.cuh"

namespace cfp {

namespace {

constexpr int TT = 64;  // transpose tile (codes), 64 x 64 bytes
constexpr int16_t NO_STEP = -32768;

// e + 2^{E-1} of a code byte (zero codes: -1).
template <int FMT>
__device__ __forceinline__ int biased_exp(uint32_t code) {
  const uint32_t m = code & (uint32_t)Fmt<FMT>::MMASK;
  return m ? (int)(m >> Fmt<FMT>::C) : -1;
}

// Exponent bytes of the 16 codes of a half step (scales a[i], the step's
// largest exponent xmax over both halves, exchanged with the partner lane
// `pmask`), and the step scale f = xmax - 15 (NO_STEP when all 32 are zero).
template <int FMT>
__device__ __forceinline__ void half_step_bytes(const uint32_t (&c)[16], const int (&a)[16], unsigned pmask,
                                                uint32_t (&dp)[4], int& f) {
  constexpr int EB = 1 << (Fmt<FMT>::E - 1);
  int x[16], xm = -100000;
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int eb = biased_exp<FMT>(c[i]);
    x[i] = eb < 0 ? -100000 : a[i] + eb - EB;
    xm = max(xm, x[i]);
  }
  xm = max(xm, __shfl_xor_sync(pmask, xm, 1));
  f = xm < -50000 ? NO_STEP : xm - 15;
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    uint32_t d = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int b = x[4 * w + j] - (xm - 15) + 16;  // plane exponent + 16
      d |= (uint32_t)(b >= 0 && b <= 31 && x[4 * w + j] > -50000 ? b : 0x80) << (8 * j);
    }
    dp[w] = d;
  }
}

// ROWS operand (codes [R x K], scales [R x K/G]): a lane pair per 32-code
// step, 16 codes per lane.
template <int FMT>
__global__ void pes_rows_kernel(const uint8_t* __restrict__ codes, const int8_t* __restrict__ s, int64_t R, int64_t K,
                                int gsh, uint8_t* __restrict__ dp, int16_t* __restrict__ fst, int* __restrict__ ref) {
  const int64_t per_row = K / 16;
  const int64_t n = R * per_row;
  const int64_t nb = K >> gsh;
  const unsigned pmask = 3u << ((threadIdx.x & 31) & ~1u);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / per_row, k = (i - r * per_row) * 16;
    const uint4 q = __ldg(reinterpret_cast<const uint4*>(codes + r * K + k));
    const int sc = (int)__ldg(s + r * nb + (k >> gsh));
    const uint32_t wv[4] = {q.x, q.y, q.z, q.w};
    uint32_t c[16];
    int a[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      c[j] = (wv[j >> 2] >> (8 * (j & 3))) & 0xFFu;
      a[j] = sc;
    }
    uint32_t d[4];
    int f;
    half_step_bytes<FMT>(c, a, pmask, d, f);
    *reinterpret_cast<uint4*>(dp + r * K + k) = make_uint4(d[0], d[1], d[2], d[3]);
    if ((i & 1) == 0) {
      fst[r * (K / 32) + (k >> 5)] = (int16_t)f;
      if (f != NO_STEP) atomicMax(ref + r, f);
    }
  }
}

// COLS operand: codes [K x R] -> codesT [R x K], with the exponent bytes and
// step scales of the transposed rows.  One 64 x 64 tile per CTA (256
// threads, 16 bytes per thread each way; lanes 2t and 2t + 1 hold the two
// halves of a 32-code step); R % 32 == 0 and K % 32 == 0, so every step is
// wholly inside or outside the matrix.
template <int FMT>
__global__ void __launch_bounds__(256) pes_cols_kernel(const uint8_t* __restrict__ codes, const int8_t* __restrict__ s,
                                                       int64_t R, int64_t K, int gsh, uint8_t* __restrict__ codesT,
                                                       uint8_t* __restrict__ dp, int16_t* __restrict__ fst,
                                                       int* __restrict__ ref) {
  __shared__ uint32_t tile[TT][TT / 4 + 1];  // [k][r / 4], one padding word per row
  __shared__ int8_t ts[TT][2];               // scales of the tile's (at most two) block columns
  const int64_t r0 = (int64_t)blockIdx.x * TT, k0 = (int64_t)blockIdx.y * TT;
  const int nq = (int)(R >> gsh);
  const int q0 = (int)(r0 >> gsh);
  const int t = threadIdx.x;
  {
    const int kk = t >> 2, seg = t & 3;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (k0 + kk < K && r0 + seg * 16 < R) v = __ldg(reinterpret_cast<const uint4*>(codes + (k0 + kk) * R + r0 + seg * 16));
    tile[kk][seg * 4 + 0] = v.x;
    tile[kk][seg * 4 + 1] = v.y;
    tile[kk][seg * 4 + 2] = v.z;
    tile[kk][seg * 4 + 3] = v.w;
    if (t < 2 * TT) {
      const int k2 = t >> 1, qq = t & 1;
      ts[k2][qq] = (k0 + k2 < K && q0 + qq < nq) ? __ldg(s + (k0 + k2) * nq + q0 + qq) : (int8_t)-128;
    }
  }
  __syncthreads();
  const int rr = t >> 2, seg = t & 3;
  const int64_t r = r0 + rr, k = k0 + seg * 16;
  if (r >= R || k >= K) return;  // a lane pair leaves together
  const int qq = (int)(r >> gsh) - q0;
  const unsigned pmask = 3u << ((threadIdx.x & 31) & ~1u);
  uint32_t c[16];
  int a[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const int kk = seg * 16 + j;
    c[j] = (tile[kk][rr >> 2] >> (8 * (rr & 3))) & 0xFFu;
    a[j] = ts[kk][qq];
  }
  uint32_t d[4];
  int f;
  half_step_bytes<FMT>(c, a, pmask, d, f);
  uint32_t cw[4];
#pragma unroll
  for (int w = 0; w < 4; ++w) cw[w] = c[4 * w] | c[4 * w + 1] << 8 | c[4 * w + 2] << 16 | c[4 * w + 3] << 24;
  *reinterpret_cast<uint4*>(codesT + r * K + k) = make_uint4(cw[0], cw[1], cw[2], cw[3]);
  *reinterpret_cast<uint4*>(dp + r * K + k) = make_uint4(d[0], d[1], d[2], d[3]);
  if ((seg & 1) == 0) {
    fst[r * (K / 32) + (k >> 5)] = (int16_t)f;
    if (f != NO_STEP) atomicMax(ref + r, f);
  }
}

int log2i(int g) {
  int s = 0;
  while ((1 << s) < g) ++s;
  return s;
}

size_t al256(size_t v) { return (v + 255) & ~(size_t)255; }

// Workspace of one operand: [codesT (COLS only)] [dp] [step scales] [ref].
size_t operand_ws(int layout, int64_t R, int64_t K) {
  return (layout == CURVEFP_LAYOUT_COLS ? al256((size_t)R * K) : 0) + al256((size_t)R * K) +
         al256((size_t)R * (K / 32) * 2) + al256((size_t)R * 4);
}

struct Prepared {
  const uint8_t* codes;
  const uint8_t* dp;
  const int16_t* f;
  const int* ref;
};

template <int FMT>
cudaError_t prepare_t(int layout, const uint8_t* codes, const int8_t* s, int64_t R, int64_t K, int G, uint8_t* ws,
                      cudaStream_t st, Prepared& out) {
  const int gsh = log2i(G);
  uint8_t* p = ws;
  uint8_t* codesT = nullptr;
  if (layout == CURVEFP_LAYOUT_COLS) {
    codesT = p;
    p += al256((size_t)R * K);
  }
  uint8_t* dp = p;
  p += al256((size_t)R * K);
  int16_t* f = reinterpret_cast<int16_t*>(p);
  p += al256((size_t)R * (K / 32) * 2);
  int* ref = reinterpret_cast<int*>(p);
  cudaError_t e = cudaMemsetAsync(ref, 0x80, (size_t)R * 4, st);  // 0x80808080: below every step scale
  if (e != cudaSuccess) return e;
  if (layout == CURVEFP_LAYOUT_ROWS) {
    const int64_t n16 = R * (K / 16);
    const int64_t want = (n16 + 255) / 256;
    const unsigned blocks = (unsigned)(want < 152 * 16 ? (want > 0 ? want : 1) : 152 * 16);
    pes_rows_kernel<FMT><<<blocks, 256, 0, st>>>(codes, s, R, K, gsh, dp, f, ref);
    out = Prepared{codes, dp, f, ref};
  } else {
    dim3 g2((unsigned)((R + TT - 1) / TT), (unsigned)((K + TT - 1) / TT));
    pes_cols_kernel<FMT><<<g2, 256, 0, st>>>(codes, s, R, K, gsh, codesT, dp, f, ref);
    out = Prepared{codesT, dp, f, ref};
  }
  return cudaGetLastError();
}

cudaError_t prepare(int fmt, int layout, const uint8_t* codes, const int8_t* s, int64_t R, int64_t K, int G,
                    uint8_t* ws, cudaStream_t st, Prepared& out) {
  if (fmt == CURVEFP_E3C3) return prepare_t<CURVEFP_E3C3>(layout, codes, s, R, K, G, ws, st, out);
  if (fmt == CURVEFP_E4C3) return prepare_t<CURVEFP_E4C3>(layout, codes, s, R, K, G, ws, st, out);
  if (fmt == CURVEFP_E5C2) return prepare_t<CURVEFP_E5C2>(layout, codes, s, R, K, G, ws, st, out);
  return cudaErrorInvalidValue;
}

}  // namespace

size_t gemm_reuse_workspace(int la, int lb, int64_t M, int64_t N, int64_t K) {
  if (la == CURVEFP_LAYOUT_ROWS && lb == CURVEFP_LAYOUT_ROWS) return 0;
  return operand_ws(la, M, K) + operand_ws(lb, N, K);
}

cudaError_t launch_gemm_tensor_reuse(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, int la,
                                     const uint8_t* b, const int8_t* sb, int lb, int64_t M, int64_t N, int64_t K,
                                     float* c, void* ws, uint32_t* status, cudaStream_t s, int sms) {
  uint8_t* w = static_cast<uint8_t*>(ws);
  Prepared pa, pb;
  cudaError_t e = prepare(fa, la, a, sa, M, K, G, w, s, pa);
  if (e != cudaSuccess) return e;
  e = prepare(fb, lb, b, sb, N, K, G, w + operand_ws(la, M, K), s, pb);
  if (e != cudaSuccess) return e;
  const PesOperands pes{pa.dp, pb.dp, pa.f, pb.f, pa.ref, pb.ref};
#define CFP_R(X, Y) \
  if (fa == X && fb == Y) return launch_tc_t<X, Y, true>(G, pa.codes, nullptr, pb.codes, nullptr, M, N, K, c, status, s, pes, sms);
  CFP_R(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_R(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_R(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_R(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_R(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_R
  return cudaErrorInvalidValue;
}

}  // namespace cfp
