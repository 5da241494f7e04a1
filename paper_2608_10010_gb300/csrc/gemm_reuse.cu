// GEMMs on reused operands (Sec. 4, training GEMMs: the backward GEMMs take
// the forward pass's quantized operands, one of them transposed).
//
// A COLS operand is a [K x R] code matrix quantized along R (scales [K x R/G])
// that the GEMM reads as R rows of K codes: the scale of an element follows
// the element, so along a GEMM row it changes with k.  The tensor-core path
// handles that with per-element scales in the producers (gemm_tc.cuh, PES):
// every operand gets a byte per element holding its scale relative to the row
// reference, dp = max(a - ref, -64) + 64 (elements 64 binades below the
// reference flush in any case), and a COLS operand's codes are transposed once
// into K-contiguous rows.  Both are written into the caller's workspace by the
// preparation kernels below, which stream the operand once (HBM-bound: R K
// bytes read, 2 R K written for a COLS operand, R K for a ROWS operand).
#include "gemm_tc.cuh"

namespace cfp {

namespace {

constexpr int TT = 64;  // transpose tile (codes), 64 x 64 bytes

// ROWS operand: ref[r] = max_b s[r][b].
__global__ void pes_ref_rows_kernel(const int8_t* __restrict__ s, int64_t R, int nb, int* __restrict__ ref) {
  const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= R) return;
  int m = -128;
  for (int b = 0; b < nb; ++b) m = max(m, (int)__ldg(s + r * nb + b));
  ref[r] = m;
}

// COLS operand: ref[q] = max_k s[k][q] over the block column q < nq (ref is
// preset to INT_MIN-like 0x80808080).  Block: 32 columns x 8 row lanes, rows
// [blockIdx.y * KCH, +KCH).
constexpr int KCH = 256;
__global__ void pes_ref_cols_kernel(const int8_t* __restrict__ s, int64_t K, int nq, int* __restrict__ ref) {
  const int q = blockIdx.x * 32 + (threadIdx.x & 31);
  if (q >= nq) return;
  const int64_t k0 = (int64_t)blockIdx.y * KCH;
  const int64_t k1 = min(K, k0 + KCH);
  int m = -128;
  for (int64_t k = k0 + (threadIdx.x >> 5); k < k1; k += 8) m = max(m, (int)__ldg(s + k * nq + q));
  atomicMax(ref + q, m);
}

__device__ __forceinline__ uint32_t rel_byte(int a, int ref) {
  const int d = a - ref;
  return (uint32_t)((d < -64 ? -64 : d) + 64);
}

// ROWS operand: dp[r][k] = rel(s[r][k >> gsh], ref[r]); 16 bytes per thread
// (G >= 32, so one scale per 16-byte run).
__global__ void pes_dp_rows_kernel(const int8_t* __restrict__ s, const int* __restrict__ ref, int64_t R, int64_t K,
                                   int gsh, uint8_t* __restrict__ dp) {
  const int64_t per_row = K / 16;
  const int64_t n = R * per_row;
  const int64_t nb = K >> gsh;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / per_row, k = (i - r * per_row) * 16;
    const uint32_t v = rel_byte((int)__ldg(s + r * nb + (k >> gsh)), __ldg(ref + r)) * 0x01010101u;
    *reinterpret_cast<uint4*>(dp + r * K + k) = make_uint4(v, v, v, v);
  }
}

// COLS operand: codes [K x R] -> codesT [R x K] and dp [R x K] with
// dp[r][k] = rel(s[k][r >> gsh], ref[r >> gsh]).  One 64 x 64 tile per CTA
// (256 threads, 16 bytes per thread each way); R % 32 == 0 and K % 16 == 0,
// so every 16-byte run is wholly inside or outside the matrix.
__global__ void __launch_bounds__(256) pes_transpose_cols_kernel(const uint8_t* __restrict__ codes,
                                                                 const int8_t* __restrict__ s,
                                                                 const int* __restrict__ refq, int64_t R, int64_t K,
                                                                 int gsh, uint8_t* __restrict__ codesT,
                                                                 uint8_t* __restrict__ dp) {
  __shared__ uint32_t tile[TT][TT / 4 + 1];  // [k][r / 4], one padding word per row
  __shared__ int8_t ts[TT][2];               // scales of the tile's (at most two) block columns
  __shared__ int tref[2];
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
    if (t < 2) tref[t] = q0 + t < nq ? __ldg(refq + q0 + t) : 0;
  }
  __syncthreads();
  const int rr = t >> 2, seg = t & 3;
  const int64_t r = r0 + rr, k = k0 + seg * 16;
  if (r >= R || k >= K) return;
  const int qq = (int)(r >> gsh) - q0;
  const int ref = tref[qq];
  uint32_t c[4], d[4];
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    uint32_t cw = 0, dw = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int kk = seg * 16 + w * 4 + j;
      const uint32_t byte = (tile[kk][rr >> 2] >> (8 * (rr & 3))) & 0xFFu;
      cw |= byte << (8 * j);
      dw |= rel_byte(ts[kk][qq], ref) << (8 * j);
    }
    c[w] = cw;
    d[w] = dw;
  }
  *reinterpret_cast<uint4*>(codesT + r * K + k) = make_uint4(c[0], c[1], c[2], c[3]);
  *reinterpret_cast<uint4*>(dp + r * K + k) = make_uint4(d[0], d[1], d[2], d[3]);
}

int log2i(int g) {
  int s = 0;
  while ((1 << s) < g) ++s;
  return s;
}

size_t al256(size_t v) { return (v + 255) & ~(size_t)255; }

// Workspace of one operand: [codesT (COLS only)] [dp] [ref].
size_t operand_ws(int layout, int64_t R, int64_t K) {
  return (layout == CURVEFP_LAYOUT_COLS ? al256((size_t)R * K) : 0) + al256((size_t)R * K) + al256((size_t)R * 4);
}

struct Prepared {
  const uint8_t* codes;
  const uint8_t* dp;
  const int* ref;
  int rsh;
};

cudaError_t prepare(int layout, const uint8_t* codes, const int8_t* s, int64_t R, int64_t K, int G, uint8_t* ws,
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
  int* ref = reinterpret_cast<int*>(p);
  if (layout == CURVEFP_LAYOUT_ROWS) {
    pes_ref_rows_kernel<<<(unsigned)((R + 255) / 256), 256, 0, st>>>(s, R, (int)(K >> gsh), ref);
    const int64_t n16 = R * (K / 16);
    const int64_t want = (n16 + 255) / 256;
    const unsigned blocks = (unsigned)(want < 152 * 16 ? (want > 0 ? want : 1) : 152 * 16);
    pes_dp_rows_kernel<<<blocks, 256, 0, st>>>(s, ref, R, K, gsh, dp);
    out = Prepared{codes, dp, ref, 0};
  } else {
    const int nq = (int)(R >> gsh);
    cudaError_t e = cudaMemsetAsync(ref, 0x80, (size_t)nq * 4, st);
    if (e != cudaSuccess) return e;
    dim3 g1((unsigned)((nq + 31) / 32), (unsigned)((K + KCH - 1) / KCH));
    pes_ref_cols_kernel<<<g1, 256, 0, st>>>(s, K, nq, ref);
    dim3 g2((unsigned)((R + TT - 1) / TT), (unsigned)((K + TT - 1) / TT));
    pes_transpose_cols_kernel<<<g2, 256, 0, st>>>(codes, s, ref, R, K, gsh, codesT, dp);
    out = Prepared{codesT, dp, ref, gsh};
  }
  return cudaGetLastError();
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
  cudaError_t e = prepare(la, a, sa, M, K, G, w, s, pa);
  if (e != cudaSuccess) return e;
  e = prepare(lb, b, sb, N, K, G, w + operand_ws(la, M, K), s, pb);
  if (e != cudaSuccess) return e;
  const PesOperands pes{pa.dp, pb.dp, pa.ref, pb.ref, pa.rsh, pb.rsh};
  constexpr int PT = PLANE_E5M2;
#define CFP_R(X, Y) \
  if (fa == X && fb == Y) return launch_tc_t<X, Y, PT, true>(G, pa.codes, nullptr, pb.codes, nullptr, M, N, K, c, status, s, pes, sms);
  CFP_R(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_R(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_R(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_R(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_R(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_R
  return cudaErrorInvalidValue;
}

}  // namespace cfp
