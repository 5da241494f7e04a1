// Quantization and dequantization for the rational-radix E4C3 formats
// (Sec. 3.1 Eq. 1 with r = 2^{p/q}; Table 7's points r = 2^{8/9} and
// r = 2^{3/4}).
//
// Levels sit at exponents lambda(n) = p n/(8q).  A scaled value y = |x| 2^{-a}
// with binade b and 23-bit mantissa mu has, on the unbounded lattice, the
// nearest level
//   n*(y) = N0[b mod PB] + floor(b / PB) NPER + #{i : mu >= THR[b mod PB][i]}
// (the count read from a 256-bucket table of the top mantissa bits: at most
// one threshold falls in a bucket)
// (the thresholds are the level midpoints inside the binade, and the pattern
// repeats every PB binades / NPER levels); the codebook then clamps n* to
// [-63, 63], and y <= L_nmin / 2 encodes as zero (R3; the tie at equality goes
// to zero).  Every threshold comes from exact integer arithmetic in
// gen_constants.py, so the decisions are exact for every FP32 input.
//
// A warp quantizes 512 values per step (16 coalesced 32-value chunks in
// flight), warp max reductions per block for the ceil-absmax scale, byte
// stores of 32 consecutive codes per chunk.
#include "cfp_common.cuh"
#include "kernels.cuh"

namespace cfp {

namespace {

static __constant__ int RX89_N0[1] = CFP_R8_9_N0_INIT;
static __constant__ int RX34_N0[3] = CFP_R3_4_N0_INIT;
// per binade class: top 8 mantissa bits -> thresholds passed by the whole
// bucket << 24 | the one threshold inside the bucket (2^23 if none)
static __constant__ uint32_t RX89_LUT[256] = CFP_R8_9_LUT_INIT;
static __constant__ uint32_t RX34_LUT[3 * 256] = CFP_R3_4_LUT_INIT;
static __constant__ uint32_t RX_C9[9] = CFP_PHASE_F32_L9_INIT;    // RN32(2^{h/9})
static __constant__ uint32_t RX_C32[32] = CFP_PHASE_F32_L32_INIT;  // RN32(2^{h/32})

__device__ __forceinline__ void split_f32r(uint32_t absb, int& F, uint32_t& mant) {
  if (absb >= 0x00800000u) {
    F = (int)(absb >> 23) - 127;
    mant = absb & 0x7FFFFFu;
  } else {
    const int p = 31 - __clz(absb);
    F = p - 149;
    mant = (absb << (23 - p)) & 0x7FFFFFu;
  }
}

__device__ __forceinline__ int floordiv_i(int a, int b) { return a >= 0 ? a / b : -((-a + b - 1) / b); }

// Ceil-absmax scale: the smallest a with amax <= 2^a 2^{lambda(63)},
// lambda(63) = F + f: a = F_amax - F, plus one if mu_amax > 2^f - 1.
template <int FMT>
__device__ __forceinline__ int radix_scale(uint32_t amaxb) {
  using R = Radix<FMT>;
  if (amaxb == 0u) return 0;
  if (amaxb >= 0x7F800000u) return 127;
  int Fx;
  uint32_t mant;
  split_f32r(amaxb, Fx, mant);
  const int a = Fx - R::F + (mant >= R::MU_SAT ? 1 : 0);
  return a < -128 ? -128 : (a > 127 ? 127 : a);
}

// Nearest-level tables of a format, staged in shared memory (lanes look up
// different binade classes, which constant memory would serialize).
struct RadixSmem {
  uint32_t lut[3 * 256];
  int n0[3];
};

template <int FMT>
__device__ __forceinline__ void radix_stage(RadixSmem& t) {
  constexpr int PB = Radix<FMT>::PB;
  for (int i = threadIdx.x; i < PB * 256; i += blockDim.x)
    t.lut[i] = FMT == CURVEFP_E4C3_R8_9 ? RX89_LUT[i] : RX34_LUT[i];
  if (threadIdx.x < PB) t.n0[threadIdx.x] = FMT == CURVEFP_E4C3_R8_9 ? RX89_N0[threadIdx.x] : RX34_N0[threadIdx.x];
}

template <int FMT>
__device__ __forceinline__ uint32_t radix_encode(const RadixSmem& t, uint32_t bits, int a, bool& nan) {
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
  split_f32r(absb, Fx, mant);
  const int b = Fx - a;
  if (b > R::F + 1) return sign | (2 * B - 1);
  if (b < R::ZB || (b == R::ZB && mant < R::ZTHR)) return 0u;
  const int k = floordiv_i(b, R::PB), c = b - k * R::PB;
  const uint32_t e = t.lut[c * 256 + (mant >> 15)];
  int n = t.n0[c] + k * R::NPER + (int)(e >> 24) + (mant >= (e & 0xFFFFFFu) ? 1 : 0);
  n = n < -NMAX ? -NMAX : (n > NMAX ? NMAX : n);
  return sign | (uint32_t)(n + B);
}

// A warp takes up to 512 elements of one row per step: 16 chunks of 32 (one
// coalesced load each, all in flight together) covering bpw = 512 / G
// consecutive blocks when the row length is a multiple of 512 (else one
// block per step).  Chunk maxima reduce with redux.sync, then across the
// G/32 chunks of a block by a butterfly.
template <int FMT, bool BF16>
__global__ void __launch_bounds__(256) quantize_radix_kernel(const void* __restrict__ x, int64_t rows, int64_t cols,
                                                             int64_t ld, int G, int lper, int bpw,
                                                             uint8_t* __restrict__ codes, int8_t* __restrict__ scales,
                                                             uint32_t* status) {
  __shared__ RadixSmem tab;
  radix_stage<FMT>(tab);
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int per = 1 << lper;  // chunks per block, G / 32
  const int nch = per * bpw;  // chunks per step (<= 16)
  const int64_t nbr = cols / G, nblk = rows * nbr;
  bool nan = false;
  for (int64_t w0 = (((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5) * bpw; w0 < nblk;
       w0 += (((int64_t)gridDim.x * blockDim.x) >> 5) * bpw) {
    const int64_t r = w0 / nbr, b0 = w0 - r * nbr;  // bpw divides nbr: one row per step
    const int64_t src = r * ld + b0 * G + lane, dst = r * cols + b0 * G + lane;
    uint32_t v[16], mx[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      v[i] = 0u;
      if (i < nch)
        v[i] = BF16 ? (uint32_t)__ldg(reinterpret_cast<const uint16_t*>(x) + src + i * 32) << 16
                    : __float_as_uint(__ldg(reinterpret_cast<const float*>(x) + src + i * 32));
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const uint32_t ab = v[i] & 0x7FFFFFFFu;
      mx[i] = __reduce_max_sync(0xffffffffu, ab <= 0x7F800000u ? ab : 0u);  // NaN left out of amax
    }
#pragma unroll
    for (int s = 1; s < 16; s <<= 1)
      if (s < per) {
        uint32_t t[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) t[i] = max(mx[i], mx[i ^ s]);
#pragma unroll
        for (int i = 0; i < 16; ++i) mx[i] = t[i];
      }
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (i < nch) {
        const int a = radix_scale<FMT>(mx[i]);
        codes[dst + i * 32] = (uint8_t)radix_encode<FMT>(tab, v[i], a, nan);
        if (lane == 0 && (i & (per - 1)) == 0) scales[w0 + (i >> lper)] = (int8_t)a;
      }
  }
  if (nan && status) atomicOr(status, CURVEFP_DEV_NAN);
}

// RN32(RN32(2^{j/N}) 2^{a + floor(p n/N)}), j = p n mod N (= h g).
template <int FMT>
__global__ void __launch_bounds__(256) dequantize_radix_kernel(const uint8_t* __restrict__ codes,
                                                               const int8_t* __restrict__ scales, int64_t n, int G,
                                                               float* __restrict__ out) {
  using R = Radix<FMT>;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t code = __ldg(codes + i);
    const uint32_t m = code & 0x7Fu;
    float v = 0.0f;
    if (m != 0u) {
      const int u = R::P * ((int)m - Fmt<FMT>::B);
      const int e = floordiv_i(u, R::N), j = u - e * R::N;
      const float cj = __uint_as_float(R::H == 9 ? RX_C9[j / R::G] : RX_C32[j / R::G]);
      v = __double2float_rn(ldexp((double)cj, (int)__ldg(scales + i / G) + e));
      if (code & 0x80u) v = -v;
    }
    out[i] = v;
  }
}

template <int FMT>
cudaError_t launch_qr(int G, const void* x, int dtype, int64_t rows, int64_t cols, int64_t ld, uint8_t* codes,
                      int8_t* scales, uint32_t* status, cudaStream_t st, int sms) {
  int lper = 0;
  while ((32 << lper) < G) ++lper;
  const int bpw = cols % 512 == 0 ? 16 >> lper : 1;  // blocks per warp step, all in one row
  const int64_t steps = rows * (cols / G) / bpw;
  const int64_t want = (steps + 7) / 8;
  const unsigned grid = (unsigned)(want < (int64_t)sms * 8 ? (want > 0 ? want : 1) : (int64_t)sms * 8);
  if (dtype == CURVEFP_BF16)
    quantize_radix_kernel<FMT, true><<<grid, 256, 0, st>>>(x, rows, cols, ld, G, lper, bpw, codes, scales, status);
  else
    quantize_radix_kernel<FMT, false><<<grid, 256, 0, st>>>(x, rows, cols, ld, G, lper, bpw, codes, scales, status);
  return cudaGetLastError();
}

}  // namespace

bool is_radix_format(int fmt) { return fmt == CURVEFP_E4C3_R8_9 || fmt == CURVEFP_E4C3_R3_4; }

cudaError_t launch_quantize_radix(int fmt, int G, const void* x, int dtype, int64_t rows, int64_t cols, int64_t ld,
                                  uint8_t* codes, int8_t* scales, uint32_t* status, cudaStream_t st, int sms) {
  if (fmt == CURVEFP_E4C3_R8_9)
    return launch_qr<CURVEFP_E4C3_R8_9>(G, x, dtype, rows, cols, ld, codes, scales, status, st, sms);
  if (fmt == CURVEFP_E4C3_R3_4)
    return launch_qr<CURVEFP_E4C3_R3_4>(G, x, dtype, rows, cols, ld, codes, scales, status, st, sms);
  return cudaErrorInvalidValue;
}

cudaError_t launch_dequantize_radix(int fmt, int G, const uint8_t* codes, const int8_t* scales, int64_t n, float* out,
                                    cudaStream_t st, int sms) {
  const int64_t want = (n + 255) / 256;
  const unsigned grid = (unsigned)(want < (int64_t)sms * 8 ? (want > 0 ? want : 1) : (int64_t)sms * 8);
  if (fmt == CURVEFP_E4C3_R8_9)
    dequantize_radix_kernel<CURVEFP_E4C3_R8_9><<<grid, 256, 0, st>>>(codes, scales, n, G, out);
  else if (fmt == CURVEFP_E4C3_R3_4)
    dequantize_radix_kernel<CURVEFP_E4C3_R3_4><<<grid, 256, 0, st>>>(codes, scales, n, G, out);
  else
    return cudaErrorInvalidValue;
  return cudaGetLastError();
}

}  // namespace cfp
