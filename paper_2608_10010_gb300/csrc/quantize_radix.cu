// Launchers for the rational-radix E4C3 formats (Sec. 3.1 Eq. 1 with
// r = 2^{p/q}; Table 2's points r = 2^{8/9} and r = 2^{3/4}): the shared
// quantizer kernels of quantize_kernels.cuh with these formats' rank tables
// and the exact encode of radix.cuh, and their dequantizer.
#include "quantize_kernels.cuh"

namespace cfp {

namespace {

template <int FMT>
__global__ void __launch_bounds__(256) dequantize_radix_kernel(const uint8_t* __restrict__ codes,
                                                               const int8_t* __restrict__ scales, int64_t n, int G,
                                                               float* __restrict__ out) {
  const int gs = __ffs(G) - 1;  // G is a power of two
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    out[i] = radix_recon_f32<FMT>(__ldg(codes + i), (int)__ldg(scales + (i >> gs)));
}

}  // namespace

bool is_radix_format(int fmt) { return fmt == CURVEFP_E4C3_R8_9 || fmt == CURVEFP_E4C3_R3_4; }

cudaError_t launch_quantize_radix(int fmt, int G, const void* x, int dtype, int64_t rows, int64_t cols, int64_t ld,
                                  int axis, uint8_t* codes, int8_t* scales, uint32_t* status, cudaStream_t st,
                                  int sms) {
#define CFP_Q(FMT)                                                                                     \
  return dtype == CURVEFP_F32                                                                          \
             ? launch_q_g<FMT, float>(G, x, rows, cols, ld, axis, codes, scales, status, st, sms)      \
             : launch_q_g<FMT, uint16_t>(G, x, rows, cols, ld, axis, codes, scales, status, st, sms);
  switch (fmt) {
    case CURVEFP_E4C3_R8_9: CFP_Q(CURVEFP_E4C3_R8_9)
    case CURVEFP_E4C3_R3_4: CFP_Q(CURVEFP_E4C3_R3_4)
  }
#undef CFP_Q
  return cudaErrorInvalidValue;
}

cudaError_t launch_quantize_static_radix(int fmt, int G, int group, int rule, const void* x, int dtype, int64_t rows,
                                         int64_t cols, uint8_t* codes, int8_t* scales, void* ws, uint32_t* status,
                                         cudaStream_t st, int sms) {
#define CFP_QS(FMT)                                                                                            \
  return dtype == CURVEFP_F32                                                                                  \
             ? launch_qs_t<FMT, float>(G, group, rule, x, rows, cols, codes, scales, ws, status, st, sms)      \
             : launch_qs_t<FMT, uint16_t>(G, group, rule, x, rows, cols, codes, scales, ws, status, st, sms);
  switch (fmt) {
    case CURVEFP_E4C3_R8_9: CFP_QS(CURVEFP_E4C3_R8_9)
    case CURVEFP_E4C3_R3_4: CFP_QS(CURVEFP_E4C3_R3_4)
  }
#undef CFP_QS
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
