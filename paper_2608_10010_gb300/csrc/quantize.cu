// Launchers of the quantizer, static-operand quantizer and dequantizer for
// the binary-radix formats (kernels in quantize_kernels.cuh).
#include "quantize_kernels.cuh"

namespace cfp {

size_t quantize_static_workspace(int64_t rows, int64_t cols, int G, int group) {
  return qs_workspace_bytes(rows, cols, G, group);
}

cudaError_t launch_quantize(int fmt, int G, const void* x, int dtype, int64_t rows, int64_t cols, int64_t ld,
                            int axis, uint8_t* codes, int8_t* scales, uint32_t* status, cudaStream_t st, int sms) {
#define CFP_Q(FMT)                                                                                     \
  return dtype == CURVEFP_F32                                                                          \
             ? launch_q_g<FMT, float>(G, x, rows, cols, ld, axis, codes, scales, status, st, sms)      \
             : launch_q_g<FMT, uint16_t>(G, x, rows, cols, ld, axis, codes, scales, status, st, sms);
  switch (fmt) {
    case CURVEFP_E3C3: CFP_Q(CURVEFP_E3C3)
    case CURVEFP_E4C3: CFP_Q(CURVEFP_E4C3)
    case CURVEFP_E5C2: CFP_Q(CURVEFP_E5C2)
  }
#undef CFP_Q
  return cudaErrorInvalidValue;
}

cudaError_t launch_quantize_static(int fmt, int G, int group, int rule, const void* x, int dtype, int64_t rows,
                                   int64_t cols, uint8_t* codes, int8_t* scales, void* ws, uint32_t* status,
                                   cudaStream_t st, int sms) {
#define CFP_QS(FMT)                                                                                            \
  return dtype == CURVEFP_F32                                                                                  \
             ? launch_qs_t<FMT, float>(G, group, rule, x, rows, cols, codes, scales, ws, status, st, sms)      \
             : launch_qs_t<FMT, uint16_t>(G, group, rule, x, rows, cols, codes, scales, ws, status, st, sms);
  switch (fmt) {
    case CURVEFP_E3C3: CFP_QS(CURVEFP_E3C3)
    case CURVEFP_E4C3: CFP_QS(CURVEFP_E4C3)
    case CURVEFP_E5C2: CFP_QS(CURVEFP_E5C2)
  }
#undef CFP_QS
  return cudaErrorInvalidValue;
}

cudaError_t launch_dequantize(int fmt, int G, const uint8_t* codes, const int8_t* scales, int64_t n, float* out,
                              cudaStream_t st, int sms) {
  int64_t grid = (n / 4 + 1023) / 1024;  // 256 threads x 4 words of 4 codes
  const int64_t cap = (int64_t)sms * 8;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  switch (fmt) {
    case CURVEFP_E3C3: dequantize_kernel<CURVEFP_E3C3><<<(unsigned)grid, 256, 0, st>>>(codes, scales, n, G, out); break;
    case CURVEFP_E4C3: dequantize_kernel<CURVEFP_E4C3><<<(unsigned)grid, 256, 0, st>>>(codes, scales, n, G, out); break;
    case CURVEFP_E5C2: dequantize_kernel<CURVEFP_E5C2><<<(unsigned)grid, 256, 0, st>>>(codes, scales, n, G, out); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace cfp
