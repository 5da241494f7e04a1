// Host-side launchers of the CurveFP kernels (argument validation is done by
// the C ABI in capi.cu before any of these is called).
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace cfp {

cudaError_t launch_quantize(int fmt, int G, const void* x, int dtype, int64_t rows, int64_t cols, int64_t ld,
                            int axis, uint8_t* codes, int8_t* scales, uint32_t* status, cudaStream_t st, int sms);
size_t quantize_static_workspace(int64_t rows, int64_t cols, int G, int group);
cudaError_t launch_quantize_static(int fmt, int G, int group, int rule, const void* x, int dtype, int64_t rows,
                                   int64_t cols, uint8_t* codes, int8_t* scales, void* ws, uint32_t* status,
                                   cudaStream_t st, int sms);
cudaError_t launch_dequantize(int fmt, int G, const uint8_t* codes, const int8_t* scales, int64_t n, float* out,
                              cudaStream_t st, int sms);
cudaError_t launch_gemm_exact(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                              const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, int64_t* phase_sums,
                              int32_t* phase_lsb, uint32_t* status, cudaStream_t st);
cudaError_t launch_selftest_wait(int arrive, long long limit, uint32_t* status, cudaStream_t s);
cudaError_t launch_gemm_tensor(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                               const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, uint32_t* status,
                               cudaStream_t st, int sms);
bool gemm_tensor_supported(int fa, int fb);
bool gemm_narrow_supported(int fa, int fb);
cudaError_t launch_gemm_tensor_narrow(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                                      const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, uint32_t* status,
                                      cudaStream_t st, int sms);
cudaError_t launch_gemm_tensor_narrow_r34(int G, const uint8_t* x, const int8_t* sx, const uint8_t* w,
                                          const int8_t* sw, int64_t M, int64_t N, int64_t K, float* c,
                                          uint32_t* st, cudaStream_t s, int sms);
bool is_radix_format(int fmt);
cudaError_t launch_gemm_skinny(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                               const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, cudaStream_t st, int sms);
cudaError_t launch_gemm_hist(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                             const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, int64_t* phase_sums,
                             int32_t* phase_lsb, uint32_t* status, cudaStream_t st, int sms);
cudaError_t launch_quantize_radix(int fmt, int G, const void* x, int dtype, int64_t rows, int64_t cols, int64_t ld,
                                  int axis, uint8_t* codes, int8_t* scales, uint32_t* status, cudaStream_t st,
                                  int sms);
cudaError_t launch_quantize_static_radix(int fmt, int G, int group, int rule, const void* x, int dtype, int64_t rows,
                                         int64_t cols, uint8_t* codes, int8_t* scales, void* ws, uint32_t* status,
                                         cudaStream_t st, int sms);
cudaError_t launch_dequantize_radix(int fmt, int G, const uint8_t* codes, const int8_t* scales, int64_t n, float* out,
                                    cudaStream_t st, int sms);
cudaError_t launch_gemm_exact_oriented(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, int la,
                                       const uint8_t* b, const int8_t* sb, int lb, int64_t M, int64_t N, int64_t K,
                                       float* c, int64_t* phase_sums, int32_t* phase_lsb, uint32_t* status,
                                       cudaStream_t st);
size_t gemm_reuse_workspace(int la, int lb, int64_t M, int64_t N, int64_t K);
cudaError_t launch_gemm_tensor_reuse(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, int la,
                                     const uint8_t* b, const int8_t* sb, int lb, int64_t M, int64_t N, int64_t K,
                                     float* c, void* ws, uint32_t* status, cudaStream_t st, int sms);
cudaError_t launch_gemm_q32(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                            const int8_t* sb, int64_t M, int64_t N, int64_t K, int64_t* out, uint32_t* status,
                            cudaStream_t s);

}  // namespace cfp
