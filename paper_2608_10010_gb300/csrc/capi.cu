// C ABI of libcurvefp: argument validation, then one asynchronous launch on
// the caller's stream.  Declarations and the full contract are in
// include/curvefp.h.  No device memory is allocated here and nothing
// synchronizes.
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/curvefp.h"
#include "kernels.cuh"

namespace {

bool fmt_ok(int f) { return f == CURVEFP_E3C3 || f == CURVEFP_E4C3 || f == CURVEFP_E5C2; }  // binary radix
bool fmt_radix(int f) { return f == CURVEFP_E4C3_R8_9 || f == CURVEFP_E4C3_R3_4; }      // rational radix
bool fmt_any(int f) { return fmt_ok(f) || fmt_radix(f); }
bool block_ok(int g) { return g == 32 || g == 64 || g == 128 || g == 256 || g == 512; }
bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
int fmt_k(int f) { return f == CURVEFP_E5C2 ? 4 : 8; }

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 148;
  return n;
}

curvefp_status_t from_cuda(cudaError_t e) { return e == cudaSuccess ? CURVEFP_OK : CURVEFP_ERR_CUDA; }

}  // namespace

extern "C" {

curvefp_status_t curvefp_quantize(curvefp_format_t fmt, int block, const void* x, curvefp_dtype_t dtype,
                                  int64_t rows, int64_t cols, int64_t ld, int block_axis, uint8_t* codes,
                                  int8_t* scales, uint32_t* device_status, void* stream) {
  if (!fmt_any(fmt) || !block_ok(block) || (dtype != CURVEFP_F32 && dtype != CURVEFP_BF16)) return CURVEFP_ERR_INVALID_ARG;
  if (block_axis != 0 && block_axis != 1) return CURVEFP_ERR_INVALID_ARG;
  if (rows < 0 || cols < 0 || ld < cols) return CURVEFP_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return CURVEFP_OK;
  if (!x || !codes || !scales) return CURVEFP_ERR_INVALID_ARG;
  const int64_t esz = dtype == CURVEFP_F32 ? 4 : 2;
  if (!al16(codes) || (reinterpret_cast<uintptr_t>(x) % esz) != 0) return CURVEFP_ERR_INVALID_ARG;
  // the row-blocked kernel reads 16-byte vectors; the column-blocked one reads elements
  if (block_axis == 0 && (!al16(x) || (ld * esz) % 16 != 0)) return CURVEFP_ERR_INVALID_ARG;
  if (block_axis == 0 && cols % block != 0) return CURVEFP_ERR_INVALID_ARG;
  if (block_axis == 1 && rows % block != 0) return CURVEFP_ERR_INVALID_ARG;
  if (block_axis == 1 && rows / block > 65535) return CURVEFP_ERR_UNSUPPORTED;
  if (rows * cols / block > (int64_t)1 << 40) return CURVEFP_ERR_UNSUPPORTED;
  if (fmt_radix(fmt))
    return from_cuda(cfp::launch_quantize_radix(fmt, block, x, dtype, rows, cols, ld, block_axis, codes, scales,
                                                device_status, static_cast<cudaStream_t>(stream), sm_count()));
  return from_cuda(cfp::launch_quantize(fmt, block, x, dtype, rows, cols, ld, block_axis, codes, scales,
                                        device_status, static_cast<cudaStream_t>(stream), sm_count()));
}

size_t curvefp_quantize_static_workspace(int64_t rows, int64_t cols, int block, curvefp_scale_group_t group) {
  if (rows <= 0 || cols <= 0 || !block_ok(block) || group < CURVEFP_SCALE_BLOCK || group > CURVEFP_SCALE_TENSOR) return 0;
  return cfp::quantize_static_workspace(rows, cols, block, group);
}

curvefp_status_t curvefp_quantize_static(curvefp_format_t fmt, int block, curvefp_scale_group_t group,
                                         curvefp_scale_rule_t rule, const void* x, curvefp_dtype_t dtype, int64_t rows,
                                         int64_t cols, uint8_t* codes, int8_t* scales, void* workspace,
                                         size_t workspace_bytes, uint32_t* device_status, void* stream) {
  if (!fmt_any(fmt) || !block_ok(block) || (dtype != CURVEFP_F32 && dtype != CURVEFP_BF16)) return CURVEFP_ERR_INVALID_ARG;
  if (group < CURVEFP_SCALE_BLOCK || group > CURVEFP_SCALE_TENSOR) return CURVEFP_ERR_INVALID_ARG;
  if (rule != CURVEFP_SCALE_CEIL_ABSMAX && rule != CURVEFP_SCALE_MSE) return CURVEFP_ERR_INVALID_ARG;
  if (rows < 0 || cols < 0) return CURVEFP_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return CURVEFP_OK;
  if (!x || !codes || !scales || cols % block != 0) return CURVEFP_ERR_INVALID_ARG;
  const int64_t esz = dtype == CURVEFP_F32 ? 4 : 2;
  if ((reinterpret_cast<uintptr_t>(x) % esz) != 0) return CURVEFP_ERR_INVALID_ARG;
  const size_t need = cfp::quantize_static_workspace(rows, cols, block, group);
  if (need && (!workspace || workspace_bytes < need || (reinterpret_cast<uintptr_t>(workspace) & 15) != 0))
    return CURVEFP_ERR_INVALID_ARG;
  if (rows * cols > (int64_t)1 << 40) return CURVEFP_ERR_UNSUPPORTED;
  // block groups with the ceil-absmax rule are the quantizer itself (R11):
  // the streaming kernels where their alignment rules hold
  if (group == CURVEFP_SCALE_BLOCK && rule == CURVEFP_SCALE_CEIL_ABSMAX && al16(x) && al16(codes) &&
      (cols * esz) % 16 == 0)
    return curvefp_quantize(fmt, block, x, dtype, rows, cols, cols, 0, codes, scales, device_status, stream);
  if (fmt_radix(fmt))
    return from_cuda(cfp::launch_quantize_static_radix(fmt, block, group, rule, x, dtype, rows, cols, codes, scales,
                                                       workspace, device_status, static_cast<cudaStream_t>(stream),
                                                       sm_count()));
  return from_cuda(cfp::launch_quantize_static(fmt, block, group, rule, x, dtype, rows, cols, codes, scales, workspace,
                                               device_status, static_cast<cudaStream_t>(stream), sm_count()));
}

/* Scratch for curvefp_quantize_static_noalloc, the entry point for callers
 * that cannot allocate device memory: a file-scope device array (reserved on
 * each GPU when the library's module loads, held until exit, never allocated
 * by a call).  In host code its name is only a host-side stand-in; kernels
 * get the device address from cudaGetSymbolAddress. */
static __device__ __align__(256) unsigned char g_static_scratch[CURVEFP_NOALLOC_SCRATCH_BYTES];

curvefp_status_t curvefp_quantize_static_noalloc(curvefp_format_t fmt, int block, curvefp_scale_group_t group,
                                                 curvefp_scale_rule_t rule, const void* x, curvefp_dtype_t dtype,
                                                 int64_t rows, int64_t cols, uint8_t* codes, int8_t* scales,
                                                 uint32_t* device_status, void* stream) {
  if (rows < 0 || cols < 0) return CURVEFP_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return CURVEFP_OK;
  if (!block_ok(block) || group < CURVEFP_SCALE_BLOCK || group > CURVEFP_SCALE_TENSOR) return CURVEFP_ERR_INVALID_ARG;
  const size_t need = cfp::quantize_static_workspace(rows, cols, block, group);
  if (need > CURVEFP_NOALLOC_SCRATCH_BYTES) return CURVEFP_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  // the current device's copy of the array, looked up on every call (nothing
  // cached: an address kept from before a device reset would be stale, and
  // concurrent callers share no host state)
  if (need && cudaGetSymbolAddress(&scratch, g_static_scratch) != cudaSuccess) return CURVEFP_ERR_CUDA;
  return curvefp_quantize_static(fmt, block, group, rule, x, dtype, rows, cols, codes, scales, scratch, need,
                                 device_status, stream);
}

curvefp_status_t curvefp_dequantize(curvefp_format_t fmt, int block, const uint8_t* codes, const int8_t* scales,
                                    int64_t rows, int64_t cols, float* out, void* stream) {
  if (!fmt_any(fmt) || !block_ok(block) || rows < 0 || cols < 0) return CURVEFP_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return CURVEFP_OK;
  if (!codes || !scales || !out || cols % block != 0 || !al16(codes) || !al16(out)) return CURVEFP_ERR_INVALID_ARG;
  if (fmt_radix(fmt))
    return from_cuda(cfp::launch_dequantize_radix(fmt, block, codes, scales, rows * cols, out,
                                                  static_cast<cudaStream_t>(stream), sm_count()));
  return from_cuda(cfp::launch_dequantize(fmt, block, codes, scales, rows * cols, out,
                                          static_cast<cudaStream_t>(stream), sm_count()));
}

static curvefp_status_t gemm_args(int fa, int fb, int block, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                                  const int8_t* sb, int64_t M, int64_t N, int64_t K) {
  if (!fmt_any(fa) || !fmt_any(fb) || !block_ok(block)) return CURVEFP_ERR_INVALID_ARG;
  if (M <= 0 || N <= 0 || K <= 0 || K % block != 0) return CURVEFP_ERR_INVALID_ARG;
  // a rational radix pairs only with itself (one lattice, App. A.1)
  if ((fmt_radix(fa) || fmt_radix(fb)) && fa != fb) return CURVEFP_ERR_UNSUPPORTED;
  if (!a || !sa || !b || !sb || !al16(a) || !al16(b)) return CURVEFP_ERR_INVALID_ARG;
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return CURVEFP_ERR_UNSUPPORTED;
  return CURVEFP_OK;
}

curvefp_status_t curvefp_gemm(curvefp_gemm_algo_t algo, curvefp_format_t fmt_a, curvefp_format_t fmt_b, int block,
                              const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb, int64_t M,
                              int64_t N, int64_t K, float* c, uint32_t* device_status, void* stream) {
  curvefp_status_t r = gemm_args(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K);
  if (r != CURVEFP_OK) return r;
  if (!c) return CURVEFP_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (algo == CURVEFP_GEMM_EXACT)
    return from_cuda(cfp::launch_gemm_exact(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K, c, nullptr, nullptr,
                                            device_status, st));
  // rational radix: EXACT, TENSOR for r = 2^{8/9}, TENSOR_NARROW for
  // r = 2^{3/4}; AUTO picks the tensor-core kernel of the format
  if (fmt_radix(fmt_a) && algo == CURVEFP_GEMM_AUTO)
    algo = fmt_a == CURVEFP_E4C3_R3_4 ? CURVEFP_GEMM_TENSOR_NARROW : CURVEFP_GEMM_TENSOR;
  if (fmt_radix(fmt_a) && algo != CURVEFP_GEMM_TENSOR && algo != CURVEFP_GEMM_TENSOR_NARROW)
    return CURVEFP_ERR_UNSUPPORTED;
  // AUTO: the fastest kernel by M (measured on the FFN and Llama-like
  // shapes and the training triplet): CUDA cores for one row; phases along N
  // (2:4-sparse pair planes) for every larger M of the pairs that kernel
  // takes; tiles for the rest
  if (algo == CURVEFP_GEMM_AUTO) {
    if (M <= CURVEFP_AUTO_SKINNY_M)
      algo = CURVEFP_GEMM_SKINNY;
    else if (cfp::gemm_narrow_supported(fmt_a, fmt_b))
      algo = CURVEFP_GEMM_TENSOR_NARROW;
    else if (M <= CURVEFP_SKINNY_MAX_M && !cfp::gemm_tensor_supported(fmt_a, fmt_b))
      algo = CURVEFP_GEMM_SKINNY;
    else
      algo = CURVEFP_GEMM_TENSOR;
  }
  if (algo == CURVEFP_GEMM_SKINNY) {
    if (M > CURVEFP_SKINNY_MAX_M) return CURVEFP_ERR_UNSUPPORTED;
    return from_cuda(cfp::launch_gemm_skinny(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K, c, st, sm_count()));
  }
  if (algo == CURVEFP_GEMM_TENSOR_NARROW) {
    if (!cfp::gemm_narrow_supported(fmt_a, fmt_b)) return CURVEFP_ERR_UNSUPPORTED;
    return from_cuda(cfp::launch_gemm_tensor_narrow(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K, c, device_status, st,
                                                    sm_count()));
  }
  if (algo == CURVEFP_GEMM_TENSOR) {
    if (!cfp::gemm_tensor_supported(fmt_a, fmt_b)) return CURVEFP_ERR_UNSUPPORTED;
    return from_cuda(cfp::launch_gemm_tensor(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K, c, device_status, st,
                                             sm_count()));
  }
  return CURVEFP_ERR_INVALID_ARG;
}

curvefp_status_t curvefp_gemm_phases(curvefp_format_t fmt_a, curvefp_format_t fmt_b, int block, const uint8_t* a,
                                     const int8_t* sa, const uint8_t* b, const int8_t* sb, int64_t M, int64_t N,
                                     int64_t K, float* c, int64_t* phase_sums, int32_t* phase_lsb,
                                     uint32_t* device_status, void* stream) {
  curvefp_status_t r = gemm_args(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K);
  if (r != CURVEFP_OK) return r;
  if (!phase_sums || !phase_lsb) return CURVEFP_ERR_INVALID_ARG;
  return from_cuda(cfp::launch_gemm_exact(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K, c, phase_sums, phase_lsb,
                                          device_status, static_cast<cudaStream_t>(stream)));
}

static bool layout_ok(int l) { return l == CURVEFP_LAYOUT_ROWS || l == CURVEFP_LAYOUT_COLS; }

static curvefp_status_t oriented_args(int fa, int fb, int block, const uint8_t* a, const int8_t* sa, int la,
                                      const uint8_t* b, const int8_t* sb, int lb, int64_t M, int64_t N, int64_t K) {
  if (fmt_radix(fa) || fmt_radix(fb)) return CURVEFP_ERR_UNSUPPORTED;
  if (!fmt_ok(fa) || !fmt_ok(fb) || !block_ok(block) || !layout_ok(la) || !layout_ok(lb))
    return CURVEFP_ERR_INVALID_ARG;
  if (M <= 0 || N <= 0 || K <= 0) return CURVEFP_ERR_INVALID_ARG;
  // the blocked extent of each operand: K for ROWS, its own row count for COLS
  if ((la == CURVEFP_LAYOUT_ROWS ? K : M) % block != 0 || (lb == CURVEFP_LAYOUT_ROWS ? K : N) % block != 0)
    return CURVEFP_ERR_INVALID_ARG;
  if (!a || !sa || !b || !sb || !al16(a) || !al16(b)) return CURVEFP_ERR_INVALID_ARG;
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return CURVEFP_ERR_UNSUPPORTED;
  return CURVEFP_OK;
}

size_t curvefp_gemm_oriented_workspace_bytes(curvefp_gemm_algo_t algo, curvefp_layout_t layout_a,
                                             curvefp_layout_t layout_b, int64_t M, int64_t N, int64_t K) {
  if (algo != CURVEFP_GEMM_TENSOR || !layout_ok(layout_a) || !layout_ok(layout_b) || M <= 0 || N <= 0 || K <= 0)
    return 0;
  return cfp::gemm_reuse_workspace(layout_a, layout_b, M, N, K);
}

curvefp_status_t curvefp_gemm_oriented(curvefp_gemm_algo_t algo, curvefp_format_t fmt_a, curvefp_format_t fmt_b,
                                       int block, const uint8_t* a, const int8_t* sa, curvefp_layout_t layout_a,
                                       const uint8_t* b, const int8_t* sb, curvefp_layout_t layout_b, int64_t M,
                                       int64_t N, int64_t K, float* c, int64_t* phase_sums, int32_t* phase_lsb,
                                       void* workspace, size_t workspace_bytes, uint32_t* device_status,
                                       void* stream) {
  curvefp_status_t r = oriented_args(fmt_a, fmt_b, block, a, sa, layout_a, b, sb, layout_b, M, N, K);
  if (r != CURVEFP_OK) return r;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (algo == CURVEFP_GEMM_EXACT) {
    if (!c && !phase_sums) return CURVEFP_ERR_INVALID_ARG;
    if (!phase_sums != !phase_lsb) return CURVEFP_ERR_INVALID_ARG;
    return from_cuda(cfp::launch_gemm_exact_oriented(fmt_a, fmt_b, block, a, sa, layout_a, b, sb, layout_b, M, N, K,
                                                     c, phase_sums, phase_lsb, device_status, st));
  }
  if (phase_sums || phase_lsb || !c) return CURVEFP_ERR_INVALID_ARG;
  if (layout_a == CURVEFP_LAYOUT_ROWS && layout_b == CURVEFP_LAYOUT_ROWS)
    return curvefp_gemm(algo, fmt_a, fmt_b, block, a, sa, b, sb, M, N, K, c, device_status, stream);
  if (algo != CURVEFP_GEMM_TENSOR) return CURVEFP_ERR_INVALID_ARG;
  if (!cfp::gemm_tensor_supported(fmt_a, fmt_b)) return CURVEFP_ERR_UNSUPPORTED;
  if (K % 32 != 0) return CURVEFP_ERR_INVALID_ARG;
  const size_t need = cfp::gemm_reuse_workspace(layout_a, layout_b, M, N, K);
  if (!workspace || workspace_bytes < need || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return CURVEFP_ERR_INVALID_ARG;
  return from_cuda(cfp::launch_gemm_tensor_reuse(fmt_a, fmt_b, block, a, sa, layout_a, b, sb, layout_b, M, N, K, c,
                                                 workspace, device_status, st, sm_count()));
}

curvefp_status_t curvefp_gemm_phases_histogram(curvefp_format_t fmt_a, curvefp_format_t fmt_b, int block,
                                               const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb,
                                               int64_t M, int64_t N, int64_t K, float* c, int64_t* phase_sums,
                                               int32_t* phase_lsb, uint32_t* device_status, void* stream) {
  curvefp_status_t r = gemm_args(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K);
  if (r != CURVEFP_OK) return r;
  if (!phase_sums || !phase_lsb) return CURVEFP_ERR_INVALID_ARG;
  return from_cuda(cfp::launch_gemm_hist(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K, c, phase_sums, phase_lsb,
                                         device_status, static_cast<cudaStream_t>(stream), sm_count()));
}

curvefp_status_t curvefp_gemm_requant(curvefp_gemm_algo_t algo, curvefp_format_t fmt_a, curvefp_format_t fmt_b,
                                      int block, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                                      const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c,
                                      curvefp_format_t fmt_c, int block_c, uint8_t* codes_c, int8_t* scales_c,
                                      uint32_t* device_status, void* stream) {
  if (!fmt_any(fmt_c) || !block_ok(block_c) || N % block_c != 0 || !c || !codes_c || !scales_c || !al16(c))
    return CURVEFP_ERR_INVALID_ARG;
  curvefp_status_t r = curvefp_gemm(algo, fmt_a, fmt_b, block, a, sa, b, sb, M, N, K, c, device_status, stream);
  if (r != CURVEFP_OK) return r;
  return curvefp_quantize(fmt_c, block_c, c, CURVEFP_F32, M, N, N, 0, codes_c, scales_c, device_status, stream);
}

curvefp_status_t curvefp_gemm_q32(curvefp_format_t fmt_a, curvefp_format_t fmt_b, int block, const uint8_t* a,
                                  const int8_t* sa, const uint8_t* b, const int8_t* sb, int64_t M, int64_t N, int64_t K,
                                  int64_t* acc, uint32_t* device_status, void* stream) {
  curvefp_status_t r = gemm_args(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K);
  if (r != CURVEFP_OK) return r;
  if (!acc) return CURVEFP_ERR_INVALID_ARG;
  if (fmt_radix(fmt_a) || !cfp::gemm_tensor_supported(fmt_a, fmt_b)) return CURVEFP_ERR_UNSUPPORTED;  // same format pairs
  if ((M + 15) / 16 > 65535) return CURVEFP_ERR_UNSUPPORTED;
  return from_cuda(cfp::launch_gemm_q32(fmt_a, fmt_b, block, a, sa, b, sb, M, N, K, acc, device_status,
                                        static_cast<cudaStream_t>(stream)));
}

int curvefp_phase_count(curvefp_format_t fmt_a, curvefp_format_t fmt_b) {
  if (fmt_radix(fmt_a) || fmt_radix(fmt_b)) {
    if (fmt_a != fmt_b) return -1;
    return fmt_a == CURVEFP_E4C3_R8_9 ? 9 : 32;  // Eq. 4: H = 8q / gcd(p, 8q)
  }
  if (!fmt_ok(fmt_a) || !fmt_ok(fmt_b)) return -1;
  const int ka = fmt_k(fmt_a), kb = fmt_k(fmt_b);
  return ka > kb ? ka : kb;
}

curvefp_status_t curvefp_selftest_bounded_wait(int arrive, int64_t limit_cycles, uint32_t* device_status,
                                               void* stream) {
  if (!device_status || limit_cycles < 1 || limit_cycles > (int64_t(1) << 31)) return CURVEFP_ERR_INVALID_ARG;
  return from_cuda(cfp::launch_selftest_wait(arrive != 0, (long long)limit_cycles, device_status,
                                             static_cast<cudaStream_t>(stream)));
}

const char* curvefp_status_string(curvefp_status_t s) {
  switch (s) {
    case CURVEFP_OK: return "ok";
    case CURVEFP_ERR_INVALID_ARG: return "invalid argument";
    case CURVEFP_ERR_UNSUPPORTED: return "unsupported configuration";
    case CURVEFP_ERR_CUDA: return "CUDA launch error";
  }
  return "unknown status";
}

const char* curvefp_version(void) { return "curvefp-gb300 0.1 (sm_103a)"; }

}  // extern "C"
