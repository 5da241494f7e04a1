// Launchers of the tensor-core GEMM (kernel in gemm_tc.cuh) for operands with
// block scales along K.
#include "gemm_tc.cuh"

namespace cfp {

bool gemm_tensor_supported(int fa, int fb) {
  return (fa == CURVEFP_E3C3 && fb == CURVEFP_E3C3) || (fa == CURVEFP_E4C3 && fb == CURVEFP_E4C3) ||
         (fa == CURVEFP_E5C2 && fb == CURVEFP_E4C3) || (fa == CURVEFP_E4C3 && fb == CURVEFP_E5C2) ||
         (fa == CURVEFP_E5C2 && fb == CURVEFP_E5C2) || (fa == CURVEFP_E4C3_R8_9 && fb == CURVEFP_E4C3_R8_9);
}

cudaError_t launch_gemm_tensor(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                               const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, uint32_t* status,
                               cudaStream_t s, int sms) {
#define CFP_T(X, Y) \
  if (fa == X && fb == Y) return launch_tc_t<X, Y, false>(G, a, sa, b, sb, M, N, K, c, status, s, PesOperands{}, sms);
  CFP_T(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_T(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_T(CURVEFP_E5C2, CURVEFP_E5C2)
  CFP_T(CURVEFP_E4C3_R8_9, CURVEFP_E4C3_R8_9)
#undef CFP_T
  return cudaErrorInvalidValue;
}

namespace {

// Failure-detection self-test of the pipeline's bounded wait (no CurveFP
// arithmetic): one warp waits on a fresh barrier of count 1, which lane 0
// completes first only when `arrive` is set.  A wait that gives up raises
// TIMEOUT and the kernel returns as the GEMM's roles do.
__global__ void __launch_bounds__(32) selftest_wait_kernel(int arrive, long long limit, uint32_t* status) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) tc::mbar_init(&bar, 1);
  __syncthreads();
  if (arrive && threadIdx.x == 0) tc::mbar_arrive(&bar);
  __syncwarp();
  const bool ok = __all_sync(0xffffffffu, tc::mbar_wait(&bar, 0, limit));
  if (!ok && threadIdx.x == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
}

}  // namespace

cudaError_t launch_selftest_wait(int arrive, long long limit, uint32_t* status, cudaStream_t s) {
  selftest_wait_kernel<<<1, 32, 0, s>>>(arrive, limit, status);
  return cudaGetLastError();
}

}  // namespace cfp
