// Decode-sized closed-product GEMM (M <= 8 activation rows) on the CUDA cores
// (Sec. 3.2, Eq. 2, Eq. 5).
//
// With a handful of activation rows the tensor-core kernel still pays for a
// full 128-row tile of plane-pair MMAs, so its time does not fall with M.
// Here every product is formed directly from the two codes, four at a time
// in byte lanes: phase h = (k_a W_A + k_b W_B) mod L, carry c, exponent
// e_a + e_b + c; the product 2^{e_a + e_b + c + a_a + a_b - ref} (+-) is an
// exact power of two that is added to the FP32 accumulator of phase h (the
// tensor-core kernel's accumulation semantics; ref = the output's largest
// scale sum, so the values stay in the FP32 normal range).  The phase
// combine C = 2^ref sum_h 2^{h/L} S_h runs in FP32 in phase order.
//
// A warp owns one weight row j (one output column) at a time: its lanes read
// 16 consecutive codes each (512 contiguous bytes per warp step), every lane
// keeps M x L accumulators in shared memory ([M L][threads], conflict-free;
// only the lane itself touches its slots), and the lane partials are summed
// by a fixed butterfly at the end.  The
// weight codes are read once; the activation rows stay in L1.
#include "cfp_common.cuh"
#include "kernels.cuh"

namespace cfp {

namespace {

constexpr int SKW = 8;  // warps per CTA
constexpr int SKM = 8;  // largest M

// 0xFF in every byte lane whose bit 7 is set
__device__ __forceinline__ uint32_t prmt_sign4(uint32_t v) {
  uint32_t r;
  asm("prmt.b32 %0, %1, 0, 0xBA98;" : "=r"(r) : "r"(v));
  return r;
}
// byte c of v in bits 24..31, zeros below
__device__ __forceinline__ uint32_t byte_to_top(uint32_t v, int c) {
  return __byte_perm(v, 0u, 0x0444u | (uint32_t)c << 12);
}

template <int FA, int FB, int MT>
__global__ void __launch_bounds__(SKW * 32) gemm_skinny_kernel(const uint8_t* __restrict__ A,
                                                               const int8_t* __restrict__ sA,
                                                               const uint8_t* __restrict__ B,
                                                               const int8_t* __restrict__ sB, int M, int N, int K,
                                                               int G, float* __restrict__ C) {
  using P = Pair<FA, FB>;
  using FAt = Fmt<FA>;
  using FBt = Fmt<FB>;
  constexpr int L = P::L, NT = SKW * 32;
  constexpr uint32_t R1 = 0x01010101u;
  constexpr uint32_t KMA = (uint32_t)(FAt::K - 1) * R1, KMB = (uint32_t)(FBt::K - 1) * R1;
  constexpr uint32_t EMA = ((1u << FAt::E) - 1u) * R1, EMB = ((1u << FBt::E) - 1u) * R1;
  constexpr uint32_t MMA = (uint32_t)FAt::MMASK * R1, MMB = (uint32_t)FBt::MMASK * R1;
  constexpr int EBIAS = (1 << (FAt::E - 1)) + (1 << (FBt::E - 1));  // of e_b,a + e_b,b
  extern __shared__ float sk_acc[];                                 // [M L][NT]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nb = K / G;
  const int gs = __ffs(G) - 1;  // G is a power of two

  for (int j = blockIdx.x * SKW + warp; j < N; j += gridDim.x * SKW) {
    // ref_i = max_b (a_i,b + b_j,b)
    int ref[MT];
#pragma unroll
    for (int i = 0; i < MT; ++i) {
      int r = -1024;
      if (i < M)
        for (int b = lane; b < nb; b += 32) r = max(r, (int)sA[(int64_t)i * nb + b] + (int)sB[(int64_t)j * nb + b]);
      ref[i] = __reduce_max_sync(0xffffffffu, r);
    }
    for (int q = 0; q < M * L; ++q) sk_acc[q * NT + tid] = 0.0f;

    const uint8_t* brow = B + (int64_t)j * K;
    uint4 wnext = lane * 16 < K ? __ldg(reinterpret_cast<const uint4*>(brow + lane * 16)) : make_uint4(0, 0, 0, 0);
    for (int k0 = lane * 16; k0 < K; k0 += 512) {
      const uint4 wv = wnext;  // the next step's codes are in flight while these are used
      if (k0 + 512 < K) wnext = __ldg(reinterpret_cast<const uint4*>(brow + k0 + 512));
      const int blk = k0 >> gs;  // G >= 32: the 16 codes share a block
      const int sb = (int)sB[(int64_t)j * nb + blk];
      const uint32_t w[4] = {wv.x, wv.y, wv.z, wv.w};
      uint32_t kb4[4], eb4[4], nzb[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        kb4[q] = (w[q] & KMB) * P::WB;
        eb4[q] = (w[q] >> FBt::C) & EMB;
        nzb[q] = ((w[q] & MMB) + 0x7F7F7F7Fu) & 0x80808080u;  // m != 0
      }
#pragma unroll
      for (int i = 0; i < MT; ++i) {
        if (i >= M) break;
        const uint4 av = __ldg(reinterpret_cast<const uint4*>(A + (int64_t)i * K + k0));
        const int k0f = (int)sA[(int64_t)i * nb + blk] + sb - ref[i] + 127 - EBIAS;  // FP32 exponent offset
        const uint32_t a[4] = {av.x, av.y, av.z, av.w};
        float* acc = sk_acc + (size_t)i * L * NT + tid;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          // byte lanes: u = k_a W_A + k_b W_B <= 2L - 2, x = e_a,b + e_b,b + carry <= 64
          const uint32_t u4 = (a[q] & KMA) * P::WA + kb4[q];
          const uint32_t h4 = u4 & ((uint32_t)(L - 1) * R1);
          const uint32_t x4 = ((a[q] >> FAt::C) & EMA) + eb4[q] + ((u4 >> P::LOG2L) & R1);
          const uint32_t nz = nzb[q] & (((a[q] & MMA) + 0x7F7F7F7Fu) & 0x80808080u);
          const uint32_t s4 = (a[q] ^ w[q]) & 0x80808080u;
          if (k0f >= 1 && k0f <= 191) {
            // common case: every FP32 exponent field x + k0f is in [1, 254], so
            // the fields form in byte lanes; zero products get field 0 (+-0.0)
            const uint32_t f4 = (x4 + (uint32_t)k0f * R1) & prmt_sign4(nz);
            // float bits of product c: byte 3 = sign | field >> 1 (from t4),
            // bit 23 = field & 1 (bit 7 of byte c of u4), nothing below
            const uint32_t t4 = ((f4 >> 1) & 0x7F7F7F7Fu) | s4;
            const uint32_t u4 = (f4 << 7) & 0x80808080u;
            const uint32_t hx4 = h4 << 2;  // phase x 4 per byte (<= 28)
            char* accb = reinterpret_cast<char*>(acc);
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              const uint32_t bits = __byte_perm(t4, u4, 0x0004u | (uint32_t)c << 12 | (uint32_t)(4 + c) << 8) & 0xFFFF0000u;
              // byte offset of slot h NT (NT = 256 floats): (4 h) << 8
              float* slot = reinterpret_cast<float*>(accb + __byte_perm(hx4, 0u, 0x4404u | (uint32_t)c << 4));
              *slot += __uint_as_float(bits);
            }
          } else {
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              const int field = (int)((x4 >> (8 * c)) & 0x7Fu) + k0f;
              if (((nz >> (8 * c)) & 0x80u) && field > 0) {
                const uint32_t bits = ((uint32_t)(field > 254 ? 254 : field) << 23) | (((s4 >> (8 * c)) & 0x80u) << 24);
                acc[((h4 >> (8 * c)) & 0xFFu) * NT] += __uint_as_float(bits);
              }
            }
          }
        }
      }
    }
    // lane partials -> phase sums (fixed butterfly), then the combine
#pragma unroll
    for (int i = 0; i < MT; ++i) {
      if (i >= M) break;
      float t = 0.0f;
      for (int h = 0; h < L; ++h) {
        float v = sk_acc[((size_t)i * L + h) * NT + tid];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        t = fmaf(__uint_as_float(L == 8 ? CFP_PHASE_F32_L8_DEV[h] : CFP_PHASE_F32_L4_DEV[h]), v, t);
      }
      if (lane == 0) C[(int64_t)i * N + j] = scalbnf(t, ref[i]);
    }
    __syncwarp();
  }
}

template <int FA, int FB, int MT>
cudaError_t launch_skinny_t(int G, const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb, int64_t M,
                            int64_t N, int64_t K, float* c, cudaStream_t s, int sms) {
  using P = Pair<FA, FB>;
  const size_t smem = (size_t)M * P::L * SKW * 32 * 4;
  auto kern = gemm_skinny_kernel<FA, FB, MT>;
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  const int64_t want = (N + SKW - 1) / SKW;
  const int64_t cap = (int64_t)sms * (smem <= 48 * 1024 ? 8 : 3);
  kern<<<(unsigned)(want < cap ? want : cap), SKW * 32, smem, s>>>(a, sa, b, sb, (int)M, (int)N, (int)K, G, c);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_skinny(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                               const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, cudaStream_t s, int sms) {
#define CFP_S(X, Y)                                                                            \
  if (fa == X && fb == Y) {                                                                    \
    if (M == 1) return launch_skinny_t<X, Y, 1>(G, a, sa, b, sb, M, N, K, c, s, sms);          \
    if (M == 2) return launch_skinny_t<X, Y, 2>(G, a, sa, b, sb, M, N, K, c, s, sms);          \
    if (M <= 4) return launch_skinny_t<X, Y, 4>(G, a, sa, b, sb, M, N, K, c, s, sms);          \
    return launch_skinny_t<X, Y, SKM>(G, a, sa, b, sb, M, N, K, c, s, sms);                    \
  }
  CFP_S(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_S(CURVEFP_E3C3, CURVEFP_E4C3)
  CFP_S(CURVEFP_E3C3, CURVEFP_E5C2)
  CFP_S(CURVEFP_E4C3, CURVEFP_E3C3)
  CFP_S(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_S(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_S(CURVEFP_E5C2, CURVEFP_E3C3)
  CFP_S(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_S(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_S
  return cudaErrorInvalidValue;
}

}  // namespace cfp
