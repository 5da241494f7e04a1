// Tensor-core closed-product GEMM (tcgen05, sm_103a): phase-plane
// decomposition with per-phase FP32 accumulation in TMEM and the phase
// combine fused into the epilogue (Sec. 3.2, Eq. 2, Eq. 5).
//
// Decomposition.  Write every decoded operand element as
//   x = 2^{k/K} * X_k,   X_k = +-2^{a_b - ref + e}  (an exact power of two),
// i.e. split each operand into K "curve planes" X_0..X_{K-1} that hold the
// element in the plane of its curve index k and zero elsewhere.  The product
// of plane k1 of A with plane k2 of B lands on the single phase
// h = (k1 WA + k2 WB) mod L with carry c = floor((k1 WA + k2 WB) / L)
// (Eq. 2 on the shared lattice), so
//   S_h = sum_{k1,k2 : phase h} 2^c  A_{k1} B_{k2}^T,
// a sum of dense products of power-of-two matrices: exactly what the tensor
// cores multiply without rounding.  Only the FP32 accumulation in TMEM rounds.
// Block scales enter the plane values as 2^{a_b - ref} (ref = largest block
// scale of the row) and 2^{ref_i + ref_j} is applied in the epilogue.
//
// Data flow per CTA (128 rows x NT columns of C, all L phases resident):
//   warps 0-3  load A codes, expand them into BF16 planes in registers and
//              store them straight into TMEM (tcgen05.st): A is the TMEM
//              operand of the MMA, so it costs no shared-memory bandwidth;
//              afterwards they run the epilogue (tcgen05.ld of the L phase
//              accumulators, C = 2^{ref_i+ref_j} sum_h 2^{h/L} S_h).
//   warps 4-7  load B codes and expand them into BF16 planes (and carry
//              copies x2) in shared memory, core-matrix K-major layout.
//   warp 8     allocates TMEM and issues tcgen05.mma (one thread) for every
//              plane pair into the accumulator of its phase.
// mbarriers hand stages between the roles; every wait is bounded.
#include "cfp_common.cuh"
#include "kernels.cuh"
#include "tc_ptx.cuh"

namespace cfp {

namespace {

template <int FA, int FB, int NT_>
struct TcCfg {
  using P = Pair<FA, FB>;
  static constexpr int KA = Fmt<FA>::K, KB = Fmt<FB>::K, L = P::L;
  static constexpr int NT = NT_;
  static constexpr int BM = 128;                       // rows per CTA (MMA M)
  static constexpr int KSTAGE = 32;                    // K per pipeline stage
  static constexpr int SUB = KSTAGE / 16;              // MMA K-steps per stage
  static constexpr int ACOLS = SUB * KA * 8;           // TMEM columns per A stage
  static constexpr int ACC_COLS = L * NT;              // TMEM columns of accumulators
  static constexpr int ACOL0 = ACC_COLS;               // first A column
  static constexpr int TMEM_COLS = 512;
  static_assert(ACC_COLS + 2 * ACOLS <= TMEM_COLS, "TMEM budget");
  static constexpr int PLANE_BYTES = NT * 32;          // NT rows x 16 BF16
  static constexpr int BSTAGE = SUB * 2 * KB * PLANE_BYTES;  // planes x {1, carry}
  static constexpr int NSB = 4;                        // B stages
  static constexpr int THREADS = 288;
  static constexpr uint32_t IDESC = tc::idesc_bf16_f32(BM, NT);
  static constexpr size_t SMEM = (size_t)NSB * BSTAGE + 1024 + 1024;
};

struct TcShared {
  uint64_t a_full[2], a_empty[2], b_full[8], b_empty[8], acc_full;
  uint32_t tmem_base;
  int abort_flag;
  int refB[64];
};

__device__ __forceinline__ void raise_flag(uint32_t* status, uint32_t bit) {
  if (status) atomicOr(status, bit);
}
__device__ __forceinline__ int read_abort(const int* f) { return *reinterpret_cast<const volatile int*>(f); }

// BF16 bits of +-2^{x} for a code (0 for the zero code or underflow).
template <int FMT>
__device__ __forceinline__ uint32_t plane_bf16(uint32_t code, int off, int& k) {
  using F = Fmt<FMT>;
  const int m = (int)(code & F::MMASK);
  const int n = m - F::B;
  k = n & (F::K - 1);
  const int ex = (n >> F::C) + off + 127;  // biased BF16 exponent
  return (m != 0 && ex >= 1) ? (((uint32_t)ex << 7) | ((code & 0x80u) << 8)) : 0u;
}

}  // namespace

template <int FA, int FB, int NT>
__global__ void __launch_bounds__(288, 1) gemm_tc_kernel(const uint8_t* __restrict__ A, const int8_t* __restrict__ sA,
                                                         const uint8_t* __restrict__ B, const int8_t* __restrict__ sB,
                                                         int M, int N, int K, int G, float* __restrict__ C,
                                                         uint32_t* status) {
  using Cfg = TcCfg<FA, FB, NT>;
  using P = typename Cfg::P;
  constexpr int KA = Cfg::KA, KB = Cfg::KB, L = Cfg::L;
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* bstage = smem;
  TcShared& sh = *reinterpret_cast<TcShared*>(smem + (size_t)Cfg::NSB * Cfg::BSTAGE);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.y * Cfg::BM, n0 = blockIdx.x * NT;
  const int nb = K / G, nkb = K / Cfg::KSTAGE;

  if (tid == 0) {
    for (int s = 0; s < 2; ++s) {
      tc::mbar_init(&sh.a_full[s], 128);
      tc::mbar_init(&sh.a_empty[s], 1);
    }
    for (int s = 0; s < Cfg::NSB; ++s) {
      tc::mbar_init(&sh.b_full[s], 128);
      tc::mbar_init(&sh.b_empty[s], 1);
    }
    tc::mbar_init(&sh.acc_full, 1);
    sh.abort_flag = 0;
  }
  if (warp == 8) {
    tc::tmem_alloc(&sh.tmem_base, Cfg::TMEM_COLS);
    tc::tmem_relinquish();
  }
  // per-row reference exponents (largest block scale of the row)
  int refA = 0;
  if (warp < 4) {
    const int r = m0 + tid;
    int mx = -128;
    if (r < M)
      for (int b = 0; b < nb; ++b) mx = max(mx, (int)sA[(int64_t)r * nb + b]);
    refA = mx;
  } else if (warp < 8 && tid - 128 < NT) {
    const int c = n0 + tid - 128;
    int mx = -128;
    if (c < N)
      for (int b = 0; b < nb; ++b) mx = max(mx, (int)sB[(int64_t)c * nb + b]);
    sh.refB[tid - 128] = mx;
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;

  if (warp < 4) {
    // ---------------- A producers: codes -> BF16 planes -> TMEM --------------
    const int r = m0 + tid;
    const bool rowok = r < M;
    const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
    auto load_a = [&](int kb, uint4 (&cv)[2], int& off) {
      cv[0] = make_uint4(0, 0, 0, 0);
      cv[1] = make_uint4(0, 0, 0, 0);
      off = 0;
      if (rowok && kb < nkb) {
        const uint4* src = reinterpret_cast<const uint4*>(A + (int64_t)r * K + (int64_t)kb * Cfg::KSTAGE);
        cv[0] = __ldg(src);
        cv[1] = __ldg(src + 1);
        off = (int)sA[(int64_t)r * nb + (kb * Cfg::KSTAGE) / G] - refA;
      }
    };
    uint4 nxt[2];
    int nxt_off;
    load_a(0, nxt, nxt_off);
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb & 1;
      uint4 cv[2] = {nxt[0], nxt[1]};
      const int off = nxt_off;
      load_a(kb + 1, nxt, nxt_off);  // prefetch the next stage
      bool fail = false;
      if (kb >= 2) {
        fail = !tc::mbar_wait(&sh.a_empty[s], ((kb >> 1) - 1) & 1);
        tc::fence_after_sync();
      }
      if (fail) {
        raise_flag(status, CURVEFP_DEV_TIMEOUT);
        sh.abort_flag = 1;
      }
      if (__any_sync(0xffffffffu, fail || read_abort(&sh.abort_flag))) break;
#pragma unroll
      for (int ss = 0; ss < Cfg::SUB; ++ss) {
        const uint4 w4 = cv[ss];
        const uint32_t w[4] = {w4.x, w4.y, w4.z, w4.w};
        uint32_t bf[16];
        int kk[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) bf[i] = plane_bf16<FA>((w[i >> 2] >> (8 * (i & 3))) & 0xFFu, off, kk[i]);
#pragma unroll
        for (int g = 0; g < KA / 4; ++g) {
          uint32_t reg[32];
#pragma unroll
          for (int pl = 0; pl < 4; ++pl) {
            const int kap = 4 * g + pl;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
              const uint32_t lo = kk[2 * c] == kap ? bf[2 * c] : 0u;
              const uint32_t hi = kk[2 * c + 1] == kap ? bf[2 * c + 1] : 0u;
              reg[pl * 8 + c] = lo | (hi << 16);
            }
          }
          const uint32_t col = Cfg::ACOL0 + s * Cfg::ACOLS + (ss * KA + 4 * g) * 8;
          tc::tmem_st32(lane_base + col, reg);
        }
      }
      tc::tmem_wait_st();
      tc::fence_before_sync();
      tc::mbar_arrive(&sh.a_full[s]);
    }
    // ---------------- epilogue -------------------------------------------------
    const bool ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.acc_full, 0));
    if (!ok) raise_flag(status, CURVEFP_DEV_TIMEOUT);
    tc::fence_after_sync();
    float cf[L];
#pragma unroll
    for (int h = 0; h < L; ++h) cf[h] = __uint_as_float(L == 8 ? CFP_PHASE_F32_L8_DEV[h] : CFP_PHASE_F32_L4_DEV[h]);
#pragma unroll 1
    for (int c0 = 0; c0 < NT; c0 += 8) {
      uint32_t acc[L][8];
#pragma unroll
      for (int h = 0; h < L; ++h) tc::tmem_ld8(lane_base + h * NT + c0, acc[h]);
      tc::tmem_wait_ld();
      if (rowok && ok) {
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const int col = n0 + c0 + c;
          if (col < N) {
            float y = 0.f;
#pragma unroll
            for (int h = 0; h < L; ++h) y = fmaf(cf[h], __uint_as_float(acc[h][c]), y);
            C[(int64_t)r * N + col] = scalbnf(y, refA + sh.refB[c0 + c]);
          }
        }
      }
    }
  } else if (warp < 8) {
    // ---------------- B producers: codes -> BF16 planes in shared memory ------
    const int t = tid - 128;
    constexpr int UPT = (NT * 4 + 127) / 128;  // units (row, 8-code chunk) per thread
    auto load_b = [&](int kb, uint2 (&cw)[UPT], int (&off)[UPT]) {
#pragma unroll
      for (int x = 0; x < UPT; ++x) {
        const int u = t + 128 * x;
        const int row = u >> 2, q = u & 3;
        const int c = n0 + row;
        cw[x] = make_uint2(0, 0);
        off[x] = 0;
        if (u < NT * 4 && c < N && kb < nkb) {
          cw[x] = __ldg(reinterpret_cast<const uint2*>(B + (int64_t)c * K + (int64_t)kb * Cfg::KSTAGE) + q);
          off[x] = (int)sB[(int64_t)c * nb + (kb * Cfg::KSTAGE) / G] - sh.refB[row];
        }
      }
    };
    uint2 nxt[UPT];
    int nxt_off[UPT];
    load_b(0, nxt, nxt_off);
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb % Cfg::NSB;
      uint2 cur[UPT];
      int cur_off[UPT];
#pragma unroll
      for (int x = 0; x < UPT; ++x) {
        cur[x] = nxt[x];
        cur_off[x] = nxt_off[x];
      }
      load_b(kb + 1, nxt, nxt_off);  // prefetch the next stage
      bool fail = false;
      if (kb >= Cfg::NSB) fail = !tc::mbar_wait(&sh.b_empty[s], ((kb / Cfg::NSB) - 1) & 1);
      if (fail) {
        raise_flag(status, CURVEFP_DEV_TIMEOUT);
        sh.abort_flag = 1;
      }
      if (fail || read_abort(&sh.abort_flag)) break;
      uint8_t* stage = bstage + (size_t)s * Cfg::BSTAGE;
#pragma unroll
      for (int x = 0; x < UPT; ++x) {
        const int u = t + 128 * x;
        if (u >= NT * 4) break;
        const int row = u >> 2, q = u & 3;
        const uint2 cw = cur[x];
        const int off = cur_off[x];
        uint32_t bf[8];
        int kk[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) bf[i] = plane_bf16<FB>(((i < 4 ? cw.x : cw.y) >> (8 * (i & 3))) & 0xFFu, off, kk[i]);
        const int ss = q >> 1, kc = q & 1;
        const uint32_t core = (uint32_t)((row >> 3) * 256 + kc * 128 + (row & 7) * 16);
#pragma unroll
        for (int carry = 0; carry < 2; ++carry)
#pragma unroll
          for (int kap = 0; kap < KB; ++kap) {
            uint32_t v[4];
#pragma unroll
            for (int wd = 0; wd < 4; ++wd) {
              uint32_t lo = kk[2 * wd] == kap ? bf[2 * wd] : 0u;
              uint32_t hi = kk[2 * wd + 1] == kap ? bf[2 * wd + 1] : 0u;
              if (carry) {
                lo = lo ? lo + (1u << 7) : 0u;
                hi = hi ? hi + (1u << 7) : 0u;
              }
              v[wd] = lo | (hi << 16);
            }
            const int plane = (ss * 2 + carry) * KB + kap;
            *reinterpret_cast<uint4*>(stage + (size_t)plane * Cfg::PLANE_BYTES + core) =
                make_uint4(v[0], v[1], v[2], v[3]);
          }
      }
      tc::fence_proxy_async_smem();
      tc::mbar_arrive(&sh.b_full[s]);
    }
  } else {
    // ---------------- MMA issuer --------------------------------------------
    if (lane == 0) {
      uint32_t inited = 0;
      uint64_t bdesc[Cfg::NSB];
#pragma unroll
      for (int s = 0; s < Cfg::NSB; ++s) bdesc[s] = tc::smem_desc(tc::smem_u32(bstage + (size_t)s * Cfg::BSTAGE), 128, 256);
      for (int kb = 0; kb < nkb; ++kb) {
        const int sa = kb & 1, sb = kb % Cfg::NSB;
        bool ok = tc::mbar_wait(&sh.a_full[sa], (kb >> 1) & 1);
        ok = ok && tc::mbar_wait(&sh.b_full[sb], (kb / Cfg::NSB) & 1);
        if (!ok || read_abort(&sh.abort_flag)) {
          raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
          break;
        }
        tc::fence_after_sync();
#pragma unroll
        for (int ss = 0; ss < Cfg::SUB; ++ss)
#pragma unroll
          for (int k1 = 0; k1 < KA; ++k1)
#pragma unroll
            for (int k2 = 0; k2 < KB; ++k2) {
              const int u = k1 * P::WA + k2 * P::WB;
              const int h = u & (L - 1), carry = u >> P::LOG2L;
              const uint32_t a_t = tmem + Cfg::ACOL0 + sa * Cfg::ACOLS + (ss * KA + k1) * 8;
              const uint64_t bd = bdesc[sb] + (uint64_t)((((ss * 2 + carry) * KB + k2) * Cfg::PLANE_BYTES) >> 4);
              const uint32_t accum = (inited >> h) & 1u;
              inited |= 1u << h;
              tc::mma_f16_ts(tmem + h * NT, a_t, bd, Cfg::IDESC, accum);
            }
        tc::mma_commit(&sh.a_empty[sa]);
        tc::mma_commit(&sh.b_empty[sb]);
      }
      tc::mma_commit(&sh.acc_full);
    }
    __syncwarp();
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == 8) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, Cfg::TMEM_COLS);
  }
}

template <int FA, int FB>
static cudaError_t launch_tc_t(int G, const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb,
                               int64_t M, int64_t N, int64_t K, float* c, uint32_t* st, cudaStream_t s) {
  constexpr int NT = 32;
  using Cfg = TcCfg<FA, FB, NT>;
  static_assert(sizeof(TcShared) <= 1024, "shared tail");
  static_assert(NT <= 64, "refB capacity");
  auto kern = gemm_tc_kernel<FA, FB, NT>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::SMEM);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((N + NT - 1) / NT), (unsigned)((M + Cfg::BM - 1) / Cfg::BM));
  kern<<<grid, Cfg::THREADS, Cfg::SMEM, s>>>(a, sa, b, sb, (int)M, (int)N, (int)K, G, c, st);
  return cudaGetLastError();
}

bool gemm_tensor_supported(int fa, int fb) {
  return (fa == CURVEFP_E3C3 && fb == CURVEFP_E3C3) || (fa == CURVEFP_E4C3 && fb == CURVEFP_E4C3) ||
         (fa == CURVEFP_E5C2 && fb == CURVEFP_E4C3) || (fa == CURVEFP_E4C3 && fb == CURVEFP_E5C2) ||
         (fa == CURVEFP_E5C2 && fb == CURVEFP_E5C2);
}

cudaError_t launch_gemm_tensor(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                               const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, uint32_t* status,
                               cudaStream_t s, int sms) {
  (void)sms;
#define CFP_T(X, Y) \
  if (fa == X && fb == Y) return launch_tc_t<X, Y>(G, a, sa, b, sb, M, N, K, c, status, s);
  CFP_T(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_T(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_T(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_T
  return cudaErrorInvalidValue;
}

}  // namespace cfp
