// Tensor-core closed-product GEMM (tcgen05, sm_103a): phase-plane
// decomposition with per-phase FP32 accumulation in TMEM and the phase
// combine fused into the epilogue (Sec. 3.2, Eq. 2, Eq. 5).
//
// Decomposition.  Write every decoded operand element as
//   x = 2^{k/K} * X_k,   X_k = +-2^{a_b - ref + e}  (an exact power of two),
// i.e. split each operand into K "curve planes" that hold the element in the
// plane of its curve index k and zero elsewhere.  Plane k1 of A times plane k2
// of B lands on the single phase h = (k1 WA + k2 WB) mod L with carry
// c = floor((k1 WA + k2 WB) / L) (Eq. 2 on the shared lattice L), so
//   S_h = sum_{k1,k2 : phase h} 2^c  A_{k1} B_{k2}^T,
// a sum of dense products of power-of-two matrices, which the tensor cores
// multiply without rounding; only the FP32 accumulation in TMEM rounds.  Block
// scales enter the plane values as 2^{a_b - ref} (ref = largest block scale of
// the row) and 2^{ref_i + ref_j} is applied in the epilogue.  Plane values are
// BF16 or FP8 E5M2 (every power of two in [2^-16, 2^15] is exact in E5M2; E5C2
// planes are stored one binade low so that the carry still fits).
//
// Shape.  A CTA owns a 128 x 128 tile of C.  tcgen05.mma runs at full rate
// only for N >= 128, and TMEM (512 columns) holds three 128-column phase
// accumulators plus two A stages, so the L phases are processed in passes of
// PP = 3 phases over the whole K; each pass adds its part of
// sum_h 2^{h/L} S_h into C.
//
// Roles (288 threads):
//   warps 0-3  A producers: codes -> planes in registers -> TMEM (tcgen05.st);
//              A is the TMEM operand of the MMA and costs no shared-memory
//              bandwidth.  At the end of each pass they run the epilogue.
//   warps 4-7  B producers: codes -> the planes (and x2 carry planes) that the
//              current pass needs -> shared memory, K-major core-matrix layout.
//   warp 8     TMEM allocation and the single MMA-issuing thread.
// mbarriers hand stages between the roles; every wait is bounded.
#include "cfp_common.cuh"
#include "kernels.cuh"
#include "tc_ptx.cuh"

#ifndef CFP_TC_PLANE
#define CFP_TC_PLANE 1  // 0: BF16 planes (K = 16 per MMA), 1: E5M2 planes (K = 32 per MMA)
#endif

namespace cfp {

namespace {

enum PlaneType { PLANE_BF16 = 0, PLANE_E5M2 = 1 };

template <int FA, int FB, int PT>
struct TcCfg {
  using P = Pair<FA, FB>;
  static constexpr int KA = Fmt<FA>::K, KB = Fmt<FB>::K, L = P::L, WA = P::WA, WB = P::WB, LOG2L = P::LOG2L;
  static constexpr int FA_ = FA, FB_ = FB;
  static constexpr int BM = 128, BN = 128;
  static constexpr int KS = PT == PLANE_BF16 ? 16 : 32;  // K per MMA = K per pipeline step (32 bytes per row)
  static constexpr int PP = 3;                            // phases per pass
  static constexpr int NP = (L + PP - 1) / PP;            // passes
  static constexpr int ACC_COLS = PP * BN;
  static constexpr int ACOLS = KA * 8;                    // TMEM columns of one A step (8 per plane)
  static constexpr int ACOL0 = ACC_COLS;
  static_assert(ACC_COLS + 2 * ACOLS <= 512, "TMEM budget");
  static constexpr int PLANE_BYTES = BN * 32;             // 128 rows x 32 bytes
  static constexpr int NSB = 4;                           // B stages
  static constexpr int PBA = FA == CURVEFP_E5C2 ? 1 : 0;  // plane exponent bias
  static constexpr int PBB = FB == CURVEFP_E5C2 ? 1 : 0;
  static constexpr int THREADS = 288;
  // D = F32, A = B = BF16 (kind::f16) or E5M2 (kind::f8f6f4): same bit pattern
  static constexpr uint32_t IDESC = tc::idesc_bf16_f32(BM, BN);

  __host__ __device__ static constexpr int phase(int k1, int k2) { return (k1 * WA + k2 * WB) & (L - 1); }
  __host__ __device__ static constexpr int carry(int k1, int k2) { return (k1 * WA + k2 * WB) >> LOG2L; }
  // Does pass p need B plane (k2, c)?
  __host__ __device__ static constexpr bool needed(int p, int c, int k2) {
    for (int k1 = 0; k1 < KA; ++k1)
      if (carry(k1, k2) == c && phase(k1, k2) / PP == p) return true;
    return false;
  }
  // Shared-memory slot of B plane (k2, c) in pass p (-1 if unused).
  __host__ __device__ static constexpr int slot(int p, int c, int k2) {
    int s = 0;
    for (int cc = 0; cc < 2; ++cc)
      for (int k = 0; k < KB; ++k) {
        const bool need = needed(p, cc, k);
        if (cc == c && k == k2) return need ? s : -1;
        if (need) ++s;
      }
    return -1;
  }
  __host__ __device__ static constexpr int nslots(int p) {
    int s = 0;
    for (int cc = 0; cc < 2; ++cc)
      for (int k = 0; k < KB; ++k) s += needed(p, cc, k) ? 1 : 0;
    return s;
  }
  __host__ __device__ static constexpr int maxslots() {
    int m = 0;
    for (int p = 0; p < NP; ++p) m = nslots(p) > m ? nslots(p) : m;
    return m;
  }
  // Is (k1, k2) the first pair of the issue order that lands on its phase?
  __host__ __device__ static constexpr bool first_of_phase(int k1, int k2) {
    for (int a = 0; a < KA; ++a)
      for (int b = 0; b < KB; ++b)
        if (phase(a, b) == phase(k1, k2)) return a == k1 && b == k2;
    return false;
  }
  static constexpr int MAXS = maxslots();
  static constexpr int BSTAGE = MAXS * PLANE_BYTES;
  static constexpr size_t SMEM = (size_t)NSB * BSTAGE + 2048;
};

struct TcShared {
  uint64_t a_full[2], a_empty[2], b_full[4], b_empty[4], acc_full, drain;
  uint32_t tmem_base;
  int abort_flag;
  int refB[128];
};

__device__ __forceinline__ void raise_flag(uint32_t* status, uint32_t bit) {
  if (status) atomicOr(status, bit);
}
__device__ __forceinline__ int read_abort(const int* f) { return *reinterpret_cast<const volatile int*>(f); }

// ---------------------------------------------------------------------------
// Producer arithmetic, four codes per 32-bit word (SIMD within a register).
//
// A code byte is s | m with m = e_b K + k (e_b = e + 2^{E-1}, App. C.1), so
//   k   = the low C bits,  e_b = the next E bits,  s = bit 7.
// Plane value +-2^{x}, x = e_b - 2^{E-1} + off (off = block scale - row
// reference - plane bias; +1 for a carry plane):
//   E5M2:  byte (x + 15) << 2 for x >= -14 (smaller values flush to zero:
//          they sit 2^14 below the row's largest element);
//   BF16:  half (x + 127) << 7 for x >= -126.
// The test "x is representable" is done with a guard bit: per lane
// u = e_b + c + (bias) has its top bit set exactly when the value is kept, so
// no lane borrows from its neighbour.

// Per-byte 0xFF where the lane's top bit (bit 7) is set.
__device__ __forceinline__ uint32_t byte_mask_from_bit7(uint32_t v7) { return ((v7 >> 7) & 0x01010101u) * 0xFFu; }
__device__ __forceinline__ uint32_t half_mask_from_bit15(uint32_t v15) {
  return ((v15 >> 15) & 0x00010001u) * 0xFFFFu;
}

template <int FMT>
struct CodeBits {
  using F = Fmt<FMT>;
  static constexpr uint32_t MM = F::MMASK * 0x01010101u;             // rank bits
  static constexpr uint32_t EBM = ((1u << F::E) - 1u) * 0x01010101u;  // e_b bits after >> C
};

// E5M2 plane bytes of four codes for exponent offset off (c = 15 - 2^{E-1} + off).
template <int FMT>
__device__ __forceinline__ uint32_t e5m2_word(uint32_t w, int off) {
  using F = Fmt<FMT>;
  int c = 15 - (1 << (F::E - 1)) + off;
  c = c < -127 ? -127 : c;                                  // everything flushes
  const uint32_t m4 = w & CodeBits<FMT>::MM;
  const uint32_t eb4 = (w >> F::C) & CodeBits<FMT>::EBM;
  const uint32_t u4 = eb4 + (uint32_t)(c + 127) * 0x01010101u;  // bit 7 <=> x >= -14
  const uint32_t nz = m4 + 0x7F7F7F7Fu;                          // bit 7 <=> m != 0
  const uint32_t keep = byte_mask_from_bit7(u4 & nz & 0x80808080u);
  const uint32_t t = ((u4 & 0x7F7F7F7Fu) + 0x01010101u) & keep;  // x + 15 where kept
  return (t << 2) | (w & 0x80808080u & keep);
}

// BF16 plane halves of two codes (bytes 0 and 1 of w2 = codes c0 | c1 << 16).
template <int FMT>
__device__ __forceinline__ uint32_t bf16_word(uint32_t w2, int off) {
  using F = Fmt<FMT>;
  const int c = 127 - (1 << (F::E - 1)) + off;               // biased exponent = e_b + c
  const uint32_t MM2 = (uint32_t)F::MMASK * 0x00010001u;
  const uint32_t EB2 = ((1u << F::E) - 1u) * 0x00010001u;
  const uint32_t m2 = w2 & MM2;
  const uint32_t eb2 = (w2 >> F::C) & EB2;
  const uint32_t u2 = eb2 + (uint32_t)(c - 1 + 0x8000) * 0x00010001u;  // bit 15 <=> e_b + c >= 1
  const uint32_t nz = m2 + 0x7FFF7FFFu;                                 // bit 15 <=> m != 0
  const uint32_t keep = half_mask_from_bit15(u2 & nz & 0x80008000u);
  const uint32_t t = ((u2 & 0x7FFF7FFFu) + 0x00010001u) & keep;       // biased exponent where kept
  return (t << 7) | ((w2 & 0x00800080u & keep) << 8);
}

// Masks of the curve-index bits (0xFF / 0xFFFF per lane where bit b of k is 1).
template <int PT, int KBITS>
__device__ __forceinline__ void k_masks(uint32_t w, uint32_t (&mk)[3]) {
#pragma unroll
  for (int b = 0; b < 3; ++b) {
    if (b >= KBITS) {
      mk[b] = 0u;
    } else if (PT == PLANE_E5M2) {
      mk[b] = ((w >> b) & 0x01010101u) * 0xFFu;
    } else {
      mk[b] = ((w >> b) & 0x00010001u) * 0xFFFFu;
    }
  }
}

// Lanes of value word v whose curve index is kap (compile-time kap; the
// compiler folds the three mask terms into 3-input logic operations).
template <int KBITS>
__device__ __forceinline__ uint32_t plane_of(uint32_t v, const uint32_t (&mk)[3], int kap) {
  uint32_t r = v;
  r &= (kap & 1) ? mk[0] : ~mk[0];
  r &= (kap & 2) ? mk[1] : ~mk[1];
  if (KBITS > 2) r &= (kap & 4) ? mk[2] : ~mk[2];
  return r;
}

// Decode one 32-byte code run (KS codes) of a row: eight value words in the
// order the MMA operands expect along K (word w holds elements 4w..4w+3 as
// E5M2 bytes, or 2w..2w+1 as BF16 halves), the x2 carry words if asked, and
// the curve-index masks of every word.
template <int FMT, int PT>
__device__ __forceinline__ void decode_run(const uint4 (&cw)[2], int off, uint32_t (&v)[8], uint32_t (&vc)[8],
                                           uint32_t (&mk)[8][3], bool want_carry) {
  constexpr int KBITS = Fmt<FMT>::C;
  if (PT == PLANE_E5M2) {
    const uint32_t w[8] = {cw[0].x, cw[0].y, cw[0].z, cw[0].w, cw[1].x, cw[1].y, cw[1].z, cw[1].w};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      v[i] = e5m2_word<FMT>(w[i], off);
      vc[i] = want_carry ? e5m2_word<FMT>(w[i], off + 1) : 0u;
      k_masks<PT, KBITS>(w[i], mk[i]);
    }
  } else {
    const uint32_t w[4] = {cw[0].x, cw[0].y, cw[0].z, cw[0].w};
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t w2 = __byte_perm(w[i >> 1], 0u, (i & 1) ? 0x4342u : 0x4140u);
      v[i] = bf16_word<FMT>(w2, off);
      vc[i] = want_carry ? bf16_word<FMT>(w2, off + 1) : 0u;
      k_masks<PT, KBITS>(w2, mk[i]);
    }
  }
}

template <class Cfg, int PT, int PASS>
__device__ __forceinline__ void write_b_planes(uint8_t* stage, int row, const uint32_t (&v)[8],
                                               const uint32_t (&vc)[8], const uint32_t (&mk)[8][3]) {
  constexpr int KBITS = Fmt<Cfg::FB_>::C;
  const uint32_t core = (uint32_t)((row >> 3) * 256 + (row & 7) * 16);
#pragma unroll
  for (int c = 0; c < 2; ++c)
#pragma unroll
    for (int k2 = 0; k2 < Cfg::KB; ++k2) {
      const int sl = Cfg::slot(PASS, c, k2);
      if (sl < 0) continue;
#pragma unroll
      for (int kc = 0; kc < 2; ++kc) {
        uint32_t o[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) o[q] = plane_of<KBITS>(c ? vc[4 * kc + q] : v[4 * kc + q], mk[4 * kc + q], k2);
        *reinterpret_cast<uint4*>(stage + (size_t)sl * Cfg::PLANE_BYTES + core + kc * 128) =
            make_uint4(o[0], o[1], o[2], o[3]);
      }
    }
}

template <class Cfg, int PT, int PASS>
__device__ __forceinline__ void issue_pass(uint32_t tmem, uint64_t bdesc0, int abuf, int bstage, bool first_step) {
#pragma unroll
  for (int k1 = 0; k1 < Cfg::KA; ++k1)
#pragma unroll
    for (int k2 = 0; k2 < Cfg::KB; ++k2) {
      const int h = Cfg::phase(k1, k2);
      if (h / Cfg::PP != PASS) continue;
      const int sl = Cfg::slot(PASS, Cfg::carry(k1, k2), k2);
      const uint32_t a_t = tmem + Cfg::ACOL0 + abuf * Cfg::ACOLS + k1 * 8;
      const uint64_t bd = bdesc0 + (uint64_t)((bstage * Cfg::BSTAGE + sl * Cfg::PLANE_BYTES) >> 4);
      const uint32_t d_t = tmem + (h - PASS * Cfg::PP) * Cfg::BN;
      const uint32_t accum = (first_step && Cfg::first_of_phase(k1, k2)) ? 0u : 1u;
      if (PT == PLANE_BF16)
        tc::mma_f16_ts(d_t, a_t, bd, Cfg::IDESC, accum);
      else
        tc::mma_f8_ts(d_t, a_t, bd, Cfg::IDESC, accum);
    }
}

}  // namespace

template <int FA, int FB, int PT>
__global__ void __launch_bounds__(288, 1) gemm_tc_kernel(const uint8_t* __restrict__ A, const int8_t* __restrict__ sA,
                                                         const uint8_t* __restrict__ B, const int8_t* __restrict__ sB,
                                                         int M, int N, int K, int G, float* __restrict__ C,
                                                         uint32_t* status) {
  using Cfg = TcCfg<FA, FB, PT>;
  constexpr int L = Cfg::L, PP = Cfg::PP, NP = Cfg::NP, BN = Cfg::BN, NSB = Cfg::NSB;
  static_assert(NP <= 3, "pass dispatch");
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* bstage = smem;
  TcShared& sh = *reinterpret_cast<TcShared*>(smem + (size_t)NSB * Cfg::BSTAGE);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.y * Cfg::BM, n0 = blockIdx.x * BN;
  const int nb = K / G, nsub = K / Cfg::KS, total = NP * nsub;

  if (tid == 0) {
    for (int s = 0; s < 2; ++s) {
      tc::mbar_init(&sh.a_full[s], 128);
      tc::mbar_init(&sh.a_empty[s], 1);
    }
    for (int s = 0; s < NSB; ++s) {
      tc::mbar_init(&sh.b_full[s], 128);
      tc::mbar_init(&sh.b_empty[s], 1);
    }
    tc::mbar_init(&sh.acc_full, 1);
    tc::mbar_init(&sh.drain, 1);
    sh.abort_flag = 0;
  }
  if (warp == 8) {
    tc::tmem_alloc(&sh.tmem_base, 512);
    tc::tmem_relinquish();
  }
  // reference exponents: largest block scale of each A row / B row
  int ref = -128;
  if (warp < 8) {
    const int r = warp < 4 ? m0 + tid : n0 + tid - 128;
    const int lim = warp < 4 ? M : N;
    const int8_t* s = warp < 4 ? sA : sB;
    if (r < lim) {
#pragma unroll 8
      for (int b = 0; b < nb; ++b) ref = max(ref, (int)__ldg(s + (int64_t)r * nb + b));
    }
    if (warp >= 4) sh.refB[tid - 128] = ref;
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;

  if (warp < 8) {
    // ------------------------------ producers ------------------------------
    const bool is_a = warp < 4;
    const int rloc = is_a ? tid : tid - 128;
    const int r = (is_a ? m0 : n0) + rloc;
    const bool rowok = r < (is_a ? M : N);
    const uint8_t* src = (is_a ? A : B) + (int64_t)r * K;
    const int8_t* srow = (is_a ? sA : sB) + (int64_t)r * nb;
    const int bias = is_a ? Cfg::PBA : Cfg::PBB;
    auto load = [&](int g, uint4 (&cw)[2], int& off) {
      cw[0] = cw[1] = make_uint4(0, 0, 0, 0);
      off = 0;
      if (rowok && g < total) {
        const int s = g % nsub;
        const uint4* p = reinterpret_cast<const uint4*>(src + (int64_t)s * Cfg::KS);
        cw[0] = __ldg(p);
        if (Cfg::KS == 32) cw[1] = __ldg(p + 1);
        off = (int)__ldg(srow + (s * Cfg::KS) / G) - ref - bias;
      }
    };
    uint4 n1[2], n2[2];
    int o1, o2;
    load(0, n1, o1);
    load(1, n2, o2);
    const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
    float cf[L];
#pragma unroll
    for (int h = 0; h < L; ++h) cf[h] = __uint_as_float(L == 8 ? CFP_PHASE_F32_L8_DEV[h] : CFP_PHASE_F32_L4_DEV[h]);

    for (int g = 0; g < total; ++g) {
      uint4 cw[2] = {n1[0], n1[1]};
      const int off = o1;
      n1[0] = n2[0];
      n1[1] = n2[1];
      o1 = o2;
      load(g + 2, n2, o2);  // keep two steps of codes in flight
      const int p = g / nsub, s = g % nsub;
      uint32_t v[8], vc[8], mk[8][3];
      if (is_a) {
        const int buf = g & 1;
        bool fail = false;
        if (g >= 2) {
          fail = !tc::mbar_wait(&sh.a_empty[buf], ((g >> 1) - 1) & 1);
          tc::fence_after_sync();
        }
        if (fail) {
          raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
        }
        if (__any_sync(0xffffffffu, fail || read_abort(&sh.abort_flag))) break;
        decode_run<FA, PT>(cw, off, v, vc, mk, false);
#pragma unroll
        for (int g4 = 0; g4 < Cfg::KA / 4; ++g4) {
          uint32_t reg[32];
#pragma unroll
          for (int pl = 0; pl < 4; ++pl)
#pragma unroll
            for (int c = 0; c < 8; ++c) reg[pl * 8 + c] = plane_of<Fmt<FA>::C>(v[c], mk[c], 4 * g4 + pl);
          tc::tmem_st32(lane_base + Cfg::ACOL0 + buf * Cfg::ACOLS + g4 * 32, reg);
        }
        tc::tmem_wait_st();
        tc::fence_before_sync();
        tc::mbar_arrive(&sh.a_full[buf]);

        if (s == nsub - 1) {
          // ---------------- epilogue of pass p -----------------------------
          const bool ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.acc_full, p & 1));
          if (!ok) {
            raise_flag(status, CURVEFP_DEV_TIMEOUT);
            sh.abort_flag = 1;
          }
          tc::fence_after_sync();
#pragma unroll 1
          for (int c0 = 0; c0 < BN; c0 += 8) {
            uint32_t acc[PP][8];
#pragma unroll
            for (int q = 0; q < PP; ++q)
              if (p * PP + q < L) tc::tmem_ld8(lane_base + q * BN + c0, acc[q]);
            tc::tmem_wait_ld();
            if (rowok && ok) {
#pragma unroll
              for (int c = 0; c < 8; ++c) {
                const int col = n0 + c0 + c;
                if (col < N) {
                  float y = 0.f;
#pragma unroll
                  for (int q = 0; q < PP; ++q)
                    if (p * PP + q < L) y = fmaf(cf[p * PP + q], __uint_as_float(acc[q][c]), y);
                  y = scalbnf(y, ref + Cfg::PBA + sh.refB[c0 + c] + Cfg::PBB);
                  float* dst = C + (int64_t)r * N + col;
                  *dst = p == 0 ? y : *dst + y;
                }
              }
            }
          }
          if (!ok) break;
        }
      } else {
        const int st = g % NSB;
        bool fail = false;
        if (g >= NSB) fail = !tc::mbar_wait(&sh.b_empty[st], ((g / NSB) - 1) & 1);
        if (fail) {
          raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
        }
        if (fail || read_abort(&sh.abort_flag)) break;
        decode_run<FB, PT>(cw, off, v, vc, mk, true);
        uint8_t* stg = bstage + (size_t)st * Cfg::BSTAGE;
        if (p == 0) write_b_planes<Cfg, PT, 0>(stg, rloc, v, vc, mk);
        if (NP > 1 && p == 1) write_b_planes<Cfg, PT, (NP > 1 ? 1 : 0)>(stg, rloc, v, vc, mk);
        if (NP > 2 && p == 2) write_b_planes<Cfg, PT, (NP > 2 ? 2 : 0)>(stg, rloc, v, vc, mk);
        tc::fence_proxy_async_smem();
        tc::mbar_arrive(&sh.b_full[st]);
      }
    }
  } else {
    // ------------------------------ MMA issuer -------------------------------
    if (lane == 0) {
      const uint64_t bdesc0 = tc::smem_desc(tc::smem_u32(bstage), 128, 256);
      for (int g = 0; g < total; ++g) {
        const int p = g / nsub, s = g % nsub;
        const int abuf = g & 1, st = g % NSB;
        bool ok = tc::mbar_wait(&sh.a_full[abuf], (g >> 1) & 1);
        ok = ok && tc::mbar_wait(&sh.b_full[st], (g / NSB) & 1);
        if (!ok || read_abort(&sh.abort_flag)) {
          raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
          break;
        }
        tc::fence_after_sync();
        if (p == 0) issue_pass<Cfg, PT, 0>(tmem, bdesc0, abuf, st, s == 0);
        if (NP > 1 && p == 1) issue_pass<Cfg, PT, (NP > 1 ? 1 : 0)>(tmem, bdesc0, abuf, st, s == 0);
        if (NP > 2 && p == 2) issue_pass<Cfg, PT, (NP > 2 ? 2 : 0)>(tmem, bdesc0, abuf, st, s == 0);
        tc::mma_commit(&sh.a_empty[abuf]);
        tc::mma_commit(&sh.b_empty[st]);
        if (s == nsub - 1) tc::mma_commit(&sh.acc_full);
      }
      // every issued MMA retires before TMEM is released (also on abort)
      tc::mma_commit(&sh.drain);
      if (!tc::mbar_wait(&sh.drain, 0)) raise_flag(status, CURVEFP_DEV_TIMEOUT);
    }
    __syncwarp();
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == 8) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

template <int FA, int FB, int PT>
static cudaError_t launch_tc_t(int G, const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb,
                               int64_t M, int64_t N, int64_t K, float* c, uint32_t* st, cudaStream_t s) {
  using Cfg = TcCfg<FA, FB, PT>;
  static_assert(sizeof(TcShared) <= 2048, "shared tail");
  static_assert(Cfg::SMEM <= 227 * 1024, "shared memory");
  auto kern = gemm_tc_kernel<FA, FB, PT>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::SMEM);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((N + Cfg::BN - 1) / Cfg::BN), (unsigned)((M + Cfg::BM - 1) / Cfg::BM));
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
  constexpr int PT = CFP_TC_PLANE;
#define CFP_T(X, Y) \
  if (fa == X && fb == Y) return launch_tc_t<X, Y, PT>(G, a, sa, b, sb, M, N, K, c, status, s);
  CFP_T(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_T(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_T(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_T
  return cudaErrorInvalidValue;
}

}  // namespace cfp
