// Tensor-core closed-product GEMM with 2:4-sparse MMAs (tcgen05.mma.sp,
// sm_103a): the phase-plane method of the dense kernel (Sec. 3.2, Eq. 2,
// Eq. 5) at half the MMA count.
//
// Every decoded element is 2^{k/K} times an exact power of two; plane k1 of A
// times plane k2 of B lands on phase h = (k1 WA + k2 WB) mod L with carry
// floor((k1 WA + k2 WB) / L).  An element lies in exactly one curve plane, so
// A planes k1 = j and k1 = j + K_A/2 (a "pair plane" j) never both hold it:
// placed at logical positions 2k (plane j) and 2k + 1 (plane j + K_A/2), they
// form a 2:4-sparse operand of logical length 2K.  Its compressed form is the
// pair plane itself (element k's value at byte k) and its sparsity metadata
// is one bit of each element's curve index.  One sparse MMA of logical K = 64
// against the interleaved B operand
//   B'[n][2k]     = the B plane that pairs with A plane j      for phase h,
//   B'[n][2k + 1] = the B plane that pairs with A plane j + K_A/2,
// adds both plane-pair products to phase h's accumulator.  A 128 x 96 x 64
// sparse FP8 MMA takes the same 48 cycles as the dense 128 x 96 x 32 one, so
// the tensor work halves.  Products stay exact (powers of two); only the FP32
// accumulation in TMEM rounds.
//
// Metadata (2:4, 8-bit types): per TMEM lane (row), 4 bits per chunk of 4
// logical positions, chunk c in bits 4c..4c+3 of a 64-bit pair of columns;
// bits 1:0 and 3:2 are the positions of the chunk's two stored values (slot 0
// = element 2c at position 0 or 1, slot 1 = element 2c + 1 at 2 or 3).
//
// Shape, roles and pipeline as in the dense kernel: 128 x 96 tiles, four
// 96-column phase accumulators per pass, 8 A-producer warps (pair planes and
// metadata -> TMEM), 6 B-producer warps (interleaved operands -> shared
// memory), one MMA warp; one full/empty barrier pair per step; bounded waits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "cfp_common.cuh"
#include "kernels.cuh"
#include "tc_planes.cuh"
#include "tc_ptx.cuh"

namespace cfp {

namespace {

template <int FA, int FB>
struct TcsCfg {
  using P = Pair<FA, FB>;
  static constexpr int KA = Fmt<FA>::K, KB = Fmt<FB>::K, L = P::L, WA = P::WA, WB = P::WB, LOG2L = P::LOG2L;
  static constexpr int FB_ = FB;
  static constexpr int BM = 128, BN = 96, KS = 32;  // KS codes per pipeline step
  static constexpr int PP = 4;                      // phases per pass
  static constexpr int NP = (L + PP - 1) / PP;      // passes
  static constexpr int HB = KA / 2;                 // partner offset inside a pair plane
  static constexpr int NJ = HB;                     // pair planes
  static constexpr int MBIT = KA == 8 ? 2 : 1;      // curve-index bit that selects the partner
  static constexpr int ACC_COLS = PP * BN;
  static constexpr int AU_COLS = NJ * 8;            // pair planes of one step, 8 columns each
  static constexpr int NAU = 2;                     // two steps of A in flight
  static constexpr int ACOL0 = ACC_COLS;
  static constexpr int MCOL0 = ACOL0 + NAU * AU_COLS;  // metadata of step unit u at MCOL0 + 8 u (2 used)
  static_assert(MCOL0 + NAU * 8 <= 512, "TMEM budget");
  static constexpr int OP_BYTES = BN * 64;          // one interleaved B operand (logical K = 64)
  static constexpr int NSB = 4;                     // B stages
  static constexpr int PBA = FA == CURVEFP_E5C2 ? 1 : 0;  // plane exponent bias
  static constexpr int PBB = FB == CURVEFP_E5C2 ? 1 : 0;
  static constexpr int NAW = 8;                     // A producer warps: two threads per row
  static constexpr int NBT = 2 * BN;                // B producer threads: two per row
  static constexpr int MMA_WARP = (NAW * 32 + NBT) / 32;
  static constexpr int TMA_WARP = MMA_WARP + 1;     // streams the code tiles
  static constexpr int THREADS = NAW * 32 + NBT + 64;
  static constexpr int NCS = 6;                     // code-tile stages (steps in flight)
  static constexpr int CODE_A = BM * KS, CODE_B = BN * KS;  // bytes of one step's code tiles
  // D = F32, A = B = E5M2, sparse flag (bit 2), sparsity selector 0
  static constexpr uint32_t IDESC = tc::idesc_bf16_f32(BM, BN) | (1u << 2);

  // B plane (k2) pairing with A plane k1 on phase h, or -1; and its carry
  __host__ __device__ static constexpr int partner(int k1, int h) {
    for (int k2 = 0; k2 < KB; ++k2)
      if (((k1 * WA + k2 * WB) & (L - 1)) == h) return k2;
    return -1;
  }
  __host__ __device__ static constexpr int partner_carry(int k1, int h) {
    return partner(k1, h) < 0 ? 0 : (k1 * WA + partner(k1, h) * WB) >> LOG2L;
  }
  // operand half: 0 = none, else 1 + 2 k2 + carry
  __host__ __device__ static constexpr int half_key(int k1, int h) {
    return partner(k1, h) < 0 ? 0 : 1 + 2 * partner(k1, h) + partner_carry(k1, h);
  }
  __host__ __device__ static constexpr int op_key(int j, int h) { return half_key(j, h) * 64 + half_key(j + HB, h); }
  __host__ __device__ static constexpr bool valid(int j, int h) { return op_key(j, h) != 0; }
  // operands of pass p in order of first use (j major, h minor)
  __host__ __device__ static constexpr int op_index(int p, int j, int h) {
    int n = 0;
    for (int jj = 0; jj < NJ; ++jj)
      for (int hh = p * PP; hh < (p + 1) * PP && hh < L; ++hh) {
        if (!valid(jj, hh)) continue;
        bool seen = false;
        for (int j2 = 0; j2 < NJ; ++j2)
          for (int h2 = p * PP; h2 < (p + 1) * PP && h2 < L; ++h2)
            if ((j2 < jj || (j2 == jj && h2 < hh)) && valid(j2, h2) && op_key(j2, h2) == op_key(jj, hh)) seen = true;
        if (seen) continue;
        if (op_key(jj, hh) == op_key(j, h)) return n;
        ++n;
      }
    return -1;
  }
  __host__ __device__ static constexpr int nops(int p) {
    int m = 0;
    for (int jj = 0; jj < NJ; ++jj)
      for (int hh = p * PP; hh < (p + 1) * PP && hh < L; ++hh)
        if (valid(jj, hh) && op_index(p, jj, hh) + 1 > m) m = op_index(p, jj, hh) + 1;
    return m;
  }
  // key of operand o of pass p
  __host__ __device__ static constexpr int key_of(int p, int o) {
    for (int jj = 0; jj < NJ; ++jj)
      for (int hh = p * PP; hh < (p + 1) * PP && hh < L; ++hh)
        if (valid(jj, hh) && op_index(p, jj, hh) == o) return op_key(jj, hh);
    return 0;
  }
  __host__ __device__ static constexpr int maxops() {
    int m = 0;
    for (int p = 0; p < NP; ++p) m = nops(p) > m ? nops(p) : m;
    return m;
  }
  // is (j, h) the first MMA of the issue order that writes phase h?
  __host__ __device__ static constexpr bool first_of_phase(int j, int h) {
    for (int jj = 0; jj < j; ++jj)
      if (valid(jj, h)) return false;
    return true;
  }
  static constexpr int MAXO = maxops();
  static constexpr int BSTAGE = MAXO * OP_BYTES;
  static constexpr size_t CODE0 = (size_t)NSB * BSTAGE;  // code ring (1024-byte aligned)
  static_assert(CODE0 % 1024 == 0, "code ring alignment");
  static constexpr size_t SMEM = CODE0 + (size_t)NCS * (CODE_A + CODE_B) + 2048;
};

__device__ __forceinline__ void mma_sp_if(uint32_t leader, uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                          uint32_t meta_tmem, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.b32 p, %5, 0;\n setp.ne.b32 q, %6, 0;\n"
      "@q tcgen05.mma.sp.cta_group::1.kind::f8f6f4 [%0], [%1], %2, [%3], %4, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(meta_tmem), "r"(idesc), "r"(accumulate), "r"(leader)
      : "memory");
}

// Interleave two plane words (elements 4q..4q+3 each) into the operand's
// logical byte order X0 Y0 X1 Y1 | X2 Y2 X3 Y3.
__device__ __forceinline__ void interleave(uint32_t x, uint32_t y, uint32_t& lo, uint32_t& hi) {
  lo = __byte_perm(x, y, 0x5140);
  hi = __byte_perm(x, y, 0x7362);
}

// Operand O (and the following ones) of pass PASS: the thread's 32 bytes
// (logical positions 32 half .. 32 half + 31 = two 16-byte core-matrix rows,
// K chunks 2 half and 2 half + 1) from the value planes pw[carry][word][k2].
template <class Cfg, int PASS, int O>
__device__ __forceinline__ void write_b_op(uint8_t* stage, uint32_t core, int half, const uint32_t (&pw)[2][4][8]) {
  if constexpr (O < Cfg::nops(PASS)) {
    constexpr int key = Cfg::key_of(PASS, O);
    constexpr int kx = key / 64, ky = key % 64;
    uint32_t w[8];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t x = kx ? pw[(kx - 1) & 1][q][(kx - 1) >> 1] : 0u;
      const uint32_t y = ky ? pw[(ky - 1) & 1][q][(ky - 1) >> 1] : 0u;
      interleave(x, y, w[2 * q], w[2 * q + 1]);
    }
    uint8_t* base = stage + (size_t)O * Cfg::OP_BYTES + core;
    *reinterpret_cast<uint4*>(base + (2 * half) * 128) = make_uint4(w[0], w[1], w[2], w[3]);
    *reinterpret_cast<uint4*>(base + (2 * half + 1) * 128) = make_uint4(w[4], w[5], w[6], w[7]);
    write_b_op<Cfg, PASS, O + 1>(stage, core, half, pw);
  }
}

template <class Cfg, int PASS>
__device__ __forceinline__ void write_b_ops(uint8_t* stage, int row, int half, const uint32_t (&v)[4],
                                            const uint32_t (&vc)[4], const uint32_t (&mk)[4][4]) {
  constexpr int KBITS = Fmt<Cfg::FB_>::C;
  uint32_t pw[2][4][8];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    planes_of<KBITS>(v[q], mk[q], pw[0][q]);
    planes_of<KBITS>(vc[q], mk[q], pw[1][q]);
  }
  const uint32_t core = (uint32_t)((row >> 3) * 512 + (row & 7) * 16);
  write_b_op<Cfg, PASS, 0>(stage, core, half, pw);
}

// The sparse MMAs of one step of pass PASS, pair plane J and phase H onwards.
template <class Cfg, int PASS, int J, int H>
__device__ __forceinline__ void issue_mmas(uint32_t leader, uint32_t tmem, uint64_t bdesc0, int abuf, int bstage,
                                           bool first_step) {
  if constexpr (J < Cfg::NJ) {
    constexpr int HEND = (PASS + 1) * Cfg::PP < Cfg::L ? (PASS + 1) * Cfg::PP : Cfg::L;
    if constexpr (H < HEND) {
      if constexpr (Cfg::valid(J, H)) {
        constexpr int o = Cfg::op_index(PASS, J, H);
        const uint32_t d_t = tmem + (H - PASS * Cfg::PP) * Cfg::BN;
        const uint32_t a_t = tmem + Cfg::ACOL0 + abuf * Cfg::AU_COLS + J * 8;
        const uint32_t m_t = tmem + Cfg::MCOL0 + abuf * 8;
        const uint64_t bd = bdesc0 + (uint64_t)((bstage * Cfg::BSTAGE + o * Cfg::OP_BYTES) >> 4);
        const uint32_t accum = (first_step && Cfg::first_of_phase(J, H)) ? 0u : 1u;
        mma_sp_if(leader, d_t, a_t, bd, m_t, Cfg::IDESC, accum);
      }
      issue_mmas<Cfg, PASS, J, H + 1>(leader, tmem, bdesc0, abuf, bstage, first_step);
    } else {
      issue_mmas<Cfg, PASS, J + 1, PASS * Cfg::PP>(leader, tmem, bdesc0, abuf, bstage, first_step);
    }
  }
}

template <class Cfg>
__device__ __forceinline__ void issue_step_sp(uint32_t leader, int p, uint32_t tmem, uint64_t bdesc0, int abuf,
                                              int bstage, bool first_step) {
  if (p == 0) issue_mmas<Cfg, 0, 0, 0>(leader, tmem, bdesc0, abuf, bstage, first_step);
  if constexpr (Cfg::NP > 1)
    if (p == 1) issue_mmas<Cfg, 1, 0, Cfg::PP>(leader, tmem, bdesc0, abuf, bstage, first_step);
}

// Metadata word of 16 codes (four code words, elements 4q..4q+3 each): per
// chunk of two elements, idx0 = bit(2c), idx1 = 2 + bit(2c + 1), where bit is
// the curve-index bit MBIT that selects the partner plane.
template <int MBIT>
__device__ __forceinline__ uint32_t sparse_meta(const uint32_t (&w)[4]) {
  uint32_t b[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint32_t t = (w[q] >> MBIT) & 0x01010101u;         // bit of element i at 8 i
    b[q] = ((t * 0x01041040u) >> 24) | 0x88u;                 // ... at 2 i, plus bit 3 of each nibble
  }
  return b[0] | (b[1] << 8) | (b[2] << 16) | (b[3] << 24);
}

}  // namespace

// Thread layout: warps 0-7 produce A (warp w: TMEM lane group w & 3, half
// w >> 2 of each 32-code run) and run the epilogue (columns [BN/2 half,
// BN/2 (half + 1))); the next 2 BN threads produce B (thread 256 + t: row
// t % BN, half t / BN); the last warp allocates TMEM and issues the MMAs.
template <int FA, int FB>
__global__ void __launch_bounds__(TcsCfg<FA, FB>::THREADS, 1)
    gemm_tcs_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
                    const int8_t* __restrict__ sA, const int8_t* __restrict__ sB, int M, int N, int K, int G,
                    int gshift, float* __restrict__ C, uint32_t* status) {
  using Cfg = TcsCfg<FA, FB>;
  constexpr int L = Cfg::L, PP = Cfg::PP, NP = Cfg::NP, BN = Cfg::BN, NSB = Cfg::NSB, NAW = Cfg::NAW;
  static_assert(NP <= 2, "pass dispatch");
  static_assert(NSB == TC_MAX_RING && Cfg::NAU == 2, "barrier rings");
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* bstage = smem;
  constexpr int NCS = Cfg::NCS, CSTAGE = Cfg::CODE_A + Cfg::CODE_B;
  static_assert(NCS <= 8, "code ring barriers");
  uint8_t* codes = smem + Cfg::CODE0;  // stage c: A tile [BM][KS] then B tile [BN][KS]
  TcShared& sh = *reinterpret_cast<TcShared*>(smem + Cfg::CODE0 + (size_t)NCS * CSTAGE);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.y * Cfg::BM, n0 = blockIdx.x * BN;
  const int nb = K / G, nsub = K / Cfg::KS, total = NP * nsub;

  if (tid == 0) {
    for (int s = 0; s < NSB; ++s) {
      tc::mbar_init(&sh.full[s], NAW + Cfg::NBT / 32);  // one arrival per producer warp
      tc::mbar_init(&sh.empty[s], 1);
    }
    for (int s = 0; s < NCS; ++s) {
      tc::mbar_init(&sh.code_full[s], 1);                        // TMA bytes
      tc::mbar_init(&sh.code_empty[s], NAW + Cfg::NBT / 32);     // producer warps done reading
    }
    tc::mbar_init(&sh.acc_full, 1);
    tc::mbar_init(&sh.drain, 1);
    sh.abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == Cfg::MMA_WARP) {
    tc::tmem_alloc(&sh.tmem_base, 512);
    tc::tmem_relinquish();
  }
  // producer geometry and the row's reference exponent (largest block scale)
  const bool is_a = warp < NAW;
  const bool is_prod = warp < Cfg::MMA_WARP;
  const int rloc = is_a ? ((warp & 3) * 32 + lane) : ((tid - NAW * 32) % BN);
  const int half = is_a ? (warp >> 2) : ((tid - NAW * 32) / BN);
  const int r = (is_a ? m0 : n0) + rloc;
  const bool rowok = is_prod && r < (is_a ? M : N);
  int ref = -128;
  if (rowok) {
    const int8_t* s = (is_a ? sA : sB) + (int64_t)r * nb;
    if ((nb & 15) == 0 && (reinterpret_cast<uintptr_t>(s) & 15) == 0) {
      uint32_t m4 = 0x80808080u;
#pragma unroll 8
      for (int b = 0; b < nb; b += 16) {
        const uint4 q = __ldg(reinterpret_cast<const uint4*>(s + b));
        m4 = __vmaxs4(m4, __vmaxs4(__vmaxs4(q.x, q.y), __vmaxs4(q.z, q.w)));
      }
      ref = max(max((int)(int8_t)(m4 & 0xFF), (int)(int8_t)((m4 >> 8) & 0xFF)),
                max((int)(int8_t)((m4 >> 16) & 0xFF), (int)(int8_t)(m4 >> 24)));
    } else {
#pragma unroll 8
      for (int b = 0; b < nb; ++b) ref = max(ref, (int)__ldg(s + b));
    }
  }
  if (!is_a && is_prod && half == 0) sh.refB[rloc] = ref;
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;

  if (is_prod) {
    // ------------------------------ producers ------------------------------
    // this thread's 16 bytes of a step's code tile in the ring
    const int cofs = (is_a ? 0 : Cfg::CODE_A) + rloc * Cfg::KS + half * 16;
    const int8_t* srow = (is_a ? sA : sB) + (int64_t)r * nb;
    const int bias = is_a ? Cfg::PBA : Cfg::PBB;
    auto pass_of = [&](int g) { return (NP > 1 && g >= nsub) ? 1 : 0; };
    // raw block scale of step g (two steps ahead, in registers; the row's
    // scales stay in L1 across the 32 steps of a sector)
    auto load = [&](int g, int& off) {
      off = 0;
      if (rowok && g < total) off = (int)__ldg(srow + ((g - pass_of(g) * nsub) >> gshift));
    };
    // the step's codes: wait for the tile and copy this thread's 16 bytes
    auto fetch = [&](int g, uint4& cw) -> bool {
      const int cs = g % NCS;
      const bool ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.code_full[cs], (g / NCS) & 1));
      cw = *reinterpret_cast<const uint4*>(codes + (size_t)cs * CSTAGE + cofs);
      return ok;
    };
    // Release the stage once every lane's shared load has returned: a shuffle
    // consumes all lanes' words and the arrival depends on its result.  (An
    // arrival issued right after the loads let the next bulk copy overwrite
    // the stage while loads were still in flight: whole lane groups then
    // decoded a later step's codes.)
    auto release = [&](int g, const uint4& cw) {
      const uint32_t dep = __shfl_xor_sync(0xffffffffu, cw.x ^ cw.y ^ cw.z ^ cw.w, 1);
      if (lane == 0) tc::mbar_arrive_after(&sh.code_empty[g % NCS], dep);
    };
    const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    // One pipeline step of this producer thread; false ends the loop (abort).
    auto step = [&](const int g, const int raw_scale) -> bool {
      uint4 cw;
      if (!fetch(g, cw)) {
        if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
        sh.abort_flag = 1;
        return false;
      }
      release(g, cw);
      if (!rowok) cw = make_uint4(0, 0, 0, 0);
      const int off = raw_scale - ref - bias;
      const int p = pass_of(g), s = g - p * nsub;
      if (is_a) {
        constexpr int KBITS = Fmt<FA>::C;
        uint32_t v[4], vc[4], mk[4][4];
        decode_words<FA, PLANE_E5M2, 4>(cw, off, v, vc, mk, false);
        const uint32_t wc[4] = {cw.x, cw.y, cw.z, cw.w};
        const uint32_t meta = sparse_meta<Cfg::MBIT>(wc);
        // pair plane j: the values whose curve index has low bits j
        uint32_t pj[4][4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          if (KBITS == 3) {
            pj[q][0] = v[q] & ~mk[q][0] & ~mk[q][1];
            pj[q][1] = v[q] & mk[q][0] & ~mk[q][1];
            pj[q][2] = v[q] & ~mk[q][0] & mk[q][1];
            pj[q][3] = v[q] & mk[q][0] & mk[q][1];
          } else {
            pj[q][0] = v[q] & ~mk[q][0];
            pj[q][1] = v[q] & mk[q][0];
            pj[q][2] = pj[q][3] = 0u;
          }
        }
        const int buf = g & 1;
        if (g >= 2) {
          // warp-uniform outcome: the TMEM stores below are warp-collective
          const int gr = g - 2;
          const bool ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.empty[gr % NSB], (gr / NSB) & 1));
          tc::fence_after_sync();
          if (!ok) {
            if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
            sh.abort_flag = 1;
            return false;
          }
        }
        // pair plane j occupies 8 columns of the unit; this thread's half of
        // the 32 codes is columns 4 half .. 4 half + 3; its metadata word is
        // column `half` of the unit's metadata pair
#pragma unroll
        for (int j = 0; j < Cfg::NJ; ++j) {
          const uint32_t reg[4] = {pj[0][j], pj[1][j], pj[2][j], pj[3][j]};
          tc::tmem_st4(lane_base + Cfg::ACOL0 + buf * Cfg::AU_COLS + j * 8 + half * 4, reg);
        }
        tc::tmem_st1(lane_base + Cfg::MCOL0 + buf * 8 + half, meta);
        tc::tmem_wait_st();
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&sh.full[g % NSB]);

        if (s == nsub - 1) {
          // ---------------- epilogue of pass p -----------------------------
          const bool ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.acc_full, p & 1));
          if (!ok) {
            raise_flag(status, CURVEFP_DEV_TIMEOUT);
            sh.abort_flag = 1;
          }
          tc::fence_after_sync();
#pragma unroll 1
          for (int c0 = half * (BN / 2); c0 < (half + 1) * (BN / 2); c0 += 8) {
            uint32_t acc[PP][8];
#pragma unroll
            for (int q = 0; q < PP; ++q)
              if (p * PP + q < L) tc::tmem_ld8(lane_base + q * BN + c0, acc[q]);
            tc::tmem_wait_ld();
            if (rowok && ok) {
              float y[8];
#pragma unroll
              for (int c = 0; c < 8; ++c) {
                float t = 0.f;
#pragma unroll
                for (int q = 0; q < PP; ++q)
                  if (p * PP + q < L) t = fmaf(phase_const(L, p * PP + q), __uint_as_float(acc[q][c]), t);
                y[c] = scalbnf(t, ref + Cfg::PBA + sh.refB[c0 + c] + Cfg::PBB);
              }
              float* dst = C + (int64_t)r * N + n0 + c0;
              const bool full8 = n0 + c0 + 8 <= N && ((reinterpret_cast<uintptr_t>(dst) & 15) == 0);
              if (full8) {
                float4* d4 = reinterpret_cast<float4*>(dst);
                float4 a0 = make_float4(y[0], y[1], y[2], y[3]), a1 = make_float4(y[4], y[5], y[6], y[7]);
                if (p > 0) {
                  const float4 b0 = d4[0], b1 = d4[1];
                  a0.x += b0.x; a0.y += b0.y; a0.z += b0.z; a0.w += b0.w;
                  a1.x += b1.x; a1.y += b1.y; a1.z += b1.z; a1.w += b1.w;
                }
                d4[0] = a0;
                d4[1] = a1;
              } else {
#pragma unroll
                for (int c = 0; c < 8; ++c)
                  if (n0 + c0 + c < N) dst[c] = p == 0 ? y[c] : dst[c] + y[c];
              }
            }
          }
          if (!ok) return false;
        }
      } else {
        const int st = g % NSB;
        bool fail = false;
        if (g >= NSB) fail = !__all_sync(0xffffffffu, tc::mbar_wait(&sh.empty[st], ((g / NSB) - 1) & 1));
        if (fail) {
          if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
          return false;
        }
        uint32_t v[4], vc[4], mk[4][4];
        decode_words<FB, PLANE_E5M2, 4>(cw, off, v, vc, mk, true);
        uint8_t* stg = bstage + (size_t)st * Cfg::BSTAGE;
        if (p == 0) write_b_ops<Cfg, 0>(stg, rloc, half, v, vc, mk);
        if constexpr (NP > 1)
          if (p == 1) write_b_ops<Cfg, 1>(stg, rloc, half, v, vc, mk);
        tc::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&sh.full[st]);
      }
      return true;
    };
    int r0, r1;
    load(0, r0);
    load(1, r1);
    for (int g = 0; g < total; g += 2) {
      if (!step(g, r0)) break;
      load(g + 2, r0);
      if (g + 1 >= total) break;
      if (!step(g + 1, r1)) break;
      load(g + 3, r1);
    }
  } else if (warp == Cfg::TMA_WARP) {
    // ------------------------------ code tiles ---------------------------------
    // one lane streams each step's A and B code tiles (rows outside the
    // matrices arrive as zeros) NCS - 1 steps ahead of the producers
    if (lane == 0) {
      int issued = 0;
      bool ok = true;
      for (int g = 0; g < total; ++g, ++issued) {
        const int cs = g % NCS;
        if (g >= NCS && !tc::mbar_wait(&sh.code_empty[cs], ((g / NCS) - 1) & 1)) {
          ok = false;
          break;
        }
        const int s = g - ((NP > 1 && g >= nsub) ? nsub : 0);
        uint8_t* dst = codes + (size_t)cs * CSTAGE;
        tc::mbar_arrive_expect_tx(&sh.code_full[cs], CSTAGE);
        tc::tma_load_2d(dst, &mapA, s * Cfg::KS, m0, &sh.code_full[cs]);
        tc::tma_load_2d(dst + Cfg::CODE_A, &mapB, s * Cfg::KS, n0, &sh.code_full[cs]);
      }
      if (!ok) {
        raise_flag(status, CURVEFP_DEV_TIMEOUT);
        sh.abort_flag = 1;
      }
      // every copy issued lands before the CTA may exit
      for (int j = issued - NCS < 0 ? 0 : issued - NCS; j < issued; ++j)
        tc::mbar_wait(&sh.code_full[j % NCS], (j / NCS) & 1);
    }
    __syncwarp();
  } else {
    // ------------------------------ MMA issuer -------------------------------
    const uint32_t leader = tc::elect_one();
    // interleaved B operands: K-major, 64 logical bytes per row = 4 core
    // matrices along K (128 bytes apart), 8-row groups 512 bytes apart
    const uint64_t bdesc0 = tc::smem_desc(tc::smem_u32(bstage), 128, 512);
    bool ok = true;
    for (int g = 0; g < total && ok; ++g) {
      const int p = (NP > 1 && g >= nsub) ? 1 : 0, s = g - p * nsub;
      const int st = g % NSB;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.full[st], (g / NSB) & 1));
      if ((g & 7) == 0) ok = ok && !read_abort(&sh.abort_flag);
      if (!ok) break;
      tc::fence_after_sync();
      issue_step_sp<Cfg>(leader, p, tmem, bdesc0, g & 1, st, s == 0);
      tc::mma_commit_if(leader, &sh.empty[st]);
      if (s == nsub - 1) tc::mma_commit_if(leader, &sh.acc_full);
    }
    if (!ok && lane == 0) {
      raise_flag(status, CURVEFP_DEV_TIMEOUT);
      sh.abort_flag = 1;
    }
    // every issued MMA retires before TMEM is released (also on abort)
    tc::mma_commit_if(leader, &sh.drain);
    if (!tc::mbar_wait(&sh.drain, 0) && lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
    __syncwarp();
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == Cfg::MMA_WARP) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

// cuTensorMapEncodeTiled from the driver, looked up once.
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}

// Tensor map of a [rows x K] code matrix (K contiguous) with boxes of
// box_rows x 32 codes.
static cudaError_t code_map(CUtensorMap* map, const uint8_t* base, int64_t rows, int64_t K, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)K};
  const cuuint32_t box[2] = {32u, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1u, 1u};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <int FA, int FB>
static cudaError_t launch_tcs_t(int G, const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb,
                                int64_t M, int64_t N, int64_t K, float* c, uint32_t* st, cudaStream_t s) {
  using Cfg = TcsCfg<FA, FB>;
  CUtensorMap mapA, mapB;
  cudaError_t me = code_map(&mapA, a, M, K, Cfg::BM);
  if (me == cudaSuccess) me = code_map(&mapB, b, N, K, Cfg::BN);
  if (me != cudaSuccess) return me;
  static_assert(sizeof(TcShared) <= 2048, "shared tail");
  static_assert(Cfg::SMEM <= 227 * 1024, "shared memory");
  auto kern = gemm_tcs_kernel<FA, FB>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::SMEM);
  if (e != cudaSuccess) return e;
  dim3 grid((unsigned)((N + Cfg::BN - 1) / Cfg::BN), (unsigned)((M + Cfg::BM - 1) / Cfg::BM));
  int gshift = 0;  // scale block of step s is s >> gshift (G / KS is a power of two)
  while ((Cfg::KS << gshift) < G) ++gshift;
  kern<<<grid, Cfg::THREADS, Cfg::SMEM, s>>>(mapA, mapB, sa, sb, (int)M, (int)N, (int)K, G, gshift, c, st);
  return cudaGetLastError();
}

cudaError_t launch_gemm_tensor_sparse(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                                      const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, uint32_t* status,
                                      cudaStream_t s) {
#define CFP_T(X, Y) \
  if (fa == X && fb == Y) return launch_tcs_t<X, Y>(G, a, sa, b, sb, M, N, K, c, status, s);
  CFP_T(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_T(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_T(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_T
  return cudaErrorInvalidValue;
}

}  // namespace cfp
