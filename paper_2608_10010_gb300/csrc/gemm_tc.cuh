// Tensor-core closed-product GEMM (tcgen05, sm_103a): phase-plane
// decomposition with per-phase FP32 accumulation in TMEM and the phase
// combine fused into the epilogue (Sec. 3.2, Eq. 2, Eq. 5).
//
// Decomposition.  Write every decoded operand element as
//   x = 2^{a_b} 2^{k/K} X_k,   X_k = +-2^e  (an exact power of two),
// i.e. split each operand into K "curve planes" that hold the element in the
// plane of its curve index k and zero elsewhere.  Plane k1 of A times plane k2
// of B lands on the single phase h = (k1 WA + k2 WB) mod L with carry
// c = floor((k1 WA + k2 WB) / L) (Eq. 2 on the shared lattice L), so
//   S_h = sum_{k1,k2 : phase h} 2^c  A_{k1} B_{k2}^T,
// a sum of dense products of power-of-two matrices, which the tensor cores
// multiply without rounding; only the FP32 accumulation in TMEM rounds.
//
// Block scales are UE8M0 scale factors of a block-scaled MMA
// (tcgen05.mma .kind::mxf8f6f4 .block_scale, tc_mx.cuh): 2^{a_b - ref + 32}
// per row and 32-code step (ref = the row's largest block scale), so every
// product is exact whatever the spread of the scales along a row, and the
// carry 2^c is the second factor byte of the B row (2^{a_b - ref + 33}): the
// B planes are stored once, not in plain and doubled copies.  The epilogue
// applies 2^{ref_i + ref_j - 64}.  Plane values are FP8 E5M2 (every code of
// the binary formats and of E4C3 with r = 2^{8/9} has an exact one).
//
// Shape.  A CTA owns a 128 x BN tile of C: BN = 96 (a 128 x 96 x 32 FP8 MMA
// runs at the full tensor rate) where TMEM holds PP phase accumulators of BN
// columns, two steps of A planes and the scale factors, else 80.  The L
// phases are processed in passes of PP phases over the whole K; each pass
// adds its part of sum_h 2^{h/L} S_h to an FP32 stash, the last writes C.
//
// Roles:
//   warps 0-7   A producers (two threads per row, 16 codes each per step):
//               codes -> planes in registers -> TMEM (tcgen05.st), and the
//               row's scale factor; at the end of each pass the epilogue.
//   next warps  B producers (two threads per row): codes -> the planes that
//               the current pass needs -> shared memory, K-major core-matrix
//               layout; the row's factor bytes -> the stage's factor block.
//   last warp   TMEM allocation, factor copies (tcgen05.cp) and MMA issue
//               (one elected lane of the converged warp).
// One mbarrier hand-off per pipeline step: every wait and commit sits on the
// path between two MMAs, so the stages are whole steps.  Every wait is
// bounded.
#pragma once
#include <functional>
#include <mutex>
#include <queue>
#include <unordered_map>
#include <vector>

#include "cfp_common.cuh"
#include "kernels.cuh"
#include "tc_mx.cuh"
#include "tc_planes.cuh"
#include "tc_ptx.cuh"

namespace cfp {

namespace {

// Planes per operand and the product lattice: binary radix on the shared
// lattice L = max(K_a, K_b) (Eq. 2); E4C3 with r = 2^{8/9}: nine planes, nine
// phases, unit weights (Eq. 4).
template <int FA, int FB>
struct TcLattice {
  using P = Pair<FA, FB>;
  static constexpr int KA = Fmt<FA>::K, KB = Fmt<FB>::K, L = P::L, WA = P::WA, WB = P::WB;
};
template <>
struct TcLattice<CURVEFP_E4C3_R8_9, CURVEFP_E4C3_R8_9> {
  static constexpr int KA = 9, KB = 9, L = 9, WA = 1, WB = 1;
};

template <int FA, int FB>
struct TcCfg {
  using T = TcLattice<FA, FB>;
  static constexpr int KA = T::KA, KB = T::KB, L = T::L, WA = T::WA, WB = T::WB;
  static constexpr int FA_ = FA, FB_ = FB;
  static constexpr int BM = 128;
  static constexpr int KS = 32;                           // K per MMA = K per pipeline step (one factor)
  static constexpr int PP = L == 9 ? 3 : 4;               // phases per pass
  static constexpr int NP = (L + PP - 1) / PP;            // passes
  // A planes of a step occupy AU_COLS TMEM columns (8 per plane); two steps
  // rotate (NAU units)
  static constexpr int AU_COLS = KA * 8;
  static constexpr int NAU = 2;
  static constexpr int NSB = 4;                           // B stages
  // TMEM: PP accumulators of BN columns, the A units, A factors (4 columns
  // per unit: quadrant q reads column q) and B factors (4 columns per stage)
  static constexpr int SF_COLS = NAU * 4 + NSB * 4;
  static constexpr int BN = PP * 96 + NAU * AU_COLS + SF_COLS <= 512 ? 96 : 80;
  static constexpr int ACC_COLS = PP * BN;
  static constexpr int ACOL0 = ACC_COLS;
  static constexpr int SFA0 = ACOL0 + NAU * AU_COLS;
  static constexpr int SFB0 = SFA0 + NAU * 4;
  static_assert(SFB0 + NSB * 4 <= 512, "TMEM budget");
  static constexpr int PLANE_BYTES = BN * 32;             // BN rows x 32 bytes
  static constexpr int ATPR = 2;                          // A producer threads per row
  static constexpr int NAW = 4 * ATPR;                    // A producer warps (4 TMEM lane groups)
  static constexpr int NWA = 8 / ATPR;                    // TMEM columns per A thread and plane
  static constexpr int NBT = 2 * BN;                      // B producer threads (two per row)
  static constexpr int THREADS = NAW * 32 + NBT + 32;     // A producers, B producers, MMA warp
  static constexpr int MMA_WARP = (NAW * 32 + NBT) / 32;
  static_assert(NBT % 32 == 0 && BN % (8 * ATPR) == 0, "producer warps");

  __host__ __device__ static constexpr int phase(int k1, int k2) { return (k1 * WA + k2 * WB) % L; }
  __host__ __device__ static constexpr int carry(int k1, int k2) { return (k1 * WA + k2 * WB) / L; }
  // Does pass p need B plane k2?
  __host__ __device__ static constexpr bool needed(int p, int k2) {
    for (int k1 = 0; k1 < KA; ++k1)
      if (phase(k1, k2) / PP == p) return true;
    return false;
  }
  // Shared-memory slot of B plane k2 in pass p (-1 if unused).
  __host__ __device__ static constexpr int slot(int p, int k2) {
    int s = 0;
    for (int k = 0; k < KB; ++k) {
      const bool need = needed(p, k);
      if (k == k2) return need ? s : -1;
      if (need) ++s;
    }
    return -1;
  }
  __host__ __device__ static constexpr int nslots(int p) {
    int s = 0;
    for (int k = 0; k < KB; ++k) s += needed(p, k) ? 1 : 0;
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
  static constexpr int SFSTAGE = 512;                       // B factor block of a stage (one copy source)
  static constexpr int BSTAGE = MAXS * PLANE_BYTES + SFSTAGE;
  // B stages, the barrier block, and the FP32 stash of the passes' partial
  // outputs (row stride SST floats)
  static constexpr int SST = BN + 4;
  static constexpr size_t STASH = (size_t)BM * SST * 4;
  static constexpr size_t SMEM = (size_t)NSB * BSTAGE + 2048 + STASH;
  // D = F32, A = B = E5M2, UE8M0 factors, M = 128, N = BN
  static constexpr uint32_t IDESC = idesc_mx_e5m2(BN, false);
};

// Plane words of 4 codes of a binary format or of E4C3 with r = 2^{8/9}:
// values +-2^e (block-scale free) and the curve-index masks.
template <int FMT>
__device__ __forceinline__ void mx_decode(uint32_t w, uint32_t& v, uint32_t (&mk)[4]) {
  if constexpr (FMT == CURVEFP_E4C3_R8_9) {
    r89_word(w, v, mk);
  } else {
    uint32_t vc;
    mx_word<FMT, 0>(w, v, vc);
    k_masks<PLANE_E5M2, Fmt<FMT>::C>(w, mk);
  }
}

// Plane words of 4 codes with per-element exponent bytes (reused operands):
// byte i of dp is x_i + 16 for the plane value 2^{x_i} (x_i in [-16, 15]), or
// 0x80 where the element has no plane value (zero code, or more than 31
// binades below the largest element of its step).
template <int FMT>
__device__ __forceinline__ void pes_decode(uint32_t w, uint32_t dp, uint32_t& v, uint32_t (&mk)[4]) {
  const uint32_t nz = prmt_sign((w & CodeBits<FMT>::MM) + 0x7F7F7F7Fu, 0xBA98u);
  const uint32_t lost = prmt_sign(dp, 0xBA98u);
  v = ((w & 0x80808080u) | e5m2_pow2(dp & 0x1F1F1F1Fu)) & nz & ~lost;
  k_masks<PLANE_E5M2, Fmt<FMT>::C>(w, mk);
}

// Plane words and masks of a thread's 16 codes.
template <int FMT, bool PES>
__device__ __forceinline__ void decode_run(const uint4& cw, const uint4& dw, uint32_t (&v)[4], uint32_t (&mk)[4][4]) {
  const uint32_t w[4] = {cw.x, cw.y, cw.z, cw.w}, d[4] = {dw.x, dw.y, dw.z, dw.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if constexpr (PES)
      pes_decode<FMT>(w[i], d[i], v[i], mk[i]);
    else
      mx_decode<FMT>(w[i], v[i], mk[i]);
  }
}

// One 16-byte core-matrix row (chunk kc of the run) of every B plane the pass needs.
template <class Cfg, int PASS>
__device__ __forceinline__ void write_b_planes(uint8_t* stage, int row, int kc, const uint32_t (&v)[4],
                                               const uint32_t (&mk)[4][4]) {
  const uint32_t core = (uint32_t)((row >> 3) * 256 + kc * 128 + (row & 7) * 16);
  uint32_t pw[4][Cfg::KB > 8 ? Cfg::KB : 8];
#pragma unroll
  for (int q = 0; q < 4; ++q) PlaneFmt<Cfg::FB_>::planes(v[q], mk[q], pw[q]);
#pragma unroll
  for (int k2 = 0; k2 < Cfg::KB; ++k2) {
    const int sl = Cfg::slot(PASS, k2);
    if (sl < 0) continue;
    *reinterpret_cast<uint4*>(stage + (size_t)sl * Cfg::PLANE_BYTES + core) =
        make_uint4(pw[0][k2], pw[1][k2], pw[2][k2], pw[3][k2]);
  }
}

template <class Cfg, int PASS>
__device__ __forceinline__ void issue_pass(uint32_t leader, uint32_t tmem, uint64_t bdesc0, int abuf, int bstage,
                                           bool first_step) {
#pragma unroll
  for (int k1 = 0; k1 < Cfg::KA; ++k1)
#pragma unroll
    for (int k2 = 0; k2 < Cfg::KB; ++k2) {
      const int h = Cfg::phase(k1, k2);
      if (h / Cfg::PP != PASS) continue;
      const int sl = Cfg::slot(PASS, k2);
      const uint32_t a_t = tmem + Cfg::ACOL0 + abuf * Cfg::AU_COLS + k1 * 8;
      const uint64_t bd = bdesc0 + (uint64_t)((bstage * Cfg::BSTAGE + sl * Cfg::PLANE_BYTES) >> 4);
      const uint32_t d_t = tmem + (h - PASS * Cfg::PP) * Cfg::BN;
      const uint32_t accum = (first_step && Cfg::first_of_phase(k1, k2)) ? 0u : 1u;
      // the carry 2^c is the B factor byte c (the row's factor times 2^c)
      const uint32_t idesc = Cfg::IDESC | ((uint32_t)Cfg::carry(k1, k2) << 4);
      mma_mx_if(leader, d_t, a_t, bd, idesc, tmem + Cfg::SFA0 + abuf * 4, tmem + Cfg::SFB0 + bstage * 4, accum);
    }
}

template <class Cfg>
__device__ __forceinline__ void issue_step(uint32_t leader, int p, uint32_t tmem, uint64_t bdesc0, int abuf,
                                           int bstage, bool first_step) {
  if (p == 0) issue_pass<Cfg, 0>(leader, tmem, bdesc0, abuf, bstage, first_step);
  if (Cfg::NP > 1 && p == 1) issue_pass<Cfg, (Cfg::NP > 1 ? 1 : 0)>(leader, tmem, bdesc0, abuf, bstage, first_step);
  if (Cfg::NP > 2 && p == 2) issue_pass<Cfg, (Cfg::NP > 2 ? 2 : 0)>(leader, tmem, bdesc0, abuf, bstage, first_step);
}

}  // namespace

// The last partial wave (tiles % SMs CTAs on an otherwise idle GPU) is
// spread out: its tiles are split in K into a larger and a smaller piece
// (steps [0, split_step) and [split_step, nsub) of every pass), launched
// after the whole tiles, so the pieces of two waves' worth of work share the
// SMs.  A piece keeps its earlier passes in shared memory and adds its total
// to C with one atomic add per output; C of those tiles is zeroed first, so
// every output receives exactly two additions onto 0 and the sum does not
// depend on their order (IEEE addition is commutative).
struct TailPlan {
  int ntiles_full;  // CTAs that own a whole tile (tiles 0 .. ntiles_full - 1)
  int nsplit;       // tiles split in K (tiles ntiles_full .. + nsplit - 1)
  int split_step;   // first step of the second piece
};

// Per-element scales of both operands (PES = true; reused operands of the
// training GEMMs), written by the preparation kernels (gemm_reuse.cu):
// dp[r][k] the element's plane exponent byte (pes_decode), f[r][s] the
// exponent of step s's largest element minus 15 (INT16_MIN for a step
// without nonzero codes), ref[r] = max_s f[r][s].
struct PesOperands {
  const uint8_t* dA;
  const uint8_t* dB;
  const int16_t* fA;
  const int16_t* fB;
  const int* refA;
  const int* refB;
};

// Thread layout: warps 0 .. NAW-1 produce A (warp w: TMEM lane group w & 3,
// share w >> 2 of each 32-byte run: NWA columns per plane) and run the
// epilogue (columns [BN/ATPR share, BN/ATPR (share + 1))); the next 2 BN
// threads produce B (thread 32 NAW + t: row t % BN, half t / BN); the last
// warp allocates TMEM and issues the factor copies and the MMAs.
template <int FA, int FB, bool PES>
__global__ void __launch_bounds__(TcCfg<FA, FB>::THREADS, 1)
    gemm_tc_kernel(const uint8_t* __restrict__ A, const int8_t* __restrict__ sA, const uint8_t* __restrict__ B,
                   const int8_t* __restrict__ sB, int M, int N, int K, int G, int gshift, float* __restrict__ C,
                   uint32_t* status, const PesOperands pes, const TailPlan plan) {
  using Cfg = TcCfg<FA, FB>;
  constexpr int L = Cfg::L, PP = Cfg::PP, NP = Cfg::NP, BN = Cfg::BN, NSB = Cfg::NSB;
  constexpr int NAW = Cfg::NAW, NWA = Cfg::NWA, ATPR = Cfg::ATPR;
  static_assert(NP <= 3, "pass dispatch");
  static_assert(NSB == TC_MAX_RING && Cfg::NAU == 2, "barrier rings");
  static_assert(NWA == 4, "16-byte runs per producer thread");
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* bstage = smem;
  TcShared& sh = *reinterpret_cast<TcShared*>(smem + (size_t)NSB * Cfg::BSTAGE);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // this CTA's job: a whole tile, or one K piece of a tail tile
  const int ntn = (N + BN - 1) / BN;
  int tile = blockIdx.x, s0 = 0, s1 = K / Cfg::KS;
  const bool split = tile >= plan.ntiles_full;
  if (split) {
    const int q = tile - plan.ntiles_full;
    if (q < plan.nsplit) {
      tile = plan.ntiles_full + q;
      s1 = plan.split_step;
    } else {
      tile = plan.ntiles_full + q - plan.nsplit;
      s0 = plan.split_step;
    }
  }
  const int m0 = (tile / ntn) * Cfg::BM, n0 = (tile % ntn) * BN;
  const int nb = K / G, nsub = s1 - s0, total = NP * nsub;  // nsub: this job's steps per pass
  float* stash = reinterpret_cast<float*>(smem + (size_t)NSB * Cfg::BSTAGE + 2048);

  if (tid == 0) {
    for (int s = 0; s < NSB; ++s) {
      tc::mbar_init(&sh.full[s], NAW + Cfg::NBT / 32);  // one arrival per producer warp
      tc::mbar_init(&sh.empty[s], 1);
    }
    tc::mbar_init(&sh.acc_full, 1);
    tc::mbar_init(&sh.drain, 1);
    sh.abort_flag = 0;
  }
  if (warp == Cfg::MMA_WARP) {
    // TMEM allocation and release are warp-collective (.sync.aligned): the
    // MMA warp reaches them, and every wait of its loop (whole-warp waits),
    // with all 32 lanes together
    __syncwarp();
    tc::tmem_alloc(&sh.tmem_base, 512);
    tc::tmem_relinquish();
  }
  // producer geometry and the row's reference exponent (largest block scale)
  const bool is_a = warp < NAW;
  const bool is_prod = warp < Cfg::MMA_WARP;
  const int rloc = is_a ? ((warp & 3) * 32 + lane) : ((tid - NAW * 32) % BN);
  const int part = is_a ? (warp >> 2) : ((tid - NAW * 32) / BN);  // share of the 32-byte run
  const int r = (is_a ? m0 : n0) + rloc;
  const bool rowok = is_prod && r < (is_a ? M : N);
  int ref = -128;
  if constexpr (PES) {
    if (rowok) ref = __ldg(is_a ? pes.refA + r : pes.refB + r);
    if (!is_a && is_prod && part == 0) sh.refB[rloc] = ref;
  } else {
    // the references of the tile's A and B rows, formed by all threads from
    // the two contiguous runs of scale rows (-128 past the ends)
    if (tid < 128) {
      sh.wref[tid] = -128;
      sh.refB[tid] = -128;
    }
    __syncthreads();
    rows_ref_coop(sA + (int64_t)m0 * nb, min(Cfg::BM, M - m0), nb, sh.wref, tid, Cfg::THREADS);
    rows_ref_coop(sB + (int64_t)n0 * nb, min(BN, N - n0), nb, sh.refB, tid, Cfg::THREADS);
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if constexpr (!PES) {
    if (rowok) ref = is_a ? sh.wref[rloc] : sh.refB[rloc];
  }
  const uint32_t tmem = sh.tmem_base;

  if (is_prod) {
    // ------------------------------ producers ------------------------------
    const uint8_t* src = (is_a ? A : B) + (int64_t)r * K + part * 16;
    const uint8_t* dsrc = PES ? (is_a ? pes.dA : pes.dB) + (int64_t)r * K + part * 16 : nullptr;
    const int8_t* srow = PES ? nullptr : (is_a ? sA : sB) + (int64_t)r * nb;
    const int16_t* frow = PES ? (is_a ? pes.fA : pes.fB) + (int64_t)r * (K / Cfg::KS) : nullptr;
    auto pass_of = [&](int g) { return (NP > 1 && g >= nsub ? 1 : 0) + (NP > 2 && g >= 2 * nsub ? 1 : 0); };
    // codes (16 bytes), per-element exponent bytes (PES) and the step's raw
    // scale (block scale, or the PES step exponent)
    auto load = [&](int g, uint4& cw, int& raw, uint4& dw) {
      cw = make_uint4(0, 0, 0, 0);
      dw = make_uint4(0, 0, 0, 0);
      raw = -32768;
      if (rowok && g < total) {
        const int s = s0 + g - pass_of(g) * nsub;  // step of the whole K
        cw = __ldg(reinterpret_cast<const uint4*>(src + (int64_t)s * Cfg::KS));
        if (PES) {
          dw = __ldg(reinterpret_cast<const uint4*>(dsrc + (int64_t)s * Cfg::KS));
          raw = (int)__ldg(frow + s);
        } else {
          raw = (int)__ldg(srow + (s >> gshift));
        }
      }
    };
    const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    // The epilogue of pass pe (A producers, after the pass's last MMA): each
    // 8-column chunk of this thread's share is read from TMEM, combined over
    // the pass's phases and added to the running total in the FP32 stash (row
    // stride BN + 4 floats: the 16-byte accesses of a warp's 32 rows hit
    // distinct banks).  The last pass writes the total to C once: stored for
    // a whole tile, added atomically to zeroed C for a K piece (two pieces
    // per output).  The total is ((y_0 + y_1) + y_2) in FP32 in every case.
    auto epilogue = [&](const int pe) -> bool {
      const bool ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.acc_full, pe & 1));
      if (!ok) {
        raise_flag(status, CURVEFP_DEV_TIMEOUT);
        sh.abort_flag = 1;
      }
      tc::fence_after_sync();
      float* strow = stash + rloc * Cfg::SST;
#pragma unroll 1
      for (int c0 = part * (BN / ATPR); c0 < (part + 1) * (BN / ATPR); c0 += 8) {
        uint32_t acc[PP][8];
#pragma unroll
        for (int q = 0; q < PP; ++q)
          if (pe * PP + q < L) tc::tmem_ld8(lane_base + q * BN + c0, acc[q]);
        tc::tmem_wait_ld();
        if (rowok && ok) {
          float y[8];
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            float t = 0.f;
#pragma unroll
            for (int q = 0; q < PP; ++q)
              if (pe * PP + q < L) t = fmaf(phase_const(L, pe * PP + q), __uint_as_float(acc[q][c]), t);
            y[c] = scale_pow2(t, ref + sh.refB[c0 + c] - 2 * MX_OFF);
          }
          float4* s4 = reinterpret_cast<float4*>(strow + c0);
          if (pe > 0) {
            const float4 b0 = s4[0], b1 = s4[1];
            y[0] = b0.x + y[0]; y[1] = b0.y + y[1]; y[2] = b0.z + y[2]; y[3] = b0.w + y[3];
            y[4] = b1.x + y[4]; y[5] = b1.y + y[5]; y[6] = b1.z + y[6]; y[7] = b1.w + y[7];
          }
          s4[0] = make_float4(y[0], y[1], y[2], y[3]);
          s4[1] = make_float4(y[4], y[5], y[6], y[7]);
        }
      }
      if (pe == NP - 1 && rowok && ok) {
#pragma unroll 1
        for (int c0 = part * (BN / ATPR); c0 < (part + 1) * (BN / ATPR); c0 += 8) {
          const float4* s4 = reinterpret_cast<const float4*>(strow + c0);
          const float4 a0 = s4[0], a1 = s4[1];
          float* dst = C + (int64_t)r * N + n0 + c0;
          if (split) {
            const float y[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
            for (int c = 0; c < 8; ++c)
              if (n0 + c0 + c < N) atomicAdd(dst + c, y[c]);
          } else if (n0 + c0 + 8 <= N && ((reinterpret_cast<uintptr_t>(dst) & 15) == 0)) {
            reinterpret_cast<float4*>(dst)[0] = a0;
            reinterpret_cast<float4*>(dst)[1] = a1;
          } else {
            const float y[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
            for (int c = 0; c < 8; ++c)
              if (n0 + c0 + c < N) dst[c] = y[c];
          }
        }
      }
      return ok;
    };
    // One pipeline step of this producer thread; false ends the loop (abort).
    auto step = [&](const int g, uint4 cw, const int raw, const uint4 dw) -> bool {
      // the step's scale factor relative to the row reference; a block too
      // far below it to have a factor byte is dropped
      bool keep = raw != -32768;
      uint32_t sf = 0;
      if (keep) sf = mx_sf(raw - ref, 0, keep);
      if (!keep) cw = make_uint4(0, 0, 0, 0);
      const int p = pass_of(g), s = g - p * nsub;
      uint32_t v[4], mk[4][4];
      if (is_a)
        decode_run<FA, PES>(cw, dw, v, mk);
      else
        decode_run<FB, PES>(cw, dw, v, mk);
      if (is_a) {
        uint32_t pl[4][Cfg::KA > 8 ? Cfg::KA : 8];
#pragma unroll
        for (int c = 0; c < 4; ++c) PlaneFmt<FA>::planes(v[c], mk[c], pl[c]);
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
        // plane k1 occupies 8 columns of the unit; this thread's share of
        // the 32-byte run is columns 4 part .. 4 part + 3
#pragma unroll
        for (int j = 0; j < Cfg::KA; ++j) {
          const uint32_t reg[4] = {pl[0][j], pl[1][j], pl[2][j], pl[3][j]};
          tc::tmem_st4(lane_base + Cfg::ACOL0 + buf * Cfg::AU_COLS + j * 8 + part * NWA, reg);
        }
        // the row's factor (quadrant q reads column q of the unit's four)
        if (part == 0) tc::tmem_st1(lane_base + Cfg::SFA0 + buf * 4 + (warp & 3), sf * 0x01010101u);
        tc::tmem_wait_st();
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&sh.full[g % NSB]);

        // the pass's epilogue after its last step (a one-trip loop: this form
        // measured faster than a plain call in the unrolled step pairs)
        const int pe_last = s == nsub - 1 ? p : -1;
#pragma unroll 1
        for (int pe = p; pe <= pe_last; ++pe)
          if (!epilogue(pe)) return false;
      } else {
        const int st = g % NSB;
        bool fail = false;
        if (g >= NSB) fail = !__all_sync(0xffffffffu, tc::mbar_wait(&sh.empty[st], ((g / NSB) - 1) & 1));
        if (fail) {
          if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
          return false;
        }
        uint8_t* stg = bstage + (size_t)st * Cfg::BSTAGE;
        if (p == 0) write_b_planes<Cfg, 0>(stg, rloc, part, v, mk);
        if (NP > 1 && p == 1) write_b_planes<Cfg, (NP > 1 ? 1 : 0)>(stg, rloc, part, v, mk);
        if (NP > 2 && p == 2) write_b_planes<Cfg, (NP > 2 ? 2 : 0)>(stg, rloc, part, v, mk);
        // factor bytes of the row: byte 0 plain, byte 1 the carry's 2x
        if (part == 0)
          *reinterpret_cast<uint32_t*>(stg + Cfg::MAXS * Cfg::PLANE_BYTES + sfb_off(rloc)) =
              keep ? (sf | (sf + 1) << 8) : 0u;
        tc::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&sh.full[st]);
      }
      return true;
    };
    // PF register sets of codes, each loaded PF steps before it is used and
    // never copied, so that no register move waits on an in-flight load.  Two
    // sets where the operands stay in L2 (the codes of one step arrive in
    // less than two steps); four for the per-element-scale operands and for
    // A with four planes (the mixed pairs of the training GEMMs), whose
    // large-K shapes miss L2 and whose short steps leave the loads exposed.
    if constexpr (PES || Cfg::KA == 4) {
      constexpr int PF = 4;
      uint4 q[PF], dq[PF];
      int rq[PF];
#pragma unroll
      for (int u = 0; u < PF; ++u) load(u, q[u], rq[u], dq[u]);
      bool run = true;
      for (int g = 0; g < total && run; g += PF) {
#pragma unroll
        for (int u = 0; u < PF; ++u) {
          if (g + u >= total || !step(g + u, q[u], rq[u], dq[u])) {
            run = false;
            break;
          }
          load(g + u + PF, q[u], rq[u], dq[u]);
        }
      }
    } else {
      uint4 q0, q1, d0, d1;
      int r0, r1;
      load(0, q0, r0, d0);
      load(1, q1, r1, d1);
      for (int g = 0; g < total; g += 2) {
        if (!step(g, q0, r0, d0)) break;
        load(g + 2, q0, r0, d0);
        if (g + 1 >= total) break;
        if (!step(g + 1, q1, r1, d1)) break;
        load(g + 3, q1, r1, d1);
      }
    }
  } else {
    // ------------------------------ MMA issuer -------------------------------
    // The whole warp runs the loop; the elected lane copies the stage's B
    // factors into TMEM, issues the MMAs and commits.
    const uint32_t leader = tc::elect_one();
    const uint64_t bdesc0 = tc::smem_desc(tc::smem_u32(bstage), 128, 256);
    bool ok = true;
    for (int g = 0; g < total && ok; ++g) {
      const int p = (NP > 1 && g >= nsub ? 1 : 0) + (NP > 2 && g >= 2 * nsub ? 1 : 0), s = g - p * nsub;
      const int st = g % NSB;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.full[st], (g / NSB) & 1));
      // a producer that gave up also stops arriving, so the wait above ends
      // the loop anyway; the flag only shortens that, and is read rarely
      // because every cycle of this loop delays the next MMA
      if ((g & 7) == 0) ok = ok && !read_abort(&sh.abort_flag);
      if (!ok) break;
      tc::fence_after_sync();
      tmem_cp_sf_if(leader, tmem + Cfg::SFB0 + st * 4,
                    bstage + (size_t)st * Cfg::BSTAGE + Cfg::MAXS * Cfg::PLANE_BYTES);
      issue_step<Cfg>(leader, p, tmem, bdesc0, g & 1, st, s == 0);
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
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

// Which tiles to split, and where.  The launch order (whole tiles, then the
// first pieces, then the second pieces) is dispatched greedily to the SMs as
// they free; the plan is the one whose simulated makespan is smallest over
// the last s = T mod P (+ P, + 2P) tiles split at 1/2, 2/3 or 3/4 of K (a
// piece costs its share of a tile's steps plus a small fixed overhead, so a
// split must gain more than that).  At the headline shape (688 tiles, 152
// SMs) this is the 80 tail tiles at 2/3: 4.67 instead of 5 waves.
inline double tail_makespan(int64_t tiles, int sms, int64_t s, double x) {
  const double ovh = 0.02;  // per-piece overhead, in tiles
  // after the whole tiles, (tiles - s) mod P SMs carry one tile more
  const int64_t w = tiles - s, base = w / sms, extra = w % sms;
  std::priority_queue<double, std::vector<double>, std::greater<double>> q;
  for (int i = 0; i < sms; ++i) q.push((double)(base + (i < extra ? 1 : 0)));
  auto run = [&](int64_t n, double d) {
    for (int64_t i = 0; i < n; ++i) {
      const double t = q.top();
      q.pop();
      q.push(t + d);
    }
  };
  run(s, x + ovh);
  run(s, 1.0 - x + ovh);
  double m = 0.0;
  while (!q.empty()) {
    m = q.top() > m ? q.top() : m;
    q.pop();
  }
  return m;
}

inline TailPlan tail_plan_search(int64_t tiles, int sms, int nsub) {
  TailPlan best{(int)tiles, 0, 0};
  if (sms <= 0 || tiles < sms || nsub < 2 || tiles % sms == 0) return best;
  double best_m = tail_makespan(tiles, sms, 0, 0.5);
  const double xs[3] = {0.5, 2.0 / 3.0, 0.75};
  for (int64_t s = tiles % sms; s <= tiles && s <= tiles % sms + 2 * (int64_t)sms; s += sms)
    for (double x : xs) {
      const int split = (int)(x * nsub + 0.5);
      if (split < 1 || split >= nsub) continue;
      const double m = tail_makespan(tiles, sms, s, (double)split / nsub);
      if (m < best_m - 1e-9) {
        best_m = m;
        best = TailPlan{(int)(tiles - s), (int)s, split};
      }
    }
  return best;
}

// The plan of a shape is searched once per process (a few hundred
// microseconds of host time) and remembered.
inline TailPlan tail_plan(int64_t tiles, int sms, int nsub) {
  static std::mutex mu;
  static std::unordered_map<uint64_t, TailPlan> memo;
  const uint64_t key = ((uint64_t)tiles << 32) ^ ((uint64_t)sms << 16) ^ (uint64_t)nsub;
  {
    std::lock_guard<std::mutex> lk(mu);
    auto it = memo.find(key);
    if (it != memo.end()) return it->second;
  }
  const TailPlan t = tail_plan_search(tiles, sms, nsub);
  std::lock_guard<std::mutex> lk(mu);
  memo[key] = t;
  return t;
}

template <int FA, int FB, bool PES>
static cudaError_t launch_tc_t(int G, const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb,
                               int64_t M, int64_t N, int64_t K, float* c, uint32_t* st, cudaStream_t s,
                               const PesOperands& pes, int sms) {
  using Cfg = TcCfg<FA, FB>;
  static_assert(sizeof(TcShared) <= 2048, "shared tail");
  static_assert(Cfg::SMEM <= 227 * 1024, "shared memory");
  auto kern = gemm_tc_kernel<FA, FB, PES>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::SMEM);
  if (e != cudaSuccess) return e;
  const int64_t ntn = (N + Cfg::BN - 1) / Cfg::BN, ntm = (M + Cfg::BM - 1) / Cfg::BM;
  const TailPlan plan = tail_plan(ntn * ntm, sms, (int)(K / Cfg::KS));
  if (plan.nsplit > 0) {
    // C of the split tiles starts at zero: whole tile rows from the first one
    const int64_t row0 = (plan.ntiles_full / ntn) * Cfg::BM;
    e = cudaMemsetAsync(c + row0 * N, 0, (size_t)((M - row0) * N) * sizeof(float), s);
    if (e != cudaSuccess) return e;
  }
  const unsigned grid = (unsigned)(plan.ntiles_full + 2 * plan.nsplit);
  int gshift = 0;  // scale block of step s is s >> gshift (G / KS is a power of two)
  while ((Cfg::KS << gshift) < G) ++gshift;
  kern<<<grid, Cfg::THREADS, Cfg::SMEM, s>>>(a, sa, b, sb, (int)M, (int)N, (int)K, G, gshift, c, st, pes, plan);
  return cudaGetLastError();
}

}  // namespace cfp
