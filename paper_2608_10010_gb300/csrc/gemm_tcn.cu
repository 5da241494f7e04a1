// Tensor-core closed-product GEMM with the phases along the MMA's N dimension
// (algo TENSOR_NARROW): Sec. 3.2, Eq. 2, Eq. 5.
//
// C = X_hat W_hat^T with X the M activation rows (the API's A operand, format
// FX) and W the N weight rows (the API's B operand, format FW).  As in the
// tile kernel, every operand splits into curve planes of exact powers of two
// (plane k holds the elements of curve index k), and plane k_x of X times
// plane k_w of W lands on phase h = (k_x WX + k_w WW) mod L with carry
// c = floor((k_x WX + k_w WW) / L) (Eq. 2 on the shared lattice L).
//
// Here the weight rows are the MMA's 128-row TMEM operand and the phase is a
// column index: the accumulator of a token group is D[w][h Mt + m] (weight
// row w, phase h, token m of the group's Mt tokens), the per-phase sums S_h
// of Eq. 5 for every token side by side.  For weight plane k_w the
// shared-memory operand must hold, in column block h, the X plane with
// k_x WX = (h - k_w WW) mod L, doubled where the sum wrapped (carry).  Lay
// out the sequence of 2L column blocks
//   Q = [ 2 X_0 ... (lattice positions 0 .. L-1, carry copies) |
//           X_0 ... (lattice positions 0 .. L-1, plain) ]
// (block u of each half holds the plane with k_x WX = u, zero where no plane
// sits on u); then the operand of weight plane k_w is the window of L blocks
// that starts at block L - k_w WW: its block h is plain for h >= k_w WW and
// the carry copy of position L - k_w WW + h otherwise.  A window is a start
// address of the MMA's shared-memory descriptor, so a pipeline step of 32
// codes costs K_W MMAs of 128 x (L Mt) x 32 on 2L Mt staged rows, against
// K_X K_W MMAs of the tile kernel.
//
// Same-format pairs (WX = WW = 1) use 2:4-sparse pair planes: an element sits
// in one plane, so weight planes j and j + K/2 share one compressed operand at
// logical positions 2k and 2k + 1, with one curve-index bit as metadata; the
// activation side stores R_b[2k] = Q_b[k], R_b[2k + 1] = Q_{b - K/2}[k] and
// the operand of pair j is the window from R block L - j: K/2 sparse MMAs of
// logical K 64 per step, half the MMAs and half the TMEM bytes.  From 512
// activation rows a CTA takes two token groups (accumulators side by side,
// a three-step ring), so each decoded weight step serves twice the tokens.
//
// Roles (15 warps for 8-phase pairs, 17 for E5C2 x E5C2; a step is short,
// so producer groups take turns):
//   warps 0-7   W producers: two groups of 4 warps taking alternate steps,
//               one thread per weight row (all 32 codes of its steps): codes
//               -> planes (pair planes and metadata) -> TMEM, prefetching
//               PFW own steps ahead; after the last step they run the
//               epilogue.
//   next warps  X producers: groups taking every NGX-th step, one 4-code word
//               of one token per work item -> the step's blocks (Q or R),
//               conflict-free stores; padding tokens are never written (the
//               stages start at zero).
//   last warp   TMEM allocation and MMA issue (one elected lane).
// With fewer weight tiles than fill the SMs' last wave, tiles are split in K
// into two pieces (the tile kernel's greedy-dispatch simulation, extended to
// grids smaller than the SM count); a piece adds its outputs to zeroed C
// atomically, two additions per output, so the result does not depend on
// their order.  Every wait is bounded.
#include "gemm_tc.cuh"

namespace cfp {

namespace {

template <int FX, int FW, bool T2>
struct TcnCfg {
  using P = Pair<FX, FW>;
  static constexpr int KW = Fmt<FW>::K, L = P::L, WX = P::WA, WW = P::WB;
  static constexpr int BM = 128;          // weight rows per CTA (TMEM lanes)
  static constexpr int KS = 32;           // codes per pipeline step (K of one FP8 MMA)
  static constexpr int MTMAX = 256 / L;   // tokens per CTA: L Mt <= 256 (MMA N)
  static constexpr int NBLK = 2 * L;      // column blocks of the doubled sequence
  static constexpr bool SP = FX == FW;     // 2:4-sparse pair planes (below)
  static constexpr bool TWO = SP && T2;    // two token groups per CTA (below)
  // pipeline depth (X stages = W TMEM units): three where TMEM also holds two
  // token groups' accumulators
  static constexpr int NSB = TWO ? 3 : 4;
  // Same-format pairs use 2:4-sparse pair planes: weight planes j and j + HB
  // share one compressed operand (an element sits in one plane), at logical
  // positions 2k and 2k + 1, with the curve-index bit MBIT as metadata.
  static constexpr int HB = KW / 2, MBIT = KW == 8 ? 2 : 1;
  static constexpr int NJ = SP ? HB : KW;  // A operands (MMAs) per step
  static constexpr int AU_COLS = NJ * 8;  // TMEM columns of one step's W planes
  // A CTA takes one token group of Mt <= MTMAX tokens or (TWO: sparse form,
  // large M) two groups of Mt <= MT2 with their accumulators side by side, so
  // each decoded weight step serves up to 2 MT2 tokens.
  static constexpr int MT2 = TWO ? 192 / L : 0;
  static constexpr int MTOK = TWO ? 2 * MT2 : MTMAX;  // tokens per CTA at most
  static constexpr int ACOL0 = TWO ? 384 : 256;       // W units after the accumulators
  static constexpr int MCOL0 = ACOL0 + NSB * AU_COLS;  // metadata of unit u at MCOL0 + 8 u (2 used)
  static_assert(MCOL0 + (SP ? NSB * 8 : 0) <= 512, "TMEM budget");
  // sparse form: R blocks RB0 .. 2L-1 of 64-byte rows, R_b[2k] = Q_b[k],
  // R_b[2k + 1] = Q_{b - HB}[k]; the operand of pair j is the window of L
  // blocks from block L - j
  static constexpr int RB0 = L - HB + 1, NRB = L + HB - 1;
  static constexpr int ROWB = SP ? 64 : 32;  // bytes of one operand row
  static_assert(L % 4 == 0 && KW % 2 == 0, "epilogue phase groups, plane pairs");
  // Producer groups take turns: W group g % NGW and X group g % NGX produce
  // step g, so each producer thread has NGW (NGX) steps of time per step.
  static constexpr int NGW = 2;                 // W groups of 4 warps (one thread per weight row)
  static constexpr int XPG = MTMAX / 16;        // X warps per group
  static constexpr int NGX = L == 8 ? 3 : 2;    // X groups
  static constexpr int NWT = NGW * 128;         // W threads
  static constexpr int NXT = NGX * XPG * 32;    // X threads
  static constexpr int THREADS = NWT + NXT + 32;
  static constexpr int MMA_WARP = (NWT + NXT) / 32;
  static constexpr int BSTAGE = (SP ? NRB * MTOK : NBLK * MTMAX) * ROWB;  // bytes of one step's X operand rows
  static constexpr int PBX = FX == CURVEFP_E5C2 ? 1 : 0;  // plane exponent bias
  static constexpr int PBW = FW == CURVEFP_E5C2 ? 1 : 0;
  static constexpr int PFW = 4;  // own steps of weight codes in flight per W thread
  static constexpr int PFX = 2;  // own steps of activation codes in flight per X thread
  static constexpr int XI = MTOK * 8 / (XPG * 32);  // X work items (4-code words) per thread and step
  // more than half of the SM's shared memory: one CTA per SM (the split plan
  // assumes it, and the CTA allocates all of TMEM)
  static constexpr size_t SMEM_USED = (size_t)NSB * BSTAGE + 2048;
  static constexpr size_t SMEM = SMEM_USED > 120 * 1024 ? SMEM_USED : 120 * 1024;
};

// Byte offset of row `row`, 16-byte chunk `kc` (of two) in a K-major
// no-swizzle stage: 8-row core-matrix groups of 256 bytes.
__device__ __forceinline__ uint32_t core_off(int row, int kc) {
  return (uint32_t)((row >> 3) * 256 + kc * 128 + (row & 7) * 16);
}

// Largest block scale of a row (the row reference of the plane values).
__device__ __forceinline__ int row_ref(const int8_t* s, int nb) {
  int ref = -128;
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
  return ref;
}

// Metadata word of 16 codes (four code words) of a 2:4 operand with 8-bit
// elements: per chunk of two elements, position bit(2c) and 2 + bit(2c + 1),
// where bit is the curve-index bit MBIT that selects the partner plane.
template <int MBIT>
__device__ __forceinline__ uint32_t pair_meta(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3) {
  const uint32_t w[4] = {w0, w1, w2, w3};
  uint32_t m = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint32_t t = (w[q] >> MBIT) & 0x01010101u;  // bit of element i at 8 i
    m |= (((t * 0x01041040u) >> 24) | 0x88u) << (8 * q);  // ... at 2 i, plus bit 3 of each nibble
  }
  return m;
}

// 2:4-sparse MMA (kind::f8f6f4), A and metadata in TMEM, issued by `leader`.
__device__ __forceinline__ void mma_sp_if(uint32_t leader, uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                          uint32_t meta_tmem, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.b32 p, %5, 0;\n setp.ne.b32 q, %6, 0;\n"
      "@q tcgen05.mma.sp.cta_group::1.kind::f8f6f4 [%0], [%1], %2, [%3], %4, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(meta_tmem), "r"(idesc), "r"(accumulate), "r"(leader)
      : "memory");
}

// Interleave two words (elements 4q..4q+3 each) into X0 Y0 X1 Y1 | X2 Y2 X3 Y3.
__device__ __forceinline__ uint2 interleave2(uint32_t x, uint32_t y) {
  return make_uint2(__byte_perm(x, y, 0x5140), __byte_perm(x, y, 0x7362));
}

__device__ __forceinline__ bool wait_all(uint64_t* bar, uint32_t parity) {
  return __all_sync(0xffffffffu, tc::mbar_wait(bar, parity));
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

}  // namespace

template <int FX, int FW, bool T2>
__global__ void __launch_bounds__(TcnCfg<FX, FW, T2>::THREADS, 1)
    gemm_tcn_kernel(const uint8_t* __restrict__ X, const int8_t* __restrict__ sX, const uint8_t* __restrict__ W,
                    const int8_t* __restrict__ sW, int M, int N, int K, int G, int gshift, int Mt, int ntg,
                    float* __restrict__ C, uint32_t* status, const TailPlan plan) {
  using Cfg = TcnCfg<FX, FW, T2>;
  constexpr int L = Cfg::L, NSB = Cfg::NSB;
  static_assert(NSB <= TC_MAX_RING && Cfg::MTOK <= 128, "barrier rings, row references");
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* xstage = smem;
  TcShared& sh = *reinterpret_cast<TcShared*>(smem + (size_t)NSB * Cfg::BSTAGE);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // this CTA's job: a whole tile (128 weight rows x Mt tokens) or one K piece
  const int ntw = (N + Cfg::BM - 1) / Cfg::BM;
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
  const int ntok = ntg * Mt;  // tokens of the CTA: ntg groups of Mt
  const int x0 = (tile / ntw) * ntok, w0 = (tile % ntw) * Cfg::BM;
  const int nb = K / G, total = s1 - s0;
  // Accumulator copies: consecutive MMAs of a step into one accumulator wait
  // for each other's accumulation, so where the accumulator is at most 128
  // columns the weight planes rotate over 2 or 4 copies (NP columns each)
  // that the epilogue adds up.
  const int NP = L * Mt, nacc0 = ntg > 1 ? 1 : (NP <= 64 ? 4 : (NP <= 128 ? 2 : 1));
  const int nacc = nacc0 < Cfg::NJ ? nacc0 : Cfg::NJ;  // every copy receives an MMA each step

  if (tid == 0) {
    for (int s = 0; s < NSB; ++s) {
      tc::mbar_init(&sh.full[s], 4 + Cfg::XPG);  // the step's W group and X group, one arrival per warp
      tc::mbar_init(&sh.empty[s], 1);
    }
    tc::mbar_init(&sh.acc_full, 1);
    tc::mbar_init(&sh.drain, 1);
    sh.abort_flag = 0;
  }
  if (warp == Cfg::MMA_WARP) {
    tc::tmem_alloc(&sh.tmem_base, 512);
    tc::tmem_relinquish();
  }
  const bool is_w = tid < Cfg::NWT, is_x = !is_w && warp < Cfg::MMA_WARP;
  // W threads: weight row (TMEM lane) and group; X threads: group.  The
  // row references: a weight row per W thread, a token per thread of the
  // first X group.  The X stages start at zero (padding tokens and empty
  // lattice positions are never written).
  const int wrow = w0 + (warp & 3) * 32 + lane, gw = warp >> 2;
  const int t_x = tid - Cfg::NWT, gx = t_x / (Cfg::XPG * 32);
  int ref = -128;
  if (is_w && wrow < N) ref = row_ref(sW + (int64_t)wrow * nb, nb);
  if (is_x && t_x < Cfg::MTOK) {
    int rx = -128;
    if (t_x < ntok && x0 + t_x < M) rx = row_ref(sX + (int64_t)(x0 + t_x) * nb, nb);
    sh.refB[t_x] = rx;
  }
  for (int o = tid * 16; o < NSB * Cfg::BSTAGE; o += Cfg::THREADS * 16)
    *reinterpret_cast<uint4*>(xstage + o) = make_uint4(0, 0, 0, 0);
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;

  if (is_w) {
    // ---------------------------- W producers -----------------------------
    constexpr int PF = Cfg::PFW, NGW = Cfg::NGW;
    const bool rowok = wrow < N;
    const uint8_t* src = W + (int64_t)wrow * K;
    const int8_t* srow = sW + (int64_t)wrow * nb;
    // own step i of this group is pipeline step g = gw + i NGW
    auto load = [&](int i, uint4& lo, uint4& hi, int& raw) {
      lo = hi = make_uint4(0, 0, 0, 0);
      raw = 0;
      const int g = gw + i * NGW;
      if (rowok && g < total) {
        const int s = s0 + g;
        const uint4* p = reinterpret_cast<const uint4*>(src + (int64_t)s * Cfg::KS);
        lo = __ldg(p);
        hi = __ldg(p + 1);
        raw = (int)__ldg(srow + (s >> gshift));
      }
    };
    const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    // The hand-over of an own step (wait for its TMEM stores, arrive) is
    // deferred until the next own step is decoded, so the store latency
    // overlaps the decode; the step before is still at least two steps
    // ahead of the empty wait that could depend on it.
    int pend = -1;  // stage of the own step not yet handed over
    auto hand_over = [&]() {
      if (pend < 0) return;
      tc::tmem_wait_st();
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&sh.full[pend]);
      pend = -1;
    };
    auto step = [&](const int g, const uint4 lo, const uint4 hi, const int raw) -> bool {
      const int st = g % NSB, off = raw - ref - Cfg::PBW;
      // the 32 codes of the row's step: value words and curve-index masks;
      // plane j of word w = p[w][j & 3] & (bit 2 of k set ? mk2 : ~mk2)
      uint32_t p[8][4], m2[8];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        uint32_t v[4], vc[4], mk[4][4];
        PlaneFmt<FW>::template decode<PLANE_E5M2, 4>(h ? hi : lo, off, v, vc, mk, false);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int w = h * 4 + c;
          p[w][0] = v[c] & ~mk[c][0] & ~mk[c][1];
          p[w][1] = v[c] & mk[c][0] & ~mk[c][1];
          p[w][2] = v[c] & ~mk[c][0] & mk[c][1];
          p[w][3] = v[c] & mk[c][0] & mk[c][1];
          m2[w] = mk[c][2];
        }
      }
      hand_over();
      if (g >= NSB) {
        // TMEM unit st is free once the MMAs of step g - NSB retired
        const bool ok = wait_all(&sh.empty[st], ((g / NSB) - 1) & 1);
        tc::fence_after_sync();
        if (!ok) {
          if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
          return false;
        }
      }
      // operands 2jp and 2jp + 1 of the step: 16 consecutive columns of the
      // unit.  Dense: plane j.  Sparse: pair plane j = the elements whose
      // curve index is j or j + HB (low bits of k equal to j), plus the
      // metadata words of codes 0-15 and 16-31.
#pragma unroll
      for (int jp = 0; jp < Cfg::NJ / 2; ++jp) {
        uint32_t r[16];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int j = 2 * jp + e;
#pragma unroll
          for (int w = 0; w < 8; ++w) {
            if constexpr (!Cfg::SP)
              r[e * 8 + w] = p[w][j & 3] & ((j & 4) ? m2[w] : ~m2[w]);
            else if constexpr (Cfg::KW == 8)
              r[e * 8 + w] = p[w][j];
            else
              r[e * 8 + w] = p[w][j] | p[w][j + 2];
          }
        }
        tmem_st16(lane_base + Cfg::ACOL0 + st * Cfg::AU_COLS + jp * 16, r);
      }
      if constexpr (Cfg::SP) {
        const uint32_t mt[2] = {pair_meta<Cfg::MBIT>(lo.x, lo.y, lo.z, lo.w), pair_meta<Cfg::MBIT>(hi.x, hi.y, hi.z, hi.w)};
        tc::tmem_st2(lane_base + Cfg::MCOL0 + st * 8, mt);
      }
      pend = st;
      return true;
    };
    // PF register sets of codes, each loaded PF own steps before its use and
    // never copied (no register move waits on an in-flight load)
    const int nown = (total - gw + NGW - 1) / NGW;
    uint4 ql[PF], qh[PF];
    int rq[PF];
#pragma unroll
    for (int u = 0; u < PF; ++u) load(u, ql[u], qh[u], rq[u]);
    bool run = true, failed = false;
    for (int i = 0; i < nown && run; i += PF) {
#pragma unroll
      for (int u = 0; u < PF; ++u) {
        if (i + u >= nown) {
          run = false;
          break;
        }
        if (!step(gw + (i + u) * NGW, ql[u], qh[u], rq[u])) {
          run = false;
          failed = true;
          break;
        }
        load(i + u + PF, ql[u], qh[u], rq[u]);
      }
    }
    if (!failed) hand_over();
    // Epilogue (after the last MMA): chunks of 8 tokens, chunk ch taken by
    // group ch % NGW; per token the phase sums D[w][h Mt + m] are combined as
    // sum_h 2^{h/L} S_h (FP32, phase order) and scaled by 2^{ref_w + ref_m}.
    // A whole tile stores C, a K piece adds to zeroed C.
    const bool aborted = __any_sync(0xffffffffu, read_abort(&sh.abort_flag) != 0);
    const bool ok = !aborted && wait_all(&sh.acc_full, 0);
    if (!ok && lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
    tc::fence_after_sync();
#pragma unroll 1
    for (int ch = gw; ch < (ntok >> 3); ch += NGW) {
      // chunk ch: tokens 8 ch .. 8 ch + 7 of token group tgp (local lt ..)
      const int tgp = (ch * 8) / Mt, lt = ch * 8 - tgp * Mt;
      float t[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) t[j] = 0.f;
#pragma unroll
      for (int h0 = 0; h0 < L; h0 += 4) {
        // S_h = the sum of the accumulator copies (copy order fixed)
        float sh4[4][8];
#pragma unroll 1
        for (int a = 0; a < nacc; ++a) {
          uint32_t acc[4][8];
#pragma unroll
          for (int h = 0; h < 4; ++h) tc::tmem_ld8(lane_base + (tgp + a) * NP + (h0 + h) * Mt + lt, acc[h]);
          tc::tmem_wait_ld();
#pragma unroll
          for (int h = 0; h < 4; ++h)
#pragma unroll
            for (int j = 0; j < 8; ++j) sh4[h][j] = a ? sh4[h][j] + __uint_as_float(acc[h][j]) : __uint_as_float(acc[h][j]);
        }
#pragma unroll
        for (int j = 0; j < 8; ++j)
#pragma unroll
          for (int h = 0; h < 4; ++h) t[j] = fmaf(phase_const(L, h0 + h), sh4[h][j], t[j]);
      }
      if (rowok && ok) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int tok = ch * 8 + j, m = x0 + tok;
          if (m < M) {
            const float y = scalbnf(t[j], ref + Cfg::PBW + sh.refB[tok] + Cfg::PBX);
            float* dst = C + (int64_t)m * N + wrow;
            if (split)
              atomicAdd(dst, y);
            else
              *dst = y;
          }
        }
      }
    }
  } else if (is_x) {
    // ---------------------------- X producers -----------------------------
    // Work item wi of a group covers one 4-code word: lane bits of wi give 8
    // tokens x 4 words of a 16-code chunk kc, so a warp's 4-byte stores fill
    // 128 consecutive bytes of a column block.  Items of padding tokens (and
    // lattice positions that hold no plane) write nothing: the stages were
    // zeroed at the start.
    constexpr int PF = Cfg::PFX, XI = Cfg::XI, NGX = Cfg::NGX;
    const int tg = t_x % (Cfg::XPG * 32);  // thread of the group
    // per item: activation row (-1: padding), its row reference and the
    // byte offset of its word in a stage (block b adds b Mt ROWB bytes)
    int xrow[XI], xref[XI];
    uint32_t xbase[XI];
    auto word_of = [&](int wi) { return ((wi >> 5) & 1) * 4 + ((wi & 31) >> 3); };  // 4-code word of the step
#pragma unroll
    for (int i = 0; i < XI; ++i) {
      const int wi = tg + i * Cfg::XPG * 32, xl = wi & 31, kc = (wi >> 5) & 1;
      const int tokc = (wi >> 6) * 8 + (xl & 7), sub = xl >> 3;  // token of the CTA
      const bool act = wi < ntok * 8 && x0 + tokc < M;
      xrow[i] = act ? x0 + tokc : -1;
      xref[i] = act ? sh.refB[tokc] : 0;
      // token group and local token; dense: word sub of 16-byte chunk kc of
      // a 32-byte row; sparse: the word's 8 interleaved bytes in 16-byte
      // chunk j >> 1 of a 64-byte row, group t's R blocks after group t - 1's
      const int t = act ? tokc / Mt : 0, tok = act ? tokc - t * Mt : 0, j = kc * 4 + sub;
      xbase[i] = Cfg::SP ? (uint32_t)(t * Cfg::NRB * Mt * 64 + (tok >> 3) * 512 + (j >> 1) * 128 + (tok & 7) * 16 +
                                      (j & 1) * 8)
                         : core_off(tok, kc) + sub * 4;
    }
    auto load = [&](int i, uint32_t (&cw)[XI], int (&raw)[XI]) {
      const int g = gx + i * NGX;
#pragma unroll
      for (int e = 0; e < XI; ++e) {
        cw[e] = 0u;
        raw[e] = 0;
        if (xrow[e] >= 0 && g < total) {
          const int s = s0 + g;
          const int wi = tg + e * Cfg::XPG * 32;
          cw[e] = __ldg(reinterpret_cast<const uint32_t*>(X + (int64_t)xrow[e] * K + (int64_t)s * Cfg::KS +
                                                          word_of(wi) * 4));
          raw[e] = (int)__ldg(sX + (int64_t)xrow[e] * nb + (s >> gshift));
        }
      }
    };
    const uint32_t bstride = (uint32_t)Mt * Cfg::ROWB;  // bytes per column block
    auto step = [&](const int g, const uint32_t (&cw)[XI], const int (&raw)[XI]) -> bool {
      const int st = g % NSB;
      if (g >= NSB) {
        const bool ok = wait_all(&sh.empty[st], ((g / NSB) - 1) & 1);
        if (!ok) {
          if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
          return false;
        }
      }
      uint8_t* stg = xstage + (size_t)st * Cfg::BSTAGE;
#pragma unroll
      for (int e = 0; e < XI; ++e) {
        if (xrow[e] < 0) continue;
        uint32_t v[1], vc[1], mk[1][4];
        PlaneFmt<FX>::template decode<PLANE_E5M2, 1>(make_uint4(cw[e], 0u, 0u, 0u), raw[e] - xref[e] - Cfg::PBX, v,
                                                     vc, mk, true);
        uint32_t pv[8], pc[8];
        PlaneFmt<FX>::planes(v[0], mk[0], pv);
        PlaneFmt<FX>::planes(vc[0], mk[0], pc);
        if constexpr (Cfg::SP) {
          // R block b interleaves Q block b (plane partner) with Q block b - HB;
          // Q block u < L is the carry copy of plane u, u >= L plane u - L
#pragma unroll
          for (int b = Cfg::RB0; b < 2 * L; ++b) {
            const uint32_t x = b < L ? pc[b] : pv[b - L];
            const uint32_t y = b - Cfg::HB < L ? pc[b - Cfg::HB] : pv[b - Cfg::HB - L];
            *reinterpret_cast<uint2*>(stg + xbase[e] + (b - Cfg::RB0) * bstride) = interleave2(x, y);
          }
        } else {
          // lattice position u holds plane u / WX where WX divides u
#pragma unroll
          for (int u = 0; u < L; u += Cfg::WX) {
            *reinterpret_cast<uint32_t*>(stg + xbase[e] + u * bstride) = pc[u / Cfg::WX];
            *reinterpret_cast<uint32_t*>(stg + xbase[e] + (L + u) * bstride) = pv[u / Cfg::WX];
          }
        }
      }
      tc::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&sh.full[st]);
      return true;
    };
    const int nown = (total - gx + NGX - 1) / NGX;
    uint32_t q[PF][XI];
    int rq[PF][XI];
#pragma unroll
    for (int u = 0; u < PF; ++u) load(u, q[u], rq[u]);
    bool run = true;
    for (int i = 0; i < nown && run; i += PF) {
#pragma unroll
      for (int u = 0; u < PF; ++u) {
        if (i + u >= nown || !step(gx + (i + u) * NGX, q[u], rq[u])) {
          run = false;
          break;
        }
        load(i + u + PF, q[u], rq[u]);
      }
    }
  } else {
    // ------------------------------ MMA issuer -------------------------------
    const uint32_t leader = tc::elect_one();
    const uint64_t bdesc0 = tc::smem_desc(tc::smem_u32(xstage), 128, Cfg::SP ? 512 : 256);
    // E5M2 x E5M2 -> F32, N = L Mt (bit 2: 2:4-sparse A)
    const uint32_t idesc = tc::idesc_bf16_f32(Cfg::BM, NP) | (Cfg::SP ? (1u << 2) : 0u);
    const int gbytes = Mt * Cfg::ROWB;  // bytes of one column block
    bool ok = true;
    for (int g = 0; g < total && ok; ++g) {
      const int st = g % NSB;
      ok = wait_all(&sh.full[st], (g / NSB) & 1);
      if ((g & 7) == 0) ok = ok && !read_abort(&sh.abort_flag);
      if (!ok) break;
      tc::fence_after_sync();
#pragma unroll 1
      for (int tg2 = 0; tg2 < ntg; ++tg2)
#pragma unroll
      for (int kw = 0; kw < Cfg::NJ; ++kw) {
        // weight plane (pair plane) k_w against the window of column blocks
        // from L - k_w WW (R block L - k_w) of token group tg2
        const uint32_t a_t = tmem + Cfg::ACOL0 + st * Cfg::AU_COLS + kw * 8;
        const uint32_t boff = (uint32_t)(st * Cfg::BSTAGE + tg2 * Cfg::NRB * gbytes +
                                         (Cfg::SP ? L - kw - Cfg::RB0 : L - kw * Cfg::WW) * gbytes);
        const uint32_t d_t = tmem + (uint32_t)((tg2 + (kw & (nacc - 1))) * NP);
        const uint32_t acc = (g == 0 && kw < nacc) ? 0u : 1u;
        if constexpr (Cfg::SP)
          mma_sp_if(leader, d_t, a_t, bdesc0 + (uint64_t)(boff >> 4), tmem + Cfg::MCOL0 + st * 8, idesc, acc);
        else
          tc::mma_f8_ts_if(leader, d_t, a_t, bdesc0 + (uint64_t)(boff >> 4), idesc, acc);
      }
      tc::mma_commit_if(leader, &sh.empty[st]);
      if (g == total - 1) tc::mma_commit_if(leader, &sh.acc_full);
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

namespace {

// Split plan of the narrow kernel: the tile kernel's tail search extended to
// grids with fewer tiles than SMs (then every tile is split), with finer
// split points (a narrow tile is short, so its pieces' fixed costs weigh
// more and the best point moves).
inline TailPlan tcn_plan_search(int64_t tiles, int sms, int nsub) {
  TailPlan best{(int)tiles, 0, 0};
  if (sms <= 0 || nsub < 2 || tiles % sms == 0) return best;
  double best_m = tail_makespan(tiles, sms, 0, 0.5);
  const double xs[5] = {0.5, 0.6, 2.0 / 3.0, 0.75, 0.8};
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

inline TailPlan tcn_plan(int64_t tiles, int sms, int nsub) {
  static std::mutex mu;
  static std::unordered_map<uint64_t, TailPlan> memo;
  const uint64_t key = ((uint64_t)tiles << 32) ^ ((uint64_t)sms << 16) ^ (uint64_t)nsub;
  {
    std::lock_guard<std::mutex> lk(mu);
    auto it = memo.find(key);
    if (it != memo.end()) return it->second;
  }
  const TailPlan t = tcn_plan_search(tiles, sms, nsub);
  std::lock_guard<std::mutex> lk(mu);
  memo[key] = t;
  return t;
}

template <int FX, int FW, bool T2>
cudaError_t launch_tcn_t(int G, const uint8_t* x, const int8_t* sx, const uint8_t* w, const int8_t* sw, int64_t M,
                         int64_t N, int64_t K, float* c, uint32_t* st, cudaStream_t s, int sms) {
  using Cfg = TcnCfg<FX, FW, T2>;
  static_assert(sizeof(TcShared) <= 2048, "shared tail");
  static_assert(Cfg::SMEM <= 227 * 1024, "shared memory");
  auto kern = gemm_tcn_kernel<FX, FW, T2>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::SMEM);
  if (e != cudaSuccess) return e;
  // token groups of equal size Mt (a multiple of 8): one per CTA of at most
  // MTMAX tokens, or (sparse form, larger M) two per CTA of at most MT2
  const int ntg = Cfg::TWO ? 2 : 1;
  const int64_t cap = ntg == 2 ? 2 * Cfg::MT2 : Cfg::MTMAX;
  int64_t ng = (M + cap - 1) / cap;
  const int Mt = (int)(((M + ng * ntg - 1) / (ng * ntg) + 7) / 8 * 8);
  ng = (M + (int64_t)ntg * Mt - 1) / ((int64_t)ntg * Mt);
  const int64_t ntw = (N + Cfg::BM - 1) / Cfg::BM, tiles = ntw * ng;
  const TailPlan plan = tcn_plan(tiles, sms, (int)(K / Cfg::KS));
  if (plan.nsplit > 0) {
    // C of the split tiles starts at zero: whole token groups from the first one
    const int64_t row0 = (plan.ntiles_full / ntw) * ntg * Mt;
    e = cudaMemsetAsync(c + row0 * N, 0, (size_t)((M - row0) * N) * sizeof(float), s);
    if (e != cudaSuccess) return e;
  }
  const unsigned grid = (unsigned)(plan.ntiles_full + 2 * plan.nsplit);
  int gshift = 0;  // scale block of step s is s >> gshift
  while ((Cfg::KS << gshift) < G) ++gshift;
  kern<<<grid, Cfg::THREADS, Cfg::SMEM, s>>>(x, sx, w, sw, (int)M, (int)N, (int)K, G, gshift, Mt, ntg, c, st, plan);
  return cudaGetLastError();
}

}  // namespace

bool gemm_narrow_supported(int fa, int fb) {
  return (fa == CURVEFP_E3C3 && fb == CURVEFP_E3C3) || (fa == CURVEFP_E4C3 && fb == CURVEFP_E4C3) ||
         (fa == CURVEFP_E5C2 && fb == CURVEFP_E4C3) || (fa == CURVEFP_E4C3 && fb == CURVEFP_E5C2) ||
         (fa == CURVEFP_E5C2 && fb == CURVEFP_E5C2);
}

cudaError_t launch_gemm_tensor_narrow(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                                      const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, uint32_t* status,
                                      cudaStream_t s, int sms) {
  // same-format pairs from 512 activation rows: two token groups per CTA
  // (measured: 2048 x 4096 x 4096 0.861 -> 0.837 ms, FFN M = 4096 5.94 ->
  // 5.54 ms; at M <= 256 the deeper one-group ring and its waves are faster)
  const bool two = fa == fb && M >= 512;
#define CFP_T(X, Y)                                                                                  \
  if (fa == X && fb == Y)                                                                           \
    return two ? launch_tcn_t<X, Y, true>(G, a, sa, b, sb, M, N, K, c, status, s, sms)             \
               : launch_tcn_t<X, Y, false>(G, a, sa, b, sb, M, N, K, c, status, s, sms);
  CFP_T(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_T(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_T(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_T
  return cudaErrorInvalidValue;
}

}  // namespace cfp
