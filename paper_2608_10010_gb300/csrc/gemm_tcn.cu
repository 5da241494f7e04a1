// Tensor-core closed-product GEMM with the phases along the MMA's N dimension
// (algo TENSOR_NARROW): Sec. 3.2, Eq. 2, Eq. 5.
//
// C = X_hat W_hat^T with X the activation ("token") operand, format FX, and
// W the weight operand, format FW.  Every operand splits into curve planes of
// exact powers of two (plane k holds the elements of curve index k), and
// plane k_x of X times plane k_w of W lands on phase h = (k_x WX + k_w WW)
// mod L with carry c = floor((k_x WX + k_w WW) / L) (Eq. 2 on the shared
// lattice L).
//
// Block scales.  A plane value is the power of two 2^e of the code alone
// (tc_mx.cuh); the block scale of every 32-code step enters the MMA as a
// UE8M0 scale factor (tcgen05.mma .kind::mxf8f6f4 .block_scale), relative to
// the row's largest block scale, so every product of the step is exact
// whatever the spread of the block scales along the row.
//
// Here the weight rows are the MMA's 128-row TMEM operand and the phase is a
// column index: the accumulator of a tile is D[w][h Mt + m] (weight row w,
// phase h, token m of the tile's Mt tokens), the per-phase sums S_h of Eq. 5
// for every token side by side.  For weight plane k_w the shared-memory
// operand must hold, in column block h, the X plane with
// k_x WX = (h - k_w WW) mod L, doubled where the sum wrapped (carry).  Lay
// out the sequence of 2L column blocks
//   Q = [ 2 X_0 ... (lattice positions 0 .. L-1, carry copies) |
//           X_0 ... (lattice positions 0 .. L-1, plain) ]
// then the operand of weight plane k_w is the window of L blocks that starts
// at block L - k_w WW: a start address of the MMA's shared-memory descriptor.
//
// 2:4-sparse pair planes: an element sits in one plane, so weight planes j
// and j + K_W/2 share one compressed operand at logical positions 2k and
// 2k + 1, with one curve-index bit as metadata.  The activation side stores
// R blocks R_b[2k] = Q_b[k], R_b[2k + 1] = Q_{b - PO}[k] (PO = K_W/2 WW, the
// lattice distance of the partner plane) and the operand of pair j is the
// window from R block L - j WW: K_W/2 sparse MMAs of logical K 64 per step.
//
// Orientation.  The tokens are A's rows and the weights B's for every pair.
// X takes the carry copies, so its planes need one binade more than W's: E5C2
// tokens store their planes one binade low (the lowest binade's plain copy,
// 2^-17, has no E5M2 value and is dropped: an element at least 2^30 below the
// top binade of its block).  E5C2 tokens against E4C3 weights put their four
// planes on every other position of the 8-phase lattice (WX = 2): half of the
// R blocks stay empty, and the W side carries the E4C3 operand's four pair
// planes, so the producers' work per MMA is lower than with the operands
// swapped (two pair planes of E5C2 weights against 8-plane tokens).
//
// Roles (15 warps for 8-phase pairs, 17 for E5C2 x E5C2):
//   warps 0-7   W producers: two groups of 4 warps taking alternate steps,
//               one thread per weight row (all 32 codes of its steps): codes
//               -> pair planes, metadata and the row's scale factor -> TMEM;
//               after the last step they run the epilogue.
//   next warps  X producers: groups taking every NGX-th step, 8 codes of one
//               token per work item -> one 16-byte chunk of each of the
//               step's R blocks; the token's scale factors -> the stage's
//               factor block (copied to TMEM by the MMA warp).
//   last warp   TMEM allocation, factor copies and MMA issue (one elected
//               lane).
// Tiles of the last partial wave may be split in K into two pieces (the plan
// in tcn_common.cuh); a piece adds its outputs to zeroed C atomically, two
// additions per output, so the result does not depend on their order.  The
// row references come from the tile's contiguous scale rows, read by all
// threads together.  Every wait is bounded.
#include "gemm_tc.cuh"
#include "tc_mx.cuh"
#include "tcn_common.cuh"

namespace cfp {

namespace {

template <int FX, int FW>
struct TcnCfg {
  using P = Pair<FX, FW>;
  static constexpr int KW = Fmt<FW>::K, L = P::L, WX = P::WA, WW = P::WB;
  static_assert(WX == 1 || (WX == 2 && Fmt<FX>::C == 2), "X planes on every (or every other) lattice position");
  static constexpr int BM = 128;          // weight rows per CTA (TMEM lanes)
  static constexpr int KS = 32;           // codes per pipeline step (one scale factor)
  static constexpr int MTMAX = 256 / L;   // tokens per CTA: L Mt <= 256 (MMA N)
  static constexpr int NSB = 4;           // pipeline depth (X stages = W TMEM units)
  static constexpr int HB = KW / 2, MBIT = KW == 8 ? 2 : 1;
  static constexpr int NJ = HB;           // sparse MMAs per step
  static constexpr int PO = HB * WW;      // lattice distance of the partner plane
  static constexpr int RB0 = L - (NJ - 1) * WW, NRB = 2 * L - RB0;
  static_assert(2 * PO == L && RB0 > PO && PO % WX == 0, "partner planes half the lattice apart");
  static constexpr int ROWB = 64;         // bytes of one operand row (logical K 64)
  static constexpr int PBX = FX == CURVEFP_E5C2 ? 1 : 0;  // X planes one binade low
  // TMEM columns: accumulators, W units, metadata (8 per unit, 2 used), A
  // factors (4 per unit: quadrant q reads column q), B factors (8 per unit)
  static constexpr int AU_COLS = NJ * 8;
  static constexpr int ACOL0 = 256;
  static constexpr int MCOL0 = ACOL0 + NSB * AU_COLS;
  static constexpr int SFA0 = MCOL0 + NSB * 8;
  static constexpr int SFB0 = (SFA0 + NSB * 4 + 31) / 32 * 32;
  static_assert(SFB0 + NSB * 8 <= 512, "TMEM budget");
  // Producer groups take turns: W group g % NGW and X group g % NGX produce
  // step g, so each producer thread has NGW (NGX) steps of time per step.
  static constexpr int NGW = 2;                 // W groups of 4 warps (one thread per weight row)
  static constexpr int XPG = MTMAX / 16;        // X warps per group
  static constexpr int NGX = L == 8 ? 3 : 2;    // X groups
  static constexpr int NWT = NGW * 128;         // W threads
  static constexpr int NXT = NGX * XPG * 32;    // X threads
  static constexpr int THREADS = NWT + NXT + 32;
  static constexpr int MMA_WARP = (NWT + NXT) / 32;
  static constexpr int BSTAGE = NRB * MTMAX * ROWB;  // bytes of one step's X operand rows
  static constexpr int SFSTAGE = 1024;               // factor block of a step (two copy sources)
  static constexpr int PFW = 4;  // own steps of weight codes in flight per W thread
  static constexpr int PFX = 2;  // own steps of activation codes in flight per X thread
  static constexpr int XI = MTMAX * 4 / (XPG * 32);  // X work items (8-code chunks) per thread and step
  // more than half of the SM's shared memory: one CTA per SM (the split plan
  // assumes it, and the CTA allocates all of TMEM)
  static constexpr size_t SMEM_USED = (size_t)NSB * (BSTAGE + SFSTAGE) + 2048;
  static constexpr size_t SMEM = SMEM_USED > 120 * 1024 ? SMEM_USED : 120 * 1024;
};

}  // namespace

// X: [Mx x K] token codes, W: [Nw x K] weight codes (K contiguous), scales
// [rows x K/G].  C: [Mx x Nw], row-major.
// FULL: every tile has MTMAX tokens (Mt == MTMAX), so the stage offsets of
// the X producers are constants.
template <int FX, int FW, bool FULL>
__global__ void __launch_bounds__(TcnCfg<FX, FW>::THREADS, 1)
    gemm_tcn_kernel(const uint8_t* __restrict__ X, const int8_t* __restrict__ sX, const uint8_t* __restrict__ W,
                    const int8_t* __restrict__ sW, int M, int N, int K, int G, int gshift, int Mt,
                    float* __restrict__ C, uint32_t* status, const TailPlan plan) {
  using Cfg = TcnCfg<FX, FW>;
  constexpr int L = Cfg::L, NSB = Cfg::NSB;
  static_assert(NSB <= TC_MAX_RING && Cfg::MTMAX <= 128, "barrier rings, row references");
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* xstage = smem;
  uint8_t* sfstage = smem + (size_t)NSB * Cfg::BSTAGE;
  TcShared& sh = *reinterpret_cast<TcShared*>(smem + (size_t)NSB * (Cfg::BSTAGE + Cfg::SFSTAGE));

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
  const int x0 = (tile / ntw) * Mt, w0 = (tile % ntw) * Cfg::BM;
  const int nb = K / G, total = s1 - s0;
  // Accumulator copies: consecutive MMAs of a step into one accumulator wait
  // for each other's accumulation, so where the accumulator is at most 128
  // columns the pair planes rotate over 2 or 4 copies (NP columns each) that
  // the epilogue adds up.
  const int NP = L * Mt, nacc0 = NP <= 64 ? 4 : (NP <= 128 ? 2 : 1);
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
    // TMEM allocation and release are warp-collective (.sync.aligned): the
    // MMA warp reaches them, and every wait of its loop (whole-warp waits),
    // with all 32 lanes together
    __syncwarp();
    tc::tmem_alloc(&sh.tmem_base, 512);
    tc::tmem_relinquish();
  }
  const bool is_w = tid < Cfg::NWT, is_x = !is_w && warp < Cfg::MMA_WARP;
  // W threads: weight row (TMEM lane) and group; X threads: group.  The row
  // references of the tile's weight rows and tokens (-128 for rows past the
  // ends) are formed by all threads together from the two contiguous runs of
  // scale rows.  The X stages and factor blocks start at zero (padding
  // tokens and empty lattice positions are never written).
  const int wrow = w0 + (warp & 3) * 32 + lane, gw = warp >> 2;
  const int t_x = tid - Cfg::NWT, gx = t_x / (Cfg::XPG * 32);
  if (tid < 128) {
    sh.wref[tid] = -128;
    sh.refB[tid] = -128;
  }
  __syncthreads();
  rows_ref_coop(sW + (int64_t)w0 * nb, min(Cfg::BM, N - w0), nb, sh.wref, tid, Cfg::THREADS);
  rows_ref_coop(sX + (int64_t)x0 * nb, min(Mt, M - x0), nb, sh.refB, tid, Cfg::THREADS);
  for (int o = tid * 16; o < NSB * (Cfg::BSTAGE + Cfg::SFSTAGE); o += Cfg::THREADS * 16)
    *reinterpret_cast<uint4*>(smem + o) = make_uint4(0, 0, 0, 0);
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  const int ref = is_w ? sh.wref[(warp & 3) * 32 + lane] : -128;  // this W thread's weight row

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
    auto step = [&](const int g, uint4 lo, uint4 hi, const int raw) -> bool {
      const int st = g % NSB;
      bool keep;
      const uint32_t sf = mx_sf(raw - ref, 0, keep) * 0x01010101u;
      if (!keep) lo = hi = make_uint4(0, 0, 0, 0);
      // the 32 codes of the row's step: plane words and curve-index masks;
      // pair plane j of word w = the elements whose low curve-index bits are j
      uint32_t p[8][4];
      const uint32_t cw[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        uint32_t v, vc, mk[4];
        mx_word<FW, 0>(cw[w], v, vc);
        k_masks<PLANE_E5M2, Fmt<FW>::C>(cw[w], mk);
        p[w][0] = v & ~mk[0] & ~mk[1];
        p[w][1] = v & mk[0] & ~mk[1];
        p[w][2] = v & ~mk[0] & mk[1];
        p[w][3] = v & mk[0] & mk[1];
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
      // pair planes 2jp and 2jp + 1 of the step: 16 consecutive columns of
      // the unit, then the metadata of codes 0-15 and 16-31 and the factor
#pragma unroll
      for (int jp = 0; jp < Cfg::NJ / 2; ++jp) {
        uint32_t r[16];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int j = 2 * jp + e;
#pragma unroll
          for (int w = 0; w < 8; ++w) r[e * 8 + w] = Cfg::KW == 8 ? p[w][j] : (p[w][j] | p[w][j + 2]);
        }
        tmem_st16(lane_base + Cfg::ACOL0 + st * Cfg::AU_COLS + jp * 16, r);
      }
      const uint32_t mt[2] = {pair_meta<Cfg::MBIT>(lo.x, lo.y, lo.z, lo.w),
                              pair_meta<Cfg::MBIT>(hi.x, hi.y, hi.z, hi.w)};
      tc::tmem_st2(lane_base + Cfg::MCOL0 + st * 8, mt);
      tc::tmem_st1(lane_base + Cfg::SFA0 + st * 4 + (warp & 3), sf);
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
    // sum_h 2^{h/L} S_h (FP32, phase order) and scaled by
    // 2^{ref_w + ref_m - 2 MX_OFF}.  A whole tile stores C, a K piece adds to
    // zeroed C.
    const bool aborted = __any_sync(0xffffffffu, read_abort(&sh.abort_flag) != 0);
    const bool ok = !aborted && wait_all(&sh.acc_full, 0);
    if (!ok && lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
    tc::fence_after_sync();
#pragma unroll 1
    for (int ch = gw; ch < (Mt >> 3); ch += NGW) {
      const int lt = ch * 8;  // tokens lt .. lt + 7 of the tile
      float t[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) t[j] = 0.f;
      if (nacc == 1) {
        // one accumulator: all L phase sums in one round of loads
        uint32_t acc[L][8];
#pragma unroll
        for (int h = 0; h < L; ++h) tc::tmem_ld8(lane_base + h * Mt + lt, acc[h]);
        tc::tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 8; ++j)
#pragma unroll
          for (int h = 0; h < L; ++h) t[j] = fmaf(phase_const(L, h), __uint_as_float(acc[h][j]), t[j]);
      } else {
#pragma unroll
        for (int h0 = 0; h0 < L; h0 += 4) {
          // S_h = the sum of the accumulator copies (copy order fixed)
          float sh4[4][8];
#pragma unroll 1
          for (int a = 0; a < nacc; ++a) {
            uint32_t acc[4][8];
#pragma unroll
            for (int h = 0; h < 4; ++h) tc::tmem_ld8(lane_base + a * NP + (h0 + h) * Mt + lt, acc[h]);
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
      }
      if (rowok && ok) {
        float y[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) y[j] = scale_pow2(t[j], ref + sh.refB[lt + j] - 2 * MX_OFF);
        const int m0 = x0 + lt;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int m = m0 + j;
          if (m < M) {
            float* dst = C + (int64_t)m * N + wrow;
            if (split)
              atomicAdd(dst, y[j]);
            else
              *dst = y[j];
          }
        }
      }
    }
  } else if (is_x) {
    // ---------------------------- X producers -----------------------------
    // Work item wi of a group covers 8 codes (16-byte chunk c of a 64-byte R
    // row) of one token: lane bits of wi give 8 tokens x the 4 chunks, so a
    // warp's 16-byte stores fill 512 consecutive bytes of an R block.  Items
    // of padding tokens (and lattice positions that hold no plane) write
    // nothing: the stages were zeroed at the start.  The item of a token's
    // first chunk also writes the token's scale factor into the factor
    // block: one word per column n = h Mt + m of the MMA (the factor ids read
    // bytes 0 and 1).
    constexpr int PF = Cfg::PFX, XI = Cfg::XI, NGX = Cfg::NGX;
    const int tg = t_x % (Cfg::XPG * 32);  // thread of the group
    // per item: activation row (-1: padding), its row reference, its token
    // and the byte offset of its chunk in a stage (block b adds b Mt 64 bytes)
    int xrow[XI], xref[XI], xtok[XI], xcol[XI];
    uint32_t xbase[XI];
#pragma unroll
    for (int i = 0; i < XI; ++i) {
      const int wi = tg + i * Cfg::XPG * 32, xl = wi & 31;
      const int tok = (wi >> 5) * 8 + (xl & 7), c = xl >> 3;  // token of the tile, chunk of the row
      const bool act = tok < Mt && x0 + tok < M;
      xrow[i] = act ? x0 + tok : -1;
      xref[i] = act ? sh.refB[tok] : 0;
      xtok[i] = c == 0 ? tok : -1;  // writes the token's factors
      xcol[i] = c * 8;
      xbase[i] = (uint32_t)((tok >> 3) * 512 + c * 128 + (tok & 7) * 16);
    }
    auto load = [&](int i, uint2 (&cw)[XI], int (&raw)[XI]) {
      const int g = gx + i * NGX;
#pragma unroll
      for (int e = 0; e < XI; ++e) {
        cw[e] = make_uint2(0u, 0u);
        raw[e] = 0;
        if (xrow[e] >= 0 && g < total) {
          const int s = s0 + g;
          cw[e] = __ldg(reinterpret_cast<const uint2*>(X + (int64_t)xrow[e] * K + (int64_t)s * Cfg::KS + xcol[e]));
          raw[e] = (int)__ldg(sX + (int64_t)xrow[e] * nb + (s >> gshift));
        }
      }
    };
    // bytes per column block (a constant for whole tiles)
    const uint32_t bstride = FULL ? (uint32_t)(Cfg::MTMAX * Cfg::ROWB) : (uint32_t)Mt * Cfg::ROWB;
    auto step = [&](const int g, const uint2 (&cw)[XI], const int (&raw)[XI]) -> bool {
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
      uint8_t* sfs = sfstage + (size_t)st * Cfg::SFSTAGE;
#pragma unroll
      for (int e = 0; e < XI; ++e) {
        if (xrow[e] < 0) continue;
        bool keep;
        const uint32_t sf = mx_sf(raw[e] - xref[e], Cfg::PBX, keep);
        constexpr int C = Fmt<FX>::C;
        if constexpr (C == 3) {
          static_assert(Fmt<FX>::K == L, "three-bit tokens sit on every lattice position");
          // Three curve-index bits.  R block b holds Q_b[k] in byte 2k and Q_{b-PO}[k] in byte 2k + 1 (Q
          // block u < L: the carry copy of plane u, u >= L: plane u - L).  With
          // PO = L/2 the two planes share their two low curve-index bits (class
          // b mod PO) and differ in the top bit T, so a code of that class sits
          // in the even byte where its T equals the top bit of b mod L, else in
          // the odd byte.  Per 16-bit lane (one code) three words place the
          // code's value by its T: qcc for b < L (carry copies on both sides;
          // b mod L has T = 1), qpc for L <= b < L + PO (plain even, carry odd;
          // T = 0) and qpp for b >= L + PO (plain, T = 1); block b is its word
          // masked to the codes of class b mod PO.
          uint32_t qcc[4], qpc[4], qpp[4], dm0[4], dm1[4];
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            const uint32_t w = q ? cw[e].y : cw[e].x;
            uint32_t v, vc;
            mx_word<FX, Cfg::PBX>(keep ? w : 0u, v, vc);
            const uint32_t wt = w << (8 - C), w0 = w << 7, w1 = w << 6;  // bits C - 1, 0, 1 -> bit 7
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              // lanes of codes 4q + 2hh and 4q + 2hh + 1: duplicated sign
              // masks, duplicated values, (plain, carry) interleaved
              const uint32_t sdup = hh ? 0xBBAAu : 0x9988u, dup = hh ? 0x3322u : 0x1100u, ilv = hh ? 0x7362u : 0x5140u;
              const int i = 2 * q + hh;
              const uint32_t dt = prmt_sign(wt, sdup);
              dm0[i] = prmt_sign(w0, sdup);
              dm1[i] = prmt_sign(w1, sdup);
              qcc[i] = __byte_perm(vc, vc, dup) & (dt ^ 0xFF00FF00u);
              qpp[i] = __byte_perm(v, v, dup) & (dt ^ 0xFF00FF00u);
              qpc[i] = __byte_perm(v, vc, ilv) & (dt ^ 0x00FF00FFu);
            }
          }
#pragma unroll
          for (int b = Cfg::RB0; b < 2 * L; ++b) {
            const int j = b % Cfg::PO;
            uint32_t r[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const uint32_t src = b < L ? qcc[i] : (b < L + Cfg::PO ? qpc[i] : qpp[i]);
              r[i] = src & ((j & 1) ? dm0[i] : ~dm0[i]) & ((j & 2) ? dm1[i] : ~dm1[i]);
            }
            *reinterpret_cast<uint4*>(stg + xbase[e] + (b - Cfg::RB0) * bstride) = make_uint4(r[0], r[1], r[2], r[3]);
          }
        } else {
          // Two curve-index bits: the tokens' planes of each word and their
          // carry copies, then per R block Q_b and Q_{b-PO} interleaved.  With
          // WX = 2 (E5C2 tokens against an 8-phase lattice) plane k sits on
          // lattice position 2k, Q blocks of odd positions are empty, and an
          // R block whose halves are both empty is never written (the stages
          // start at zero).
          uint32_t pv[2][8], pc[2][8];
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            const uint32_t w = q ? cw[e].y : cw[e].x;
            uint32_t v, vc, mk[4];
            mx_word<FX, Cfg::PBX>(keep ? w : 0u, v, vc);
            k_masks<PLANE_E5M2, C>(w, mk);
            planes_of<C>(v, mk, pv[q]);
            planes_of<C>(vc, mk, pc[q]);
          }
          constexpr int WXc = Cfg::WX;
          // Q block u: the carry copy (u < L) or the plane (u >= L) of the
          // token plane on lattice position u mod L, zero where none sits
          auto qb = [&](int q, int u) -> uint32_t {
            const int pos = u < L ? u : u - L;
            if (pos % WXc) return 0u;
            return u < L ? pc[q][pos / WXc] : pv[q][pos / WXc];
          };
#pragma unroll
          for (int b = Cfg::RB0; b < 2 * L; ++b) {
            if ((b % WXc) != 0 && ((b - Cfg::PO) % WXc) != 0) continue;
            const uint2 lo = interleave2(qb(0, b), qb(0, b - Cfg::PO));
            const uint2 hi = interleave2(qb(1, b), qb(1, b - Cfg::PO));
            *reinterpret_cast<uint4*>(stg + xbase[e] + (b - Cfg::RB0) * bstride) = make_uint4(lo.x, lo.y, hi.x, hi.y);
          }
        }
        if (xtok[e] >= 0) {
          const uint32_t sw = sf * 0x01010101u;
          if constexpr (FULL && Cfg::MTMAX == 32) {
            // n = 32 h + m: row m of both copy sources, all four words
#pragma unroll
            for (int c = 0; c < L / 4; ++c)
              *reinterpret_cast<uint4*>(sfs + c * 512 + xtok[e] * 16) = make_uint4(sw, sw, sw, sw);
          } else {
#pragma unroll
            for (int h = 0; h < L; ++h) *reinterpret_cast<uint32_t*>(sfs + sfb_off(h * Mt + xtok[e])) = sw;
          }
        }
      }
      tc::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&sh.full[st]);
      return true;
    };
    const int nown = (total - gx + NGX - 1) / NGX;
    uint2 q[PF][XI];
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
    const uint64_t bdesc0 = tc::smem_desc(tc::smem_u32(xstage), 128, 512);
    const uint32_t idesc = idesc_mx_e5m2(NP, true);
    const int gbytes = Mt * Cfg::ROWB;  // bytes of one column block
    // per pair plane: its accumulator copy and the descriptor of its window
    // of R blocks (from L - kw WW) in stage 0; the loop below is unrolled
    // over the stages, so every other offset is a constant of its body
    uint32_t d_kw[Cfg::NJ];
    uint64_t b_kw[Cfg::NJ];
#pragma unroll
    for (int kw = 0; kw < Cfg::NJ; ++kw) {
      d_kw[kw] = tmem + (uint32_t)((kw & (nacc - 1)) * NP);
      b_kw[kw] = bdesc0 + (uint64_t)((uint32_t)((L - kw * Cfg::WW - Cfg::RB0) * gbytes) >> 4);
    }
    bool ok = true;
    for (int g0 = 0, par = 0; g0 < total && ok; g0 += NSB, par ^= 1) {
#pragma unroll
      for (int st = 0; st < NSB; ++st) {
        const int g = g0 + st;
        if (g >= total) break;
        ok = wait_all(&sh.full[st], (uint32_t)par);
        if ((g & 7) == 0) ok = ok && !read_abort(&sh.abort_flag);
        if (!ok) break;
        tc::fence_after_sync();
        // the step's B factors: columns 0..127 and, for N > 128, 128..255
        const uint8_t* sfs = sfstage + (size_t)st * Cfg::SFSTAGE;
        tmem_cp_sf_if(leader, tmem + Cfg::SFB0 + st * 8, sfs);
        if (NP > 128) tmem_cp_sf_if(leader, tmem + Cfg::SFB0 + st * 8 + 4, sfs + 512);
#pragma unroll
        for (int kw = 0; kw < Cfg::NJ; ++kw) {
          const uint32_t acc = (g == 0 && kw < nacc) ? 0u : 1u;
          mma_sp_mx_if(leader, d_kw[kw], tmem + Cfg::ACOL0 + st * Cfg::AU_COLS + kw * 8,
                       b_kw[kw] + (uint64_t)((st * Cfg::BSTAGE) >> 4), tmem + Cfg::MCOL0 + st * 8, idesc,
                       tmem + Cfg::SFA0 + st * 4, tmem + Cfg::SFB0 + st * 8, acc);
        }
        tc::mma_commit_if(leader, &sh.empty[st]);
        if (g == total - 1) tc::mma_commit_if(leader, &sh.acc_full);
      }
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

namespace {

// x: [Mx x K] token codes, w: [Nw x K] weight codes; c: [Mx x Nw].
template <int FX, int FW>
cudaError_t launch_tcn_t(int G, const uint8_t* x, const int8_t* sx, const uint8_t* w, const int8_t* sw, int64_t Mx,
                         int64_t Nw, int64_t K, float* c, uint32_t* st, cudaStream_t s, int sms) {
  using Cfg = TcnCfg<FX, FW>;
  static_assert(sizeof(TcShared) <= 2048, "shared tail");
  static_assert(Cfg::SMEM <= 227 * 1024, "shared memory");
  // token groups of equal size Mt (a multiple of 8) of at most MTMAX tokens
  int64_t ng = (Mx + Cfg::MTMAX - 1) / Cfg::MTMAX;
  const int Mt = (int)(((Mx + ng - 1) / ng + 7) / 8 * 8);
  ng = (Mx + Mt - 1) / Mt;
  auto kern = Mt == Cfg::MTMAX ? gemm_tcn_kernel<FX, FW, true> : gemm_tcn_kernel<FX, FW, false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::SMEM);
  if (e != cudaSuccess) return e;
  const int64_t ntw = (Nw + Cfg::BM - 1) / Cfg::BM, tiles = ntw * ng;
  const TailPlan plan = tcn_plan(tiles, sms, (int)(K / Cfg::KS));
  if (plan.nsplit > 0) {
    // C of the split tiles starts at zero: the token rows from the first
    // split tile's group on
    const int64_t row0 = (plan.ntiles_full / ntw) * Mt;
    e = cudaMemsetAsync(c + row0 * Nw, 0, (size_t)((Mx - row0) * Nw) * sizeof(float), s);
    if (e != cudaSuccess) return e;
  }
  const unsigned grid = (unsigned)(plan.ntiles_full + 2 * plan.nsplit);
  int gshift = 0;  // scale block of step s is s >> gshift
  while ((Cfg::KS << gshift) < G) ++gshift;
  kern<<<grid, Cfg::THREADS, Cfg::SMEM, s>>>(x, sx, w, sw, (int)Mx, (int)Nw, (int)K, G, gshift, Mt, c, st, plan);
  return cudaGetLastError();
}

}  // namespace

bool gemm_narrow_supported(int fa, int fb) {
  return (fa == CURVEFP_E3C3 && fb == CURVEFP_E3C3) || (fa == CURVEFP_E4C3 && fb == CURVEFP_E4C3) ||
         (fa == CURVEFP_E5C2 && fb == CURVEFP_E4C3) || (fa == CURVEFP_E4C3 && fb == CURVEFP_E5C2) ||
         (fa == CURVEFP_E5C2 && fb == CURVEFP_E5C2) || (fa == CURVEFP_E4C3_R3_4 && fb == CURVEFP_E4C3_R3_4);
}

// C = A_hat B_hat^T, A [M x K] (format fa), B [N x K] (format fb): the
// tokens are A's rows and the weights B's.
cudaError_t launch_gemm_tensor_narrow(int fa, int fb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                                      const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c, uint32_t* status,
                                      cudaStream_t s, int sms) {
  if (fa == CURVEFP_E3C3 && fb == CURVEFP_E3C3)
    return launch_tcn_t<CURVEFP_E3C3, CURVEFP_E3C3>(G, a, sa, b, sb, M, N, K, c, status, s, sms);
  if (fa == CURVEFP_E4C3 && fb == CURVEFP_E4C3)
    return launch_tcn_t<CURVEFP_E4C3, CURVEFP_E4C3>(G, a, sa, b, sb, M, N, K, c, status, s, sms);
  if (fa == CURVEFP_E4C3 && fb == CURVEFP_E5C2)
    return launch_tcn_t<CURVEFP_E4C3, CURVEFP_E5C2>(G, a, sa, b, sb, M, N, K, c, status, s, sms);
  if (fa == CURVEFP_E5C2 && fb == CURVEFP_E4C3)
    return launch_tcn_t<CURVEFP_E5C2, CURVEFP_E4C3>(G, a, sa, b, sb, M, N, K, c, status, s, sms);
  if (fa == CURVEFP_E5C2 && fb == CURVEFP_E5C2)
    return launch_tcn_t<CURVEFP_E5C2, CURVEFP_E5C2>(G, a, sa, b, sb, M, N, K, c, status, s, sms);
  if (fa == CURVEFP_E4C3_R3_4 && fb == CURVEFP_E4C3_R3_4)  // 32 phases: gemm_tcn_r34.cu
    return launch_gemm_tensor_narrow_r34(G, a, sa, b, sb, M, N, K, c, status, s, sms);
  return cudaErrorInvalidValue;
}

}  // namespace cfp
