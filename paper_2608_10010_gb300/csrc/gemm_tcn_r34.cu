// Tensor-core closed-product GEMM for E4C3 with the rational radix
// r = 2^{3/4} (Sec. 3.1 Eq. 4, Table 2; App. A.1), phases along the MMA's N
// dimension as in gemm_tcn.cu (algo TENSOR_NARROW / AUTO for this format).
//
// The level of index n (n = m - 64, m the 7-bit rank) is 2^{3n/32}.  With
// 3n = 32 q + j (j in [0, 32)) an element is 2^q 2^{j/32}: it sits in curve
// plane j with the power-of-two value 2^q (q in [-6, 5]; the block scale is
// the MMA's UE8M0 scale factor), and plane j1 times plane j2 lands on phase
// h = (j1 + j2) mod 32 with carry (j1 + j2) >= 32: the 32 phases of Table 2.
// Per byte, 3m in a 16-bit lane gives j = 3m mod 32 and q = floor(3m/32) - 6
// (3 * 64 = 6 * 32).
//
// Layout (the narrow kernel's with L = 32): the weight rows are the MMA's
// 128-row TMEM operand; planes j and j + 16 share one 2:4-sparse compressed
// operand (pair plane j, bit 4 of the curve index as metadata); the tokens'
// planes and their carry copies form the sequence Q of 64 column blocks
// (carry copies of lattice positions 0..31, then plain copies), stored as R
// blocks R_b[2k] = Q_b[k], R_b[2k + 1] = Q_{b-16}[k] (b in [17, 64)), and pair
// plane p reads the window of 32 blocks from R block 32 - p.  Mt = 8 tokens
// (the MMA's 8-row core matrices): N = 256, 16 sparse block-scaled MMAs of
// 128 x 256 x 64 (logical K) per 32-code step.
//
// TMEM holds the 256-column accumulator, one weight unit of 16 x 8 columns,
// its metadata and the scale factors: a single weight stage.  Its producers
// decode the next step while the step before is in the tensor pipe and
// store once those MMAs retire, the 16 pair planes split between two warp
// halves; the token stages form a ring of two in shared memory.
//
// Roles (352 threads): warps 0-7 weight producers (warp w: rows 32 (w & 3)
// .. + 31 of the tile, pair planes 8 (w >> 2) .. + 7; all 32 codes of a step
// per thread) and, after the last step, the epilogue (tokens 4 (w >> 2) ..
// + 3); warps 8-9 token producers taking alternate steps (one work item of 8
// codes of one token per lane); warp 10 TMEM allocation, factor copies and
// MMA issue.  The tail of the last wave is split in K as in gemm_tcn.cu.
// Every wait is bounded.
#include "gemm_tc.cuh"
#include "tc_mx.cuh"
#include "tcn_common.cuh"

namespace cfp {

namespace {

static __constant__ uint32_t CFP_PHASE_F32_L32_TCN[32] = CFP_PHASE_F32_L32_INIT;  // RN32(2^{h/32})

struct R34 {
  static constexpr int L = 32, NJ = 16, PO = 16, RB0 = 17, NRB = 2 * L - RB0;  // 47 R blocks
  static constexpr int BM = 128, KS = 32, MT = 8, ROWB = 64;
  static constexpr int NP = L * MT;                               // 256 MMA columns
  static constexpr int BSTAGE = (NRB * MT * ROWB + 1023) / 1024 * 1024;
  static constexpr int SFSTAGE = 1024;
  static constexpr int NSX = 2;                                   // token stages
  static constexpr int ACOL0 = 256, MCOL0 = 384, SFA0 = 416, SFB0 = 448;  // TMEM columns
  static constexpr int NWT = 256, MMA_WARP = 10, THREADS = 352;  // 8 weight warps, 2 token warps, MMA warp
  static constexpr int PFW = 4, PFX = 2;
  static constexpr size_t SMEM_USED = (size_t)NSX * (BSTAGE + SFSTAGE) + 1024;
  static constexpr size_t SMEM = SMEM_USED > 120 * 1024 ? SMEM_USED : 120 * 1024;  // one CTA per SM
};
static_assert(R34::ACOL0 + R34::NJ * 8 <= R34::MCOL0 && R34::SFB0 + 8 <= 512, "TMEM budget");

struct R34Shared {
  uint64_t wfull, wempty, xfull[2], xempty[2], acc_full, drain;
  uint32_t tmem_base;
  int abort_flag;
  int refB[8];
  int wref[128];
};

// Plane bytes of four codes: v = the E5M2 byte of +-2^q (0 for the zero
// code), nz = 0xFF where the code is not zero, j4 = the curve plane j of
// each code.
__device__ __forceinline__ void r34_word(uint32_t w, uint32_t& v, uint32_t& nz, uint32_t& j4) {
  const uint32_t m4 = w & 0x7F7F7F7Fu;
  nz = prmt_sign(m4 + 0x7F7F7F7Fu, 0xBA98u);
  const uint32_t lo = (m4 & 0x00FF00FFu) * 3u, hi = ((m4 >> 8) & 0x00FF00FFu) * 3u;  // 3m (<= 381) per 16-bit lane
  j4 = (lo & 0x001F001Fu) | ((hi & 0x001F001Fu) << 8);
  const uint32_t q4 = ((lo >> 5) & 0x000F000Fu) | (((hi >> 5) & 0x000F000Fu) << 8);  // floor(3m/32)
  v = ((w & 0x80808080u) | ((q4 + 0x09090909u) << 2)) & nz;  // exponent field q + 15 = floor(3m/32) + 9
}

// The codes of a 4-bit class c (low bits of j) given the sign masks of its
// four bits.
template <int C>
__device__ __forceinline__ uint32_t class_mask(uint32_t m0, uint32_t m1, uint32_t m2, uint32_t m3) {
  return ((C & 1) ? m0 : ~m0) & ((C & 2) ? m1 : ~m1) & ((C & 4) ? m2 : ~m2) & ((C & 8) ? m3 : ~m3);
}

// Pair planes P and P + 1 of a row's step (8 words each) into a 16-column store.
template <int P>
__device__ __forceinline__ void pair_words2(const uint32_t (&v)[8], const uint32_t (&mk)[8][4], uint32_t (&out)[16]) {
#pragma unroll
  for (int w = 0; w < 8; ++w) {
    out[w] = v[w] & class_mask<P>(mk[w][0], mk[w][1], mk[w][2], mk[w][3]);
    out[8 + w] = v[w] & class_mask<P + 1>(mk[w][0], mk[w][1], mk[w][2], mk[w][3]);
  }
}

}  // namespace

// X: [M x K] token codes, W: [N x K] weight codes (K contiguous), scales
// [rows x K/G]; C: [M x N] row-major.
__global__ void __launch_bounds__(R34::THREADS, 1)
    gemm_tcn_r34_kernel(const uint8_t* __restrict__ X, const int8_t* __restrict__ sX, const uint8_t* __restrict__ W,
                        const int8_t* __restrict__ sW, int M, int N, int K, int G, int gshift,
                        float* __restrict__ C, uint32_t* status, const TailPlan plan) {
  using Cf = R34;
  constexpr int L = Cf::L, MT = Cf::MT;
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* xstage = smem;
  uint8_t* sfstage = smem + (size_t)Cf::NSX * Cf::BSTAGE;
  R34Shared& sh = *reinterpret_cast<R34Shared*>(smem + (size_t)Cf::NSX * (Cf::BSTAGE + Cf::SFSTAGE));

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // this CTA's job: a whole tile (128 weight rows x 8 tokens) or one K piece
  const int ntw = (N + Cf::BM - 1) / Cf::BM;
  int tile = blockIdx.x, s0 = 0, s1 = K / Cf::KS;
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
  const int x0 = (tile / ntw) * MT, w0 = (tile % ntw) * Cf::BM;
  const int nb = K / G, total = s1 - s0;

  if (tid == 0) {
    tc::mbar_init(&sh.wfull, 8);  // the 8 weight warps
    tc::mbar_init(&sh.wempty, 1);
    for (int s = 0; s < Cf::NSX; ++s) {
      tc::mbar_init(&sh.xfull[s], 1);  // the step's token warp
      tc::mbar_init(&sh.xempty[s], 1);
    }
    tc::mbar_init(&sh.acc_full, 1);
    tc::mbar_init(&sh.drain, 1);
    sh.abort_flag = 0;
  }
  if (warp == Cf::MMA_WARP) {
    __syncwarp();  // TMEM allocation and release are warp-collective: a converged warp
    tc::tmem_alloc(&sh.tmem_base, 512);
    tc::tmem_relinquish();
  }
  const bool is_w = tid < Cf::NWT, is_x = !is_w && warp < Cf::MMA_WARP;
  const int q4 = warp & 3, hf = (warp >> 2) & 1;  // W: row quadrant, half (pair planes 8 hf ..)
  const int wrow = w0 + q4 * 32 + lane;
  // the references of the tile's weight rows and tokens, formed by all
  // threads from the two contiguous runs of scale rows (-128 past the ends)
  if (tid < 128) sh.wref[tid] = -128;
  if (tid < MT) sh.refB[tid] = -128;
  __syncthreads();
  rows_ref_coop(sW + (int64_t)w0 * nb, min(Cf::BM, N - w0), nb, sh.wref, tid, Cf::THREADS);
  rows_ref_coop(sX + (int64_t)x0 * nb, min(MT, M - x0), nb, sh.refB, tid, Cf::THREADS);
  for (int o = tid * 16; o < Cf::NSX * (Cf::BSTAGE + Cf::SFSTAGE); o += Cf::THREADS * 16)
    *reinterpret_cast<uint4*>(smem + o) = make_uint4(0, 0, 0, 0);
  tc::fence_proxy_async_smem();
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  const int ref = is_w ? sh.wref[q4 * 32 + lane] : -128;  // this W thread's weight row

  if (is_w) {
    // ---------------------------- weight producers ---------------------------
    constexpr int PF = Cf::PFW;
    const bool rowok = wrow < N;
    const uint8_t* src = W + (int64_t)(rowok ? wrow : 0) * K;
    const int8_t* srow = sW + (int64_t)(rowok ? wrow : 0) * nb;
    const uint32_t lane_base = tmem + ((uint32_t)(q4 * 32) << 16);
    auto load = [&](int g, uint4& lo, uint4& hi, int& raw) {
      lo = hi = make_uint4(0, 0, 0, 0);
      raw = 0;
      if (rowok && g < total) {
        const int s = s0 + g;
        const uint4* p = reinterpret_cast<const uint4*>(src + (int64_t)s * Cf::KS);
        lo = __ldg(p);
        hi = __ldg(p + 1);
        raw = (int)__ldg(srow + (s >> gshift));
      }
    };
    auto step = [&](const int g, uint4 lo, uint4 hi, const int raw) -> bool {
      bool keep;
      const uint32_t sf = mx_sf(raw - ref, 0, keep) * 0x01010101u;
      if (!keep) lo = hi = make_uint4(0, 0, 0, 0);
      // the step's 32 codes: plane bytes, curve planes and the sign masks of
      // the class bits (bits 0-3 of j); decoded while the step before is
      // still in the tensor pipe
      const uint32_t cw[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
      uint32_t v[8], j4[8], mk[8][4];
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        uint32_t nz;
        r34_word(cw[w], v[w], nz, j4[w]);
#pragma unroll
        for (int b = 0; b < 4; ++b) mk[w][b] = prmt_sign(j4[w] << (7 - b), 0xBA98u);
      }
      if (g >= 1) {
        // the weight unit is free once the MMAs of step g - 1 retired
        const bool ok = wait_all(&sh.wempty, (g - 1) & 1);
        tc::fence_after_sync();
        if (!ok) {
          if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
          return false;
        }
      }
      // this half's 8 pair planes (8 columns each), two per store
      uint32_t r[16];
      if (hf == 0) {
        pair_words2<0>(v, mk, r);
        tmem_st16(lane_base + Cf::ACOL0 + 0 * 8, r);
        pair_words2<2>(v, mk, r);
        tmem_st16(lane_base + Cf::ACOL0 + 2 * 8, r);
        pair_words2<4>(v, mk, r);
        tmem_st16(lane_base + Cf::ACOL0 + 4 * 8, r);
        pair_words2<6>(v, mk, r);
        tmem_st16(lane_base + Cf::ACOL0 + 6 * 8, r);
        // metadata: bit 4 of j picks plane j or j + 16 of the pair
        const uint32_t mt[2] = {pair_meta<4>(j4[0], j4[1], j4[2], j4[3]), pair_meta<4>(j4[4], j4[5], j4[6], j4[7])};
        tc::tmem_st2(lane_base + Cf::MCOL0, mt);
        tc::tmem_st1(lane_base + Cf::SFA0 + q4, sf);
      } else {
        pair_words2<8>(v, mk, r);
        tmem_st16(lane_base + Cf::ACOL0 + 8 * 8, r);
        pair_words2<10>(v, mk, r);
        tmem_st16(lane_base + Cf::ACOL0 + 10 * 8, r);
        pair_words2<12>(v, mk, r);
        tmem_st16(lane_base + Cf::ACOL0 + 12 * 8, r);
        pair_words2<14>(v, mk, r);
        tmem_st16(lane_base + Cf::ACOL0 + 14 * 8, r);
      }
      tc::tmem_wait_st();
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&sh.wfull);
      return true;
    };
    uint4 ql[PF], qh[PF];
    int rq[PF];
#pragma unroll
    for (int u = 0; u < PF; ++u) load(u, ql[u], qh[u], rq[u]);
    bool run = true;
    for (int i = 0; i < total && run; i += PF) {
#pragma unroll
      for (int u = 0; u < PF; ++u) {
        if (i + u >= total || !step(i + u, ql[u], qh[u], rq[u])) {
          run = false;
          break;
        }
        load(i + u + PF, ql[u], qh[u], rq[u]);
      }
    }
    // Epilogue (after the last MMA): this half's 4 tokens; per token the
    // phase sums D[w][8 h + m] are combined as sum_h 2^{h/32} S_h (FP32,
    // phase order) and scaled by 2^{ref_w + ref_m - 2 MX_OFF}.  A whole tile
    // stores C, a K piece adds to zeroed C.
    const bool aborted = __any_sync(0xffffffffu, read_abort(&sh.abort_flag) != 0);
    const bool ok = !aborted && wait_all(&sh.acc_full, 0);
    if (!ok && lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
    tc::fence_after_sync();
    float t[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
    for (int h0 = 0; h0 < L; h0 += 4) {
      uint32_t acc[4][8];
#pragma unroll
      for (int h = 0; h < 4; ++h) tc::tmem_ld8(lane_base + (uint32_t)((h0 + h) * MT), acc[h]);
      tc::tmem_wait_ld();
#pragma unroll
      for (int h = 0; h < 4; ++h) {
        const float c = __uint_as_float(CFP_PHASE_F32_L32_TCN[h0 + h]);
#pragma unroll
        for (int m = 0; m < 4; ++m) t[m] = fmaf(c, __uint_as_float(hf ? acc[h][4 + m] : acc[h][m]), t[m]);
      }
    }
    if (rowok && ok) {
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        const int tok = 4 * hf + m, row = x0 + tok;
        if (row < M) {
          const float y = scale_pow2(t[m], ref + sh.refB[tok] - 2 * MX_OFF);
          float* dst = C + (int64_t)row * N + wrow;
          if (split)
            atomicAdd(dst, y);
          else
            *dst = y;
        }
      }
    }
  } else if (is_x) {
    // ---------------------------- token producers ----------------------------
    // Lane l: token l & 7 of the tile, codes 8 (l >> 3) .. + 7 of a step (a
    // 16-byte chunk of each 64-byte R row); warp 8 + (g & 1) takes step g.
    constexpr int PF = Cf::PFX;
    const int gx = warp - Cf::NWT / 32;
    const int tok = lane & 7, c = lane >> 3;
    const int xrow = x0 + tok < M ? x0 + tok : -1;
    const int xref = xrow >= 0 ? sh.refB[tok] : 0;
    const uint32_t xbase = (uint32_t)(c * 128 + tok * 16);
    auto load = [&](int i, uint2& cw, int& raw) {
      cw = make_uint2(0u, 0u);
      raw = 0;
      const int g = gx + 2 * i;
      if (xrow >= 0 && g < total) {
        const int s = s0 + g;
        cw = __ldg(reinterpret_cast<const uint2*>(X + (int64_t)xrow * K + (int64_t)s * Cf::KS + c * 8));
        raw = (int)__ldg(sX + (int64_t)xrow * nb + (s >> gshift));
      }
    };
    auto step = [&](const int g, const uint2 cw, const int raw) -> bool {
      const int xs = g & 1;
      if (g >= Cf::NSX) {
        const bool ok = wait_all(&sh.xempty[xs], ((g >> 1) - 1) & 1);
        if (!ok) {
          if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
          return false;
        }
      }
      uint8_t* stg = xstage + (size_t)xs * Cf::BSTAGE;
      uint8_t* sfs = sfstage + (size_t)xs * Cf::SFSTAGE;
      if (xrow >= 0) {
        bool keep;
        const uint32_t sf = mx_sf(raw - xref, 0, keep);
        // R block b holds Q_b[k] in byte 2k and Q_{b-16}[k] in byte 2k + 1;
        // the two planes share their class (bits 0-3 of j) and differ in bit
        // 4 (T), so per 16-bit lane (one code) three words place the code's
        // value by its T: carry copies on both sides (b < 32, T(b) = 1),
        // plain even / carry odd (32 <= b < 48), plain on both (b >= 48);
        // block b is its word masked to the codes of class b mod 16
        uint32_t qcc[4], qpc[4], qpp[4], dm[4][4];
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          uint32_t v, nz, j4;
          r34_word(keep ? (q ? cw.y : cw.x) : 0u, v, nz, j4);
          const uint32_t vc = v + (nz & 0x04040404u);  // the carry copy 2^{q + 1}
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const uint32_t sdup = hh ? 0xBBAAu : 0x9988u, dup = hh ? 0x3322u : 0x1100u, ilv = hh ? 0x7362u : 0x5140u;
            const int i = 2 * q + hh;
            const uint32_t dt = prmt_sign(j4 << 3, sdup);
#pragma unroll
            for (int b = 0; b < 4; ++b) dm[i][b] = prmt_sign(j4 << (7 - b), sdup);
            qcc[i] = __byte_perm(vc, vc, dup) & (dt ^ 0xFF00FF00u);
            qpp[i] = __byte_perm(v, v, dup) & (dt ^ 0xFF00FF00u);
            qpc[i] = __byte_perm(v, vc, ilv) & (dt ^ 0x00FF00FFu);
          }
        }
#pragma unroll
        for (int b = Cf::RB0; b < 2 * L; ++b) {
          const int cls = b & 15;
          uint32_t rr[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const uint32_t srcw = b < L ? qcc[i] : (b < L + Cf::PO ? qpc[i] : qpp[i]);
            rr[i] = srcw & ((cls & 1) ? dm[i][0] : ~dm[i][0]) & ((cls & 2) ? dm[i][1] : ~dm[i][1]) &
                    ((cls & 4) ? dm[i][2] : ~dm[i][2]) & ((cls & 8) ? dm[i][3] : ~dm[i][3]);
          }
          *reinterpret_cast<uint4*>(stg + xbase + (b - Cf::RB0) * (MT * Cf::ROWB)) =
              make_uint4(rr[0], rr[1], rr[2], rr[3]);
        }
        if (c == 0) {
          // the token's factor in every column n = 8 h + tok of the MMA
          const uint32_t sw = sf * 0x01010101u;
#pragma unroll
          for (int h = 0; h < L; ++h) *reinterpret_cast<uint32_t*>(sfs + sfb_off(h * MT + tok)) = sw;
        }
      }
      tc::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) tc::mbar_arrive(&sh.xfull[xs]);
      return true;
    };
    const int nown = (total - gx + 1) / 2;
    uint2 q[PF];
    int rq[PF];
#pragma unroll
    for (int u = 0; u < PF; ++u) load(u, q[u], rq[u]);
    bool run = true;
    for (int i = 0; i < nown && run; i += PF) {
#pragma unroll
      for (int u = 0; u < PF; ++u) {
        if (i + u >= nown || !step(gx + 2 * (i + u), q[u], rq[u])) {
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
    const uint32_t idesc = idesc_mx_e5m2(Cf::NP, true);
    constexpr int gbytes = MT * Cf::ROWB;  // bytes of one column block
    bool ok = true;
    for (int g = 0; g < total && ok; ++g) {
      const int xs = g & 1;
      ok = wait_all(&sh.wfull, g & 1) && wait_all(&sh.xfull[xs], (g >> 1) & 1);
      if ((g & 7) == 0) ok = ok && !read_abort(&sh.abort_flag);
      if (!ok) break;
      tc::fence_after_sync();
      // the step's token factors: columns 0..127 and 128..255
      const uint8_t* sfs = sfstage + (size_t)xs * Cf::SFSTAGE;
      tmem_cp_sf_if(leader, tmem + Cf::SFB0, sfs);
      tmem_cp_sf_if(leader, tmem + Cf::SFB0 + 4, sfs + 512);
#pragma unroll
      for (int p = 0; p < Cf::NJ; ++p) {
        // pair plane p against the window of R blocks from 32 - p
        const uint32_t boff = (uint32_t)(xs * Cf::BSTAGE + (L - p - Cf::RB0) * gbytes);
        mma_sp_mx_if(leader, tmem, tmem + Cf::ACOL0 + p * 8, bdesc0 + (uint64_t)(boff >> 4), tmem + Cf::MCOL0,
                     idesc, tmem + Cf::SFA0, tmem + Cf::SFB0, (g == 0 && p == 0) ? 0u : 1u);
      }
      tc::mma_commit_if(leader, &sh.wempty);
      tc::mma_commit_if(leader, &sh.xempty[xs]);
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
  if (warp == Cf::MMA_WARP) {
    __syncwarp();
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

// x: [M x K] token codes, w: [N x K] weight codes; c: [M x N].
cudaError_t launch_gemm_tensor_narrow_r34(int G, const uint8_t* x, const int8_t* sx, const uint8_t* w,
                                          const int8_t* sw, int64_t M, int64_t N, int64_t K, float* c,
                                          uint32_t* st, cudaStream_t s, int sms) {
  using Cf = R34;
  static_assert(sizeof(R34Shared) <= 1024, "shared tail");
  static_assert(Cf::SMEM <= 227 * 1024, "shared memory");
  cudaError_t e = cudaFuncSetAttribute(gemm_tcn_r34_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cf::SMEM);
  if (e != cudaSuccess) return e;
  const int64_t ntw = (N + Cf::BM - 1) / Cf::BM, ng = (M + Cf::MT - 1) / Cf::MT, tiles = ntw * ng;
  const TailPlan plan = tcn_plan(tiles, sms, (int)(K / Cf::KS));
  if (plan.nsplit > 0) {
    // C of the split tiles starts at zero: the token rows from the first split tile's group on
    const int64_t row0 = (plan.ntiles_full / ntw) * Cf::MT;
    e = cudaMemsetAsync(c + row0 * N, 0, (size_t)((M - row0) * N) * sizeof(float), s);
    if (e != cudaSuccess) return e;
  }
  const unsigned grid = (unsigned)(plan.ntiles_full + 2 * plan.nsplit);
  int gshift = 0;  // scale block of step s is s >> gshift
  while ((Cf::KS << gshift) < G) ++gshift;
  gemm_tcn_r34_kernel<<<grid, Cf::THREADS, Cf::SMEM, s>>>(x, sx, w, sw, (int)M, (int)N, (int)K, G, gshift, c, st,
                                                          plan);
  return cudaGetLastError();
}

}  // namespace cfp
