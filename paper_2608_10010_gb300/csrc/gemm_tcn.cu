// Tensor-core closed-product GEMM for few activation rows (algo
// TENSOR_NARROW): the phases of Eq. 5 run along the MMA's N dimension.
//
// C = X_hat W_hat^T with X the M activation rows (the API's A operand, format
// FX) and W the N weight rows (the API's B operand, format FW).  As in the
// tile kernel, every operand splits into curve planes of exact powers of two
// (plane k holds the elements of curve index k), and plane k_x of X times
// plane k_w of W lands on phase h = (k_x WX + k_w WW) mod L with carry
// c = floor((k_x WX + k_w WW) / L) (Eq. 2 on the shared lattice L).
//
// Here the weight rows are the MMA's 128-row TMEM operand and the phase is a
// column index: the accumulator of a CTA is D[w][h Mt + m] (weight row w,
// phase h, token m of the CTA's Mt tokens), the per-phase sums S_h of Eq. 5
// for every token side by side.  For weight plane k_w the shared-memory
// operand must hold, in column block h, the X plane with k_x WX =
// (h - k_w WW) mod L, doubled where the sum wrapped (carry).  Lay out the
// sequence of 2L column blocks
//   Q = [ 2 X_0 ... (lattice positions 0 .. L-1, carry copies) |
//           X_0 ... (lattice positions 0 .. L-1, plain) ]
// (block u of each half holds the plane with k_x WX = u, zero where no plane
// sits on u); then the operand of weight plane k_w is the window of L blocks
// that starts at block L - k_w WW: its block h is plain for h >= k_w WW and
// the carry copy of position L - k_w WW + h otherwise.  A window is a start
// address of the MMA's shared-memory descriptor, so each pipeline step of 32
// codes costs K_W MMAs of 128 x (L Mt) x 32 (8 for 8-curve weights) on 2L Mt
// rows of staged X planes, against K_X K_W MMAs of the tile kernel, whose
// 128-row activation tile is mostly empty when M is small.
//
// Roles (8 + NXT/32 + 1 warps):
//   warps 0-7   W producers, two threads per weight row (16 codes each per
//               step): codes -> planes -> TMEM (as the tile kernel's A
//               producers), prefetching PF steps ahead (the weights stream
//               from HBM); after the last step they run the epilogue.
//   next warps  X producers, two threads per token: codes -> plane and
//               carry-plane words -> the 2L blocks of the step's stage.
//   last warp   TMEM allocation and MMA issue (one elected lane).
// With fewer weight tiles than SMs every tile is split in K into two pieces
// (chosen by the same greedy-dispatch simulation as the tile kernel's tail);
// a piece adds its outputs to zeroed C atomically, two additions per output,
// so the result does not depend on their order.  Every wait is bounded.
#include "gemm_tc.cuh"

namespace cfp {

namespace {

template <int FX, int FW>
struct TcnCfg {
  using P = Pair<FX, FW>;
  static constexpr int KW = Fmt<FW>::K, L = P::L, WX = P::WA, WW = P::WB;
  static constexpr int BM = 128;         // weight rows per CTA (TMEM lanes)
  static constexpr int KS = 32;          // codes per pipeline step (K of one FP8 MMA)
  static constexpr int MTMAX = 256 / L;  // tokens per CTA: L Mt <= 256 (MMA N)
  static constexpr int NBLK = 2 * L;     // column blocks of the doubled sequence
  static constexpr int NSB = 4;          // pipeline depth (X stages = W TMEM units)
  static constexpr int AU_COLS = KW * 8; // TMEM columns of one step's W planes
  static constexpr int ACOL0 = 256;      // W units after the accumulator
  static_assert(ACOL0 + NSB * AU_COLS <= 512, "TMEM budget");
  static constexpr int NAW = 8;              // W producer warps
  static constexpr int NXT = 2 * MTMAX;      // X producer threads
  static constexpr int THREADS = NAW * 32 + NXT + 32;
  static constexpr int MMA_WARP = (NAW * 32 + NXT) / 32;
  static_assert(NXT % 32 == 0, "X producer warps");
  static constexpr int BSTAGE = NBLK * MTMAX * 32;  // bytes of one step's X planes
  static constexpr int PBX = FX == CURVEFP_E5C2 ? 1 : 0;  // plane exponent bias
  static constexpr int PBW = FW == CURVEFP_E5C2 ? 1 : 0;
  static constexpr int PF = 8;  // steps of codes in flight per producer thread
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

}  // namespace

template <int FX, int FW>
__global__ void __launch_bounds__(TcnCfg<FX, FW>::THREADS, 1)
    gemm_tcn_kernel(const uint8_t* __restrict__ X, const int8_t* __restrict__ sX, const uint8_t* __restrict__ W,
                    const int8_t* __restrict__ sW, int M, int N, int K, int G, int gshift, int Mt,
                    float* __restrict__ C, uint32_t* status, const TailPlan plan) {
  using Cfg = TcnCfg<FX, FW>;
  constexpr int L = Cfg::L, NSB = Cfg::NSB, NAW = Cfg::NAW, PF = Cfg::PF;
  static_assert(NSB == TC_MAX_RING, "barrier rings");
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
  const int x0 = (tile / ntw) * Mt, w0 = (tile % ntw) * Cfg::BM;
  const int nb = K / G, total = s1 - s0;

  if (tid == 0) {
    for (int s = 0; s < NSB; ++s) {
      tc::mbar_init(&sh.full[s], NAW + Cfg::NXT / 32);  // one arrival per producer warp
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
  // producer geometry and the row's reference exponent (largest block scale)
  const bool is_w = warp < NAW;
  const bool is_prod = warp < Cfg::MMA_WARP;
  const int t_x = tid - NAW * 32;
  const int rloc = is_w ? ((warp & 3) * 32 + lane) : (t_x >> 1);  // weight row / token of the CTA
  const int part = is_w ? (warp >> 2) : (t_x & 1);                // 16-byte half of the step's 32 codes
  const int r = (is_w ? w0 : x0) + rloc;
  const bool rowok = is_prod && (is_w ? r < N : (rloc < Mt && r < M));
  int ref = -128;
  if (rowok) {
    const int8_t* s = (is_w ? sW : sX) + (int64_t)r * nb;
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
  if (!is_w && is_prod && part == 0 && rloc < Cfg::MTMAX) sh.refB[rloc] = ref;
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;

  if (is_prod) {
    // ------------------------------ producers ------------------------------
    const uint8_t* src = (is_w ? W : X) + (int64_t)r * K + part * 16;
    const int8_t* srow = (is_w ? sW : sX) + (int64_t)r * nb;
    const int bias = is_w ? Cfg::PBW : Cfg::PBX;
    auto load = [&](int g, uint4& cw, int& raw) {
      cw = make_uint4(0, 0, 0, 0);
      raw = 0;
      if (rowok && g < total) {
        const int s = s0 + g;
        cw = __ldg(reinterpret_cast<const uint4*>(src + (int64_t)s * Cfg::KS));
        raw = (int)__ldg(srow + (s >> gshift));
      }
    };
    const uint32_t lane_base = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    // Epilogue (W producers, after the last MMA): chunks of 8 tokens, this
    // thread's half taking every other chunk; per token the phase sums
    // D[w][h Mt + m] are combined as sum_h 2^{h/L} S_h (FP32, phase order)
    // and scaled by 2^{ref_w + ref_m}.  A whole tile stores C, a K piece adds
    // to zeroed C.
    auto epilogue = [&]() -> bool {
      const bool ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.acc_full, 0));
      if (!ok) {
        if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
        sh.abort_flag = 1;
      }
      tc::fence_after_sync();
      const int nch = Mt >> 3;
#pragma unroll 1
      for (int ch = part; ch < nch; ch += 2) {
        uint32_t acc[L][8];
#pragma unroll
        for (int h = 0; h < L; ++h) tc::tmem_ld8(lane_base + h * Mt + ch * 8, acc[h]);
        tc::tmem_wait_ld();
        if (rowok && ok) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int tok = ch * 8 + j, m = x0 + tok;
            if (m < M) {
              float t = 0.f;
#pragma unroll
              for (int h = 0; h < L; ++h) t = fmaf(phase_const(L, h), __uint_as_float(acc[h][j]), t);
              const float y = scalbnf(t, ref + Cfg::PBW + sh.refB[tok] + Cfg::PBX);
              float* dst = C + (int64_t)m * N + r;
              if (split)
                atomicAdd(dst, y);
              else
                *dst = y;
            }
          }
        }
      }
      return ok;
    };
    // One pipeline step of this producer thread; false ends the loop.
    auto step = [&](const int g, const uint4 cw, const int raw) -> bool {
      const int off = raw - ref - bias;
      const int st = g % NSB;
      if (g >= NSB) {
        // stage / TMEM unit st is free once the MMAs of step g - NSB retired
        const bool ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.empty[st], ((g / NSB) - 1) & 1));
        tc::fence_after_sync();
        if (!ok) {
          if (lane == 0) raise_flag(status, CURVEFP_DEV_TIMEOUT);
          sh.abort_flag = 1;
          return false;
        }
      }
      if (is_w) {
        uint32_t v[4], vc[4], mk[4][4];
        PlaneFmt<FW>::template decode<PLANE_E5M2, 4>(cw, off, v, vc, mk, false);
        uint32_t pl[4][8];
#pragma unroll
        for (int c = 0; c < 4; ++c) PlaneFmt<FW>::planes(v[c], mk[c], pl[c]);
        // plane k_w: 8 columns of the unit, this thread's half = 4 of them
#pragma unroll
        for (int j = 0; j < Cfg::KW; ++j) {
          const uint32_t reg[4] = {pl[0][j], pl[1][j], pl[2][j], pl[3][j]};
          tc::tmem_st4(lane_base + Cfg::ACOL0 + st * Cfg::AU_COLS + j * 8 + part * 4, reg);
        }
        tc::tmem_wait_st();
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&sh.full[st]);
        if (g == total - 1) return epilogue();
      } else {
        uint32_t v[4], vc[4], mk[4][4];
        PlaneFmt<FX>::template decode<PLANE_E5M2, 4>(cw, off, v, vc, mk, true);
        uint32_t pv[4][8], pc[4][8];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          PlaneFmt<FX>::planes(v[c], mk[c], pv[c]);
          PlaneFmt<FX>::planes(vc[c], mk[c], pc[c]);
        }
        if (rloc < Mt) {
          uint8_t* stg = xstage + (size_t)st * Cfg::BSTAGE;
          // lattice position u holds plane u / WX where WX divides u
#pragma unroll
          for (int u = 0; u < L; ++u) {
            const bool on = (u % Cfg::WX) == 0;
            const int k = u / Cfg::WX;
            const uint4 cq = on ? make_uint4(pc[0][k], pc[1][k], pc[2][k], pc[3][k]) : make_uint4(0, 0, 0, 0);
            const uint4 pq = on ? make_uint4(pv[0][k], pv[1][k], pv[2][k], pv[3][k]) : make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(stg + core_off(u * Mt + rloc, part)) = cq;
            *reinterpret_cast<uint4*>(stg + core_off((L + u) * Mt + rloc, part)) = pq;
          }
        }
        tc::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&sh.full[st]);
      }
      return true;
    };
    // PF register sets of codes, each loaded PF steps before its use (the
    // weights stream from HBM and a narrow step is short)
    uint4 q[PF];
    int rq[PF];
#pragma unroll
    for (int u = 0; u < PF; ++u) load(u, q[u], rq[u]);
    bool run = true;
    for (int g = 0; g < total && run; g += PF) {
#pragma unroll
      for (int u = 0; u < PF; ++u) {
        if (g + u >= total || !step(g + u, q[u], rq[u])) {
          run = false;
          break;
        }
        load(g + u + PF, q[u], rq[u]);
      }
    }
  } else {
    // ------------------------------ MMA issuer -------------------------------
    const uint32_t leader = tc::elect_one();
    const uint64_t bdesc0 = tc::smem_desc(tc::smem_u32(xstage), 128, 256);
    const uint32_t idesc = tc::idesc_bf16_f32(Cfg::BM, L * Mt);  // E5M2 x E5M2 -> F32, N = L Mt
    const int gbytes = (Mt >> 3) * 256;                          // bytes of one column block
    bool ok = true;
    for (int g = 0; g < total && ok; ++g) {
      const int st = g % NSB;
      ok = __all_sync(0xffffffffu, tc::mbar_wait(&sh.full[st], (g / NSB) & 1));
      if ((g & 7) == 0) ok = ok && !read_abort(&sh.abort_flag);
      if (!ok) break;
      tc::fence_after_sync();
#pragma unroll
      for (int kw = 0; kw < Cfg::KW; ++kw) {
        // weight plane k_w against the window of column blocks from L - k_w WW
        const uint32_t a_t = tmem + Cfg::ACOL0 + st * Cfg::AU_COLS + kw * 8;
        const uint32_t boff = (uint32_t)(st * Cfg::BSTAGE + (L - kw * Cfg::WW) * gbytes);
        tc::mma_f8_ts_if(leader, tmem, a_t, bdesc0 + (uint64_t)(boff >> 4), idesc, (g == 0 && kw == 0) ? 0u : 1u);
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

template <int FX, int FW>
cudaError_t launch_tcn_t(int G, const uint8_t* x, const int8_t* sx, const uint8_t* w, const int8_t* sw, int64_t M,
                         int64_t N, int64_t K, float* c, uint32_t* st, cudaStream_t s, int sms) {
  using Cfg = TcnCfg<FX, FW>;
  static_assert(sizeof(TcShared) <= 2048, "shared tail");
  static_assert(Cfg::SMEM <= 227 * 1024, "shared memory");
  auto kern = gemm_tcn_kernel<FX, FW>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::SMEM);
  if (e != cudaSuccess) return e;
  // token groups of equal size Mt (a multiple of 8, at most MTMAX)
  int64_t ng = (M + Cfg::MTMAX - 1) / Cfg::MTMAX;
  const int Mt = (int)(((M + ng - 1) / ng + 7) / 8 * 8);
  ng = (M + Mt - 1) / Mt;
  const int64_t ntw = (N + Cfg::BM - 1) / Cfg::BM, tiles = ntw * ng;
  const TailPlan plan = tcn_plan(tiles, sms, (int)(K / Cfg::KS));
  if (plan.nsplit > 0) {
    // C of the split tiles starts at zero: whole token groups from the first one
    const int64_t row0 = (plan.ntiles_full / ntw) * Mt;
    e = cudaMemsetAsync(c + row0 * N, 0, (size_t)((M - row0) * N) * sizeof(float), s);
    if (e != cudaSuccess) return e;
  }
  const unsigned grid = (unsigned)(plan.ntiles_full + 2 * plan.nsplit);
  int gshift = 0;  // scale block of step s is s >> gshift
  while ((Cfg::KS << gshift) < G) ++gshift;
  kern<<<grid, Cfg::THREADS, Cfg::SMEM, s>>>(x, sx, w, sw, (int)M, (int)N, (int)K, G, gshift, Mt, c, st, plan);
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
#define CFP_T(X, Y) \
  if (fa == X && fb == Y) return launch_tcn_t<X, Y>(G, a, sa, b, sb, M, N, K, c, status, s, sms);
  CFP_T(CURVEFP_E3C3, CURVEFP_E3C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E4C3)
  CFP_T(CURVEFP_E5C2, CURVEFP_E4C3)
  CFP_T(CURVEFP_E4C3, CURVEFP_E5C2)
  CFP_T(CURVEFP_E5C2, CURVEFP_E5C2)
#undef CFP_T
  return cudaErrorInvalidValue;
}

}  // namespace cfp
