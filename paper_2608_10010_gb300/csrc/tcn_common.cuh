// Helpers shared by the phases-along-N tensor-core kernels (gemm_tcn.cu:
// binary formats; gemm_tcn_r34.cu: r = 2^{3/4}): the 2:4 metadata of pair
// planes, whole-warp bounded waits, TMEM stores and the K-split plan of the
// last wave.
#pragma once
#include <mutex>
#include <unordered_map>

#include "gemm_tc.cuh"

namespace cfp {

namespace {

// Interleave two words (elements 4q..4q+3 each) into X0 Y0 X1 Y1 | X2 Y2 X3 Y3.
__device__ __forceinline__ uint2 interleave2(uint32_t x, uint32_t y) {
  return make_uint2(__byte_perm(x, y, 0x5140), __byte_perm(x, y, 0x7362));
}

// Metadata word of 16 codes (four code words) of a 2:4 operand with 8-bit
// elements: per chunk of two elements, position bit(2c) and 2 + bit(2c + 1),
// where bit is bit MBIT of each byte (the curve-index bit that selects the
// partner plane).  Element c = 4q + i (byte i of word q) puts its bit at
// bit 2c = 8q + 2i: gathering the four words' bits side by side puts it at
// 8i + 2q, a 4 x 4 matrix of 2-bit cells stored transposed, which two delta
// swaps (the off-diagonal 2 x 2 blocks, then the off-diagonal cells of each
// block) transpose.
template <int MBIT>
__device__ __forceinline__ uint32_t pair_meta(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3) {
  const uint32_t w[4] = {w0, w1, w2, w3};
  uint32_t a = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int sh = MBIT - 2 * q;  // bit MBIT of byte i -> bit 8 i + 2 q
    a |= (sh >= 0 ? w[q] >> sh : w[q] << -sh) & (0x01010101u << (2 * q));
  }
  uint32_t t = (a ^ (a >> 12)) & 0x0000F0F0u;
  a ^= t ^ (t << 12);
  t = (a ^ (a >> 6)) & 0x00CC00CCu;
  a ^= t ^ (t << 6);
  return a | 0x88888888u;  // bit 3 of each nibble: the second element's position is 2 + bit
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

// Split plan of the narrow kernel: the tile kernel's tail search with finer
// split points (a narrow tile is short, so its pieces' fixed costs weigh
// more and the best point moves).  With fewer tiles than SMs every tile is
// split in halves when all pieces fit in one wave, and none is split
// otherwise: a CTA's fixed cost (about 6 us of set-up and first decode, a
// sixth of a 128-step tile at few tokens) makes a second wave of short
// pieces slower than the whole tiles (measured at 112 tiles on 152 SMs:
// 44.6 us unsplit, 49-53 us with the pieces at 1/2 or 3/4).
inline TailPlan tcn_plan_search(int64_t tiles, int sms, int nsub) {
  TailPlan best{(int)tiles, 0, 0};
  if (sms <= 0 || nsub < 2 || tiles % sms == 0) return best;
  if (tiles < sms) return 2 * tiles <= sms ? TailPlan{0, (int)tiles, nsub / 2} : best;
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

}  // namespace

}  // namespace cfp
