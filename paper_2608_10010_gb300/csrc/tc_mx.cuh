// Block-scaled (MX) form of the tensor-core planes: the plane value of an
// element is the power of two 2^e of its code alone, and the block scale
// enters the MMA as a UE8M0 scale factor per 32-code step (Sec. 3.1 Eq. 1:
// x = (-1)^s 2^{a_b} 2^{e + k/K}; Sec. 3.2 Eq. 2, Eq. 5).  Every code of the
// three binary formats has an exact E5M2 plane value (E5C2's two lowest
// binades as E5M2 subnormals), so nothing is flushed relative to the row's
// other blocks: a block's scale relative to the row reference only changes
// its scale factor.
//
// Scale factors (UE8M0: byte b stands for 2^{b - 127}).  With d = a_b - ref
// (ref = the row's largest block scale, d <= 0) a block's factor is
// 2^{d + MX_OFF}, byte d + MX_SF0, MX_SF0 = 127 + MX_OFF.  MX_OFF = 32 puts
// the largest products near 2^{2 MX_OFF + 32} so that a K of up to 2^20
// products stays below FP32's overflow, and keeps every product down to
// 2^{-190} of 2^{ref_a + ref_b} inside FP32's normal range.  Blocks with
// d < -MX_SF0 (no byte) are dropped: their elements are below 2^{-143} of
// 2^{ref}.
//
// TMEM layout of the factors of an M = 128 MMA (found by a layout probe of
// tcgen05.mma.kind::mxf8f6f4.block_scale on sm_103a; a 2:4-sparse MMA of
// logical K 64 reads bytes id and id + 1):
//   A: row m reads lane m, column base + m / 32, byte id (four columns).
//   B: column n reads lane 32 q + n % 32 of every lane quadrant q (the four
//      quadrants hold copies), column base + n / 32, byte id; a
//      tcgen05.cp .32x128b.warpx4 from 512 contiguous bytes of shared memory
//      (row i = 16 bytes = four columns of lane i) writes four columns.
#pragma once
#include "tc_planes.cuh"
#include "tc_ptx.cuh"

namespace cfp {

constexpr int MX_OFF = 32;
constexpr int MX_SF0 = 127 + MX_OFF;

// E5M2 bytes of 2^{x - 16} for four lanes x in [0, 31]: (x - 1) << 2 from
// x = 2 (normal), 0x02 and 0x01 for x = 1 and 0 (subnormal 2^-15, 2^-16).
// No lane borrows from or carries into a neighbour (x <= 31).
__device__ __forceinline__ uint32_t e5m2_pow2(uint32_t x) {
  const uint32_t ge2 = prmt_sign(x + 0x7E7E7E7Eu, 0xBA98u);
  const uint32_t nrm = ((((x | 0x80808080u) - 0x01010101u) & 0x1F1F1F1Fu) << 2) & ge2;
  return nrm | ((x + 0x01010101u) & ~ge2);
}

// Plane bytes of four codes: v = +-2^{e - BIAS} where the code is nonzero
// (and, for BIAS = 1, representable), and the x2 carry copy vc = +-2^{e -
// BIAS + 1} (every nonzero code).  BIAS = 1 only for E5C2 operands that take
// the carry copies: there the plain copy of the lowest binade (e = -16,
// 2^-17) has no E5M2 value and is dropped; every other value is exact.
template <int FMT, int BIAS>
__device__ __forceinline__ void mx_word(uint32_t w, uint32_t& v, uint32_t& vc) {
  using F = Fmt<FMT>;
  const uint32_t sgn = w & 0x80808080u;
  const uint32_t nz = prmt_sign((w & CodeBits<FMT>::MM) + 0x7F7F7F7Fu, 0xBA98u);  // rank m != 0
  const uint32_t eb = (w >> F::C) & (((1u << F::E) - 1u) * 0x01010101u);         // e + 2^{E-1}
  if constexpr (F::E < 5) {
    static_assert(BIAS == 0, "E3/E4 planes are exact without a bias");
    // e5 = e + 15 in [7, 22]: always a normal E5M2 exponent, carry included
    v = (sgn | ((eb + (uint32_t)(15 - (1 << (F::E - 1))) * 0x01010101u) << 2)) & nz;
    vc = v + (nz & 0x04040404u);
  } else {
    if constexpr (BIAS == 0) {
      v = (sgn | e5m2_pow2(eb)) & nz;  // 2^{eb - 16} = 2^e
      vc = 0u;                         // (no carry copies on this side)
    } else {
      const uint32_t ge1 = prmt_sign(eb + 0x7F7F7F7Fu, 0xBA98u);  // eb >= 1
      const uint32_t x = ((eb | 0x80808080u) - 0x01010101u) & 0x1F1F1F1Fu;
      v = (sgn | e5m2_pow2(x)) & nz & ge1;  // 2^{e - 1}
      vc = (sgn | e5m2_pow2(eb)) & nz;      // 2^{e}
    }
  }
}

// t 2^e, the epilogue's output scaling: a multiply by the normal float 2^e
// where e is in [-126, 127] (one correctly rounded product, the value
// scalbnf returns), scalbnf itself outside that range.
__device__ __forceinline__ float scale_pow2(float t, int e) {
  return (e >= -126 && e <= 127) ? t * __int_as_float((e + 127) << 23) : scalbnf(t, e);
}

// Scale-factor byte of a block scale relative to its row reference, and
// whether the block is kept (see the header).
__device__ __forceinline__ uint32_t mx_sf(int d, int bias, bool& keep) {
  const int b = d + MX_SF0 + bias;
  keep = b >= 0;
  return keep ? (uint32_t)b : 0u;
}

// Instruction descriptor of tcgen05.mma .kind::mxf8f6f4 .block_scale: D F32,
// A and B E5M2, K-major, UE8M0 factors, M = 128, factor ids 0, 2:4-sparse A
// when `sparse`.
__host__ __device__ constexpr uint32_t idesc_mx_e5m2(int N, bool sparse) {
  return (sparse ? (1u << 2) : 0u)  // sparse A
         | (1u << 7)                // A: E5M2
         | (1u << 10)               // B: E5M2
         | ((uint32_t)(N >> 3) << 17)
         | (1u << 23)               // scale factors UE8M0
         | (1u << 27);              // M >> 7 = 1
}

// 2:4-sparse block-scaled MMA, A, metadata and factors in TMEM, B in shared
// memory; issued by `leader`.
__device__ __forceinline__ void mma_sp_mx_if(uint32_t leader, uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                             uint32_t meta_tmem, uint32_t idesc, uint32_t sfa_tmem,
                                             uint32_t sfb_tmem, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.b32 p, %7, 0;\n setp.ne.b32 q, %8, 0;\n"
      "@q tcgen05.mma.sp.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], [%1], %2, [%3], %4, [%5], [%6], "
      "p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(meta_tmem), "r"(idesc), "r"(sfa_tmem), "r"(sfb_tmem), "r"(accumulate),
      "r"(leader)
      : "memory");
}

// Dense block-scaled MMA, A and factors in TMEM, B in shared memory.
__device__ __forceinline__ void mma_mx_if(uint32_t leader, uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                          uint32_t idesc, uint32_t sfa_tmem, uint32_t sfb_tmem, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.b32 p, %6, 0;\n setp.ne.b32 q, %7, 0;\n"
      "@q tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], [%1], %2, %3, [%4], [%5], p;\n}\n" ::"r"(
          d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(sfa_tmem), "r"(sfb_tmem), "r"(accumulate), "r"(leader)
      : "memory");
}

// Shared memory -> TMEM copy of 32 rows of 16 bytes (512 contiguous bytes)
// into four columns of every lane quadrant, issued by `leader`; ordered
// before the MMAs the same thread issues after it.
__device__ __forceinline__ void tmem_cp_sf_if(uint32_t leader, uint32_t tmem_col, const void* src) {
  const uint64_t d = tc::smem_desc(tc::smem_u32(src), 128, 128);
  asm volatile(
      "{\n .reg .pred q;\n setp.ne.b32 q, %2, 0;\n"
      "@q tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;\n}\n" ::"r"(tmem_col),
      "l"(d), "r"(leader)
      : "memory");
}

// Byte offset of B column n's factor word in the copy sources of one stage
// (512 bytes per four TMEM columns).
__device__ __forceinline__ uint32_t sfb_off(int n) {
  return (uint32_t)((n >> 7) * 512 + (n & 31) * 16 + ((n >> 5) & 3) * 4);
}

}  // namespace cfp
