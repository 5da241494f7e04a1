// CurveFP block-scaled quantization and dequantization (Sec. 3.1, Eq. 1).
//
// Quantizer: one HBM streaming pass.  Each block of G values is reduced to
// max|x| (16-bit SIMD max for BF16, warp shuffles across the lanes that share
// the block), the ceil-absmax scale a_b comes from the max's exponent and one
// mantissa compare (App. A.2), and every element is encoded without a search:
// its scaled magnitude |x| 2^{-a_b} is a binade offset from the zero boundary
// F_z plus a mantissa, and an exact rank table indexed by (binade offset, top
// 7 mantissa bits) gives the nearest level's rank (BF16: the whole decision,
// its mantissa has 7 bits; FP32: plus one compare against the bucket's
// threshold).  m = 0 below L_nmin/2; code = sign << 7 | m, zero always 0x00.
// All thresholds are irrational, so no input ties; the tables are generated
// in exact integer arithmetic.  Blocks containing NaN, Inf or values that
// need subnormal care take an exact slow path.
//
// Dense rows with G = 32 (the common case) are fed by bulk (TMA) copies into a
// shared-memory ring; other shapes use a register-fed kernel of the same
// arithmetic.
#pragma once
#include "cfp_common.cuh"
#include "kernels.cuh"
#include "radix.cuh"
#include "tc_ptx.cuh"

namespace cfp {

// Unsigned exponent/mantissa split of a positive finite FP32 bit pattern,
// normalizing subnormals.
__device__ __forceinline__ void split_f32(uint32_t absb, int& F, uint32_t& mant) {
  if (absb >= 0x00800000u) {
    F = (int)(absb >> 23) - 127;
    mant = absb & 0x7FFFFFu;
  } else {
    int p = 31 - __clz(absb);
    F = p - 149;
    mant = (absb << (23 - p)) & 0x7FFFFFu;
  }
}

// Number of midpoint thresholds at or below a 23-bit mantissa.
__device__ __forceinline__ int mid_count(const uint32_t* lut, uint32_t mant) {
  uint32_t e = lut[mant >> 15];
  return (int)(e >> 24) + (mant >= (e & 0xFFFFFFu) ? 1 : 0);
}

// Ceil-absmax block scale from the bit pattern of max|x| (NaN excluded).
// (Rational radix: the floor F and mantissa threshold of lambda(63) from the
// generated tables in place of E_max and 2^{(K-1)/K}.)
template <int FMT>
__device__ __forceinline__ int block_scale(uint32_t amaxb) {
  using F = Fmt<FMT>;
  if (amaxb == 0u) return 0;
  if (amaxb >= 0x7F800000u) return 127;
  int Fx;
  uint32_t mant;
  split_f32(amaxb, Fx, mant);
  int a;
  if constexpr (IsRadix<FMT>::value)
    a = Fx - Radix<FMT>::F + (mant >= Radix<FMT>::MU_SAT ? 1 : 0);
  else
    a = Fx - F::EMAX + (mant >= RadixConst<F::K>::MU_SAT ? 1 : 0);
  return a < -128 ? -128 : (a > 127 ? 127 : a);
}

// Lowest binade of the fast path's rank table (keys of smaller values clamp
// into it and read rank 0).
template <int FMT>
__host__ __device__ constexpr int rank_fz() {
  if constexpr (IsRadix<FMT>::value)
    return Radix<FMT>::ZB - 1;
  else
    return ZeroBoundary<FMT>::FZ;
}

// Fast-path encode: finite input, block scale a in [-100, 127].
template <int FMT>
__device__ __forceinline__ uint32_t encode_fast(const uint32_t* lut, uint32_t bits, int32_t ashift) {
  using F = Fmt<FMT>;
  if constexpr (IsRadix<FMT>::value) {
    bool nan = false;  // finite blocks only
    return radix_encode<FMT>(bits, ashift >> 23, nan);
  }
  constexpr int32_t T0 = ((ZeroBoundary<FMT>::FZ + 127) << 23) | (int32_t)RadixConst<F::K>::MU_Z;
  int32_t t = (int32_t)(bits & 0x7FFFFFFFu) - ashift;
  uint32_t e = lut[(t >> 15) & 0xFF];
  int j = (int)(e >> 24) + (((uint32_t)t & 0x7FFFFFu) >= (e & 0xFFFFFFu) ? 1 : 0);
  int m = ((t >> 23) << F::C) + j + (F::B - 127 * F::K);
  m = m < 1 ? 1 : m;
  const uint32_t code = (uint32_t)m | ((bits >> 24) & 0x80u);
  return t < T0 ? 0u : code;  // zero is always 0x00, whatever the sign
}

// Exact encode for any input and scale.  Sets *nan if the input is NaN.
template <int FMT>
__device__ __forceinline__ uint32_t encode_slow(const uint32_t* lut, uint32_t bits, int a, bool& nan) {
  using F = Fmt<FMT>;
  if constexpr (IsRadix<FMT>::value) return radix_encode<FMT>(bits, a, nan);
  uint32_t absb = bits & 0x7FFFFFFFu;
  int m;
  if (absb > 0x7F800000u) {
    nan = true;
    return 0u;
  } else if (absb == 0x7F800000u) {
    m = 2 * F::B - 1;
  } else if (absb == 0u) {
    return 0u;
  } else {
    int Fx;
    uint32_t mant;
    split_f32(absb, Fx, mant);
    int Fv = Fx - a;
    int j = mid_count(lut, mant);
    if (Fv > F::EMAX || (Fv == F::EMAX && j == F::K)) {
      m = 2 * F::B - 1;
    } else if (Fv < ZeroBoundary<FMT>::FZ || (Fv == ZeroBoundary<FMT>::FZ && mant < RadixConst<F::K>::MU_Z)) {
      return 0u;
    } else {
      m = F::K * Fv + j + F::B;
      m = m < 1 ? 1 : m;
    }
  }
  return (uint32_t)m | ((bits >> 24) & 0x80u);
}

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  static constexpr int VEC = 4;
  __device__ static __forceinline__ uint32_t bits(const uint4& v, int i) {
    return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
  }
};
template <>
struct Elem<uint16_t> {  // BF16 storage
  static constexpr int VEC = 8;
  __device__ static __forceinline__ uint32_t bits(const uint4& v, int i) {
    uint32_t w = (i >> 1) == 0 ? v.x : (i >> 1) == 1 ? v.y : (i >> 1) == 2 ? v.z : v.w;
    return (i & 1) ? (w & 0xFFFF0000u) : (w << 16);
  }
};

template <int K>
__device__ __forceinline__ const uint32_t* lut_src();

// Rank tables of the fast path, indexed by (binade offset, top 7 mantissa bits)
// of the scaled value; entry = rank below | rank above << 8 | the in-bucket
// threshold's low 16 mantissa bits << 16 (generated exactly on the host).
// (global memory, not __constant__: every thread copies a different entry)
static __device__ const uint32_t CFP_RANK_E3C3_DEV[CFP_RANK_E3C3_NBIN * 128] = CFP_RANK_E3C3_INIT;
static __device__ const uint32_t CFP_RANK_E4C3_DEV[CFP_RANK_E4C3_NBIN * 128] = CFP_RANK_E4C3_INIT;
static __device__ const uint32_t CFP_RANK_E5C2_DEV[CFP_RANK_E5C2_NBIN * 128] = CFP_RANK_E5C2_INIT;
static __device__ const uint32_t CFP_RANK_E4C3_R8_9_DEV[CFP_RANK_E4C3_R8_9_NBIN * 128] = CFP_RANK_E4C3_R8_9_INIT;
static __device__ const uint32_t CFP_RANK_E4C3_R3_4_DEV[CFP_RANK_E4C3_R3_4_NBIN * 128] = CFP_RANK_E4C3_R3_4_INIT;
static __device__ const uint32_t CFP_LUT_K4_G[256] = CFP_LUT_K4_INIT;
static __device__ const uint32_t CFP_LUT_K8_G[256] = CFP_LUT_K8_INIT;

template <>
__device__ __forceinline__ const uint32_t* lut_src<4>() {
  return CFP_LUT_K4_G;
}
template <>
__device__ __forceinline__ const uint32_t* lut_src<8>() {
  return CFP_LUT_K8_G;
}

template <int FMT>
struct RankTab;
template <>
struct RankTab<CURVEFP_E3C3> {
  static constexpr int NBIN = CFP_RANK_E3C3_NBIN;
  __device__ static const uint32_t* src() { return CFP_RANK_E3C3_DEV; }
};
template <>
struct RankTab<CURVEFP_E4C3> {
  static constexpr int NBIN = CFP_RANK_E4C3_NBIN;
  __device__ static const uint32_t* src() { return CFP_RANK_E4C3_DEV; }
};
template <>
struct RankTab<CURVEFP_E5C2> {
  static constexpr int NBIN = CFP_RANK_E5C2_NBIN;
  __device__ static const uint32_t* src() { return CFP_RANK_E5C2_DEV; }
};
template <>
struct RankTab<CURVEFP_E4C3_R8_9> {
  static constexpr int NBIN = CFP_RANK_E4C3_R8_9_NBIN;
  __device__ static const uint32_t* src() { return CFP_RANK_E4C3_R8_9_DEV; }
};
template <>
struct RankTab<CURVEFP_E4C3_R3_4> {
  static constexpr int NBIN = CFP_RANK_E4C3_R3_4_NBIN;
  __device__ static const uint32_t* src() { return CFP_RANK_E4C3_R3_4_DEV; }
};

// FP32 compare form of a rank-table entry r_lo | r_hi << 8 | t16 << 16 (a
// bucket with a decision threshold has r_hi = r_lo + 1 and t16 >= 1, checked
// by the table's generator): (t16 - 1) << 16 | r_lo with a threshold,
// 0xFFFF0000 | r_lo without.  For a value with FP32 bits w, (w << 16) > entry
// holds iff its low 16 mantissa bits are >= t16 (never without a threshold),
// so its rank is r_lo + that comparison.
__device__ __forceinline__ uint32_t rank_cmp_entry(uint32_t e) {
  const uint32_t lo = e & 0xFFu;
  return ((e >> 8) & 0xFFu) != lo ? (((e >> 16) - 1u) << 16) | lo : 0xFFFF0000u | lo;
}

// Table key of a magnitude bit pattern (FP32 bits >> 16, or BF16 bits) for
// block scale a: (binade - F_z) * 128 + top 7 mantissa bits, clamped at 0
// (everything below binade F_z encodes as zero).  kb = (127 + a + F_z) << 7.
__device__ __forceinline__ int rank_key(uint32_t hi16, int kb) {
  const int k = (int)hi16 - kb;
  return k < 0 ? 0 : k;
}

// Merge signs into four packed ranks: a sign bit is kept only on nonzero codes
// (zero is always 0x00).  s4 holds each element's sign in bit 7 of its byte.
__device__ __forceinline__ uint32_t merge_signs(uint32_t r4, uint32_t s4) {
  const uint32_t nz = (r4 + 0x7F7F7F7Fu) & 0x80808080u;  // rank >= 1
  return r4 | (s4 & nz);
}

__device__ __forceinline__ uint32_t max_u16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.u16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// Ranks of four FP32 values (bits w[0..3]) from the compare-form table: the
// table keys of two values at a time in 16-bit lanes (kb2 = the block's key
// base in both lanes), then r = r_lo + [(w << 16) > entry].
__device__ __forceinline__ uint32_t ranks4_f32(const uint32_t* tab, const uint32_t (&w)[4], uint32_t kb2) {
  uint32_t r[4];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const uint32_t k2 = max_u16x2(__byte_perm(w[2 * h], w[2 * h + 1], 0x7632) & 0x7FFF7FFFu, kb2) - kb2;
    const uint32_t e0 = tab[k2 & 0xFFFFu], e1 = tab[k2 >> 16];
    r[2 * h] = (e0 & 0xFFu) + ((w[2 * h] << 16) > e0 ? 1u : 0u);
    r[2 * h + 1] = (e1 & 0xFFu) + ((w[2 * h + 1] << 16) > e1 ? 1u : 0u);
  }
  return __byte_perm(__byte_perm(r[0], r[1], 0x0040), __byte_perm(r[2], r[3], 0x0040), 0x5410);
}

// ---------------------------------------------------------------------------
// block_axis 0: blocks of G consecutive elements along a row.
// TPB lanes cooperate on one block; each lane holds VPT 16-byte vectors.
// Fast path (finite block, scale >= -100): one shared-memory rank lookup per
// element (BF16: the byte itself; FP32: plus one 16-bit compare), signs merged
// four at a time.  Other blocks take the exact per-element slow path.
// With gscale (static operands with row or tensor scale groups) the scale of
// block b is gscale[b / bpg] instead of the block's own ceil-absmax scale.
template <int FMT, typename T, int G>
__global__ void __launch_bounds__(256) quantize_rows_kernel(const T* __restrict__ x, int64_t rows, int64_t cols,
                                                            int64_t ld, uint8_t* __restrict__ codes,
                                                            int8_t* __restrict__ scales, uint32_t* status,
                                                            const int8_t* __restrict__ gscale, int64_t bpg) {
  using F = Fmt<FMT>;
  constexpr int VEC = Elem<T>::VEC;
  constexpr bool BF16 = sizeof(T) == 2;
  constexpr int VPB = G / VEC;              // vectors per block
  // BF16 blocks of 32: two lanes share a block (two 16-byte vectors each), which
  // keeps every load instruction on whole 32-byte sectors while halving the
  // per-block work (one shuffle, the scale computed by two lanes); otherwise up
  // to 8 lanes share a block
  constexpr int TPB = (BF16 && G == 32) ? 2 : (VPB < 8 ? VPB : 8);  // lanes per block
  constexpr int VPT = VPB / TPB;            // vectors per lane
  constexpr int BPW = 32 / TPB;             // blocks per warp step
  constexpr int UNROLL = VPT >= 4 ? 1 : 4 / VPT;
  constexpr int NTAB = RankTab<FMT>::NBIN * 128;

  __shared__ uint32_t lut[256];
  // FP32: full entries; BF16: the low byte of each entry only (its low 16
  // mantissa bits are zero, so the in-bucket compare never fires)
  __shared__ __align__(16) uint32_t tab[BF16 ? 1 : NTAB];
  __shared__ __align__(16) uint8_t tab8[BF16 ? NTAB : 1];
  for (int i = threadIdx.x; i < 256; i += blockDim.x) lut[i] = __ldg(lut_src<F::K>() + i);
  for (int i = threadIdx.x; i < NTAB; i += blockDim.x) {
    const uint32_t e = __ldg(RankTab<FMT>::src() + i);
    if (BF16)
      tab8[i] = (uint8_t)(e & 0xFFu);
    else
      tab[i] = rank_cmp_entry(e);
  }
  __syncthreads();

  const int lane = threadIdx.x & 31;
  const int sub = lane % TPB;
  const int64_t nbc = cols / G;
  const int64_t nblk = rows * nbc;
  const int64_t warp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const bool dense = (ld == cols);
  bool saw_nan = false;

  for (int64_t base = warp * BPW * UNROLL; base < nblk; base += nwarps * BPW * UNROLL) {
    uint4 v[UNROLL][VPT];
    int64_t blk[UNROLL];
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      blk[u] = base + (int64_t)u * BPW + lane / TPB;
      const bool ok = blk[u] < nblk;
      int64_t off = 0;
      if (ok) off = dense ? blk[u] * G : (blk[u] / nbc) * ld + (blk[u] % nbc) * G;
      const uint4* src = reinterpret_cast<const uint4*>(x + off);
#pragma unroll
      for (int q = 0; q < VPT; ++q) v[u][q] = ok ? __ldcs(src + q * TPB + sub) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      // max |x| over the block as an unsigned bit pattern (NaN sorts above Inf)
      uint32_t mx = 0u;
#pragma unroll
      for (int q = 0; q < VPT; ++q) {
        const uint32_t w[4] = {v[u][q].x, v[u][q].y, v[u][q].z, v[u][q].w};
        if (BF16) {
          uint32_t m2 = 0u;
#pragma unroll
          for (int i = 0; i < 4; ++i) m2 = max_u16x2(m2, w[i] & 0x7FFF7FFFu);
          mx = max(mx, max(m2 & 0xFFFFu, m2 >> 16) << 16);
        } else {
#pragma unroll
          for (int i = 0; i < 4; ++i) mx = max(mx, w[i] & 0x7FFFFFFFu);
        }
      }
#pragma unroll
      for (int o = TPB / 2; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      const bool ok = blk[u] < nblk;
      const bool grouped = gscale != nullptr;
      int a = grouped ? (ok ? (int)gscale[blk[u] / bpg] : 0) : block_scale<FMT>(mx);
      const bool fast = mx < 0x7F800000u && a >= -100;
      if (!grouped && __any_sync(0xffffffffu, !fast)) {  // rare: NaN / Inf / subnormal-scale blocks
        uint32_t mx2 = 0u;
#pragma unroll
        for (int q = 0; q < VPT; ++q)
#pragma unroll
          for (int i = 0; i < VEC; ++i) {
            uint32_t b = Elem<T>::bits(v[u][q], i) & 0x7FFFFFFFu;
            mx2 = max(mx2, b > 0x7F800000u ? 0u : b);
          }
#pragma unroll
        for (int o = TPB / 2; o > 0; o >>= 1) mx2 = max(mx2, __shfl_xor_sync(0xffffffffu, mx2, o));
        if (!fast) a = block_scale<FMT>(mx2);
      }
      if (!ok) continue;
      uint8_t* dst = codes + blk[u] * G;
      if (sub == 0) scales[blk[u]] = (int8_t)a;
      const int kb = (127 + a + rank_fz<FMT>()) << 7;
#pragma unroll
      for (int q = 0; q < VPT; ++q) {
        const uint32_t w[4] = {v[u][q].x, v[u][q].y, v[u][q].z, v[u][q].w};
        uint8_t* d = dst + (q * TPB + sub) * VEC;
        if (fast) {
          if (BF16) {
            // two keys per word: clamp each 16-bit magnitude at kb with a
            // SIMD max, then one 32-bit subtract (no lane can borrow)
            const uint32_t kb2 = (uint32_t)kb * 0x00010001u;
            uint32_t out[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const uint32_t w0 = w[2 * h], w1 = w[2 * h + 1];
              const uint32_t k0 = max_u16x2(w0 & 0x7FFF7FFFu, kb2) - kb2;
              const uint32_t k1 = max_u16x2(w1 & 0x7FFF7FFFu, kb2) - kb2;
              const uint32_t r0 = tab8[k0 & 0xFFFFu], r1 = tab8[k0 >> 16];
              const uint32_t r2 = tab8[k1 & 0xFFFFu], r3 = tab8[k1 >> 16];
              const uint32_t r4 = __byte_perm(__byte_perm(r0, r1, 0x0040), __byte_perm(r2, r3, 0x0040), 0x5410);
              out[h] = merge_signs(r4, __byte_perm(w0, w1, 0x7531));
            }
            *reinterpret_cast<uint2*>(d) = make_uint2(out[0], out[1]);
          } else {
            const uint32_t r4 = ranks4_f32(tab, w, (uint32_t)kb * 0x00010001u);
            const uint32_t s4 = __byte_perm(__byte_perm(w[0], w[1], 0x0073), __byte_perm(w[2], w[3], 0x7300), 0x7610);
            *reinterpret_cast<uint32_t*>(d) = merge_signs(r4, s4);
          }
        } else {
          uint32_t c[VEC];
#pragma unroll
          for (int i = 0; i < VEC; ++i) c[i] = encode_slow<FMT>(lut, Elem<T>::bits(v[u][q], i), a, saw_nan);
          if (VEC == 4) {
            *reinterpret_cast<uint32_t*>(d) = c[0] | (c[1] << 8) | (c[2] << 16) | (c[3] << 24);
          } else {
            uint2 wv;
            wv.x = c[0] | (c[1] << 8) | (c[2] << 16) | (c[3] << 24);
            wv.y = c[4] | (c[5] << 8) | (c[6] << 16) | (c[7] << 24);
            *reinterpret_cast<uint2*>(d) = wv;
          }
        }
      }
    }
  }
  if (saw_nan && status) atomicOr(status, CURVEFP_DEV_NAN);
}

// ---------------------------------------------------------------------------
// block_axis 0, dense rows, G = 32: the same encoder fed by bulk (TMA) copies.
// One producer lane streams 16 KB chunks of the input into a ring of NST
// shared-memory stages (completion counted in mbarrier transaction bytes);
// 16 consumer warps each take 1 KB of every chunk with conflict-free 16-byte
// shared loads, release the stage at once, encode, and write codes and scales
// straight to global memory.  The input stream never waits on the encoder's
// arithmetic, which the register-fed kernel above cannot avoid.
constexpr int QB_CHUNK = 16384;  // bytes per stage
constexpr int QB_NCW = 16;       // consumer warps, 1 KB of each chunk each

template <int FMT, typename T>
struct BulkQ {
  static constexpr int NTAB = RankTab<FMT>::NBIN * 128;
  static constexpr bool BF16 = sizeof(T) == 2;
  static constexpr size_t smem(int nst) {
    return (size_t)nst * QB_CHUNK + 256 * 4 + (size_t)NTAB * (BF16 ? 1 : 4) + (size_t)2 * nst * 8;
  }
};

#ifndef CFP_QB_NST
#define CFP_QB_NST 3  // stages of the bulk-fed quantizer
#endif
#ifndef CFP_QB_CTAS
#define CFP_QB_CTAS 2  // its resident CTAs per SM (at most)
#endif

template <int FMT, typename T, int NST>
__global__ void __launch_bounds__((QB_NCW + 1) * 32, CFP_QB_CTAS) quantize_rows_bulk_kernel(const T* __restrict__ x, int64_t nblk,
                                                                              uint8_t* __restrict__ codes,
                                                                              int8_t* __restrict__ scales,
                                                                              uint32_t* status) {
  using F = Fmt<FMT>;
  constexpr int G = 32;
  constexpr bool BF16 = sizeof(T) == 2;
  constexpr int VEC = 16 / (int)sizeof(T);  // elements per 16-byte vector
  constexpr int TPB = G / VEC;              // lanes per block: 4 (BF16) or 8 (FP32)
  constexpr int BLK_BYTES = G * (int)sizeof(T);
  constexpr int CH_BLK = QB_CHUNK / BLK_BYTES;  // blocks per chunk
  constexpr int NTAB = BulkQ<FMT, T>::NTAB;
  extern __shared__ __align__(128) uint8_t qsm[];
  uint8_t* ring = qsm;
  uint32_t* lut = reinterpret_cast<uint32_t*>(qsm + (size_t)NST * QB_CHUNK);
  uint32_t* tab = lut + 256;  // FP32: full entries; BF16: rank bytes (tab8)
  uint8_t* tab8 = reinterpret_cast<uint8_t*>(tab);
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(tab) + (size_t)NTAB * (BF16 ? 1 : 4));
  uint64_t* empty = full + NST;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < NST; ++i) {
      tc::mbar_init(&full[i], 1);
      tc::mbar_init(&empty[i], QB_NCW);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  // the first copies are issued while the consumers load the tables; the
  // consumers then meet on named barrier 1 (the producer warp does not take
  // part), so the table loads' latency hides behind the first chunks'
  if (warp < QB_NCW) {
    for (int i = threadIdx.x; i < 256; i += QB_NCW * 32) lut[i] = __ldg(lut_src<F::K>() + i);
    for (int i = threadIdx.x; i < NTAB; i += QB_NCW * 32) {
      const uint32_t e = __ldg(RankTab<FMT>::src() + i);
      if (BF16)
        tab8[i] = (uint8_t)(e & 0xFFu);
      else
        tab[i] = rank_cmp_entry(e);
    }
    asm volatile("bar.sync 1, %0;" ::"n"(QB_NCW * 32) : "memory");
  }

  const int64_t nchunks = (nblk + CH_BLK - 1) / CH_BLK;
  if (warp == QB_NCW) {
    // ------------------------------ producer ---------------------------------
    if (lane == 0) {
      int issued = 0;
      bool ok = true;
      for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x, ++issued) {
        const int st = issued % NST;
        if (issued >= NST && !tc::mbar_wait(&empty[st], ((issued / NST) - 1) & 1)) {
          ok = false;
          break;
        }
        const int64_t b0 = c * CH_BLK;
        const int64_t left = nblk - b0;
        const uint32_t bytes = (uint32_t)(left < CH_BLK ? left : CH_BLK) * BLK_BYTES;
        tc::mbar_arrive_expect_tx(&full[st], bytes);
        tc::bulk_g2s(ring + (size_t)st * QB_CHUNK, reinterpret_cast<const uint8_t*>(x) + b0 * BLK_BYTES, bytes,
                     &full[st]);
      }
      if (!ok) {
        if (status) atomicOr(status, CURVEFP_DEV_TIMEOUT);
        // the copies already issued land before the CTA may exit
        for (int j = issued - NST < 0 ? 0 : issued - NST; j < issued; ++j) tc::mbar_wait(&full[j % NST], (j / NST) & 1);
      }
    }
    return;
  }

  // ------------------------------ consumers ----------------------------------
  bool saw_nan = false;
  const int sub = lane % TPB;
  int it = 0;
  for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x, ++it) {
    const int st = it % NST;
    if (!__all_sync(0xffffffffu, tc::mbar_wait(&full[st], (it / NST) & 1))) {
      if (lane == 0 && status) atomicOr(status, CURVEFP_DEV_TIMEOUT);
      break;
    }
    const uint4* src = reinterpret_cast<const uint4*>(ring + (size_t)st * QB_CHUNK + warp * 1024);
    uint4 v[2];
    v[0] = src[lane];
    v[1] = src[32 + lane];
    // refill the stage as soon as every lane's loads have returned: a shuffle
    // consumes a word of each load and the arrival depends on its result (an
    // arrival right after the loads could let the next bulk copy overwrite
    // the stage while a load is still in flight)
    const uint32_t dep = __shfl_xor_sync(0xffffffffu, v[0].x ^ v[1].x, 1);
    if (lane == 0) tc::mbar_arrive_after(&empty[st], dep);
    const int64_t b0 = c * CH_BLK;
    const int64_t left = nblk - b0;
    const int nb = (int)(left < CH_BLK ? left : CH_BLK);
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int lb = (warp * 64 + q * 32 + lane) / TPB;  // block within the chunk
      const uint32_t w[4] = {v[q].x, v[q].y, v[q].z, v[q].w};
      uint32_t mx = 0u;
      if (BF16) {
        uint32_t m2 = 0u;
#pragma unroll
        for (int i = 0; i < 4; ++i) m2 = max_u16x2(m2, w[i] & 0x7FFF7FFFu);
        mx = max(m2 & 0xFFFFu, m2 >> 16) << 16;
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) mx = max(mx, w[i] & 0x7FFFFFFFu);
      }
#pragma unroll
      for (int o = TPB / 2; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      int a = block_scale<FMT>(mx);
      const bool fast = mx < 0x7F800000u && a >= -100;
      if (__any_sync(0xffffffffu, !fast)) {  // rare: NaN / Inf / subnormal-scale blocks
        uint32_t mx2 = 0u;
#pragma unroll
        for (int i = 0; i < VEC; ++i) {
          const uint32_t b = Elem<T>::bits(v[q], i) & 0x7FFFFFFFu;
          mx2 = max(mx2, b > 0x7F800000u ? 0u : b);
        }
#pragma unroll
        for (int o = TPB / 2; o > 0; o >>= 1) mx2 = max(mx2, __shfl_xor_sync(0xffffffffu, mx2, o));
        if (!fast) a = block_scale<FMT>(mx2);
      }
      if (lb >= nb) continue;
      const int64_t blk = b0 + lb;
      if (sub == 0) scales[blk] = (int8_t)a;
      uint8_t* d = codes + blk * G + sub * VEC;
      const int kb = (127 + a + rank_fz<FMT>()) << 7;
      if (fast) {
        if (BF16) {
          const uint32_t kb2 = (uint32_t)kb * 0x00010001u;
          uint32_t out[2];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const uint32_t w0 = w[2 * h], w1 = w[2 * h + 1];
            const uint32_t k0 = max_u16x2(w0 & 0x7FFF7FFFu, kb2) - kb2;
            const uint32_t k1 = max_u16x2(w1 & 0x7FFF7FFFu, kb2) - kb2;
            const uint32_t r0 = tab8[k0 & 0xFFFFu], r1 = tab8[k0 >> 16];
            const uint32_t r2 = tab8[k1 & 0xFFFFu], r3 = tab8[k1 >> 16];
            const uint32_t r4 = __byte_perm(__byte_perm(r0, r1, 0x0040), __byte_perm(r2, r3, 0x0040), 0x5410);
            out[h] = merge_signs(r4, __byte_perm(w0, w1, 0x7531));
          }
          *reinterpret_cast<uint2*>(d) = make_uint2(out[0], out[1]);
        } else {
          const uint32_t r4 = ranks4_f32(tab, w, (uint32_t)kb * 0x00010001u);
          const uint32_t s4 = __byte_perm(__byte_perm(w[0], w[1], 0x0073), __byte_perm(w[2], w[3], 0x7300), 0x7610);
          *reinterpret_cast<uint32_t*>(d) = merge_signs(r4, s4);
        }
      } else {
        uint32_t cc[VEC];
#pragma unroll
        for (int i = 0; i < VEC; ++i) cc[i] = encode_slow<FMT>(lut, Elem<T>::bits(v[q], i), a, saw_nan);
        if constexpr (VEC == 4) {
          *reinterpret_cast<uint32_t*>(d) = cc[0] | (cc[1] << 8) | (cc[2] << 16) | (cc[3] << 24);
        } else {
          *reinterpret_cast<uint2*>(d) = make_uint2(cc[0] | (cc[1] << 8) | (cc[2] << 16) | (cc[3] << 24),
                                                    cc[4] | (cc[5] << 8) | (cc[6] << 16) | (cc[7] << 24));
        }
      }
    }
  }
  if (saw_nan && status) atomicOr(status, CURVEFP_DEV_NAN);
}

// ---------------------------------------------------------------------------
// block_axis 1: blocks of G consecutive rows of one column; the output is the
// transposed operand (codes [cols x rows]).  One lane owns one column and one
// row-block: its loads are coalesced across the warp (consecutive columns),
// its G codes are one contiguous run of the output row.
template <int FMT, typename T, int G>
__global__ void __launch_bounds__(256) quantize_cols_kernel(const T* __restrict__ x, int64_t rows, int64_t cols,
                                                            int64_t ld, uint8_t* __restrict__ codes,
                                                            int8_t* __restrict__ scales, uint32_t* status) {
  using F = Fmt<FMT>;
  __shared__ uint32_t lut[256];
  for (int i = threadIdx.x; i < 256; i += blockDim.x) lut[i] = __ldg(lut_src<F::K>() + i);
  __syncthreads();
  const int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const int64_t rb = blockIdx.y;
  if (c >= cols) return;
  const int64_t nrb = rows / G;
  const T* src = x + rb * G * ld + c;
  auto load_bits = [&](int i) -> uint32_t {
    if (sizeof(T) == 4) return __float_as_uint(__ldcs(reinterpret_cast<const float*>(src) + i * ld));
    return (uint32_t)__ldcs(reinterpret_cast<const unsigned short*>(src) + i * ld) << 16;
  };
  uint32_t mx = 0u, mxn = 0u;
  constexpr int KEEP = G <= 32 ? G : 1;
  uint32_t keep[KEEP];
#pragma unroll 8
  for (int i = 0; i < G; ++i) {
    uint32_t b = load_bits(i);
    if (G <= 32) keep[i % KEEP] = b;
    uint32_t ab = b & 0x7FFFFFFFu;
    mx = max(mx, ab);
    mxn = max(mxn, ab > 0x7F800000u ? 0u : ab);
  }
  const int a = block_scale<FMT>(mxn);
  const bool fast = mx < 0x7F800000u && a >= -100;
  scales[c * nrb + rb] = (int8_t)a;
  const int32_t ashift = a * (1 << 23);
  bool saw_nan = false;
  uint8_t* dst = codes + c * rows + rb * G;
#pragma unroll 1
  for (int i0 = 0; i0 < G; i0 += 16) {
    uint32_t w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint32_t acc = 0;
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int i = i0 + 4 * q + r;
        uint32_t b = G <= 32 ? keep[i % KEEP] : load_bits(i);
        uint32_t code = fast ? encode_fast<FMT>(lut, b, ashift) : encode_slow<FMT>(lut, b, a, saw_nan);
        acc |= code << (8 * r);
      }
      w[q] = acc;
    }
    *reinterpret_cast<uint4*>(dst + i0) = make_uint4(w[0], w[1], w[2], w[3]);
  }
  if (saw_nan && status) atomicOr(status, CURVEFP_DEV_NAN);
}

// ---------------------------------------------------------------------------
// Dequantization: 16 codes per lane (one 16-byte load, four 16-byte stores).
// Fast path: RN32(2^{k/K}) 2^{e} comes from a 128-entry table indexed by the
// rank and the block scale is added to the exponent field; blocks whose
// results could leave the normal FP32 range multiply twice with one rounding.
template <int FMT>
__global__ void __launch_bounds__(256) dequantize_kernel(const uint8_t* __restrict__ codes,
                                                         const int8_t* __restrict__ scales, int64_t n, int G,
                                                         float* __restrict__ out) {
  using F = Fmt<FMT>;
  constexpr int EMIN = -(F::EMAX + 1);
  __shared__ uint32_t tab[128];
  for (int m = threadIdx.x; m < 128; m += blockDim.x) {
    uint32_t v = 0u;
    if (m >= 1 && m <= 2 * F::B - 1) {
      int nn = m - F::B;
      int e = nn >> F::C, k = nn & (F::K - 1);
      uint32_t ck = F::K == 8 ? CFP_CK_F32_K8_DEV[k] : CFP_CK_F32_K4_DEV[k];
      v = ck + (uint32_t)(e * (1 << 23));
    }
    tab[m] = v;
  }
  __syncthreads();
  // A thread takes words of 4 codes, U at a time (all loads issued first); the
  // warp's loads cover 128 contiguous bytes and its stores 512 contiguous
  // bytes per instruction.  n is a multiple of the block size (>= 32).
  constexpr int U = 4;
  const int64_t nw = n >> 2;
  const int64_t tile = (int64_t)blockDim.x * U;
  const int gs = __ffs(G) - 1;  // G is a power of two: block of code i = i >> gs
  const uint32_t* codes32 = reinterpret_cast<const uint32_t*>(codes);
  uint4* out4 = reinterpret_cast<uint4*>(out);
  for (int64_t t0 = (int64_t)blockIdx.x * tile; t0 < nw; t0 += (int64_t)gridDim.x * tile) {
    uint32_t cw[U];
    int sc[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t w = t0 + u * (int64_t)blockDim.x + threadIdx.x;
      cw[u] = w < nw ? __ldcs(codes32 + w) : 0u;
      sc[u] = w < nw ? (int)scales[(w << 2) >> gs] : 0;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t w = t0 + u * (int64_t)blockDim.x + threadIdx.x;
      if (w >= nw) continue;
      const int a = sc[u];
      const bool fast = (a + EMIN >= -126) && (a + F::EMAX <= 126);
      uint32_t o[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t code = (cw[u] >> (8 * i)) & 0xFFu;
        const uint32_t m = code & F::MMASK;
        uint32_t r;
        if (fast) {
          r = m ? tab[m] + (uint32_t)(a * (1 << 23)) : 0u;
        } else if (m == 0u) {
          r = 0u;
        } else {
          const int nn = (int)m - F::B;
          const int e = nn >> F::C, k = nn & (F::K - 1);
          const float ck = __uint_as_float(F::K == 8 ? CFP_CK_F32_K8_DEV[k] : CFP_CK_F32_K4_DEV[k]);
          const int E = a + e;
          const int E1 = E < -126 ? -126 : (E > 127 ? 127 : E);
          const int E2 = E - E1;  // in [-18, 15]
          float y = __fmul_rn(ck, __uint_as_float((uint32_t)(E1 + 127) << 23));
          y = __fmul_rn(y, __uint_as_float((uint32_t)(E2 + 127) << 23));
          r = __float_as_uint(y);
        }
        o[i] = m ? (r | ((code & 0x80u) << 24)) : 0u;
      }
      __stcs(out4 + w, make_uint4(o[0], o[1], o[2], o[3]));
    }
  }
}

// ---------------------------------------------------------------------------
// Static operands (Sec. 3.1: a fixed operand's power-of-two scale is picked
// by the reconstruction error it gives; Sec. 4.2 compares per-tensor,
// per-row and per-block scales).  A scale group is a block of G elements, a row
// or the whole tensor; its scale is the ceil-absmax scale a_c, or, for the MSE
// rule, the candidate a in [a_c - 3, a_c + 1] with the smallest
//   D(a) = sum_i floor((x_i - xhat_i)^2 2^{60 - 2 a_c}),
// xhat_i the FP32 reconstruction (Eq. 1, RN32(RN32(2^{k/K}) 2^{a+e})) of the
// element's nearest level at scale a; an exact integer, so the choice does
// not depend on the order of the sum; ties go to the larger a.  NaN elements
// are left out; groups with Inf or an all-zero max keep a_c.

template <typename T>
__device__ __forceinline__ uint32_t load_bits(const T* x, int64_t i) {
  if constexpr (sizeof(T) == 2)
    return (uint32_t)__ldg(reinterpret_cast<const uint16_t*>(x) + i) << 16;
  else
    return __float_as_uint(__ldg(reinterpret_cast<const float*>(x) + i));
}

// Eq. 1 reconstruction in FP32 of a code at scale a: one rounding of the
// exact product RN32(2^{k/K}) 2^{a+e}.  Where 2^{a+e} keeps the product in
// FP32's normal range the product is exact and is formed on the exponent
// field (integer arithmetic only: FP64 is a slow pipe on this GPU); the
// other cases round once through FP64.
template <int FMT>
__device__ __forceinline__ float recon_f32(uint32_t code, int a) {
  using F = Fmt<FMT>;
  if constexpr (IsRadix<FMT>::value) return radix_recon_f32<FMT>(code, a);
  const uint32_t m = code & 0x7Fu;
  if (m == 0u) return 0.0f;
  const int n = (int)m - F::B;
  const int e = n >= 0 ? n / F::K : -((-n + F::K - 1) / F::K);
  const int k = n - e * F::K;
  const uint32_t ckb = F::K == 8 ? CFP_CK_F32_K8_DEV[k] : CFP_CK_F32_K4_DEV[k];  // in [1, 2): exponent field 127
  const int E = a + e;
  uint32_t vb;
  if (E >= -126 && E <= 127) {
    vb = ckb + ((uint32_t)E << 23);
  } else {
    vb = __float_as_uint(__double2float_rn(ldexp((double)__uint_as_float(ckb), E)));
  }
  return __uint_as_float(vb | ((code & 0x80u) << 24));
}

// The same term through FP64 (x - xhat is exact in FP64 while the two
// exponents differ by less than 29).
__device__ __forceinline__ unsigned __int128 sq_term_f64(float x, float xhat, int ac) {
  const double e = fabs((double)x - (double)xhat);
  if (e == 0.0) return 0;
  int E;
  const double fr = frexp(e, &E);
  const unsigned long long M = (unsigned long long)ldexp(fr, 53);
  const unsigned __int128 sq = (unsigned __int128)M * M;
  const int sh = 2 * E - 106 + 60 - 2 * ac;
  if (sh >= 0) return sh >= 128 ? (unsigned __int128)0 : sq << sh;
  return sh <= -128 ? (unsigned __int128)0 : sq >> (-sh);
}

// A finite FP32 value as M 2^E with a signed integer M (|M| < 2^24).
__device__ __forceinline__ void f32_int(float v, int& M, int& E) {
  const uint32_t b = __float_as_uint(v);
  const int ef = (int)((b >> 23) & 0xFFu);
  const int mm = (int)(b & 0x7FFFFFu);
  M = ef ? (mm | 0x800000) : mm;
  E = ef ? ef - 150 : -149;
  if (b >> 31) M = -M;
}

// floor((x - xhat)^2 2^{60 - 2 ac}) exactly, in integer arithmetic: with
// x = Mx 2^Ex, xhat = Mh 2^Eh and Emin = min(Ex, Eh), x - xhat =
// (Mx 2^{Ex - Emin} - Mh 2^{Eh - Emin}) 2^Emin.  xhat is the nearest level to
// x or the saturation level of a scale at most 3 binades below the group's
// ceil-absmax scale, so the exponents differ by at most a few binades (more
// only when xhat = 0, where the difference is x itself); the integer
// difference then needs at most 32 bits and its square 64.
__device__ __forceinline__ unsigned __int128 sq_term(float x, float xhat, int ac) {
  int Mx, Ex, Mh, Eh;
  f32_int(x, Mx, Ex);
  f32_int(xhat, Mh, Eh);
  long long d;
  int E;
  if (Mh == 0) {
    d = Mx;
    E = Ex;
  } else if (Mx == 0) {
    d = Mh;
    E = Eh;
  } else {
    E = min(Ex, Eh);
    const int sx = Ex - E, sh2 = Eh - E;
    if (sx > 30 || sh2 > 30) return sq_term_f64(x, xhat, ac);  // not reached by the callers (see above)
    d = ((long long)Mx << sx) - ((long long)Mh << sh2);
  }
  if (d == 0) return 0;
  const unsigned long long ad = (unsigned long long)(d < 0 ? -d : d);
  const unsigned __int128 sq = (unsigned __int128)ad * ad;
  const int sh = 2 * E + 60 - 2 * ac;
  if (sh >= 0) return sh >= 128 ? (unsigned __int128)0 : sq << sh;
  return sh <= -128 ? (unsigned __int128)0 : sq >> (-sh);
}

// ---- the five MSE candidates of one element, sharing the scale-free work --
// The code of x at scale a (encode_slow) depends on a only through the binade
// test of Fv = Fx - a: the saturation code, zero, the smallest level (m
// clamped to 1) or the interior code K Fv + j + B, whose reconstruction
// (recon_f32) RN32(2^{k/K}) 2^{a + e} has a + e = Fx + [j = K] and
// k = j mod K whatever a is.  So an element needs one midpoint count and one
// interior value, and per candidate a class and one exact term.

// |v| of a finite FP32 bit pattern as M 2^E (M >= 0; f32_int's split).
__device__ __forceinline__ void f32_mag(uint32_t absb, int& M, int& E) {
  const int ef = (int)(absb >> 23);
  const int mm = (int)(absb & 0x7FFFFFu);
  M = ef ? (mm | 0x800000) : mm;
  E = ef ? ef - 150 : -149;
}

// The candidates of one group (scale ac): their scales and, as M 2^E, their
// saturation level (code 2B - 1) and smallest level (code 1).
struct MseCands {
  int ac, a[5], Ms[5], Es[5], Ml[5], El[5];
  bool valid[5];
};
template <int FMT>
__device__ __forceinline__ MseCands mse_cands(int ac) {
  MseCands c;
  c.ac = ac;
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    const int a = ac - 3 + k;
    c.a[k] = a;
    c.valid[k] = a >= -128 && a <= 127;
    f32_mag(__float_as_uint(recon_f32<FMT>((uint32_t)(2 * Fmt<FMT>::B - 1), a)) & 0x7FFFFFFFu, c.Ms[k], c.Es[k]);
    f32_mag(__float_as_uint(recon_f32<FMT>(1u, a)) & 0x7FFFFFFFu, c.Ml[k], c.El[k]);
  }
  return c;
}

// floor(q 2^sh) for q = ad^2 as a 128-bit integer (sq_term's shift; sh >= 128
// reads 0 as there).
__device__ __forceinline__ unsigned __int128 sq_shift(uint32_t ad, int sh) {
  const unsigned long long q = (unsigned long long)ad * ad;
  unsigned long long lo = 0ull, hi = 0ull;
  if (sh >= 0) {
    if (sh < 64) {
      lo = q << sh;
      hi = sh ? q >> (64 - sh) : 0ull;
    } else if (sh < 128) {
      hi = q << (sh - 64);
    }
  } else if (sh > -64) {
    lo = q >> -sh;
  }
  return ((unsigned __int128)hi << 64) | lo;
}

// Adds the five terms floor((x - xhat_a)^2 2^{60 - 2 ac}) of a finite, non-NaN
// element (bits b) to acc, exactly as sq_term(x, recon_f32(encode_slow(x, a),
// a), ac) per candidate.  Returns false, adding nothing, where the element
// takes the general path: an interior value outside FP32's normal range, or
// a reconstruction more than 8 binades from x (the integer difference then
// needs more than 32 bits).  ck: the K values RN32(2^{k/K}) as FP32 bits.
template <int FMT>
__device__ __forceinline__ bool mse_add5(const uint32_t* lut, const uint32_t* ck, uint32_t b, const MseCands& c,
                                         unsigned __int128 (&acc)[5]) {
  using F = Fmt<FMT>;
  const uint32_t absb = b & 0x7FFFFFFFu;
  if (absb == 0u) return true;  // x = 0 reconstructs as 0 at every scale
  int Fx;
  uint32_t mant;
  split_f32(absb, Fx, mant);
  const int j = mid_count(lut, mant);
  const int Ei = Fx + (j == F::K ? 1 : 0);
  if (Ei < -126 || Ei > 127) return false;
  // x = Mx 2^Ex; the interior value RN32(2^{k/K}) 2^Ei (normal) = Mi 2^{Ei - 23}
  int Mx, Ex;
  f32_mag(absb, Mx, Ex);
  const int Mi = (int)((ck[j & (F::K - 1)] & 0x7FFFFFu) | 0x800000u), Eiv = Ei - 23;
  // Classes by threshold on a (encode_slow's tests with Fv = Fx - a):
  // saturated for a < as, zero for a > az, clamped to the smallest level for
  // a > acl (and not zero), interior otherwise.
  const int as = Fx - F::EMAX + (j == F::K ? 1 : 0);
  const int az = Fx - ZeroBoundary<FMT>::FZ - (mant < RadixConst<F::K>::MU_Z ? 1 : 0);
  const int acl = Fx + (j + F::B - 1) / F::K;  // K (Fx - a) + j + B < 1; j + B - 1 >= 0
  // the interior term (x and its interior value are within one binade)
  unsigned __int128 tint;
  {
    const int E = min(Ex, Eiv), sx = Ex - E, s2 = Eiv - E;
    const long long d = (long long)((uint32_t)Mx << sx) - (long long)((uint32_t)Mi << s2);
    tint = sq_shift((uint32_t)(d < 0 ? -d : d), 2 * E + 60 - 2 * c.ac);
  }
  unsigned __int128 t[5];
  bool ok = true;
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    const int a = c.a[k];
    const bool sat = a < as, zero = !sat && a > az, clamp = !sat && !zero && a > acl;
    const bool own = sat || zero || clamp;
    t[k] = tint;
    // a candidate's own term only where the element is not interior there
    // (mostly the saturating scales below a_c); a warp skips the branch when
    // none of its lanes takes it
    if (own) {
      int Mh = sat ? c.Ms[k] : (clamp ? c.Ml[k] : 0);
      int Eh = sat ? c.Es[k] : (clamp ? c.El[k] : Ex);
      const int E = min(Ex, Eh), sx = Ex - E, s2 = Eh - E;
      ok = ok && sx <= 8 && s2 <= 8;
      const long long d = (long long)((uint32_t)Mx << (sx & 15)) - (long long)((uint32_t)Mh << (s2 & 15));
      t[k] = sq_shift((uint32_t)(d < 0 ? -d : d), 2 * E + 60 - 2 * c.ac);
    }
  }
  if (!ok) return false;
#pragma unroll
  for (int k = 0; k < 5; ++k)
    if (c.valid[k]) acc[k] += t[k];
  return true;
}

// Exact 128-bit accumulation into global memory ([lo, hi] words).
__device__ __forceinline__ void atomic_add_u128(unsigned long long* p, unsigned __int128 v) {
  const unsigned long long lo = (unsigned long long)v, hi = (unsigned long long)(v >> 64);
  const unsigned long long old = atomicAdd(p, lo);
  const unsigned long long carry = (old + lo < old) ? 1ull : 0ull;
  if (hi + carry) atomicAdd(p + 1, hi + carry);
}

// Row and tensor groups are cut into spans of at most QS_SPAN elements; one
// CTA per span (span c of group g = blockIdx.x: g = bid / cpg, c = bid % cpg)
// reads it with coalesced loads and raises its group's result once.
constexpr int64_t QS_SPAN = 16384;

// Group maxima: max |x| as an FP32 bit pattern (NaN left out; Inf =
// 0x7F800000), one atomic max per CTA.
template <typename T>
__global__ void __launch_bounds__(256) qs_gmax_kernel(const T* __restrict__ x, int64_t glen, int64_t cpg,
                                                      uint32_t* amax, uint32_t* status) {
  __shared__ uint32_t red[8];
  const int64_t g = blockIdx.x / cpg, c = blockIdx.x - g * cpg;
  const int64_t i0 = g * glen + c * QS_SPAN, i1 = g * glen + min(glen, (c + 1) * QS_SPAN);
  bool nan = false;
  uint32_t m = 0u;
  constexpr int VEC = 16 / (int)sizeof(T);
  const bool vec = ((i0 | i1) % VEC) == 0 && (reinterpret_cast<uintptr_t>(x) & 15) == 0;
  if (vec) {
    const uint4* p = reinterpret_cast<const uint4*>(x + i0);
    const int64_t nv = (i1 - i0) / VEC;
    for (int64_t v = threadIdx.x; v < nv; v += blockDim.x) {
      const uint4 q = __ldcs(p + v);
      const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if constexpr (sizeof(T) == 2) {
          const uint32_t lo = (w[k] << 16) & 0x7FFFFFFFu, hi = w[k] & 0x7FFF0000u;
          nan |= lo > 0x7F800000u || hi > 0x7F800000u;
          m = max(m, max(lo > 0x7F800000u ? 0u : lo, hi > 0x7F800000u ? 0u : hi));
        } else {
          const uint32_t b = w[k] & 0x7FFFFFFFu;
          nan |= b > 0x7F800000u;
          m = max(m, b > 0x7F800000u ? 0u : b);
        }
      }
    }
  } else {
    for (int64_t i = i0 + threadIdx.x; i < i1; i += blockDim.x) {
      const uint32_t b = load_bits(x, i) & 0x7FFFFFFFu;
      nan |= b > 0x7F800000u;
      m = max(m, b > 0x7F800000u ? 0u : b);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) m = max(m, red[w]);
    if (m) atomicMax(&amax[g], m);
  }
  if (__any_sync(0xffffffffu, nan) && (threadIdx.x & 31) == 0 && status) atomicOr(status, CURVEFP_DEV_NAN);
}

// 128-bit sum of a warp's lanes (exact; carries from the low words).
__device__ __forceinline__ unsigned __int128 warp_sum_u128(unsigned __int128 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long lo = __shfl_xor_sync(0xffffffffu, (unsigned long long)v, o);
    const unsigned long long hi = __shfl_xor_sync(0xffffffffu, (unsigned long long)(v >> 64), o);
    v += ((unsigned __int128)hi << 64) | lo;
  }
  return v;
}

// Per group and candidate: D(a) over the CTA's span, one exact 128-bit
// atomic add per warp and candidate.
template <int FMT, typename T>
__global__ void __launch_bounds__(256, 3) qs_mse_kernel(const T* __restrict__ x, int64_t glen, int64_t cpg,
                                                     const uint32_t* __restrict__ amax, unsigned long long* D) {
  __shared__ uint32_t lut[256], ck[8];
  for (int i = threadIdx.x; i < 256; i += blockDim.x) lut[i] = __ldg(lut_src<Fmt<FMT>::K>() + i);
  if (threadIdx.x < 8) ck[threadIdx.x] = Fmt<FMT>::K == 8 ? CFP_CK_F32_K8_DEV[threadIdx.x] : CFP_CK_F32_K4_DEV[threadIdx.x & 3];
  __syncthreads();
  const int64_t g = blockIdx.x / cpg, c = blockIdx.x - g * cpg;
  const uint32_t am = amax[g];
  if (am == 0u || am >= 0x7F800000u) return;  // the group keeps a_c
  const int ac = block_scale<FMT>(am);
  const int64_t i0 = g * glen + c * QS_SPAN, i1 = g * glen + min(glen, (c + 1) * QS_SPAN);
  unsigned __int128 acc[5] = {0, 0, 0, 0, 0};
  bool dummy = false;
  [[maybe_unused]] const MseCands cand = mse_cands<FMT>(ac);
  auto element = [&](uint32_t b) {
    if ((b & 0x7FFFFFFFu) > 0x7F800000u) return;  // NaN: left out
    if constexpr (!IsRadix<FMT>::value)
      if (mse_add5<FMT>(lut, ck, b, cand, acc)) return;
    const float xv = __uint_as_float(b);
#pragma unroll
    for (int k = 0; k < 5; ++k) {
      const int a = ac - 3 + k;
      if (a < -128 || a > 127) continue;
      acc[k] += sq_term(xv, recon_f32<FMT>(encode_slow<FMT>(lut, b, a, dummy), a), ac);
    }
  };
  constexpr int VEC = Elem<T>::VEC;
  if (((i0 | i1) % VEC) == 0 && (reinterpret_cast<uintptr_t>(x) & 15) == 0) {
    // 16-byte loads: VEC independent elements per thread and iteration
    const uint4* p = reinterpret_cast<const uint4*>(x + i0);
    const int64_t nv = (i1 - i0) / VEC;
    for (int64_t v = threadIdx.x; v < nv; v += blockDim.x) {
      const uint4 q = __ldcs(p + v);
#pragma unroll
      for (int e = 0; e < VEC; ++e) element(Elem<T>::bits(q, e));
    }
  } else {
    for (int64_t i = i0 + threadIdx.x; i < i1; i += blockDim.x) element(load_bits(x, i));
  }
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    const unsigned __int128 s = warp_sum_u128(acc[k]);
    if ((threadIdx.x & 31) == 0 && s) atomic_add_u128(D + (g * 5 + k) * 2, s);
  }
}

// The group's scale: a_c, or the MSE candidate with the smallest D (ties: the
// larger a).
template <int FMT>
__device__ __forceinline__ int choose_scale(uint32_t am, const unsigned long long* Dg, int rule) {
  const int ac = block_scale<FMT>(am);
  if (rule == 0 || am == 0u || am >= 0x7F800000u) return ac;
  int best = ac;
  unsigned __int128 bestD = 0;
  bool first = true;
  for (int c = 0; c < 5; ++c) {
    const int a = ac - 3 + c;
    if (a < -128 || a > 127) continue;
    const unsigned __int128 d = ((unsigned __int128)Dg[2 * c + 1] << 64) | Dg[2 * c];
    if (first || d <= bestD) {
      bestD = d;
      best = a;
      first = false;
    }
  }
  return best;
}

// Encode with one scale per group, element by element: the fallback for
// inputs that are not 16-byte aligned (the block quantizer loads 16-byte
// vectors).
template <int FMT, typename T>
__global__ void __launch_bounds__(256) qs_encode_scalar_kernel(const T* __restrict__ x, int64_t n, int64_t glen, int G,
                                                               const int8_t* __restrict__ gscale, uint8_t* codes,
                                                               int8_t* scales, uint32_t* status) {
  __shared__ uint32_t lut[256];
  for (int i = threadIdx.x; i < 256; i += blockDim.x) lut[i] = __ldg(lut_src<Fmt<FMT>::K>() + i);
  __syncthreads();
  const int gs = __ffs(G) - 1;
  bool nan = false;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int a = gscale[i / glen];
    codes[i] = (uint8_t)encode_slow<FMT>(lut, load_bits(x, i), a, nan);
    if ((i & (G - 1)) == 0) scales[i >> gs] = (int8_t)a;  // G is a power of two
  }
  if (nan && status) atomicOr(status, CURVEFP_DEV_NAN);
}

// One scale per group (the encode pass then takes it per block).
template <int FMT>
__global__ void qs_choose_kernel(const uint32_t* __restrict__ amax, const unsigned long long* __restrict__ D,
                                 int rule, int64_t ngroups, int8_t* __restrict__ gscale) {
  for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < ngroups; g += (int64_t)gridDim.x * blockDim.x)
    gscale[g] = (int8_t)choose_scale<FMT>(amax[g], D ? D + g * 10 : nullptr, D ? rule : 0);
}

// Block groups: one thread per block of G elements does everything in
// registers (no workspace).
template <int FMT, typename T>
__global__ void __launch_bounds__(256, 3) qs_block_kernel(const T* __restrict__ x, int64_t nblk, int G, int rule,
                                                       uint8_t* codes, int8_t* scales, uint32_t* status) {
  __shared__ uint32_t lut[256], ck[8];
  for (int i = threadIdx.x; i < 256; i += blockDim.x) lut[i] = __ldg(lut_src<Fmt<FMT>::K>() + i);
  if (threadIdx.x < 8) ck[threadIdx.x] = Fmt<FMT>::K == 8 ? CFP_CK_F32_K8_DEV[threadIdx.x] : CFP_CK_F32_K4_DEV[threadIdx.x & 3];
  __syncthreads();
  bool nan = false, dummy = false;
  // a thread's block with 16-byte loads where the input allows (G is a power
  // of two >= 32), element by element otherwise
  constexpr int VEC = Elem<T>::VEC;
  const bool vec = (reinterpret_cast<uintptr_t>(x) & 15) == 0 && (reinterpret_cast<uintptr_t>(codes) & 7) == 0;
  auto for_block = [&](int64_t i0, auto&& f) {  // f(element index in the block, bits)
    if (vec) {
      const uint4* p = reinterpret_cast<const uint4*>(x + i0);
      for (int v = 0; v < G / VEC; ++v) {
        const uint4 q = __ldg(p + v);
#pragma unroll
        for (int e = 0; e < VEC; ++e) f(v * VEC + e, Elem<T>::bits(q, e));
      }
    } else {
      for (int i = 0; i < G; ++i) f(i, load_bits(x, i0 + i));
    }
  };
  for (int64_t blk = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; blk < nblk;
       blk += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i0 = blk * G;
    uint32_t am = 0u;
    for_block(i0, [&](int, uint32_t bits) {
      const uint32_t b = bits & 0x7FFFFFFFu;
      if (b > 0x7F800000u) nan = true;
      else am = max(am, b);
    });
    unsigned long long Dg[10];
    const bool search = rule == 1 && am != 0u && am < 0x7F800000u;
    if (search) {
      const int ac = block_scale<FMT>(am);
      unsigned __int128 acc[5] = {0, 0, 0, 0, 0};
      [[maybe_unused]] const MseCands cand = mse_cands<FMT>(ac);
      for_block(i0, [&](int, uint32_t b) {
        if ((b & 0x7FFFFFFFu) > 0x7F800000u) return;
        if constexpr (!IsRadix<FMT>::value)
          if (mse_add5<FMT>(lut, ck, b, cand, acc)) return;
        const float xv = __uint_as_float(b);
#pragma unroll
        for (int k = 0; k < 5; ++k) {
          const int a = ac - 3 + k;
          if (a < -128 || a > 127) continue;
          acc[k] += sq_term(xv, recon_f32<FMT>(encode_slow<FMT>(lut, b, a, dummy), a), ac);
        }
      });
      for (int c = 0; c < 5; ++c) {
        Dg[2 * c] = (unsigned long long)acc[c];
        Dg[2 * c + 1] = (unsigned long long)(acc[c] >> 64);
      }
    }
    const int a = choose_scale<FMT>(am, Dg, search ? 1 : 0);
    scales[blk] = (int8_t)a;
    if (vec) {
      const uint4* p = reinterpret_cast<const uint4*>(x + i0);
      for (int v = 0; v < G / VEC; ++v) {
        const uint4 q = __ldg(p + v);
        uint32_t w[2] = {0u, 0u};
#pragma unroll
        for (int e = 0; e < VEC; ++e) w[e >> 2] |= encode_slow<FMT>(lut, Elem<T>::bits(q, e), a, dummy) << (8 * (e & 3));
        if constexpr (VEC == 4)
          *reinterpret_cast<uint32_t*>(codes + i0 + v * VEC) = w[0];
        else
          *reinterpret_cast<uint2*>(codes + i0 + v * VEC) = make_uint2(w[0], w[1]);
      }
    } else {
      for (int i = 0; i < G; ++i) codes[i0 + i] = (uint8_t)encode_slow<FMT>(lut, load_bits(x, i0 + i), a, dummy);
    }
  }
  if (nan && status) atomicOr(status, CURVEFP_DEV_NAN);
}

// ---------------------------------------------------------------------------
// Host-side launchers (called by the C ABI after argument validation).
// Templates shared by the per-format launcher files.


template <int FMT, typename T>
static cudaError_t launch_q_bulk(const void* x, int64_t nblk, uint8_t* codes, int8_t* scales, uint32_t* status,
                                 cudaStream_t st, int sms) {
  constexpr int NST = CFP_QB_NST;
  const size_t smem = BulkQ<FMT, T>::smem(NST);
  auto kern = quantize_rows_bulk_kernel<FMT, T, NST>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int64_t ch_blk = QB_CHUNK / (32 * (int64_t)sizeof(T));
  const int64_t nchunks = (nblk + ch_blk - 1) / ch_blk;
  // persistent CTAs take chunks round-robin, so the grid must be resident at once
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, (QB_NCW + 1) * 32, smem);
  if (e != cudaSuccess) return e;
  if (per_sm > CFP_QB_CTAS) per_sm = CFP_QB_CTAS;
  if (per_sm < 1) per_sm = 1;
  int64_t grid = (int64_t)sms * per_sm;
  if (grid > nchunks) grid = nchunks;
  kern<<<(unsigned)grid, (QB_NCW + 1) * 32, smem, st>>>(static_cast<const T*>(x), nblk, codes, scales, status);
  return cudaGetLastError();
}

template <int FMT, typename T, int G>
static cudaError_t launch_q(const void* x, int64_t rows, int64_t cols, int64_t ld, int axis, uint8_t* codes,
                            int8_t* scales, uint32_t* status, cudaStream_t st, int sms) {
  // dense rows of 32-element blocks: the bulk-fed kernel (16-byte aligned
  // input is checked by the caller for block_axis 0)
  if (axis == 0 && G == 32 && ld == cols)
    return launch_q_bulk<FMT, T>(x, rows * (cols / G), codes, scales, status, st, sms);
  if (axis == 0) {
    constexpr int VEC = Elem<T>::VEC;
    constexpr int TPB = (sizeof(T) == 2 && G == 32) ? 2 : ((G / VEC) < 8 ? (G / VEC) : 8);
    const int64_t nblk = rows * (cols / G);
    constexpr int VPT = (G / VEC) / TPB;
    constexpr int PER_WARP = (32 / TPB) * (VPT >= 4 ? 1 : 4 / VPT);
    const int64_t warps_needed = (nblk + PER_WARP - 1) / PER_WARP;
    int64_t grid = (warps_needed + 7) / 8;
    const int64_t cap = (int64_t)sms * 8;  // 8 resident CTAs of 256 lanes per SM
    if (grid > cap) grid = cap;
    if (grid < 1) grid = 1;
    quantize_rows_kernel<FMT, T, G><<<(unsigned)grid, 256, 0, st>>>(static_cast<const T*>(x), rows, cols, ld,
                                                                      codes, scales, status, nullptr, 1);
  } else {
    dim3 grid((unsigned)((cols + 255) / 256), (unsigned)(rows / G));
    quantize_cols_kernel<FMT, T, G><<<grid, 256, 0, st>>>(static_cast<const T*>(x), rows, cols, ld, codes, scales,
                                                           status);
  }
  return cudaGetLastError();
}

template <int FMT, typename T>
static cudaError_t launch_q_g(int G, const void* x, int64_t rows, int64_t cols, int64_t ld, int axis,
                              uint8_t* codes, int8_t* scales, uint32_t* status, cudaStream_t st, int sms) {
  switch (G) {
    case 32: return launch_q<FMT, T, 32>(x, rows, cols, ld, axis, codes, scales, status, st, sms);
    case 64: return launch_q<FMT, T, 64>(x, rows, cols, ld, axis, codes, scales, status, st, sms);
    case 128: return launch_q<FMT, T, 128>(x, rows, cols, ld, axis, codes, scales, status, st, sms);
    case 256: return launch_q<FMT, T, 256>(x, rows, cols, ld, axis, codes, scales, status, st, sms);
    case 512: return launch_q<FMT, T, 512>(x, rows, cols, ld, axis, codes, scales, status, st, sms);
  }
  return cudaErrorInvalidValue;
}

// The register-fed block quantizer with a scale per group of bpg blocks.
template <int FMT, typename T, int G>
static cudaError_t launch_q_grp(const T* x, int64_t rows, int64_t cols, uint8_t* codes, int8_t* scales,
                                uint32_t* status, cudaStream_t st, int sms, const int8_t* gscale, int64_t bpg) {
  constexpr int VEC = Elem<T>::VEC;
  constexpr int TPB = (sizeof(T) == 2 && G == 32) ? 2 : ((G / VEC) < 8 ? (G / VEC) : 8);
  const int64_t nblk = rows * (cols / G);
  constexpr int VPT = (G / VEC) / TPB;
  constexpr int PER_WARP = (32 / TPB) * (VPT >= 4 ? 1 : 4 / VPT);
  const int64_t warps_needed = (nblk + PER_WARP - 1) / PER_WARP;
  int64_t grid = (warps_needed + 7) / 8;
  const int64_t cap = (int64_t)sms * 8;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  quantize_rows_kernel<FMT, T, G><<<(unsigned)grid, 256, 0, st>>>(x, rows, cols, cols, codes, scales, status, gscale,
                                                                    bpg);
  return cudaGetLastError();
}

template <int FMT, typename T>
static cudaError_t launch_q_grouped(int G, const T* x, int64_t rows, int64_t cols, uint8_t* codes, int8_t* scales,
                                    uint32_t* status, cudaStream_t st, int sms, const int8_t* gscale, int64_t bpg) {
  switch (G) {
    case 32: return launch_q_grp<FMT, T, 32>(x, rows, cols, codes, scales, status, st, sms, gscale, bpg);
    case 64: return launch_q_grp<FMT, T, 64>(x, rows, cols, codes, scales, status, st, sms, gscale, bpg);
    case 128: return launch_q_grp<FMT, T, 128>(x, rows, cols, codes, scales, status, st, sms, gscale, bpg);
    case 256: return launch_q_grp<FMT, T, 256>(x, rows, cols, codes, scales, status, st, sms, gscale, bpg);
    case 512: return launch_q_grp<FMT, T, 512>(x, rows, cols, codes, scales, status, st, sms, gscale, bpg);
  }
  return cudaErrorInvalidValue;
}

// Workspace of row / tensor groups: group maxima (4 bytes), group scales
// (1 byte) and the MSE sums (5 candidates x 16 bytes) per group.
inline size_t qs_workspace_bytes(int64_t rows, int64_t cols, int G, int group) {
  if (group == 0) return 0;
  const int64_t ngroups = group == 1 ? rows : 1;
  return (size_t)((ngroups * 4 + 15) / 16 * 16) + (size_t)((ngroups + 15) / 16 * 16) + (size_t)ngroups * 80;
}

template <int FMT, typename T>
static cudaError_t launch_qs_t(int G, int group, int rule, const void* xv, int64_t rows, int64_t cols, uint8_t* codes,
                               int8_t* scales, void* ws, uint32_t* status, cudaStream_t st, int sms) {
  const T* x = static_cast<const T*>(xv);
  const int64_t n = rows * cols;
  if (group == 0) {
    const int64_t nblk = n / G;
    int64_t grid = (nblk + 255) / 256;
    if (grid > (int64_t)sms * 8) grid = (int64_t)sms * 8;
    qs_block_kernel<FMT, T><<<(unsigned)(grid < 1 ? 1 : grid), 256, 0, st>>>(x, nblk, G, rule, codes, scales, status);
    return cudaGetLastError();
  }
  const int64_t glen = group == 1 ? cols : n;
  const int64_t ngroups = n / glen;
  uint8_t* w8 = static_cast<uint8_t*>(ws);
  uint32_t* amax = reinterpret_cast<uint32_t*>(w8);
  int8_t* gscale = reinterpret_cast<int8_t*>(w8 + (ngroups * 4 + 15) / 16 * 16);
  unsigned long long* D =
      reinterpret_cast<unsigned long long*>(w8 + (ngroups * 4 + 15) / 16 * 16 + (ngroups + 15) / 16 * 16);
  cudaError_t e = cudaMemsetAsync(ws, 0, qs_workspace_bytes(rows, cols, G, group), st);
  if (e != cudaSuccess) return e;
  const int64_t cpg = (glen + QS_SPAN - 1) / QS_SPAN;  // spans per group
  const unsigned nspan = (unsigned)(ngroups * cpg);
  qs_gmax_kernel<T><<<nspan, 256, 0, st>>>(x, glen, cpg, amax, status);
  if (rule == 1) qs_mse_kernel<FMT, T><<<nspan, 256, 0, st>>>(x, glen, cpg, amax, D);
  int64_t cg = (ngroups + 255) / 256;
  qs_choose_kernel<FMT><<<(unsigned)(cg < 1024 ? cg : 1024), 256, 0, st>>>(amax, rule == 1 ? D : nullptr, rule,
                                                                        ngroups, gscale);
  // encode: the register-fed block quantizer with the group's scale per block
  // (16-byte aligned input), else element by element
  if ((reinterpret_cast<uintptr_t>(x) & 15) == 0) {
    const int64_t bpg = glen / G;
    return launch_q_grouped<FMT, T>(G, x, rows, cols, codes, scales, status, st, sms, gscale, bpg);
  }
  int64_t grid = (n + 255) / 256;
  if (grid > (int64_t)sms * 8) grid = (int64_t)sms * 8;
  qs_encode_scalar_kernel<FMT, T><<<(unsigned)(grid < 1 ? 1 : grid), 256, 0, st>>>(x, n, glen, G, gscale, codes,
                                                                                   scales, status);
  return cudaGetLastError();
}

}  // namespace cfp
