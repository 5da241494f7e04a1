/*
 * CurveFP oracle — TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously-correct CPU restatement of what the CurveFP hot
 * path computes.  Only the tests, the smoke check and the benchmark's
 * CPU-baseline leg may load this file's library; the product path never does.
 * It shares no code, header, table or constant with the CUDA library: every
 * level and phase constant here comes from libm's exp2 at run time, and every
 * decision (nearest level, block scale, phase address) is taken by brute
 * force or by the plain definition.
 *
 * Paper references are to "CurveFP: Co-Designing Numerical Representation
 * and Product Arithmetic for Language Models":
 *   Eq. 1  element value          x = (-1)^s 2^{a_b} r^{e+k/K}      (Sec. 3.1)
 *   Eq. 2  curve-index product    l = (i+j) mod K, c = floor((i+j)/K) (Sec. 3.2)
 *   Eq. 4  phase count            H = qK / gcd(p, qK)               (Sec. 3.2)
 *   Eq. 5  binned accumulation    x.w = sum_h 2^{h/H} sum_t n_{h,t} 2^t
 *   App. A.1 closed-product addressing (delta, h, t)
 *   App. C.1 rank packing: sign in bit 7, magnitude rank m in bits 6:0,
 *            m = 0 is zero.
 * Binary radix (p = q = 1) throughout, as in every principal format.
 *
 * Readings taken where the paper is silent (each one is listed in the design
 * notes and mirrored by the CUDA library's header):
 *   R1 code byte = (s << 7) | m, m = n + B, n = eK + k, B = 2^{E+C-1};
 *      m = 0 is the zero sentinel; zero is emitted as 0x00.
 *   R2 "ceil-absmax" scale: a_b = the smallest integer in [-128, 127] with
 *      amax <= 2^{a_b} * L_{nmax}; amax = 0 gives a_b = 0; no such integer
 *      (amax = Inf) gives 127.  NaN elements are left out of amax.
 *   R3 nearest level over the codebook {0} U {2^{n/K}}; zero is a codebook
 *      entry, so values below L_{nmin}/2 become zero; values above L_{nmax}
 *      saturate; NaN encodes to 0x00 and raises a flag.
 *   R4 dequantized FP32 value = RN32( RN32(2^{k/K}) * 2^{a_b + e} ).
 *   R5 mixed formats share the lattice L = lcm(K_a, K_b): u = n_a L/K_a +
 *      n_b L/K_b, h = u mod L, t = floor(u / L), H = L phases.
 *   R6 exported per-phase sums are integers S_h at the per-output LSB
 *      lambda = min_b(sa_b + sb_b) + t_min.
 *   R11, R12 static-operand scale groups and MSE-search scales (below).
 *   R14 rational radix r = 2^{p/q} (Sec. 3.1, Eq. 4, Table 2's E4C3 points
 *      r = 2^{8/9} and r = 2^{3/4}): the level of index n is 2^{p n/(qK)};
 *      the closed product of two codes of the same format has
 *      u = p (n_a + n_b), phase h = (u mod qK)/g and bin t = floor(u/qK)
 *      (App. A.1), H = qK/g phases weighted 2^{h/H}; FP32 dequantization is
 *      RN32(2^{j/(qK)}) 2^{a + floor(p n/(qK))}, j = p n mod qK (R4 with the
 *      fractional exponent in place of k/K).  Only same-format pairs.  An
 *      exact tie in the nearest-level search (possible only between zero and
 *      L_nmin when L_nmin is a power of two, as for r = 2^{8/9}) goes to the
 *      smaller magnitude.
 *   R13 reused operands (Sec. 4, training GEMMs: the backward GEMMs take the
 *      forward pass's quantized operands, one of them transposed) keep each
 *      element's own code and block scale, so a GEMM operand may carry a
 *      scale per element; the accumulation is Eq. 5 with per-element scales
 *      (oracle_gemm_elem below).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef __int128 i128;

/* Format ids follow Table 1: E3C3 (CurveFP7), E4C3 and E5C2 (CurveFP8). */
typedef struct {
  int E;    /* exponent width                         */
  int C;    /* curve-index width                      */
  int K;    /* curves per exponent, K = 2^C           */
  int B;    /* rank bias 2^{E+C-1}                    */
  int nmax; /* largest lattice index, nmin = -nmax    */
  int p, q; /* radix r = 2^{p/q} (R14); 1, 1 = binary  */
} ofmt;

static int ofmt_get(int id, ofmt* f) {
  switch (id) {
    case 0: f->E = 3; f->C = 3; break; /* E3C3 */
    case 1: f->E = 4; f->C = 3; break; /* E4C3 */
    case 2: f->E = 5; f->C = 2; break; /* E5C2 */
    case 3: f->E = 4; f->C = 3; break; /* E4C3, r = 2^{8/9} (R14) */
    case 4: f->E = 4; f->C = 3; break; /* E4C3, r = 2^{3/4} (R14) */
    default: return -1;
  }
  f->p = id == 3 ? 8 : (id == 4 ? 3 : 1);
  f->q = id == 3 ? 9 : (id == 4 ? 4 : 1);
  f->K = 1 << f->C;
  f->B = 1 << (f->E + f->C - 1);
  /* Sec. 3.1: exponents e in [-2^{E-1}, 2^{E-1}-1], k in [0, K-1]; the
   * smallest combination (e = -2^{E-1}, k = 0) is dropped, leaving
   * 2^{E+C} - 1 positive magnitudes n = eK + k in [-(B-1), B-1]. */
  f->nmax = f->B - 1;
  return 0;
}

static int floordiv(int a, int b) { int q = a / b; if ((a % b) && ((a < 0) != (b < 0))) q--; return q; }
static int floormod(int a, int b) { int r = a % b; if (r && ((r < 0) != (b < 0))) r += b; return r; }

/* ---- Element value, Eq. 1 ------------------------------------------- */

/* Unscaled level for lattice index n: r^{n/K} = 2^{p n/(q K)}, evaluated as
 * 2^{j/(qK)} 2^e with e = floor(p n/(qK)), j = p n mod qK (the exponent's
 * fractional part is then the only rounded input of exp2). */
static double olevel(const ofmt* f, int n) {
  int den = f->q * f->K;
  return ldexp(exp2((double)floormod(f->p * n, den) / den), floordiv(f->p * n, den));
}

/* R4 (R14): RN32 of the fractional power times the integer power. */
static double odequant_exact(const ofmt* f, int n, int a) {
  int den = f->q * f->K;
  int e = floordiv(f->p * n, den), j = floormod(f->p * n, den);
  float cj = (float)exp2((double)j / den); /* RN32(2^{j/(qK)}) */
  return ldexp((double)cj, a + e);        /* exact in fp64     */
}

int oracle_format(int id, int* E, int* C, int* K, int* B, int* nmax) {
  ofmt f;
  if (ofmt_get(id, &f)) return -1;
  *E = f.E; *C = f.C; *K = f.K; *B = f.B; *nmax = f.nmax;
  return 0;
}

/* All 2B-1 positive levels, index n + nmax.  Table 1 counts them. */
int oracle_levels(int id, double* out) {
  ofmt f;
  if (ofmt_get(id, &f)) return -1;
  for (int n = -f.nmax; n <= f.nmax; ++n) out[n + f.nmax] = olevel(&f, n);
  return 2 * f.nmax + 1;
}

/* Eq. 4: number of phase classes for radix 2^{p/q} with K curves. */
static long gcdl(long a, long b) { while (b) { long t = a % b; a = b; b = t; } return a < 0 ? -a : a; }
long oracle_phase_count(long p, long q, long K) { return q * K / gcdl(p, q * K); }

/* Field view of a code (App. C.1 packing).  Returns 0 for the zero code. */
static int odecode(const ofmt* f, uint8_t code, int* s, int* n) {
  int m = code & (f->E + f->C == 6 ? 0x3F : 0x7F);
  if (m == 0) return 0;
  *s = code >> 7;
  *n = m - f->B;
  return 1;
}

int oracle_decode_fields(int id, uint8_t code, int* s, int* e, int* k, int* m) {
  ofmt f;
  if (ofmt_get(id, &f)) return -1;
  int n;
  *m = code & (f.E + f.C == 6 ? 0x3F : 0x7F);
  if (!odecode(&f, code, s, &n)) { *s = 0; *e = 0; *k = 0; return 0; }
  *e = floordiv(n, f.K);
  *k = floormod(n, f.K);
  return 1;
}

/* ---- Block scale, Sec. 3.1 ("dynamic training operands use ceil-absmax
 * scaling"), reading R2: brute-force search over the int8 container. ---- */
int oracle_block_scale(int id, double amax) {
  ofmt f;
  if (ofmt_get(id, &f)) return 0;
  if (amax == 0.0) return 0;
  double top = olevel(&f, f.nmax);
  for (int a = -128; a <= 127; ++a)
    if (amax <= ldexp(top, a)) return a;
  return 127;
}

/* ---- Nearest level, Sec. 3.1, reading R3: scan every codebook entry ---- */
static int onearest_rank(const ofmt* f, double v) {
  if (isinf(v)) return 2 * f->B - 1; /* above every level: saturate */
  int best = 0;                       /* rank 0 = zero                */
  double bestd = fabs(v);
  for (int n = -f->nmax; n <= f->nmax; ++n) {
    double d = fabs(v - olevel(f, n));
    if (d < bestd) { bestd = d; best = n + f->B; }
  }
  return best;
}

/* Quantize one tensor.  x is FP32 (BF16 callers widen exactly first).
 * block_axis 0: blocks of G along columns; codes [rows x cols], scales
 *               [rows x cols/G].
 * block_axis 1: blocks of G along rows; the output is the transposed
 *               operand: codes [cols x rows], scales [cols x rows/G].
 * Returns a flag word: bit 0 = a NaN was seen. */
int oracle_quantize(int id, int G, const float* x, int64_t rows, int64_t cols, int64_t ld,
                    int block_axis, uint8_t* codes, int8_t* scales) {
  ofmt f;
  if (ofmt_get(id, &f)) return -1;
  int64_t R = block_axis ? cols : rows; /* output rows    */
  int64_t Cc = block_axis ? rows : cols; /* output columns */
  int64_t nb = Cc / G;
  int flags = 0;
#pragma omp parallel for schedule(static) reduction(| : flags)
  for (int64_t r = 0; r < R; ++r) {
    for (int64_t b = 0; b < nb; ++b) {
      double amax = 0.0;
      for (int64_t i = 0; i < G; ++i) {
        int64_t c = b * G + i;
        float xv = block_axis ? x[c * ld + r] : x[r * ld + c];
        if (isnan(xv)) continue;
        double av = fabs((double)xv);
        if (av > amax) amax = av;
      }
      int a = oracle_block_scale(id, amax);
      scales[r * nb + b] = (int8_t)a;
      for (int64_t i = 0; i < G; ++i) {
        int64_t c = b * G + i;
        float xv = block_axis ? x[c * ld + r] : x[r * ld + c];
        uint8_t code = 0;
        if (isnan(xv)) {
          flags |= 1;
        } else {
          double v = ldexp(fabs((double)xv), -a); /* exact: power-of-two scaling */
          int m = onearest_rank(&f, v);
          if (m) code = (uint8_t)(((signbit(xv) ? 1 : 0) << 7) | m);
        }
        codes[r * Cc + c] = code;
      }
    }
  }
  return flags;
}

/* Element encode with given block scales (Sec. 3.1: with the block scale
 * fixed, an element keeps its sign and takes the magnitude level whose
 * reconstruction lies closest to it).  x is [R x Cc] row-major, blocks of G
 * along columns, scales [R x Cc/G].  Returns the NaN flag. */
int oracle_encode(int id, int G, const float* x, int64_t R, int64_t Cc, const int8_t* scales,
                  uint8_t* codes) {
  ofmt f;
  if (ofmt_get(id, &f)) return -1;
  int64_t nb = Cc / G;
  int flags = 0;
#pragma omp parallel for schedule(static) reduction(| : flags)
  for (int64_t r = 0; r < R; ++r)
    for (int64_t c = 0; c < Cc; ++c) {
      float xv = x[r * Cc + c];
      uint8_t code = 0;
      if (isnan(xv)) {
        flags |= 1;
      } else {
        int m = onearest_rank(&f, ldexp(fabs((double)xv), -scales[r * nb + c / G]));
        if (m) code = (uint8_t)(((signbit(xv) ? 1 : 0) << 7) | m);
      }
      codes[r * Cc + c] = code;
    }
  return flags;
}

/* ---- Static operands: scale granularity and MSE-search scales ----------
 * Sec. 3.1: a static operand's power-of-two scale is picked by the
 * reconstruction error it gives, a dynamic (training) operand's by the
 * ceil-absmax rule; Sec. 4.2 compares per-tensor, per-row and fixed-size
 * block scales.
 * Readings (listed with the others):
 *   R11 a scale group is a block of G elements of a row, a whole row, or the
 *       whole tensor; scales are stored per block of G ([rows x cols/G]),
 *       every block of a group holding the group's scale.
 *   R12 MSE search: candidates a in [a_c - 3, a_c + 1] (clamped to int8),
 *       a_c the group's ceil-absmax scale; each element is encoded at scale a
 *       (nearest level, R3, saturating) and reconstructed as in R4; the
 *       criterion is D(a) = sum_i floor((x_i - xhat_i)^2 * 2^{60 - 2 a_c}),
 *       an exact integer (every squared FP32 reconstruction error on a grid
 *       of 2^{2 a_c - 60}); the smallest D wins, ties go to the larger a.
 *       NaN elements are left out; groups with Inf, or with amax = 0, keep
 *       a_c. */

/* Reading R4 for one code under scale a (0.0f for the zero code). */
static float odequant_one(const ofmt* f, uint8_t code, int a) {
  int s, n;
  if (!odecode(f, code, &s, &n)) return 0.0f;
  double exact = odequant_exact(f, n, a);
  return (float)(s ? -exact : exact);
}

static uint8_t oencode_one(const ofmt* f, float xv, int a) {
  if (isnan(xv)) return 0;
  int m = onearest_rank(f, ldexp(fabs((double)xv), -a));
  return m ? (uint8_t)(((signbit(xv) ? 1 : 0) << 7) | m) : 0;
}

/* floor((x - xhat)^2 * 2^{60 - 2 ac}), exact.  x - xhat is exact in fp64
 * (both FP32, within a factor 16 of each other unless xhat = 0), so
 * e = M 2^{E-53} with an integer M < 2^53 and e^2 = M^2 2^{2E-106}. */
static unsigned __int128 osq_term(float x, float xhat, int ac) {
  double e = fabs((double)x - (double)xhat);
  if (e == 0.0) return 0;
  int E;
  double fr = frexp(e, &E);                   /* e = fr 2^E, fr in [0.5, 1) */
  unsigned long long M = (unsigned long long)ldexp(fr, 53);
  unsigned __int128 sq = (unsigned __int128)M * M;
  int sh = 2 * E - 106 + 60 - 2 * ac;          /* term = sq * 2^sh */
  if (sh >= 0) return sh >= 128 ? 0 : sq << sh; /* (never taken: |e| < 2^{ac+18}) */
  return sh <= -128 ? 0 : sq >> (-sh);
}

/* Quantize with a scale per group (R11) chosen by ceil-absmax (rule 0) or by
 * MSE search (rule 1, R12).  granularity: 0 block of G, 1 row, 2 tensor.
 * x [rows x cols] (ld = cols), blocks along columns (cols % G == 0); codes
 * [rows x cols], scales [rows x cols/G].  Returns the NaN flag. */
int oracle_quantize_static(int id, int G, const float* x, int64_t rows, int64_t cols, int granularity, int rule,
                           uint8_t* codes, int8_t* scales) {
  ofmt f;
  if (ofmt_get(id, &f) || G <= 0 || cols % G) return -1;
  int64_t nb = cols / G;
  int64_t glen = granularity == 0 ? G : (granularity == 1 ? cols : rows * cols);
  int64_t ngroups = (rows * cols) / glen;
  int flags = 0;
#pragma omp parallel for schedule(dynamic) reduction(| : flags)
  for (int64_t g = 0; g < ngroups; ++g) {
    /* group g covers flat elements [g glen, (g + 1) glen) of the row-major tensor */
    const int64_t i0 = g * glen;
    double amax = 0.0;
    int has_inf = 0;
    for (int64_t i = i0; i < i0 + glen; ++i) {
      float xv = x[i];
      if (isnan(xv)) { flags |= 1; continue; }
      if (isinf(xv)) has_inf = 1;
      double av = fabs((double)xv);
      if (av > amax) amax = av;
    }
    int ac = oracle_block_scale(id, amax);
    int best = ac;
    if (rule == 1 && !has_inf && amax != 0.0) {
      unsigned __int128 bestD = 0;
      int first = 1;
      for (int a = ac - 3; a <= ac + 1; ++a) {
        if (a < -128 || a > 127) continue;
        unsigned __int128 D = 0;
        for (int64_t i = i0; i < i0 + glen; ++i) {
          float xv = x[i];
          if (isnan(xv)) continue;
          D += osq_term(xv, odequant_one(&f, oencode_one(&f, xv, a), a), ac);
        }
        if (first || D <= bestD) { bestD = D; best = a; first = 0; } /* ties: the larger a */
      }
    }
    for (int64_t i = i0; i < i0 + glen; ++i) codes[i] = oencode_one(&f, x[i], best);
    for (int64_t i = i0; i < i0 + glen; i += G) scales[i / G] = (int8_t)best;
  }
  (void)nb;
  return flags;
}

/* Real value of each code under its block scale, in fp64 (Eq. 1). */
int oracle_decode(int id, int G, const uint8_t* codes, const int8_t* scales, int64_t R, int64_t Cc,
                  double* out) {
  ofmt f;
  if (ofmt_get(id, &f)) return -1;
  int64_t nb = Cc / G;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < R; ++r)
    for (int64_t c = 0; c < Cc; ++c) {
      int s, n;
      double v = 0.0;
      if (odecode(&f, codes[r * Cc + c], &s, &n))
        v = (s ? -1.0 : 1.0) * ldexp(olevel(&f, n), scales[r * nb + c / G]);
      out[r * Cc + c] = v;
    }
  return 0;
}

/* Reading R4: FP32 dequantization. */
int oracle_dequantize(int id, int G, const uint8_t* codes, const int8_t* scales, int64_t R, int64_t Cc,
                      float* out) {
  ofmt f;
  if (ofmt_get(id, &f)) return -1;
  int64_t nb = Cc / G;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < R; ++r)
    for (int64_t c = 0; c < Cc; ++c) {
      int s, n;
      float v = 0.0f;
      if (odecode(&f, codes[r * Cc + c], &s, &n)) {
        double exact = odequant_exact(&f, n, scales[r * nb + c / G]); /* exact in fp64 */
        v = (float)(s ? -exact : exact);                               /* one RN32 rounding */
      }
      out[r * Cc + c] = v;
    }
  return 0;
}

/* ---- Closed product, Eq. 2 and App. A.1, readings R5 and R14 ---------
 * A product of lattice indices n_a, n_b sits at u = P (n_a wa + n_b wb) on a
 * lattice of N steps per binade: phase h = (u mod N)/g, bin t = floor(u/N),
 * L = N/g phases.  Binary radix (R5): N = max(K_a, K_b) (the lcm of two
 * powers of two), wa = N/K_a, wb = N/K_b, P = g = 1.  Rational radix, same
 * format on both sides (R14): N = qK, wa = wb = 1, P = p, g = gcd(p, qK). */
typedef struct { int wa, wb, P, N, g, L, ok; } olattice;

static olattice olattice_of(const ofmt* fa, const ofmt* fb) {
  olattice l;
  if (fa->p == 1 && fa->q == 1 && fb->p == 1 && fb->q == 1) {
    l.N = fa->K > fb->K ? fa->K : fb->K;
    l.wa = l.N / fa->K;
    l.wb = l.N / fb->K;
    l.P = 1;
    l.g = 1;
    l.ok = 1;
  } else {
    l.ok = fa->p == fb->p && fa->q == fb->q && fa->K == fb->K;
    l.N = fa->q * fa->K;
    l.wa = l.wb = 1;
    l.P = fa->p;
    l.g = (int)gcdl(fa->p, l.N);
  }
  l.L = l.N / l.g;
  return l;
}

static void oaddr(const olattice* l, int na, int nb, int* h, int* t) {
  int u = l->P * (na * l->wa + nb * l->wb);
  *h = floormod(u, l->N) / l->g;
  *t = floordiv(u, l->N);
}

/* Product of two codes: returns 0 if either is zero (no update), else sets
 * delta = +-1, phase h in [0, L) and bin offset t = floor(u / L). */
int oracle_closed_product(int ida, int idb, uint8_t ca, uint8_t cb, int* delta, int* h, int* t) {
  ofmt fa, fb;
  if (ofmt_get(ida, &fa) || ofmt_get(idb, &fb)) return -1;
  int sa, na, sb, nb;
  if (!odecode(&fa, ca, &sa, &na) || !odecode(&fb, cb, &sb, &nb)) return 0;
  olattice l = olattice_of(&fa, &fb);
  if (!l.ok) return -1;
  *delta = (sa ^ sb) ? -1 : 1;
  oaddr(&l, na, nb, h, t);
  return 1;
}

/* Smallest and largest bin offset t over nonzero products of a pair (every
 * pair of lattice indices tried). */
static void otrange(const ofmt* fa, const ofmt* fb, int* tmin, int* tmax) {
  olattice l = olattice_of(fa, fb);
  *tmin = 1 << 20;
  *tmax = -(1 << 20);
  for (int na = -fa->nmax; na <= fa->nmax; ++na)
    for (int nb = -fb->nmax; nb <= fb->nmax; ++nb) {
      int h, t;
      oaddr(&l, na, nb, &h, &t);
      if (t < *tmin) *tmin = t;
      if (t > *tmax) *tmax = t;
    }
}

int oracle_pair_info(int ida, int idb, int* L, int* tmin, int* tmax) {
  ofmt fa, fb;
  if (ofmt_get(ida, &fa) || ofmt_get(idb, &fb)) return -1;
  olattice l = olattice_of(&fa, &fb);
  if (!l.ok) return -1;
  *L = l.L;
  otrange(&fa, &fb, tmin, tmax);
  return 0;
}

static int obitlen(int64_t v) { int b = 0; while (v) { b++; v >>= 1; } return b; }

/* ---- Per-phase accumulation (Eq. 5, App. A.1) and phase combine -------
 * A: [M x K] codes (K contiguous), sa: [M x K/G]; B: [N x K], sb: [N x K/G].
 * For each output (i, j):
 *   lambda = min_b (sa[i,b] + sb[j,b]) + t_min                   (R6)
 *   S_h    = sum over nonzero products with phase h of
 *            delta * 2^{sa + sb + t - lambda}   (exact integer)
 *   C      = sum_h 2^{h/L} * S_h * 2^lambda      (fp64 combine)
 * The int128 window is declared out of range when
 *   bitlen(K) + spread + (t_max - t_min) > 127,
 * spread = max_b(sa+sb) - min_b(sa+sb); then rflag = 1 and S, C are not
 * defined (C is set to NaN).
 * S (may be NULL): M*N*L int128 as (lo, hi) int64 pairs; lsb (may be NULL):
 * M*N int32; rflag (may be NULL): M*N bytes.  Returns the number of
 * out-of-range outputs. */
int64_t oracle_gemm(int ida, int idb, int G, const uint8_t* A, const int8_t* sA, const uint8_t* B,
                    const int8_t* sB, int64_t M, int64_t N, int64_t K, double* C, int64_t* S,
                    int32_t* lsb, uint8_t* rflag) {
  ofmt fa, fb;
  if (ofmt_get(ida, &fa) || ofmt_get(idb, &fb)) return -1;
  olattice l = olattice_of(&fa, &fb);
  if (!l.ok) return -1;
  int tmin, tmax;
  otrange(&fa, &fb, &tmin, &tmax);
  int64_t nb = K / G;
  int64_t bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(+ : bad)
  for (int64_t i = 0; i < M; ++i) {
    i128 acc[32];
    for (int64_t j = 0; j < N; ++j) {
      int smin = 1 << 20, smax = -(1 << 20);
      for (int64_t b = 0; b < nb; ++b) {
        int s = sA[i * nb + b] + sB[j * nb + b];
        if (s < smin) smin = s;
        if (s > smax) smax = s;
      }
      int lambda = smin + tmin;
      int out_of_range = obitlen(K) + (smax - smin) + (tmax - tmin) > 127;
      for (int h = 0; h < l.L; ++h) acc[h] = 0;
      if (!out_of_range) {
        for (int64_t d = 0; d < K; ++d) {
          int s1, n1, s2, n2;
          if (!odecode(&fa, A[i * K + d], &s1, &n1)) continue;
          if (!odecode(&fb, B[j * K + d], &s2, &n2)) continue;
          int h, t;
          oaddr(&l, n1, n2, &h, &t);
          t += sA[i * nb + d / G] + sB[j * nb + d / G];
          i128 term = (i128)1 << (t - lambda);
          acc[h] += (s1 ^ s2) ? -term : term;
        }
      }
      double c = 0.0;
      for (int h = 0; h < l.L; ++h)
        c += exp2((double)h / l.L) * ldexp((double)acc[h], lambda);
      if (out_of_range) { c = NAN; bad++; }
      C[i * N + j] = c;
      if (S)
        for (int h = 0; h < l.L; ++h) {
          S[((i * N + j) * l.L + h) * 2 + 0] = (int64_t)(uint64_t)((unsigned __int128)acc[h]);
          S[((i * N + j) * l.L + h) * 2 + 1] = (int64_t)(acc[h] >> 64);
        }
      if (lsb) lsb[i * N + j] = lambda;
      if (rflag) rflag[i * N + j] = (uint8_t)out_of_range;
    }
  }
  return bad;
}

/* ---- Per-element scales (R13) ----------------------------------------
 * As oracle_gemm, with a scale per operand element: ea [M x K], eb [N x K]
 * (int8, K contiguous).  For output (i, j) and index d:
 *   t      = floor(u / L) + ea[i,d] + eb[j,d]
 *   lambda = min_d (ea[i,d] + eb[j,d]) + t_min
 * and the int128 window check takes spread = max_d - min_d of the same sum.
 * With block scales broadcast to every element of their block this is
 * oracle_gemm's definition (the min and max over d run over the same set of
 * values as over blocks). */
int64_t oracle_gemm_elem(int ida, int idb, const uint8_t* A, const int8_t* eA, const uint8_t* B,
                         const int8_t* eB, int64_t M, int64_t N, int64_t K, double* C, int64_t* S,
                         int32_t* lsb, uint8_t* rflag) {
  ofmt fa, fb;
  if (ofmt_get(ida, &fa) || ofmt_get(idb, &fb)) return -1;
  olattice l = olattice_of(&fa, &fb);
  if (!l.ok) return -1;
  int tmin, tmax;
  otrange(&fa, &fb, &tmin, &tmax);
  int64_t bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(+ : bad)
  for (int64_t i = 0; i < M; ++i) {
    i128 acc[32];
    for (int64_t j = 0; j < N; ++j) {
      int smin = 1 << 20, smax = -(1 << 20);
      for (int64_t d = 0; d < K; ++d) {
        int s = eA[i * K + d] + eB[j * K + d];
        if (s < smin) smin = s;
        if (s > smax) smax = s;
      }
      int lambda = smin + tmin;
      int out_of_range = obitlen(K) + (smax - smin) + (tmax - tmin) > 127;
      for (int h = 0; h < l.L; ++h) acc[h] = 0;
      if (!out_of_range) {
        for (int64_t d = 0; d < K; ++d) {
          int s1, n1, s2, n2;
          if (!odecode(&fa, A[i * K + d], &s1, &n1)) continue;
          if (!odecode(&fb, B[j * K + d], &s2, &n2)) continue;
          int h, t;
          oaddr(&l, n1, n2, &h, &t);
          t += eA[i * K + d] + eB[j * K + d];
          i128 term = (i128)1 << (t - lambda);
          acc[h] += (s1 ^ s2) ? -term : term;
        }
      }
      double c = 0.0;
      for (int h = 0; h < l.L; ++h)
        c += exp2((double)h / l.L) * ldexp((double)acc[h], lambda);
      if (out_of_range) { c = NAN; bad++; }
      C[i * N + j] = c;
      if (S)
        for (int h = 0; h < l.L; ++h) {
          S[((i * N + j) * l.L + h) * 2 + 0] = (int64_t)(uint64_t)((unsigned __int128)acc[h]);
          S[((i * N + j) * l.L + h) * 2 + 1] = (int64_t)(acc[h] >> 64);
        }
      if (lsb) lsb[i * N + j] = lambda;
      if (rflag) rflag[i * N + j] = (uint8_t)out_of_range;
    }
  }
  return bad;
}

/* Histogram layout (Eq. 5, App. A.1: products with the same address may be
 * merged into one signed count): signed counts n_{h,t} for ONE output, t in
 * [tlo, tlo + nt).  Used by the tests to check that both accumulation
 * layouts give the same phase sums.  Returns -1 if a t falls outside. */
int oracle_histogram(int ida, int idb, int G, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                     const int8_t* sb, int64_t K, int tlo, int nt, int64_t* counts /* L*nt */) {
  ofmt fa, fb;
  if (ofmt_get(ida, &fa) || ofmt_get(idb, &fb)) return -1;
  olattice l = olattice_of(&fa, &fb);
  if (!l.ok) return -1;
  memset(counts, 0, sizeof(int64_t) * (size_t)l.L * (size_t)nt);
  for (int64_t d = 0; d < K; ++d) {
    int delta, h, t;
    int nz = oracle_closed_product(ida, idb, a[d], b[d], &delta, &h, &t);
    if (nz <= 0) continue;
    t += sa[d / G] + sb[d / G];
    if (t < tlo || t >= tlo + nt) return -1;
    counts[h * nt + (t - tlo)] += delta;
  }
  return 0;
}

/* Euclidean norms of the dequantized rows (fp64), for the normalised
 * error bound |C_gpu - C| <= tol * ||a_i|| * ||b_j||. */
int oracle_row_norms(int id, int G, const uint8_t* codes, const int8_t* scales, int64_t R, int64_t Cc,
                     double* out) {
  ofmt f;
  if (ofmt_get(id, &f)) return -1;
  int64_t nb = Cc / G;
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < R; ++r) {
    double s2 = 0.0;
    for (int64_t c = 0; c < Cc; ++c) {
      int s, n;
      if (odecode(&f, codes[r * Cc + c], &s, &n)) {
        double v = ldexp(olevel(&f, n), scales[r * nb + c / G]);
        s2 += v * v;
      }
    }
    out[r] = sqrt(s2);
  }
  return 0;
}

int oracle_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
