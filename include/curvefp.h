/*
 * curvefp.h — C ABI of the CurveFP GB300 library (libcurvefp.so).
 *
 * CurveFP ("CurveFP: Co-Designing Numerical Representation and Product
 * Arithmetic for Language Models") stores each element of a block of G values
 * as a sign, an exponent and a curve index under one power-of-two block scale
 * (Sec. 3.1, Eq. 1), multiplies codes exactly by adding curve indices with a
 * carry into the exponent (Sec. 3.2, Eq. 2), accumulates products per phase
 * of the radix's phase schedule (Eq. 4, Eq. 5, App. A.1) and combines the
 * phases with fixed constants 2^{h/H}.  Binary radix (r = 2) throughout, and
 * the two rational-radix E4C3 variants of the radix frontier (see
 * curvefp_format_t).
 *
 * Conventions for every entry point
 *   - All tensor pointers are DEVICE pointers to caller-owned memory.  The
 *     library allocates no device memory, never synchronizes, and enqueues its
 *     kernels on `stream` (a cudaStream_t; NULL = the legacy default stream).
 *   - Host-checkable errors (NULL pointers, unknown enums, bad sizes or
 *     alignment) are returned synchronously and nothing is enqueued.
 *     CURVEFP_ERR_CUDA means a launch failed.
 *   - Data-dependent conditions are OR-ed into `device_status` (a device
 *     uint32_t the caller zeroes; may be NULL): CURVEFP_DEV_NAN,
 *     CURVEFP_DEV_RANGE, CURVEFP_DEV_TIMEOUT.  Read it after the stream has
 *     synchronized.
 *   - Row-major layouts; sizes in elements.
 *
 * Code byte (App. C.1 packing; reading of Sec. 3.1):
 *   code = (s << 7) | m,  m = n + B,  n = e*K + k,  B = 2^{E+C-1},
 *   K = 2^C, e in [-2^{E-1}, 2^{E-1}-1], k in [0, K-1], n in [-(B-1), B-1].
 *   m = 0 is the zero sentinel (the smallest combination e = -2^{E-1}, k = 0
 *   is omitted); zero is written as 0x00.  Decoders read m = code & 0x7F
 *   (E4C3, E5C2) or code & 0x3F (E3C3, whose bit 6 is always 0 in a byte
 *   container).  Value: x = (-1)^s 2^{a_b} 2^{n/K}.
 * Block scale a_b (int8, "ceil-absmax", Sec. 3.1 and App. A.2): the smallest
 *   integer in [-128, 127] with max|x| <= 2^{a_b} 2^{(B-1)/K} over the block
 *   (NaN excluded); 0 for an all-zero block; 127 if no integer qualifies (Inf).
 */
#ifndef CURVEFP_H
#define CURVEFP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* E3C3 (CurveFP7, 7 bits, 63 positive levels, H = 8), E4C3 and E5C2
 * (CurveFP8, 8 bits, 127 positive levels, H = 8 and 4): Table 1, binary radix.
 * E4C3_R8_9, E4C3_R3_4: E4C3 codes with the rational radices r = 2^{8/9}
 * (9 phases) and r = 2^{3/4} (32 phases) of the radix frontier (Sec. 3.1
 * Eq. 1 with r = 2^{p/q}, Eq. 4, Table 2): level x = (-1)^s 2^{a_b}
 * 2^{p n/(8q)}; block scale = the smallest a_b with max|x| <= 2^{a_b}
 * 2^{63 p/(8q)}; an exact tie in the nearest-level search (only between zero
 * and L_nmin = 2^{-7} for r = 2^{8/9}) goes to zero; dequantization is
 * RN32(RN32(2^{j/(8q)}) 2^{a_b + floor(p n/(8q))}), j = p n mod 8q.  They are
 * accepted by curvefp_quantize, curvefp_quantize_static (and its variants),
 * curvefp_dequantize, curvefp_gemm_requant's destination, the EXACT GEMMs
 * (curvefp_gemm, curvefp_gemm_phases, curvefp_gemm_phases_histogram; both
 * operands of the same format), for r = 2^{8/9} curvefp_gemm TENSOR (nine
 * planes per operand, 81 plane pairs, three passes of three phases) and for
 * r = 2^{3/4} curvefp_gemm TENSOR_NARROW (32 planes per operand, 16 pair
 * planes, the 32 phases along the MMA's N dimension), AUTO picking those;
 * the other algorithms, curvefp_gemm_q32 and curvefp_gemm_oriented return
 * CURVEFP_ERR_UNSUPPORTED for them. */
typedef enum {
  CURVEFP_E3C3 = 0,
  CURVEFP_E4C3 = 1,
  CURVEFP_E5C2 = 2,
  CURVEFP_E4C3_R8_9 = 3,
  CURVEFP_E4C3_R3_4 = 4
} curvefp_format_t;

typedef enum { CURVEFP_F32 = 0, CURVEFP_BF16 = 1 } curvefp_dtype_t;

typedef enum {
  CURVEFP_OK = 0,
  CURVEFP_ERR_INVALID_ARG = 1,
  CURVEFP_ERR_UNSUPPORTED = 2,
  CURVEFP_ERR_CUDA = 3
} curvefp_status_t;

/* GEMM kernels.  EXACT: integer-ALU kernel whose per-phase sums are exact
 * integers (bit-identical to the definition).  TENSOR: tcgen05 tensor-core
 * kernel over power-of-two phase planes with FP32 per-phase accumulation, one
 * plane pair per dense MMA of a 128-row tile.  SKINNY: decode-sized GEMMs
 * (M <= CURVEFP_SKINNY_MAX_M) on the CUDA cores with the same FP32 per-phase
 * accumulation, every product formed from the two codes.  TENSOR_NARROW: the
 * tensor-core method with the weight rows as the 128-row operand and the L
 * phases of every token (row) along the MMA's N dimension (Sec. 3.2, Eq. 2,
 * Eq. 5): a step of 32 codes takes K_w/2 2:4-sparse MMAs of 128 x (L Mt)
 * (weight curve planes j and j + K_w/2 share one compressed operand; Mt <=
 * 256/L tokens per CTA), against K_a K_b dense MMAs of a 128-row tile; the
 * fastest tensor-core kernel at every M.  For r = 2^{3/4} (32 phases) the
 * same layout with Mt = 8 tokens: 16 sparse MMAs of 128 x 256 x 64 per step,
 * one weight stage in TMEM (the 256-column accumulator leaves room for no
 * second).  In both tensor-core kernels the
 * block scales enter the MMAs as UE8M0 scale factors (block-scaled MMAs), so
 * the plane values are the codes' own powers of two.
 * AUTO (measured on the FFN shapes, N = 14336, K = 4096, the
 * 2048 x 4096 x 4096 linear and the training triplet's three GEMMs): SKINNY
 * for M <= CURVEFP_AUTO_SKINNY_M; TENSOR_NARROW for every pair it supports;
 * TENSOR for r = 2^{8/9} and TENSOR_NARROW for r = 2^{3/4} at every M;
 * SKINNY up to CURVEFP_SKINNY_MAX_M for pairs without a tensor-core kernel.
 * (Value 2 is not an algorithm.) */
typedef enum {
  CURVEFP_GEMM_EXACT = 0,
  CURVEFP_GEMM_TENSOR = 1,
  CURVEFP_GEMM_SKINNY = 3,
  CURVEFP_GEMM_AUTO = 4,
  CURVEFP_GEMM_TENSOR_NARROW = 5
} curvefp_gemm_algo_t;
#define CURVEFP_SKINNY_MAX_M 8
#define CURVEFP_AUTO_SKINNY_M 1

/* Bits of the device status word. */
#define CURVEFP_DEV_NAN 1u     /* quantize: a NaN input was encoded as 0x00        */
#define CURVEFP_DEV_RANGE 2u   /* gemm: an output's scale spread exceeds the exact
                                  int128 window (see curvefp_gemm_phases)          */
#define CURVEFP_DEV_TIMEOUT 4u /* gemm: a pipeline wait gave up (internal error)   */

/* Block-scaled quantization Q(X) (Sec. 3.1; ceil-absmax scale, nearest level in
 * absolute error over {0} U {2^{n/K}}, saturation at 2^{(B-1)/K}).
 *   x        : [rows x cols] FP32 or BF16 with leading dimension ld >= cols
 *              (elements), aligned to its element size; for block_axis 0 also
 *              16-byte aligned with ld * element size a multiple of 16.
 *   block    : G in {32, 64, 128, 256, 512}.
 *   block_axis 0: blocks of G consecutive elements of a row (cols % G == 0);
 *              codes [rows x cols] dense, scales [rows x cols/G].
 *   block_axis 1: blocks of G consecutive rows of a column (rows % G == 0);
 *              the output is the transposed operand, blocked axis contiguous:
 *              codes [cols x rows] dense, scales [cols x rows/G].
 *   codes    : 16-byte aligned.
 * NaN inputs encode as 0x00 and raise CURVEFP_DEV_NAN. */
curvefp_status_t curvefp_quantize(curvefp_format_t fmt, int block, const void* x, curvefp_dtype_t dtype,
                                  int64_t rows, int64_t cols, int64_t ld, int block_axis, uint8_t* codes,
                                  int8_t* scales, uint32_t* device_status, void* stream);

/* Static operands (Sec. 3.1: the scale of a weight, fixed ahead of time, is
 * picked among representable powers of two by the reconstruction error it
 * gives; Sec. 4.2 compares scales per tensor, per row and per block).  A
 * scale group is a block of `block` elements of a row, a whole row, or the
 * whole tensor. */
typedef enum { CURVEFP_SCALE_BLOCK = 0, CURVEFP_SCALE_ROW = 1, CURVEFP_SCALE_TENSOR = 2 } curvefp_scale_group_t;
/* CEIL_ABSMAX: the group's ceil-absmax scale a_c (as curvefp_quantize).
 * MSE: the candidate a in [a_c - 3, a_c + 1] (clamped to int8) with the
 *   smallest D(a) = sum_i floor((x_i - xhat_i)^2 * 2^{60 - 2 a_c}), xhat_i the
 *   FP32 reconstruction (as curvefp_dequantize) of x_i encoded at scale a;
 *   D is an exact integer, so the choice is independent of summation order;
 *   ties go to the larger a.  NaN elements are left out of D; groups with an
 *   Inf element or an all-zero max keep a_c. */
typedef enum { CURVEFP_SCALE_CEIL_ABSMAX = 0, CURVEFP_SCALE_MSE = 1 } curvefp_scale_rule_t;

/* Bytes of device workspace curvefp_quantize_static needs (0 for block
 * groups; a few bytes per group for rows and the tensor); 0 for bad arguments. */
size_t curvefp_quantize_static_workspace(int64_t rows, int64_t cols, int block, curvefp_scale_group_t group);

/* Quantize a static operand with one scale per group.
 *   x      : [rows x cols] FP32 or BF16, dense (ld = cols), aligned to its element.
 *   codes  : [rows x cols]; scales: [rows x cols/block], every block of a group
 *            holding the group's scale (the layout every GEMM call takes).
 *   workspace : device memory of at least curvefp_quantize_static_workspace()
 *            bytes, 16-byte aligned, owned by the caller (contents clobbered);
 *            may be NULL when that size is 0.
 * Requirements: cols % block == 0.  NaN inputs encode as 0x00 and raise
 * CURVEFP_DEV_NAN.  The library allocates nothing. */
curvefp_status_t curvefp_quantize_static(curvefp_format_t fmt, int block, curvefp_scale_group_t group,
                                         curvefp_scale_rule_t rule, const void* x, curvefp_dtype_t dtype, int64_t rows,
                                         int64_t cols, uint8_t* codes, int8_t* scales, void* workspace,
                                         size_t workspace_bytes, uint32_t* device_status, void* stream);

/* curvefp_quantize_static without a workspace argument, for callers that
 * cannot allocate device memory: code running where cudaMalloc is not
 * allowed or would stall other work (it can synchronize the device), code
 * whose device memory is owned by a host framework's own pool, and hosts
 * with a fixed memory budget that reserve everything up front.  The paper
 * has no counterpart; this is an interface variant of the static quantizer.
 *   The scratch lives in a fixed file-scope device array of the library,
 *   CURVEFP_NOALLOC_SCRATCH_BYTES (8 MiB) on every GPU that loads the library,
 *   held until the process exits.  That is enough for row groups of up to
 *   about 98,000 rows; tensor and block groups need almost none.  The call makes
 *   no cudaMalloc, cudaFree or other allocating call.
 *   Returns CURVEFP_ERR_UNSUPPORTED, before any device work, when the groups
 *   need more scratch than the array holds.
 *   The array is shared by every call on a device and keeps the last call's
 *   contents; each call clears the part it uses before its kernels.  Calls
 *   that overlap on the GPU (different streams without ordering) race on it.
 *   Every call looks the array's device address up on the current device
 *   (cudaGetSymbolAddress; nothing is cached, so a device reset between
 *   calls is harmless); the first call on a device also loads the library's
 *   module there, so make that first call before any stream capture.  Other
 *   arguments, results and errors as curvefp_quantize_static. */
#define CURVEFP_NOALLOC_SCRATCH_BYTES (8u << 20)
curvefp_status_t curvefp_quantize_static_noalloc(curvefp_format_t fmt, int block, curvefp_scale_group_t group,
                                                 curvefp_scale_rule_t rule, const void* x, curvefp_dtype_t dtype,
                                                 int64_t rows, int64_t cols, uint8_t* codes, int8_t* scales,
                                                 uint32_t* device_status, void* stream);

/* Dequantization to FP32 (Eq. 1): out = RN32( RN32(2^{k/K}) * 2^{a_b + e} ) with
 * the sign applied; zero codes give +0.0.
 *   codes [rows x cols] (16-byte aligned, cols % block == 0), scales
 *   [rows x cols/block], out [rows x cols] FP32 (16-byte aligned). */
curvefp_status_t curvefp_dequantize(curvefp_format_t fmt, int block, const uint8_t* codes, const int8_t* scales,
                                    int64_t rows, int64_t cols, float* out, void* stream);

/* Closed-product GEMM C = A_hat * B_hat^T (Sec. 3.2, Eq. 2, Eq. 5, App. A.1;
 * the forward/backward operators of Sec. 3.3 and App. A.2 are all of this form
 * once each operand is quantized along its own reduction axis).
 *   a  : [M x K] codes of format fmt_a, K contiguous; sa: [M x K/block].
 *   b  : [N x K] codes of format fmt_b, K contiguous; sb: [N x K/block].
 *   c  : [M x N] FP32 output, row-major.
 * Every nonzero product a (x) b has sign s_a xor s_b, scale a_a + a_b and
 * lattice exponent u = n_a L/K_a + n_b L/K_b with L = max(K_a, K_b); it lands on
 * phase h = u mod L with weight 2^{floor(u/L)}.  Per-phase sums S_h are combined
 * as C = sum_h 2^{h/L} S_h in the epilogue.
 * Requirements: K % block == 0; a, b 16-byte aligned.
 * EXACT: S_h exact, combine in FP64, one FP32 rounding; outputs whose scale
 *   spread leaves the int128 window raise CURVEFP_DEV_RANGE (values undefined).
 * TENSOR, TENSOR_NARROW: S_h accumulated in FP32 on the tensor cores, combine
 *   in FP32.  Every product is exact before the FP32 accumulation: a plane
 *   value is the code's power of two 2^e and the block scale is the MMA's
 *   scale factor 2^{a_b - ref + 32} (ref = the row's largest block scale),
 *   so the spread of the block scales along a row costs nothing.  Lost are
 *   only (1) products below FP32's normal range, i.e. below 2^{-190} of
 *   2^{ref_a + ref_b}; (2) blocks more than 159 binades below their row's
 *   largest block scale; (3) TENSOR_NARROW with E5C2 x E5C2: the tokens'
 *   elements of the lowest binade (e = -16) in the products without carry
 *   (an element at least 2^30 below its block's top binade).  Within 1e-5 of
 *   ||a_i|| ||b_j|| whenever, per row, the largest element lies within about
 *   75 binades of the row's largest block scale on both operands (the
 *   quantizer writes 0 as the scale of an all-zero block, so this holds
 *   unless both operands' data lie below about 2^-75).  Format pairs: E3C3 x
 *   E3C3, E4C3 x E4C3, E5C2 x E4C3, E4C3 x E5C2, E5C2 x E5C2, (TENSOR)
 *   E4C3_R8_9 x E4C3_R8_9 and (TENSOR_NARROW) E4C3_R3_4 x E4C3_R3_4 (others
 *   return CURVEFP_ERR_UNSUPPORTED).  TENSOR and
 *   TENSOR_NARROW zero parts of C with cudaMemsetAsync before adding split-K
 *   pieces to them (two additions per output, so results do not depend on
 *   their order).
 * SKINNY (M <= CURVEFP_SKINNY_MAX_M, else CURVEFP_ERR_UNSUPPORTED), AUTO:
 *   S_h accumulated in FP32 per output (products relative to the output's
 *   largest scale sum; products below the FP32 normal range relative to it
 *   flush), combine in FP32; every binary-radix format pair. */
curvefp_status_t curvefp_gemm(curvefp_gemm_algo_t algo, curvefp_format_t fmt_a, curvefp_format_t fmt_b, int block,
                              const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb, int64_t M,
                              int64_t N, int64_t K, float* c, uint32_t* device_status, void* stream);

/* Validation form of the EXACT GEMM that also exports the per-phase integer
 * accumulators (Eq. 5: the signed integer counts of each phase, summed with
 * their bin weights; App. A.1).
 *   phase_sums : M*N*H two's-complement int128 values stored as (lo, hi) int64
 *                pairs, [M][N][H]; S_h at LSB 2^{lsb}.
 *   phase_lsb  : [M x N] int32, lsb = min_b(sa[i,b] + sb[j,b]) + t_min with
 *                t_min = floor(-((B_a-1) L/K_a + (B_b-1) L/K_b) / L).
 *   An output is out of range (CURVEFP_DEV_RANGE, its sums undefined) when
 *   bitlen(K) + spread + (t_max - t_min) > 127, spread = max_b - min_b of
 *   sa[i,b] + sb[j,b].
 *   c may be NULL. */
curvefp_status_t curvefp_gemm_phases(curvefp_format_t fmt_a, curvefp_format_t fmt_b, int block, const uint8_t* a,
                                     const int8_t* sa, const uint8_t* b, const int8_t* sb, int64_t M, int64_t N,
                                     int64_t K, float* c, int64_t* phase_sums, int32_t* phase_lsb,
                                     uint32_t* device_status, void* stream);

/* Operand layouts of curvefp_gemm_oriented (Sec. 4, training GEMMs: the
 * backward pass reuses the forward pass's quantized operands, one of them
 * transposed: dgrad = Q(dY) Q(W), wgrad = Q(dY)^T Q(X)).  For an operand with
 * R GEMM rows (R = M for A, N for B):
 *   ROWS: codes [R x K] (K contiguous), scales [R x K/block]: quantized along
 *         the GEMM's K, as curvefp_gemm takes it.  K % block == 0.
 *   COLS: codes [K x R] (R contiguous), scales [K x R/block]: a matrix
 *         quantized along R (curvefp_quantize with block_axis 0 on a [K x R]
 *         matrix) and used transposed.  Every element keeps its own block
 *         scale, so along a GEMM row the scale changes with k.  R % block == 0. */
typedef enum { CURVEFP_LAYOUT_ROWS = 0, CURVEFP_LAYOUT_COLS = 1 } curvefp_layout_t;

/* Bytes of device workspace curvefp_gemm_oriented needs (0 for EXACT and for
 * ROWS x ROWS); for TENSOR with a COLS operand:
 *   sum over operands of [R K (COLS only)] + R K + R K / 16 + 4 R, each
 *   rounded up to 256. */
size_t curvefp_gemm_oriented_workspace_bytes(curvefp_gemm_algo_t algo, curvefp_layout_t layout_a,
                                             curvefp_layout_t layout_b, int64_t M, int64_t N, int64_t K);

/* C = A_hat B_hat^T with each operand in either layout; every product is the
 * closed product of Eq. 2 with both elements' own scales, accumulated per
 * phase (Eq. 5 with per-element scales: lambda = min_k(a(i,k) + b(j,k)) +
 * t_min, the window check on the spread of the same sums).
 *   EXACT : integer ALUs, phase sums bit-identical to the definition;
 *           phase_sums / phase_lsb as curvefp_gemm_phases (both or neither);
 *           c may be NULL when phase_sums is given.  No workspace.
 *   TENSOR: the tensor-core kernel with per-element scales: per 32-code step
 *           of a row the scale factor follows the step's largest element and
 *           each element's plane value is its power of two relative to it;
 *           an element more than 31 binades below the largest element of
 *           its step (2^-31 of it) is dropped, so the error bound is
 *           2^-31 sqrt(K) ||a_i|| ||b_j|| beyond curvefp_gemm TENSOR's;
 *           phase_sums and phase_lsb must be NULL; K % 32 == 0; workspace
 *           (256-byte aligned, at least curvefp_gemm_oriented_workspace_bytes)
 *           receives the transposed codes of COLS operands, an exponent byte
 *           per element and a scale per step, written by preparation kernels
 *           on the same stream.  ROWS x ROWS is curvefp_gemm (no workspace).
 * Codes pointers 16-byte aligned; M, N, K > 0. */
curvefp_status_t curvefp_gemm_oriented(curvefp_gemm_algo_t algo, curvefp_format_t fmt_a, curvefp_format_t fmt_b,
                                       int block, const uint8_t* a, const int8_t* sa, curvefp_layout_t layout_a,
                                       const uint8_t* b, const int8_t* sb, curvefp_layout_t layout_b, int64_t M,
                                       int64_t N, int64_t K, float* c, int64_t* phase_sums, int32_t* phase_lsb,
                                       void* workspace, size_t workspace_bytes, uint32_t* device_status,
                                       void* stream);

/* curvefp_gemm_phases computed with the histogram layout (Eq. 5, App. A.1:
 * products with equal addresses merge into one signed count): every product's
 * address (phase h, bin t) is counted in a per-output histogram n_{h,t}
 * (lanes of a warp with equal addresses merge by signed popcount), and
 * S_h = sum_t n_{h,t} 2^t.  Same outputs, requirements and format pairs as
 * curvefp_gemm_phases (rational radices included); the phase sums are
 * bit-identical to it.  Validation kernel (one warp per output). */
curvefp_status_t curvefp_gemm_phases_histogram(curvefp_format_t fmt_a, curvefp_format_t fmt_b, int block,
                                               const uint8_t* a, const int8_t* sa, const uint8_t* b, const int8_t* sb,
                                               int64_t M, int64_t N, int64_t K, float* c, int64_t* phase_sums,
                                               int32_t* phase_lsb, uint32_t* device_status, void* stream);

/* GEMM followed by output requantization (Sec. 3.2: closure holds on the
 * widened product coordinates; the explicit requantization to an E-bit
 * destination comes after the phase combine): C = A_hat B_hat^T as
 * curvefp_gemm, then Q(C) as curvefp_quantize with blocks of block_c along N
 * (the layout of the next layer's activation operand).
 *   c        : [M x N] FP32 (16-byte aligned), written; the requantizer reads it
 *              back (one extra HBM round trip of 4 M N bytes).
 *   codes_c  : [M x N] codes of fmt_c; scales_c: [M x N/block_c].
 * Requirements: those of both calls, and N % block_c == 0. */
curvefp_status_t curvefp_gemm_requant(curvefp_gemm_algo_t algo, curvefp_format_t fmt_a, curvefp_format_t fmt_b,
                                      int block, const uint8_t* a, const int8_t* sa, const uint8_t* b,
                                      const int8_t* sb, int64_t M, int64_t N, int64_t K, float* c,
                                      curvefp_format_t fmt_c, int block_c, uint8_t* codes_c, int8_t* scales_c,
                                      uint32_t* device_status, void* stream);

/* The spatial tile's integer semantics as a second bit-exact GEMM (App. C.1,
 * C.2): every nonzero product, with lattice exponent u = L e + k (as in
 * curvefp_gemm), adds (-1)^{s_a xor s_b} round(2^{k/L} 2^16) 2^{16+e+sa+sb} to a
 * signed 64-bit Q32 accumulator (value = acc * 2^-32), with no intermediate
 * rounding; for E4C3 x E4C3 this is the tile's Q16 coefficient select on
 * q_p = m_a + m_b - 128 = 8e + k followed by the shift into Q32.
 *   acc : [M x N] int64, row-major.
 * A product needing a shift below 0 or above 45, or an accumulator outside
 * int64, raises CURVEFP_DEV_RANGE (that output's value is undefined).
 * Operands, layouts and format pairs as curvefp_gemm with algo TENSOR. */
curvefp_status_t curvefp_gemm_q32(curvefp_format_t fmt_a, curvefp_format_t fmt_b, int block, const uint8_t* a,
                                  const int8_t* sa, const uint8_t* b, const int8_t* sb, int64_t M, int64_t N, int64_t K,
                                  int64_t* acc, uint32_t* device_status, void* stream);

/* Number of phases H of a format pair (Eq. 4 with binary radix, on the shared
 * lattice L = max(K_a, K_b)); -1 for an unknown format. */
int curvefp_phase_count(curvefp_format_t fmt_a, curvefp_format_t fmt_b);

/* Failure-detection self-test (an interface of this library, not from the
 * paper; no CurveFP arithmetic).  One warp waits on a fresh mbarrier of count
 * 1 with the bounded wait that every pipeline hand-off of the TENSOR GEMM
 * uses, limited here to limit_cycles SM clock cycles (1 .. 2^31; the GEMM's
 * own limit is 2^31, about a second).  arrive != 0: lane 0 completes the
 * barrier's phase first, the wait succeeds and *device_status is unchanged.
 * arrive == 0: nothing completes it; the wait gives up after the limit, ORs
 * CURVEFP_DEV_TIMEOUT into *device_status and the kernel returns normally
 * (no trap), so the context stays usable.
 *   device_status : device uint32_t, required.
 * Errors: CURVEFP_ERR_INVALID_ARG for a NULL status or a limit out of range
 * (nothing enqueued). */
curvefp_status_t curvefp_selftest_bounded_wait(int arrive, int64_t limit_cycles, uint32_t* device_status,
                                               void* stream);

/* Static description of a status code. */
const char* curvefp_status_string(curvefp_status_t status);

/* Library version string. */
const char* curvefp_version(void);

#ifdef __cplusplus
}
#endif

#endif /* CURVEFP_H */
