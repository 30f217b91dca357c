/*
 * sss_oracle.h -- the plain CPU oracle for group-wise few-bit weight
 * quantization with signed symmetric, unsigned symmetric and min-max
 * asymmetric grids (Colbert, Dash et al., "Signed Symmetric Quantization
 * for Few-Bit Integers").
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * CPU-baseline leg of the benchmark may load this library.  The product
 * path (the CUDA library) shares no code, header, table or constant with
 * it.  This header is the oracle's own and is included by nothing else.
 *
 * Everything here follows the paper's definitions in plain, single-threaded
 * C.  Floating point: fp32 where the method defines an fp32 quantity (the
 * scale, the dequantised weight), fp64 for the exact RNE quotient and the
 * matmul reference.  Build with -O2 -ffp-contract=off and no fast-math.
 */
#ifndef SSS_ORACLE_H
#define SSS_ORACLE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* grid selectors (same numeric values as the product ABI so the tests can
 * pass one integer to both; the values are restated here, not shared) */
#define ORC_GRID_UNSIGNED_SYM 0 /* absmax, s > 0 (eq:absmax)                 */
#define ORC_GRID_SIGNED_SYM 1   /* signed absmax, s = gamma* alpha (eq:sign_rule) */
#define ORC_GRID_ASYM 2         /* min-max, unsigned alphabet (eq:minmax)    */

/* status bits (OR-ed) */
#define ORC_FLAG_NONFINITE 1 /* a weight of the group is NaN or +-Inf       */
#define ORC_FLAG_RANGE 2     /* the stored fp16 scale/min is infinite, or the
                                fp32 asymmetric step overflowed             */

/* IEEE 754 binary16, round to nearest even, written from the format's
 * definition (sign, 5-bit biased exponent, 10-bit fraction, subnormals). */
uint16_t orc_f32_to_f16(float x);
float orc_f16_to_f32(uint16_t h);
/* bfloat16 -> fp32 (the upper 16 bits of an fp32) */
float orc_bf16_to_f32(uint16_t b);

/* Per-group result of the quantizer, all fields filled by
 * orc_quantize_group / orc_quantize_group_gamma. */
typedef struct {
  float s32;        /* the fp32 scale s used for rounding (eq:quantizer)      */
  float alpha;      /* |s| for symmetric grids (alpha = M / 2^(q-1))          */
  float mx, mn;     /* max_j w_j, min_j w_j                                   */
  float M;          /* ||w||_inf                                             */
  int32_t gamma;    /* +1/-1 for symmetric grids, 0 for ASYM                  */
  uint16_t s16;     /* stored fp16 scale                                      */
  uint16_t m16;     /* stored fp16 minimum (ASYM), else 0                     */
  int32_t n_self;   /* |C_gamma|  = #{c_pre == +2^(q-1)} (def:clipped-set)    */
  int32_t n_other;  /* |C_-gamma| = #{c_pre == -2^(q-1)}                      */
  int32_t flags;    /* ORC_FLAG_*                                             */
} orc_group_t;

/* Quantize one group w[0..g-1] with the given grid.  Writes the pre-clip
 * integer c_pre (nullable), the clipped integer c on the grid's alphabet
 * (signed alphabet for SYM, {0..2^q-1} for ASYM) and the stored offset
 * code u (u = c + 2^(q-1) for SYM, u = c for ASYM). Returns flags. */
int32_t orc_quantize_group(const float* w, int32_t g, int32_t q, int32_t grid,
                           int32_t* c_pre, int32_t* c, uint8_t* u,
                           orc_group_t* info);

/* Symmetric quantizer Q(w; gamma*alpha, 0) with alpha = M/2^(q-1) and a
 * caller-chosen sign gamma (eq:signed_sym_quant).  Used for brute force over
 * both scale signs.  Same outputs as orc_quantize_group. */
int32_t orc_quantize_group_gamma(const float* w, int32_t g, int32_t q,
                                 int32_t gamma, int32_t* c_pre, int32_t* c,
                                 uint8_t* u, orc_group_t* info);

/* Pack the stored codes u[0..g-1] of one group into the canonical byte
 * layout (g*q/8 bytes):
 *   q=4: element j in byte j>>1, low nibble for even j, high for odd j;
 *   q=2: element j in byte j>>2 at bit 2*(j&3);
 *   q=3: a low plane of g/4 bytes holding (u & 3) in the q=2 layout, then a
 *        high plane of g/8 bytes with bit (j&7) of byte (j>>3) = u>>2.      */
void orc_pack_group(const uint8_t* u, int32_t g, int32_t q, uint8_t* out);
void orc_unpack_group(const uint8_t* in, int32_t g, int32_t q, uint8_t* u);

/* Whole matrix W[n][k] (row-major fp32), groups of g along k.
 * codes: n*k*q/8 bytes; scales, mins: n*(k/g) fp16 (mins may be NULL unless
 * ASYM); clip_counts: nullable, n*(k/g)*2 bytes {n_self, n_other}.
 * Returns the OR of all group flags. */
int32_t orc_quantize(const float* W, int64_t n, int64_t k, int32_t q,
                     int32_t g, int32_t grid, uint8_t* codes, uint16_t* scales,
                     uint16_t* mins, uint8_t* clip_counts);

/* Dequantised weight: SYM w^ = f16(s)*c (exact in fp32);
 * ASYM w^ = fl32(fl32(f16(s)*u) + f16(m)).  out: fp32 [n][k]. */
void orc_dequantize(const uint8_t* codes, const uint16_t* scales,
                    const uint16_t* mins, int64_t n, int64_t k, int32_t q,
                    int32_t g, int32_t grid, float* out);

/* Dequantise rows [r0, r0+nr) only (for sampled checks at full size). */
void orc_dequantize_rows(const uint8_t* codes, const uint16_t* scales,
                         const uint16_t* mins, int64_t n, int64_t k, int32_t q,
                         int32_t g, int32_t grid, int64_t r0, int64_t nr,
                         float* out);

/* fp64 matmul reference y[b][j] = sum_k (double)What[j][k]*(double)x[b][k],
 * x given as bf16 bits [nb][k], What fp32 [n][k], y fp64 [nb][n]. */
void orc_matmul_f64(const float* What, const uint16_t* x_bf16, int64_t nb,
                    int64_t n, int64_t k, double* y);

/* The packed-weight decode GEMV of the oracle: dequantise each row of the
 * packed tensor and dot it with x in fp64 (the two steps above, one row at a
 * time).  y fp64 [nb][n]. */
void orc_gemv(const uint8_t* codes, const uint16_t* scales,
              const uint16_t* mins, int64_t n, int64_t k, int32_t q, int32_t g,
              int32_t grid, const uint16_t* x_bf16, int64_t nb, double* y);

/* Dynamic Q8_0 activation quantization, the narrow-range 8-bit quantizer
 * the paper pairs with the few-bit weight formats at inference (Sec. 5,
 * "Composition with PTQ methods"; Appendix C, "Algorithm details"): the
 * alphabet {-K..K}, K = 2^(8-1) - 1 = 127, one scale per block of 32
 * consecutive activations of a token (the GGUF block).  Per block:
 *   M = max_i |x_i|;  d = fl32(M / 127);
 *   q_i = clip(RNE(x_i / d), -127, 127) of the exact quotient;
 *   stored scale d16 = fp16(d).  An all-zero block gives d = 0, q = 0.
 * x given as bf16 bits [nb][k], k % 32 == 0; q int8 [nb][k]; d16
 * [nb][k/32].  Returns ORC_FLAG_NONFINITE if an activation is NaN/Inf
 * (that block's outputs are q = 0, d16 = +0) and ORC_FLAG_RANGE if a
 * stored d16 is infinite. */
int32_t orc_quantize_act_q8(const uint16_t* x_bf16, int64_t nb, int64_t k,
                            int8_t* q, uint16_t* d16);

/* The decode GEMV with Q8_0 activations: y[b][j] = sum_k w^[j][k] * x^[b][k]
 * in fp64, where w^ is the dequantised weight (orc_dequantize) and
 * x^ = f16(d) * q the dequantised activation.  y fp64 [nb][n]. */
void orc_gemv_q8(const uint8_t* codes, const uint16_t* scales,
                 const uint16_t* mins, int64_t n, int64_t k, int32_t q,
                 int32_t g, int32_t grid, const int8_t* xq,
                 const uint16_t* xd16, int64_t nb, double* y);

/* ---------------------------------------------------------------------- */
/* Normalized Hadamard rotation of the weights before quantization (Sec. 5  */
/* "Composition with PTQ methods"; Appendix C: rotations merged into the    */
/* weights, grids computed on the rotated weights).                         */
/* ---------------------------------------------------------------------- */

/* The normalized Walsh-Hadamard transform of x[0..b) (b a power of two,
 * Sylvester order H_2m = [[H_m, H_m], [H_m, -H_m]]), in the arithmetic this
 * build takes for it (reading: the paper names the rotation, not its
 * arithmetic): the in-place fast transform in IEEE fp32 with strides
 * h = 1, 2, ..., b/2, each butterfly (a, c) -> (a + c, a - c), then every
 * element times the fp32 nearest to 1/sqrt(b). */
void orc_fwht_f32(float* x, int32_t b);

/* W [n][k] rotated on its input side, W <- W (I (x) H_b/sqrt(b)): every
 * block of b consecutive elements of a row transformed as above
 * (b | k).  out may equal W. */
void orc_rotate_rows(const float* W, int64_t n, int64_t k, int32_t b, float* out);

/* W [n][k] rotated on its output side, W <- (I (x) H_b/sqrt(b)) W: every
 * block of b consecutive rows transformed column by column (b | n). */
void orc_rotate_cols(const float* W, int64_t n, int64_t k, int32_t b, float* out);

/* ---------------------------------------------------------------------- */
/* Signed LSQ scale refinement (Sec. 5 "Composition with learned rotations  */
/* and grid parameters"; Appendix C: LSQ with s != 0 for the signed         */
/* formats, s > 0 for the conventional ones).  The paper learns the scales  */
/* on calibration data through the model loss; this is the data-free        */
/* reading on each group's own reconstruction loss (see orc_lsq_scale).     */
/* ---------------------------------------------------------------------- */

/* The refined scale of one group w[0..g-1] (g a power of two, 32..128):
 * s_0 = the signed absmax scale gamma* alpha (signed_grid != 0) or the
 * absmax scale alpha; then `steps` LSQ steps on L(s) = sum (s c_i - w_i)^2,
 * all in IEEE fp32 without fused multiply-add:
 *   v_i = w_i / s, c_i = clip(rint(v_i), -2^(q-1), 2^(q-1) - 1),
 *   d_i = dw^_i/ds, LSQ's straight-through estimate: c_i - v_i when v_i
 *         lies strictly inside (-2^(q-1), 2^(q-1) - 1), else the clip value,
 *   e_i = s c_i - w_i,   t_i = (2 e_i) d_i,
 *   G = sum t_i in the pairwise order: t_i <- t_i + t_{i+h} for
 *       h = g/2, g/4, ..., 1, G = t_0,
 *   s' = s - (lr * (1/sqrt(g (2^(q-1) - 1)))) * G  (LSQ's gradient scale),
 *   and s' keeps the sign of s: if s' s <= 0 then s' = s / 2.
 * An all-zero (or underflowed) or non-finite group keeps s = 0.  */
float orc_lsq_scale(const float* w, int32_t g, int32_t q, int32_t signed_grid,
                    int32_t steps, float lr);

/* Quantize W [n][k] on the symmetric grid with every group's scale refined
 * by orc_lsq_scale: codes c = clip(RNE(w/s)) of the exact quotient with the
 * refined fp32 scale s, packed as orc_quantize packs them, fp16 scales.
 * grid: ORC_GRID_SIGNED_SYM or ORC_GRID_UNSIGNED_SYM.  Returns OR-ed flags. */
int32_t orc_lsq_quantize(const float* W, int64_t n, int64_t k, int32_t q,
                         int32_t g, int32_t grid, int32_t steps, float lr,
                         uint8_t* codes, uint16_t* scales);

#ifdef __cplusplus
}
#endif
#endif
