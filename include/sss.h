/*
 * sss.h -- C ABI of the GB300 (sm_103a) signed-symmetric few-bit weight
 * library: group-wise q-bit weight quantization with a signed per-group scale
 * and no zero point, and the decode GEMV / prefill GEMM that consume the
 * packed codes with dequantisation fused in.
 *
 * Source of the operations: Colbert, Dash et al., "Signed Symmetric
 * Quantization for Few-Bit Integers": the integer quantizer (eq:quantizer,
 * Sec. 1), the min-max grid (eq:minmax) and absmax grid (eq:absmax) of
 * Sec. 3, the signed symmetric family (eq:signed_sym_quant) and the signed
 * absmax sign rule (eq:sign_rule), the direct-casting protocol (Appendix C.1)
 * and the deployed block formats and quantized GEMM expansion (Appendix B).
 *
 * Conventions for every entry point:
 *  - All tensor pointers are DEVICE pointers owned by the caller.  No entry
 *    point allocates device memory; the library keeps only small host-side
 *    per-device records (SM count, raised shared-memory limits of kernels).
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Every call is asynchronous on that stream; none synchronises.
 *  - The return value reports synchronous argument checks and launch errors.
 *    Data-dependent conditions (NaN/Inf weights, a scale that overflows
 *    fp16, a wait that timed out) are OR-ed as SSS_FLAG_* bits into the
 *    optional device word `dev_status` (uint32), which the caller zeroes and
 *    reads back after synchronising.
 *  - No C++ exception crosses the ABI.  Functions are thread-safe.
 *
 * Weight layout: W is row-major fp32 [n][k] (n = output features, k = input
 * features, the quantized axis); groups are `group` consecutive elements
 * along k, so group G = row*(k/group) + j starts at element G*group.
 * Packed codes are stored per group, groups back to back (codes of group G
 * start at byte G*group*q/8):
 *   q=4: element j in byte j>>1, low nibble for even j, high for odd j;
 *   q=2: element j in byte j>>2 at bits 2*(j&3);
 *   q=3: a plane of group/4 bytes holding (u & 3) in the q=2 layout, then a
 *        plane of group/8 bytes with bit (j&7) of byte (j>>3) = (u >> 2).
 * The stored code is u = c + 2^(q-1) for the symmetric grids (c in the signed
 * alphabet {-2^(q-1) .. 2^(q-1)-1}) and u = c in {0 .. 2^q-1} for ASYM.
 * scales: IEEE fp16 [n][k/group], the signed scale s = gamma*alpha for the
 * symmetric grids (Appendix B.1 lets the stored scale be negative), the step
 * for ASYM.
 * mins: fp16 [n][k/group], ASYM only (the stored minimum m; w^ = s*u + m).
 */
#ifndef SSS_H
#define SSS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SSS_GRID_UNSIGNED_SYM = 0, /* absmax grid, s = ||w||_inf / 2^(q-1) > 0 (eq:absmax)      */
  SSS_GRID_SIGNED_SYM = 1,   /* signed absmax, s = gamma* alpha (eq:signed_sym_quant,
                                eq:sign_rule); gamma = +1 when max w == -min w            */
  SSS_GRID_ASYM = 2          /* min-max grid on {0..2^q-1} (eq:minmax)                  */
} sss_grid_t;

typedef enum {
  SSS_OK = 0,
  SSS_E_ARG = 1,         /* a size or enum argument is out of range / NULL         */
  SSS_E_UNSUPPORTED = 2, /* a combination this build does not implement            */
  SSS_E_ALIGN = 3,       /* a pointer is not aligned as documented                 */
  SSS_E_CUDA = 4,        /* a CUDA runtime/driver call or launch failed            */
  SSS_E_WORKSPACE = 5    /* workspace too small (see sss_workspace_bytes)          */
} sss_status_t;

/* bits OR-ed into *dev_status by the kernels */
#define SSS_FLAG_NONFINITE 0x1u /* a weight group contains NaN or +-Inf; that group's
                                   codes/scale are placeholders (u = 2^(q-1) and s = +0
                                   for symmetric grids, u = 0 and s = +0 for ASYM)     */
#define SSS_FLAG_RANGE 0x2u     /* sss_quantize: a stored fp16 scale or min is infinite
                                   (|s| >= 65520), or the fp32 ASYM step overflowed
                                   (codes then 0).  sss_gemv at batch 2..16 and
                                   sss_gemm: a group's fp16 weight operand may overflow
                                   (see those calls); their outputs may then hold
                                   inf or NaN                                         */
#define SSS_FLAG_TIMEOUT 0x4u   /* a bounded pipeline wait of sss_gemm (or
                                   sss_gemm_noalloc) expired; the output is
                                   incomplete                                         */

typedef enum { SSS_OUT_F32 = 0, SSS_OUT_F16 = 1, SSS_OUT_BF16 = 2 } sss_dtype_t;

/* A packed weight tensor.  Plain descriptor; the library never frees it. */
typedef struct {
  int64_t n;         /* rows (output features), 0 .. 2^31                           */
  int64_t k;         /* columns (input features), 0 .. 2^31, multiple of `group`  */
  int32_t q;         /* bits per code: 2, 3 or 4                                   */
  int32_t group;     /* group size along k: 32, 64 or 128                          */
  int32_t grid;      /* sss_grid_t                                                 */
  int32_t reserved;  /* must be 0                                                  */
  uint8_t* codes;    /* [n][k*q/8] bytes, layout above                             */
  uint16_t* scales;  /* [n][k/group] fp16                                          */
  uint16_t* mins;    /* [n][k/group] fp16 for SSS_GRID_ASYM, else ignored (NULL)   */
} sss_qtensor_t;

/* Bytes of packed codes for an [n][k] tensor at q bits: n*k*q/8. */
size_t sss_codes_bytes(int64_t n, int64_t k, int32_t q);

/* Human-readable name of a status code (static storage). */
const char* sss_status_string(sss_status_t status);

/* Text of the last CUDA error seen by this thread inside the library
 * (static thread-local storage; "" if none). */
const char* sss_last_error(void);

/*
 * sss_quantize -- direct casting of an fp32 weight matrix (Appendix C.1):
 * for every group, M = ||w||_inf, the grid's scale (eq:absmax; eq:sign_rule
 * for SIGNED: gamma* = -sign(w_i*), so the dominant outlier lands exactly on
 * the code -2^(q-1); eq:minmax for ASYM), codes c = clip(RNE(w/s)) of the
 * exact quotient (ties to even), packed as above, and the fp16 scale (and
 * min).  Bit-exact with the reference definition.
 *
 *   w           [in]  device fp32 [n][k], 16-byte aligned, row-major contiguous.
 *   out         [in]  descriptor of the outputs (n, k, q, group, grid and the
 *                     device buffers codes (16-byte aligned), scales, mins);
 *                     not retained.
 *   clip_counts [out] nullable device uint8 [n][k/group][2]: for symmetric
 *                     grids {|C_gamma|, |C_-gamma|} (def:clipped-set): the
 *                     number of pre-clip codes equal to +2^(q-1) and to
 *                     -2^(q-1); for ASYM {0, 0}.
 *   dev_status  [out] nullable device uint32; SSS_FLAG_NONFINITE/RANGE OR-ed.
 * Errors: SSS_E_ARG (q, group, grid, k % group, NULL buffers), SSS_E_ALIGN
 * (w or codes not 16-byte aligned), SSS_E_CUDA.  n == 0 is a no-op.
 */
sss_status_t sss_quantize(const float* w, const sss_qtensor_t* out,
                          uint8_t* clip_counts, uint32_t* dev_status,
                          void* stream);

/*
 * sss_dequantize -- w^ = f16(s)*c (symmetric; exact in fp32) or
 * w^ = fl32(fl32(f16(s)*u) + f16(m)) (ASYM), the value eq:quantizer assigns
 * to each weight, written as [n][k] in out_dtype (fp16/bf16 outputs are the
 * round-to-nearest-even of the fp32 value).
 *   qt   [in]  packed tensor (device buffers).
 *   out  [out] device [n][k] of sss_dtype_t out_dtype, 16-byte aligned.
 * Errors: SSS_E_ARG, SSS_E_ALIGN, SSS_E_CUDA.
 */
sss_status_t sss_dequantize(const sss_qtensor_t* qt, void* out,
                            int32_t out_dtype, void* stream);

/*
 * sss_gemv -- decode GEMV y[b][r] = sum_k w^[r][k] * x[b][k] with the
 * dequantisation fused (Appendix B.3: y = sum_b s * (integer dot) for the
 * symmetric formats, plus the row-sum term sum_b m * sum_{k in b} x for
 * ASYM).  fp32 accumulation; deterministic (no atomics).  At batch 1 the
 * integer codes meet the activations exactly and the group scale is applied
 * in fp32.  At batch 2..16 (k a multiple of 256), the batch fills the
 * tensor-core columns, so each weight enters the product as w^ rounded once
 * to fp16 (<= 2^-11 relative, as in sss_gemm), times 2^p (p = 0, 2 or 4, the
 * bit offset of the code's field).  That operand fits fp16 while
 * |w^| * 2^p < 65520; every group whose scale could break this raises
 * SSS_FLAG_RANGE (checked per scale, conservatively: |s| * 2^(q-1) * 16 >=
 * 65520 for the symmetric grids, (|s| * (2^q - 1) + |m|) * 16 >= 65520 for
 * ASYM).
 *   qt        [in]  packed tensor; codes 16-byte aligned, scales/mins 4-byte
 *                   aligned.
 *   x_bf16    [in]  device bf16 [batch][k], 16-byte aligned.
 *   batch     [in]  1..16.
 *   y         [out] device fp32 [batch][n].
 *   workspace [in]  device scratch of ws_bytes >= sss_workspace_bytes(qt,
 *                   batch, SSS_OP_GEMV) bytes, 16-byte aligned, or NULL when
 *                   that size is 0.  Its contents on entry are ignored.
 *   dev_status [out] nullable; SSS_FLAG_RANGE as above (batch 2..16).  The
 *                   GEMV kernels have no waits that could time out.
 * Errors: SSS_E_ARG, SSS_E_ALIGN, SSS_E_WORKSPACE, SSS_E_CUDA.
 */
sss_status_t sss_gemv(const sss_qtensor_t* qt, const uint16_t* x_bf16,
                      int32_t batch, float* y, void* workspace,
                      size_t ws_bytes, uint32_t* dev_status, void* stream);

/* flags of sss_gemv_multi */
#define SSS_GEMV_PDL 0x1u           /* launch as a programmatic dependent launch: the kernel
                                       may start while the preceding kernel in the stream
                                       drains; it reads x (and writes y) only after that
                                       kernel has completed                                */
#define SSS_GEMV_WEIGHTS_READY 0x2u /* with SSS_GEMV_PDL: the packed weights are not written
                                       by the preceding work in the stream, so they may be
                                       streamed in before it completes                     */
#define SSS_GEMV_ACT_Q8 0x4u        /* quantize x to Q8_0 on the fly (see
                                       sss_quantize_act_q8) and multiply the packed
                                       weights with the Q8_0 values: y_j[r] =
                                       sum_blocks fl16(d) * sum_k w^_j[r][k] * q[k]; the
                                       integer dot of codes and int8 values is exact */

/*
 * sss_gemv_multi -- batch-1 decode GEMV of several packed matrices that
 * share one activation vector (e.g. the q/k/v or gate/up projections of a
 * layer) in one launch: y_j[r] = sum_k w^_j[r][k] * x[k] (same arithmetic as
 * sss_gemv).  Every lane loads the packed bytes it multiplies straight into
 * registers (a ring one unit ahead of its use); only the activations are
 * staged in shared memory.
 *   qts     [in]  count pointers to packed tensors with equal k, q, group and
 *                 grid; codes, scales (and mins) 16-byte aligned.
 *   ys      [out] count device fp32 pointers, y_j of length qts[j]->n.
 *   count   [in]  1..4.
 *   x_bf16  [in]  device bf16 [k], 16-byte aligned.
 *   flags   [in]  SSS_GEMV_* bits.
 *   dev_status [out] nullable; with SSS_GEMV_ACT_Q8 the Q8_0 flags of x
 *                 (the streaming kernel has no waits that could time out).
 * Shapes with k % 256 != 0 or k % (8*group) != 0, or unaligned buffers, run
 * as one sss_gemv per matrix (flags then have no effect, and SSS_GEMV_ACT_Q8
 * returns SSS_E_UNSUPPORTED).
 * Errors: SSS_E_ARG, SSS_E_ALIGN, SSS_E_UNSUPPORTED, SSS_E_CUDA.
 */
sss_status_t sss_gemv_multi(const sss_qtensor_t* const* qts, float* const* ys,
                            int32_t count, const uint16_t* x_bf16, uint32_t flags,
                            uint32_t* dev_status, void* stream);

/*
 * sss_gemm -- prefill GEMM Y[m][r] = sum_k w^[r][k] * X[m][k] (Appendix B.3;
 * prefill is the phase where the matrix products set the time), dequantising
 * weight tiles on chip and accumulating on the tcgen05 tensor cores in fp32
 * (tensor memory).  Tile operands are fp16: w^ rounded to fp16 and X
 * converted from bf16 (exact for 2^-17 <= |x| <= 65504).  The weight
 * operand fits fp16 while |w^| < 65520; every group whose scale could break
 * this raises SSS_FLAG_RANGE (checked per scale, conservatively: |s| *
 * 2^(q-1) >= 65520, or |s| * (2^q - 1) + |m| >= 65520 for ASYM).
 *   qt        [in]  packed tensor, symmetric grids or ASYM; k % 64 == 0;
 *                   codes 16-byte aligned.
 *   x_bf16    [in]  device bf16 [m][k], 16-byte aligned.
 *   m         [in]  0 .. 2^24 tokens.
 *   y         [out] device fp32 [m][n], 16-byte aligned, n % 4 == 0.
 *   workspace [in]  device scratch, 16-byte aligned, of ws_bytes >= m * k * 2
 *                   (rounded up to 256); sss_workspace_bytes(qt, m,
 *                   SSS_OP_GEMM) bytes enable split K (see there).  Its
 *                   contents on entry are ignored.
 *   dev_status [out] nullable; SSS_FLAG_TIMEOUT if a bounded wait expired,
 *                   SSS_FLAG_RANGE as above.
 * Errors: SSS_E_ARG, SSS_E_ALIGN, SSS_E_UNSUPPORTED, SSS_E_WORKSPACE, SSS_E_CUDA.
 */
sss_status_t sss_gemm(const sss_qtensor_t* qt, const uint16_t* x_bf16,
                      int64_t m, float* y, void* workspace, size_t ws_bytes,
                      uint32_t* dev_status, void* stream);

/*
 * sss_gemm_multi -- sss_gemm for several packed matrices that share one
 * activation matrix (e.g. the q/k/v or gate/up projections of a layer) in
 * one launch: Y_j[m][r] = sum_k w^_j[r][k] * X[m][k] (same arithmetic as
 * sss_gemm, Appendix B.3).  X is converted to fp16 once, and the output
 * tiles of all the matrices share one grid, so small matrices (k/v) fill
 * the SMs together with the others instead of splitting K.
 *   qts   [in]  count pointers to packed tensors with equal k, q, group and
 *               grid; each n % 4 == 0; codes 16-byte aligned.  Tensors with
 *               n == 0 are skipped.
 *   ys    [out] count device fp32 pointers, Y_j [m][n_j], 16-byte aligned.
 *   count [in]  1..4.
 *   x_bf16, m, workspace, ws_bytes, dev_status, stream: as sss_gemm, with
 *               the workspace sized by sss_gemm_multi_workspace_bytes (the
 *               fp16 copy of X, m*k*2 bytes, is enough to run unsplit).
 * Errors: SSS_E_ARG (count, mismatched tensors), SSS_E_ALIGN,
 * SSS_E_UNSUPPORTED, SSS_E_WORKSPACE, SSS_E_CUDA.
 */
sss_status_t sss_gemm_multi(const sss_qtensor_t* const* qts, float* const* ys,
                            int32_t count, const uint16_t* x_bf16, int64_t m,
                            void* workspace, size_t ws_bytes,
                            uint32_t* dev_status, void* stream);

/* Workspace bytes that let sss_gemm_multi take its preferred plan (0 for
 * invalid arguments or an empty call). */
size_t sss_gemm_multi_workspace_bytes(const sss_qtensor_t* const* qts,
                                      int32_t count, int64_t m);

/*
 * sss_gemm_q8 -- sss_gemm on Q8_0 activations: each token's X is quantized
 * per block of 32 (sss_quantize_act_q8) and the GEMM multiplies the packed
 * weights with fl16(fl16(d) * q), the fp16 operand of the tensor cores (one
 * rounding, <= 2^-11 relative).  This is the runtime pairing of few-bit
 * weights with 8-bit activations the paper deploys (Sec. 5 "Composition with
 * PTQ methods"; Appendix B.3 product).  Arguments, layouts, workspace and
 * errors as sss_gemm; dev_status also receives the activation flags of
 * sss_quantize_act_q8.
 */
sss_status_t sss_gemm_q8(const sss_qtensor_t* qt, const uint16_t* x_bf16,
                         int64_t m, float* y, void* workspace, size_t ws_bytes,
                         uint32_t* dev_status, void* stream);

/*
 * sss_quantize_act_q8 -- Q8_0 activations, the narrow-range 8-bit format the
 * paper pairs with its weight formats (Sec. 5 "Composition with PTQ
 * methods"; Appendix C "Algorithm details"): per block of 32 consecutive
 * values of a row, M = max |x|, d = fl32(M / 127), q = clip(RNE(x / d) of
 * the exact quotient, -127, 127), stored scale fl16(d).  A zero block gives
 * q = 0, d = +0; a block with NaN/Inf gives q = 0, d = +0 and
 * SSS_FLAG_NONFINITE; an fp16 overflow of d raises SSS_FLAG_RANGE.
 *   x_bf16 [in]  device bf16 [rows][k], 16-byte aligned; k % 32 == 0.
 *   q      [out] device int8 [rows][k], 8-byte aligned.
 *   d      [out] device fp16 [rows][k/32].
 * Errors: SSS_E_ARG, SSS_E_ALIGN, SSS_E_CUDA.
 */
sss_status_t sss_quantize_act_q8(const uint16_t* x_bf16, int64_t rows, int64_t k,
                                 int8_t* q, uint16_t* d, uint32_t* dev_status,
                                 void* stream);

/*
 * Normalized Hadamard rotation of the weights before quantization: the
 * mergeable rotations of the paper's PTQ pipeline (Sec. 5 "Composition with
 * PTQ methods"; Appendix C, the rotation graph), folded into the weights so
 * that the grids are computed on the rotated weights and the runtime path
 * is unchanged.  The transform of a block of b values (b a power of two,
 * 2 <= b <= 8192) is the normalized Walsh-Hadamard transform H_b/sqrt(b)
 * (Sylvester order) computed as the in-place fast transform in IEEE fp32:
 * strides h = 1, 2, ..., b/2, butterflies (a, c) -> (a + c, a - c), then
 * every value times the fp32 nearest to 1/sqrt(b).  H_b/sqrt(b) is
 * symmetric and orthogonal: W x = (W R)(R x) for R = I (x) H_b/sqrt(b).
 */
#define SSS_ROTATE_INPUT 0  /* W <- W R: every block of b consecutive values of a row (b | k,
                               k a multiple of 4)                                            */
#define SSS_ROTATE_OUTPUT 1 /* W <- R W: every block of b consecutive rows, per column
                               (b | n, and k a multiple of 8192/b)                          */

/*
 * sss_hadamard -- rotate the fp32 matrix w [n][k] into out [n][k] (out may
 * equal w).  Both 16-byte aligned.
 * Errors: SSS_E_ARG (block, side or shape), SSS_E_ALIGN, SSS_E_CUDA.
 */
sss_status_t sss_hadamard(const float* w, float* out, int64_t n, int64_t k,
                          int32_t block, int32_t side, void* stream);

/*
 * sss_quantize_rotated -- sss_quantize of the input-side rotation of w:
 * bit for bit sss_hadamard(w, tmp, n, k, block, SSS_ROTATE_INPUT) followed
 * by sss_quantize(tmp, out, ...), in one pass that never writes the rotated
 * fp32 weights (block | k).  Arguments and errors as sss_quantize.
 */
sss_status_t sss_quantize_rotated(const float* w, int32_t block, const sss_qtensor_t* out,
                                  uint8_t* clip_counts, uint32_t* dev_status,
                                  void* stream);

/*
 * sss_quantize_lsq -- symmetric-grid quantization with every group's scale
 * refined by LSQ steps (Sec. 5 "Composition with learned rotations and grid
 * parameters"; Appendix C: LSQ, the scale constrained to s != 0 for the
 * signed formats and s > 0 for the conventional ones).  The paper learns
 * the scales through the model loss on calibration data; this is the
 * data-free reading on each group's reconstruction loss L(s) =
 * sum (s c_i - w_i)^2, in IEEE fp32 without fused multiply-add:
 *   s_0 = gamma* alpha (SIGNED) or alpha (UNSIGNED), as sss_quantize;
 *   each step: v_i = w_i / s, c_i = clip(rint(v_i)), d_i = c_i - v_i inside
 *   the alphabet and the clip value outside (LSQ's straight-through
 *   derivative of w^_i = s c_i), t_i = (2 (s c_i - w_i)) d_i, G = the
 *   pairwise sum t_i <- t_i + t_{i+h} (h = g/2, ..., 1),
 *   s <- s - (lr / sqrt(g (2^(q-1) - 1))) G, and a step that would cross or
 *   reach zero halves s instead, so the sign is kept;
 *   then codes c = clip(RNE(w / s)) of the exact quotient and fp16 s, in the
 *   layout of sss_quantize.  steps = 0 reproduces sss_quantize.
 *   out   [in]  as sss_quantize; grid SIGNED_SYM or UNSIGNED_SYM.
 *   steps [in]  >= 0;  lr [in] >= 0.
 * Errors: SSS_E_ARG, SSS_E_ALIGN, SSS_E_UNSUPPORTED (ASYM), SSS_E_CUDA.
 */
sss_status_t sss_quantize_lsq(const float* w, const sss_qtensor_t* out, int32_t steps,
                              float lr, uint32_t* dev_status, void* stream);

/*
 * sss_sign_diagnostics -- the cardinality margin and the realised l2 gain of
 * the signed absmax sign rule on every group (Sec. 4, rem:cardinality-margin
 * and fig:theory-diagnostics), on any fp32 weights: for the sign gamma* of
 * eq:sign_rule and the clipped sets of def:clipped-set,
 *   margin m = |C_-gamma*| - |C_gamma*|            (in -group .. group)
 *   gain   g = ||w - Q_-gamma*(w)||^2 - ||w - Q_gamma*(w)||^2
 * with the weights each sign's stored fp16 scale dequantises to.  g is
 * exact (fp64).  Groups with NaN/Inf are skipped and raise
 * SSS_FLAG_NONFINITE; all-zero groups count as m = 0, g = 0.
 *   w      [in]  device fp32 [n][k], 16-byte aligned; k % group == 0.
 *   q      [in]  2, 3 or 4;  group 32, 64 or 128.
 *   margin [out] nullable device int16 [n][k/group].
 *   gain   [out] nullable device fp64 [n][k/group].
 *   hist   [in,out] nullable device uint64 [2*group+1][3], ADDED to: row
 *                m + group, column 0 (g < 0), 1 (g == 0) or 2 (g > 0).
 * Errors: SSS_E_ARG, SSS_E_ALIGN, SSS_E_CUDA.
 */
sss_status_t sss_sign_diagnostics(const float* w, int64_t n, int64_t k, int32_t q,
                                  int32_t group, int16_t* margin, double* gain,
                                  uint64_t* hist, uint32_t* dev_status, void* stream);

#define SSS_OP_GEMV 0
#define SSS_OP_GEMM 1
/* Workspace bytes sss_gemv (op SSS_OP_GEMV, m_or_batch = batch) or sss_gemm
 * (op SSS_OP_GEMM, m_or_batch = m) needs for this tensor; 0 if none (or an
 * invalid tensor).  For sss_gemm this is the size that lets the call take
 * its fastest plan: the fp16 copy of X (m * k * 2 bytes, rounded up to 256),
 * plus, when the weight tiles are fewer than the SMs, room for fp32 partial
 * tiles of K split across CTAs (summed in a fixed order, so the result does
 * not depend on timing).  sss_gemm runs with any workspace that holds the
 * fp16 copy of X, unsplit when the partials do not fit. */
size_t sss_workspace_bytes(const sss_qtensor_t* qt, int64_t m_or_batch,
                           int32_t op);

/*
 * sss_gemm_noalloc -- sss_gemm with its scratch (the fp16 copy of X, m*k*2
 * bytes) in a static 32 MiB device array of the library instead of a
 * caller workspace.  The paper has no counterpart: this is a library
 * convenience for callers that cannot allocate device memory when they
 * call, e.g. a plain C host with no device allocator, or a serving loop
 * that must not call cudaMalloc (it synchronises the device and can fail
 * under memory pressure).  Nothing is allocated at call time.
 *   Arguments, layouts and errors as sss_gemm, without workspace/ws_bytes.
 *   Limit: m * k * 2 <= sss_gemm_noalloc_max_scratch_bytes() (33554432);
 *          larger calls return SSS_E_WORKSPACE (sss_last_error() says why).
 *   The first call on each device looks up the array's device address with
 *   that device current (set-up); make that first call before any stream
 *   capture begins.  Nothing in the scratch needs to start at zero.
 *   All calls on a device share the one array: calls that overlap in time
 *   (other streams, other host threads) race on it; callers serialise them.
 */
sss_status_t sss_gemm_noalloc(const sss_qtensor_t* qt, const uint16_t* x_bf16,
                              int64_t m, float* y, uint32_t* dev_status,
                              void* stream);
size_t sss_gemm_noalloc_max_scratch_bytes(void);

/*
 * sss_test_set_stall -- test hook for the bounded waits; the paper has no
 * counterpart.  While a bit below is set, every later launch of that kernel
 * family leaves one mbarrier one arrive short: the GEMM on the first
 * stage's weight tile.  The decode GEMV kernels (batch 1 and batched) have
 * no data-dependent waits (their warps meet only at CTA-wide barriers), so
 * their bits have no effect.  The wait on that barrier then runs out after
 * its bound (about one second), the kernel raises SSS_FLAG_TIMEOUT in
 * dev_status, lets its own copies and MMAs in flight finish, releases its
 * tensor memory and returns; its output is incomplete.  Nothing faults or
 * hangs.  mask = 0 (the default) restores normal launches.  Process-wide;
 * affects launches issued (or captured) after the call on every thread.
 */
#define SSS_TEST_STALL_GEMV 0x1u       /* gemv_stream_kernel: no waits, no effect               */
#define SSS_TEST_STALL_GEMV_BATCH 0x2u /* gemv_batch_kernel: no waits, no effect                */
#define SSS_TEST_STALL_GEMM 0x4u       /* gemm_kernel (sss_gemm, sss_gemm_noalloc)             */
void sss_test_set_stall(uint32_t mask);

#ifdef __cplusplus
}
#endif
#endif /* SSS_H */
