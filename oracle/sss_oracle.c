/*
 * sss_oracle.c -- plain CPU oracle (TEST INFRASTRUCTURE ONLY; see the
 * header).  Each function cites the passage of the paper it follows.
 *
 * Readings of points the paper leaves open (also listed in the design notes):
 *  - Sign tie: when max w == -min w the dominant outlier is ambiguous
 *    (Sec. 3 after eq:sign_rule asks for a deterministic tie-break but names
 *    no rule); we take
 *    gamma = +1, the standard convention.
 *  - RTN tie (w/s exactly a half-integer, assumed away in Sec. 4): round
 *    half to even of the EXACT quotient.  The fp64 quotient of two fp32
 *    numbers decides RNE of the exact quotient correctly (see
 *    orc_rne_quotient).
 *  - M == 0: all codes 0 and stored scale +0 (the paper requires M > 0).
 *    The same holds when alpha = M / 2^(q-1) underflows to zero in fp32
 *    (M <= 2^(q-151)), where the paper's s != 0 cannot be met.
 *  - Asymmetric grid (eq:minmax): s = fl32(fl32(max-min)/(2^q-1)), the code
 *    is RNE(fl32(w-min)/s) clipped to {0..2^q-1}, i.e. eq:quantizer with
 *    z = -min/s written as (w-min)/s; the minimum is stored as fp16 and the
 *    dequantised weight is s*u + min.
 */
#include "sss_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* IEEE binary16 from its definition.                                        */
/* ------------------------------------------------------------------------ */

uint16_t orc_f32_to_f16(float x) {
  uint16_t sign = signbit(x) ? 0x8000u : 0u;
  if (isnan(x)) return (uint16_t)(sign | 0x7e00u);
  double a = fabs((double)x);
  if (isinf(x)) return (uint16_t)(sign | 0x7c00u);
  if (a == 0.0) return sign;
  /* binary16: normal numbers are (1 + f/1024) * 2^(e-15), e in 1..30;
   * subnormals are f * 2^-24, f in 1..1023. */
  int e2;
  (void)frexp(a, &e2); /* a = m * 2^e2, m in [0.5, 1) => a in [2^(e2-1), 2^e2) */
  int e = e2 - 1;      /* a in [2^e, 2^(e+1)) */
  if (e < -14) {
    /* subnormal range: quantum 2^-24 */
    double m = nearbyint(ldexp(a, 24)); /* exact scaling, RNE */
    /* m may reach 1024, which is exactly the smallest normal's encoding */
    return (uint16_t)(sign | (uint16_t)m);
  }
  /* normal range: 11 significant bits, quantum 2^(e-10) */
  double m = nearbyint(ldexp(a, 10 - e)); /* in [1024, 2048] */
  int biased = e + 15;
  long bits = ((long)biased << 10) + ((long)m - 1024); /* carry into exponent */
  if (bits >= 0x7c00) return (uint16_t)(sign | 0x7c00u); /* overflow -> inf */
  return (uint16_t)(sign | (uint16_t)bits);
}

float orc_f16_to_f32(uint16_t h) {
  int s = (h >> 15) & 1;
  int e = (h >> 10) & 0x1f;
  int f = h & 0x3ff;
  double v;
  if (e == 0x1f) {
    v = f ? NAN : INFINITY;
  } else if (e == 0) {
    v = ldexp((double)f, -24);
  } else {
    v = ldexp(1024.0 + (double)f, e - 25);
  }
  return (float)(s ? -v : v);
}

float orc_bf16_to_f32(uint16_t b) {
  uint32_t bits = ((uint32_t)b) << 16;
  float f;
  memcpy(&f, &bits, sizeof f);
  return f;
}

/* ------------------------------------------------------------------------ */
/* Rounding of the exact quotient.                                          */
/* ------------------------------------------------------------------------ */

/* RNE(a / b) of the exact real quotient of two fp32 numbers (eq:quantizer's
 * rounding).  Both fit in fp64 exactly.  If a/b is a half-integer it is a
 * short dyadic number, representable in fp64, so the correctly rounded fp64
 * division returns it exactly and nearbyint breaks the tie to even.
 * Otherwise a/b lies at least 2^-27 * |a/b|-ish away from every
 * half-integer (24-bit significands), far more than the fp64 division error
 * (2^-53 relative), so fp64 rounding cannot move it across one. */
static double orc_rne_quotient(float a, float b) {
  return nearbyint((double)a / (double)b);
}

static int32_t clampi(int32_t v, int32_t lo, int32_t hi) {
  return v < lo ? lo : (v > hi ? hi : v);
}

/* ------------------------------------------------------------------------ */
/* Symmetric grids: eq:quantizer with z = 0, s = gamma * alpha,             */
/* alpha = ||w||_inf / 2^(q-1) (eq:absmax, eq:signed_sym_quant).            */
/* ------------------------------------------------------------------------ */

static int32_t scan_group(const float* w, int32_t g, float* mx, float* mn) {
  int32_t flags = 0;
  float hi = w[0], lo = w[0];
  for (int32_t j = 0; j < g; ++j) {
    if (!isfinite(w[j])) flags |= ORC_FLAG_NONFINITE;
    if (w[j] > hi) hi = w[j];
    if (w[j] < lo) lo = w[j];
  }
  *mx = hi;
  *mn = lo;
  return flags;
}

int32_t orc_quantize_group_gamma(const float* w, int32_t g, int32_t q,
                                 int32_t gamma, int32_t* c_pre, int32_t* c,
                                 uint8_t* u, orc_group_t* info) {
  orc_group_t r;
  memset(&r, 0, sizeof r);
  r.flags = scan_group(w, g, &r.mx, &r.mn);
  /* M := ||w||_inf (Sec. 3, signed absmax grid) */
  r.M = (r.mx > -r.mn) ? r.mx : -r.mn;
  r.gamma = gamma;
  const int32_t half = 1 << (q - 1);           /* 2^(q-1)              */
  const int32_t amin = -half, amax = half - 1; /* A_q = {-2^(q-1)..2^(q-1)-1} */
  /* alpha := M / 2^(q-1): exact power-of-two scaling of M, except that a
   * subnormal M can round it (to zero when M <= 2^(q-151)) */
  const float alpha = ldexpf(r.M, -(q - 1));
  if (r.M == 0.0f || alpha == 0.0f || (r.flags & ORC_FLAG_NONFINITE)) {
    /* all-zero group: codes 0, stored scale +0 (reading; the paper assumes
     * M > 0 and s != 0).  A group whose alpha underflows to zero has no
     * usable scale and is given the same outputs (reading).  A group
     * holding NaN/Inf is flagged and given the same placeholder outputs;
     * its content is not meaningful. */
    r.alpha = 0.0f;
    r.s32 = 0.0f;
    for (int32_t j = 0; j < g; ++j) {
      if (c_pre) c_pre[j] = 0;
      if (c) c[j] = 0;
      if (u) u[j] = (uint8_t)half;
    }
  } else {
    r.alpha = alpha;
    r.s32 = (float)gamma * r.alpha; /* s := gamma * alpha */
    for (int32_t j = 0; j < g; ++j) {
      /* round-to-nearest of w/s, then clip to A_q (eq:quantizer, z = 0) */
      int32_t cp = (int32_t)orc_rne_quotient(w[j], r.s32);
      int32_t cc = clampi(cp, amin, amax);
      if (cp == half) r.n_self++;   /* index in C_gamma (def:clipped-set) */
      if (cp == -half) r.n_other++; /* index in C_-gamma (odd symmetry of RNE) */
      if (c_pre) c_pre[j] = cp;
      if (c) c[j] = cc;
      if (u) u[j] = (uint8_t)(cc + half);
    }
  }
  r.s16 = orc_f32_to_f16(r.s32);
  if ((r.s16 & 0x7fffu) == 0x7c00u) r.flags |= ORC_FLAG_RANGE;
  if (info) *info = r;
  return r.flags;
}

/* ------------------------------------------------------------------------ */
/* Asymmetric min-max grid (eq:minmax) on the unsigned alphabet.            */
/* ------------------------------------------------------------------------ */

static int32_t quantize_group_asym(const float* w, int32_t g, int32_t q,
                                   int32_t* c_pre, int32_t* c, uint8_t* u,
                                   orc_group_t* info) {
  orc_group_t r;
  memset(&r, 0, sizeof r);
  r.flags = scan_group(w, g, &r.mx, &r.mn);
  /* reading: a zero minimum is stored as +0 (the sign of zero of a group
   * mixing +0 and -0 is otherwise an artefact of the scan order) */
  if (r.mn == 0.0f) r.mn = 0.0f;
  if (r.mx == 0.0f) r.mx = 0.0f;
  r.M = (r.mx > -r.mn) ? r.mx : -r.mn;
  r.gamma = 0;
  const int32_t umax = (1 << q) - 1;
  int zero_codes = 0;
  if (r.mx == r.mn || (r.flags & ORC_FLAG_NONFINITE)) {
    r.s32 = 0.0f; /* constant group: every weight equals min */
    zero_codes = 1;
  } else {
    float range = r.mx - r.mn;                  /* fl32(max - min)          */
    r.s32 = range / (float)umax;                /* s = (max-min)/(2^q - 1)  */
    if (!isfinite(r.s32)) {
      r.flags |= ORC_FLAG_RANGE;
      zero_codes = 1;
    } else if (r.s32 == 0.0f) {
      zero_codes = 1; /* the step underflowed to zero: codes 0 (reading) */
    }
  }
  for (int32_t j = 0; j < g; ++j) {
    int32_t cp = 0;
    if (!zero_codes) {
      float d = w[j] - r.mn;                       /* fl32(w - min) >= 0   */
      cp = (int32_t)orc_rne_quotient(d, r.s32);    /* RNE((w - min)/s)     */
    }
    int32_t cc = clampi(cp, 0, umax);
    if (c_pre) c_pre[j] = cp;
    if (c) c[j] = cc;
    if (u) u[j] = (uint8_t)cc;
  }
  r.s16 = orc_f32_to_f16(r.s32);
  r.m16 = orc_f32_to_f16(r.mn);
  if ((r.s16 & 0x7fffu) == 0x7c00u || (r.m16 & 0x7fffu) == 0x7c00u)
    r.flags |= ORC_FLAG_RANGE;
  if (info) *info = r;
  return r.flags;
}

int32_t orc_quantize_group(const float* w, int32_t g, int32_t q, int32_t grid,
                           int32_t* c_pre, int32_t* c, uint8_t* u,
                           orc_group_t* info) {
  if (grid == ORC_GRID_ASYM) return quantize_group_asym(w, g, q, c_pre, c, u, info);
  int32_t gamma = 1; /* unsigned convention: s > 0 (eq:absmax) */
  if (grid == ORC_GRID_SIGNED_SYM) {
    /* gamma* = -sign(w_i*), i* in argmax |w_i| (eq:sign_rule).  The dominant
     * outlier is positive iff max w > -min w; on a tie gamma = +1. */
    float mx, mn;
    (void)scan_group(w, g, &mx, &mn);
    gamma = (mx > -mn) ? -1 : 1;
  }
  return orc_quantize_group_gamma(w, g, q, gamma, c_pre, c, u, info);
}

/* ------------------------------------------------------------------------ */
/* Canonical packed layout (our choice; the paper fixes 4-bit and 2-bit      */
/* block contents, Appendix "Formats and block layout", not a GPU layout).  */
/* ------------------------------------------------------------------------ */

void orc_pack_group(const uint8_t* u, int32_t g, int32_t q, uint8_t* out) {
  int32_t nbytes = g * q / 8;
  memset(out, 0, (size_t)nbytes);
  if (q == 4) {
    for (int32_t j = 0; j < g; ++j)
      out[j >> 1] |= (uint8_t)((u[j] & 0xf) << (4 * (j & 1)));
  } else if (q == 2) {
    for (int32_t j = 0; j < g; ++j)
      out[j >> 2] |= (uint8_t)((u[j] & 0x3) << (2 * (j & 3)));
  } else if (q == 3) {
    uint8_t* lo = out;
    uint8_t* hi = out + g / 4;
    for (int32_t j = 0; j < g; ++j) {
      lo[j >> 2] |= (uint8_t)((u[j] & 0x3) << (2 * (j & 3)));
      hi[j >> 3] |= (uint8_t)(((u[j] >> 2) & 0x1) << (j & 7));
    }
  }
}

void orc_unpack_group(const uint8_t* in, int32_t g, int32_t q, uint8_t* u) {
  for (int32_t j = 0; j < g; ++j) {
    if (q == 4) {
      u[j] = (uint8_t)((in[j >> 1] >> (4 * (j & 1))) & 0xf);
    } else if (q == 2) {
      u[j] = (uint8_t)((in[j >> 2] >> (2 * (j & 3))) & 0x3);
    } else {
      const uint8_t* lo = in;
      const uint8_t* hi = in + g / 4;
      uint8_t l = (uint8_t)((lo[j >> 2] >> (2 * (j & 3))) & 0x3);
      uint8_t h = (uint8_t)((hi[j >> 3] >> (j & 7)) & 0x1);
      u[j] = (uint8_t)(l | (h << 2));
    }
  }
}

/* ------------------------------------------------------------------------ */
/* Whole-matrix drivers.                                                    */
/* ------------------------------------------------------------------------ */

int32_t orc_quantize(const float* W, int64_t n, int64_t k, int32_t q,
                     int32_t g, int32_t grid, uint8_t* codes, uint16_t* scales,
                     uint16_t* mins, uint8_t* clip_counts) {
  int32_t flags = 0;
  int64_t ngroups = n * (k / g);
  int64_t gbytes = (int64_t)g * q / 8;
  uint8_t* u = (uint8_t*)malloc((size_t)g);
  for (int64_t G = 0; G < ngroups; ++G) {
    orc_group_t info;
    flags |= orc_quantize_group(W + G * g, g, q, grid, NULL, NULL, u, &info);
    orc_pack_group(u, g, q, codes + G * gbytes);
    scales[G] = info.s16;
    if (mins) mins[G] = (grid == ORC_GRID_ASYM) ? info.m16 : 0;
    if (clip_counts) {
      clip_counts[2 * G] = (uint8_t)info.n_self;
      clip_counts[2 * G + 1] = (uint8_t)info.n_other;
    }
  }
  free(u);
  return flags;
}

void orc_dequantize_rows(const uint8_t* codes, const uint16_t* scales,
                         const uint16_t* mins, int64_t n, int64_t k, int32_t q,
                         int32_t g, int32_t grid, int64_t r0, int64_t nr,
                         float* out) {
  (void)n;
  int64_t gpr = k / g;
  int64_t gbytes = (int64_t)g * q / 8;
  uint8_t* u = (uint8_t*)malloc((size_t)g);
  const int32_t half = 1 << (q - 1);
  for (int64_t r = 0; r < nr; ++r) {
    for (int64_t jg = 0; jg < gpr; ++jg) {
      int64_t G = (r0 + r) * gpr + jg;
      orc_unpack_group(codes + G * gbytes, g, q, u);
      float s = orc_f16_to_f32(scales[G]);
      float* o = out + r * k + jg * g;
      if (grid == ORC_GRID_ASYM) {
        float m = orc_f16_to_f32(mins[G]);
        for (int32_t j = 0; j < g; ++j) {
          float t = s * (float)u[j]; /* exact: 11-bit x 4-bit significands */
          o[j] = t + m;              /* one rounding: s*u + min           */
        }
      } else {
        for (int32_t j = 0; j < g; ++j) o[j] = s * (float)((int32_t)u[j] - half);
      }
    }
  }
  free(u);
}

void orc_dequantize(const uint8_t* codes, const uint16_t* scales,
                    const uint16_t* mins, int64_t n, int64_t k, int32_t q,
                    int32_t g, int32_t grid, float* out) {
  orc_dequantize_rows(codes, scales, mins, n, k, q, g, grid, 0, n, out);
}

void orc_matmul_f64(const float* What, const uint16_t* x_bf16, int64_t nb,
                    int64_t n, int64_t k, double* y) {
  for (int64_t b = 0; b < nb; ++b) {
    const uint16_t* xb = x_bf16 + b * k;
    for (int64_t j = 0; j < n; ++j) {
      const float* wr = What + j * k;
      double acc = 0.0;
      for (int64_t i = 0; i < k; ++i)
        acc += (double)wr[i] * (double)orc_bf16_to_f32(xb[i]);
      y[b * n + j] = acc;
    }
  }
}

void orc_gemv(const uint8_t* codes, const uint16_t* scales,
              const uint16_t* mins, int64_t n, int64_t k, int32_t q, int32_t g,
              int32_t grid, const uint16_t* x_bf16, int64_t nb, double* y) {
  float* row = (float*)malloc((size_t)k * sizeof(float));
  double* yr = (double*)malloc((size_t)nb * sizeof(double));
  for (int64_t j = 0; j < n; ++j) {
    orc_dequantize_rows(codes, scales, mins, n, k, q, g, grid, j, 1, row);
    orc_matmul_f64(row, x_bf16, nb, 1, k, yr);
    for (int64_t b = 0; b < nb; ++b) y[b * n + j] = yr[b];
  }
  free(yr);
  free(row);
}

/* ------------------------------------------------------------------------ */
/* Q8_0 activations (narrow range, blocks of 32)                            */
/* ------------------------------------------------------------------------ */

int32_t orc_quantize_act_q8(const uint16_t* x_bf16, int64_t nb, int64_t k,
                            int8_t* q, uint16_t* d16) {
  int32_t flags = 0;
  const int64_t nblk = k / 32;
  for (int64_t b = 0; b < nb; ++b) {
    for (int64_t j = 0; j < nblk; ++j) {
      const uint16_t* xs = x_bf16 + b * k + j * 32;
      int8_t* qs = q + b * k + j * 32;
      float x[32];
      float M = 0.0f;
      int bad = 0;
      for (int i = 0; i < 32; ++i) {
        x[i] = orc_bf16_to_f32(xs[i]);
        if (isnan(x[i]) || isinf(x[i])) bad = 1;
        const float a = fabsf(x[i]);
        if (a > M) M = a;
      }
      if (bad || M == 0.0f) {
        for (int i = 0; i < 32; ++i) qs[i] = 0;
        d16[b * nblk + j] = 0;
        if (bad) flags |= ORC_FLAG_NONFINITE;
        continue;
      }
      const float d = M / 127.0f; /* one IEEE fp32 division */
      for (int i = 0; i < 32; ++i)
        qs[i] = (int8_t)clampi((int32_t)orc_rne_quotient(x[i], d), -127, 127);
      const uint16_t h = orc_f32_to_f16(d);
      if ((h & 0x7fffu) == 0x7c00u) flags |= ORC_FLAG_RANGE;
      d16[b * nblk + j] = h;
    }
  }
  return flags;
}

void orc_gemv_q8(const uint8_t* codes, const uint16_t* scales,
                 const uint16_t* mins, int64_t n, int64_t k, int32_t q,
                 int32_t g, int32_t grid, const int8_t* xq,
                 const uint16_t* xd16, int64_t nb, double* y) {
  float* row = (float*)malloc((size_t)k * sizeof(float));
  for (int64_t j = 0; j < n; ++j) {
    orc_dequantize_rows(codes, scales, mins, n, k, q, g, grid, j, 1, row);
    for (int64_t b = 0; b < nb; ++b) {
      double acc = 0.0;
      for (int64_t i = 0; i < k; ++i) {
        const double xh = (double)orc_f16_to_f32(xd16[b * (k / 32) + i / 32]) *
                          (double)xq[b * k + i];
        acc += (double)row[i] * xh;
      }
      y[b * n + j] = acc;
    }
  }
  free(row);
}

/* ------------------------------------------------------------------------ */
/* Normalized Hadamard rotation (Sec. 5 composition; Appendix C).            */
/* ------------------------------------------------------------------------ */

void orc_fwht_f32(float* x, int32_t b) {
  for (int32_t h = 1; h < b; h *= 2) {
    for (int32_t i = 0; i < b; i += 2 * h) {
      for (int32_t j = i; j < i + h; ++j) {
        const float a = x[j], c = x[j + h];
        x[j] = a + c;
        x[j + h] = a - c;
      }
    }
  }
  const float norm = (float)(1.0 / sqrt((double)b)); /* the fp32 nearest 1/sqrt(b) */
  for (int32_t j = 0; j < b; ++j) x[j] = x[j] * norm;
}

void orc_rotate_rows(const float* W, int64_t n, int64_t k, int32_t b, float* out) {
  if (out != W) memcpy(out, W, (size_t)n * (size_t)k * sizeof(float));
  for (int64_t r = 0; r < n; ++r)
    for (int64_t c0 = 0; c0 < k; c0 += b) orc_fwht_f32(out + r * k + c0, b);
}

void orc_rotate_cols(const float* W, int64_t n, int64_t k, int32_t b, float* out) {
  float* col = (float*)malloc((size_t)b * sizeof(float));
  for (int64_t r0 = 0; r0 < n; r0 += b) {
    for (int64_t c = 0; c < k; ++c) {
      for (int32_t i = 0; i < b; ++i) col[i] = W[(r0 + i) * k + c];
      orc_fwht_f32(col, b);
      for (int32_t i = 0; i < b; ++i) out[(r0 + i) * k + c] = col[i];
    }
  }
  free(col);
}

/* ------------------------------------------------------------------------ */
/* Signed LSQ scale refinement (Sec. 5 learned grids; Appendix C).           */
/* ------------------------------------------------------------------------ */

float orc_lsq_scale(const float* w, int32_t g, int32_t q, int32_t signed_grid,
                    int32_t steps, float lr) {
  orc_group_t info;
  const int32_t grid = signed_grid ? ORC_GRID_SIGNED_SYM : ORC_GRID_UNSIGNED_SYM;
  (void)orc_quantize_group(w, g, q, grid, NULL, NULL, NULL, &info);
  float s = info.s32; /* the (signed) absmax initialisation */
  if (s == 0.0f) return s;
  const float qn = (float)(-(1 << (q - 1))), qp = (float)((1 << (q - 1)) - 1);
  const float gscale = (float)(1.0 / sqrt((double)g * (double)qp)); /* LSQ gradient scale */
  const float step = lr * gscale;
  float* t = (float*)malloc((size_t)g * sizeof(float));
  for (int32_t it = 0; it < steps; ++it) {
    for (int32_t i = 0; i < g; ++i) {
      const float v = w[i] / s;
      float c = rintf(v);
      float d;
      if (v <= qn) {
        c = qn;
        d = qn;
      } else if (v >= qp) {
        c = qp;
        d = qp;
      } else {
        if (c < qn) c = qn; /* v > qn but rint(v) may still equal qn */
        if (c > qp) c = qp;
        d = c - v;
      }
      const float e = s * c - w[i];
      t[i] = (2.0f * e) * d;
    }
    for (int32_t h = g / 2; h >= 1; h /= 2)
      for (int32_t i = 0; i < h; ++i) t[i] = t[i] + t[i + h];
    float sn = s - step * t[0];
    if (sn * s <= 0.0f) sn = s * 0.5f; /* keep the sign; never reach zero */
    s = sn;
  }
  free(t);
  return s;
}

int32_t orc_lsq_quantize(const float* W, int64_t n, int64_t k, int32_t q,
                         int32_t g, int32_t grid, int32_t steps, float lr,
                         uint8_t* codes, uint16_t* scales) {
  int32_t flags = 0;
  const int64_t ngroups = n * (k / g);
  const int32_t half = 1 << (q - 1);
  uint8_t* u = (uint8_t*)malloc((size_t)g);
  for (int64_t G = 0; G < ngroups; ++G) {
    const float* w = W + G * g;
    orc_group_t info;
    /* NaN/Inf and all-zero groups: the placeholder codes; RANGE is judged
     * on the refined scale that is stored, below */
    flags |= orc_quantize_group(w, g, q, grid, NULL, NULL, u, &info) & ORC_FLAG_NONFINITE;
    const float s = orc_lsq_scale(w, g, q, grid == ORC_GRID_SIGNED_SYM, steps, lr);
    if (s != 0.0f) {
      for (int32_t j = 0; j < g; ++j) {
        int32_t c = (int32_t)orc_rne_quotient(w[j], s);
        c = clampi(c, -half, half - 1);
        u[j] = (uint8_t)(c + half);
      }
    }
    scales[G] = orc_f32_to_f16(s);
    if ((scales[G] & 0x7fffu) == 0x7c00u) flags |= ORC_FLAG_RANGE;
    orc_pack_group(u, g, q, codes + G * (int64_t)(g * q / 8));
  }
  free(u);
  return flags;
}
