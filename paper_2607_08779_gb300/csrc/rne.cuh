// rne.cuh -- round-to-nearest-even of the exact quotient w / s in fp32
// arithmetic, shared by the quantizer and the sign diagnostics (the
// rounding of eq:quantizer; ties of the exact quotient go to even).
#pragma once

#include "sss_internal.cuh"

namespace sss {

// 1.5 * 2^23: adding it to |v| < 2^22 rounds v to an integer (ties to even)
// held in the low mantissa bits.
constexpr float kMagic = 12582912.0f;

// The exact-residual side decision for one weight whose rounded code is
// u (c = u - OFF the integer w*r rounded to): when w*r lies within 2^-18
// of the half-integer h between c and its neighbour, the sign of the
// single-rounding residual w - h*s places the exact quotient; a zero
// residual is an exact tie -> even.  Returns the corrected code.
template <int OFF>
__device__ __forceinline__ int fix_tie(float w, float s, float r, int u) {
  const float c = static_cast<float>(u - OFF);
  const float dd = __fmaf_rn(w, r, -c);  // w*r - c
  if (fabsf(__fsub_rn(fabsf(dd), 0.5f)) <= 0x1p-18f) {
    const float h = __fadd_rn(c, copysignf(0.5f, dd));   // the half-integer at stake
    const float e = __fmaf_rn(-h, s, w);                  // w - h*s, one rounding
    const float side = (s > 0.f) ? e : -e;                // sign of (w/s - h)
    const float lo = __fsub_rn(h, 0.5f), hi = __fadd_rn(h, 0.5f);
    float cc;
    if (side > 0.f) {
      cc = hi;
    } else if (side < 0.f) {
      cc = lo;
    } else {  // exact tie: to even
      cc = (static_cast<int>(lo) & 1) ? hi : lo;
    }
    u += static_cast<int>(__fsub_rn(cc, c));
  }
  return u;
}

// Stored code u = RNE(w / s) + OFF of the EXACT quotient, given r = RN(1/s)
// (OFF = 2^(q-1) for the symmetric grids, 0 for the min-max grid; OFF is
// even, so the parity of the rounded sum is that of the code).  One FMA
// rounds w*r straight to an integer; a second FMA gives the remainder
// w*r - c.  Only when that remainder is within 2^-18 of +-1/2 can the exact
// quotient fall on the other side of the half-integer (|w*r - w/s| <=
// 16 * 2^-24 here); fix_tie then decides it.
template <int OFF>
__device__ __forceinline__ int code_of(float w, float s, float r) {
  constexpr float MAGIC = kMagic + static_cast<float>(OFF);
  const float t = __fmaf_rn(w, r, MAGIC);
  const int u = __float_as_int(t) - __float_as_int(kMagic);
  const float dd = __fmaf_rn(w, r, __fsub_rn(MAGIC, t));  // w*r - c; MAGIC - t = -c exactly
  if (fabsf(__fsub_rn(fabsf(dd), 0.5f)) <= 0x1p-18f) return fix_tie<OFF>(w, s, r, u);
  return u;
}

// The same for N weights at once (the same codes as N calls of code_of):
// every weight's rounding in one straight line, so the N chains
// interleave, and a single branch, taken only when some weight lies within
// 2^-18 of a half-integer, into the exact side decisions.  That branch
// takes weight e from wat(e), which must return the value w[e] held, so
// that w need not stay in registers past the straight line.
template <int OFF, int N, class Wat>
__device__ __forceinline__ void codes_of(const float (&w)[N], float s, float r, int (&u)[N],
                                         Wat wat) {
  constexpr float MAGIC = kMagic + static_cast<float>(OFF);
  float near = 1.f;
#pragma unroll
  for (int e = 0; e < N; ++e) {
    const float t = __fmaf_rn(w[e], r, MAGIC);
    u[e] = __float_as_int(t) - __float_as_int(kMagic);
    const float dd = __fmaf_rn(w[e], r, __fsub_rn(MAGIC, t));
    near = fminf(near, fabsf(__fsub_rn(fabsf(dd), 0.5f)));
  }
  if (near <= 0x1p-18f) {  // unrolled: u stays in registers
#pragma unroll
    for (int e = 0; e < N; ++e) u[e] = fix_tie<OFF>(wat(e), s, r, u[e]);
  }
}

}  // namespace sss
