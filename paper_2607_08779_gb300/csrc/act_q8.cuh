// act_q8.cuh -- Q8_0 activation quantization (narrow range, blocks of 32):
// the 8-bit activation format the paper's runtime pairs with the few-bit
// weight formats (Sec. 5, "Composition with PTQ methods"; Appendix C).
//
// Per block of 32 consecutive activations of one token:
//   M = max |x|,  d = fl32(M / 127)                (one IEEE fp32 division)
//   q = clip(RNE(x / d), -127, 127)                 (exact quotient, ties to even)
//   stored scale fl16(d); the block's value is fl16(d) * q.
// A block of zeros gives q = 0 and d = +0; a block holding NaN or Inf gives
// q = 0, d = +0 and SSS_FLAG_NONFINITE; a d that overflows fp16 raises
// SSS_FLAG_RANGE.
#pragma once

#include <stdint.h>

#include "sss_internal.cuh"

namespace sss {

// RNE(x / d) of the exact quotient clipped to [-127, 127], given
// r = RN(1/d): x*r is within 127 * 2^-24 < 2^-17 of x/d, so away from a
// half-integer (farther than 2^-14) the fused multiply-add rounding of x*r
// decides it; near one the sign of the single-rounding residual x - h*d
// does (a zero residual is an exact tie -> even).
__device__ __forceinline__ int q8_code(float x, float d, float r) {
  constexpr float MAGIC = 12582912.0f;  // 1.5 * 2^23
  const float t = __fmaf_rn(x, r, MAGIC);
  const float c = __fsub_rn(t, MAGIC);
  int q = __float_as_int(t) - __float_as_int(MAGIC);
  const float dd = __fmaf_rn(x, r, -c);  // x*r - c
  if (fabsf(__fsub_rn(fabsf(dd), 0.5f)) <= 0x1p-14f) {
    const float h = __fadd_rn(c, copysignf(0.5f, dd));  // the half-integer at stake
    const float e = __fmaf_rn(-h, d, x);                 // x - h*d, one rounding (d > 0)
    const float lo = __fsub_rn(h, 0.5f), hi = __fadd_rn(h, 0.5f);
    float cc;
    if (e > 0.f) {
      cc = hi;
    } else if (e < 0.f) {
      cc = lo;
    } else {
      cc = (static_cast<int>(lo) & 1) ? hi : lo;
    }
    q += static_cast<int>(__fsub_rn(cc, c));
  }
  return max(-127, min(127, q));
}

// The block's scale from its max |x| and non-finite flag: fp32 d (0 for a
// zero or non-finite block) and its fp16 bits; flags as above.
__device__ __forceinline__ float q8_scale(float amax, bool bad, uint16_t* d16, unsigned* flags) {
  if (bad || amax == 0.f) {
    *d16 = 0;
    if (bad) *flags |= SSS_FLAG_NONFINITE;
    return 0.f;
  }
  const float d = __fdiv_rn(amax, 127.f);
  *d16 = __half_as_ushort(__float2half_rn(d));
  if ((*d16 & 0x7fffu) == 0x7c00u) *flags |= SSS_FLAG_RANGE;
  return d;
}

}  // namespace sss
