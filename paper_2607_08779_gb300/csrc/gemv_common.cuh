// gemv_common.cuh -- pieces shared by the decode GEMV kernels
// (gemv_stream.cu, gemv_batch.cu): mma.sync m16n8k16 wrappers,
// shared-memory loads, and the code-pair unpack of the batched kernel
// (fields at bit 0, 2 or 4 of each fp16 half).
#pragma once

#include <stdint.h>

#include "sss_internal.cuh"

namespace sss {
namespace gv {

// fp16 pairs per 32-code sub-chunk: every width uses 16 (q=3 merges its two
// bit planes into 3-bit fields before the mma)
constexpr int NP = 16;

__device__ __forceinline__ uint32_t su32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// the same with a zero accumulator in (the first mma of a chain)
__device__ __forceinline__ void mma16816_z(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                           uint32_t a3, uint32_t b0, uint32_t b1) {
  const float z = 0.f;
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%10,%10,%10};\n"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(z));
}
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr));
  return v;
}

// Activation pair p (0..15) of a 32-code sub-chunk: its two elements and
// the multiplier that undoes the power of two the code's bit position
// carries in the fp16 subnormal.
//   q=4: p = 4w + i covers elements 8w+i and 8w+i+4 (nibble i&1 of a byte
//        pair, so odd i sits 4 bits up: multiplier 1/16);
//   q=2 and q=3: p = 8w + e covers elements 16w+e and 16w+e+8, whose 2-bit
//        fields land at bit 2(e mod 3) after the unpack's shift.
template <int Q>
__device__ __forceinline__ void pair_desc(int p, int& ea, int& eb, float& mult) {
  if (Q == 4) {
    const int w = p >> 2, i = p & 3;
    ea = 8 * w + i;
    eb = ea + 4;
    mult = (i & 1) ? 0.0625f : 1.f;
  } else {
    const int w = p >> 3, e = p & 7;
    ea = 16 * w + e;
    eb = ea + 8;
    const int m3 = e % 3;
    mult = (m3 == 0) ? 1.f : (m3 == 1 ? 0.25f : 0.0625f);
  }
}

// Pair p of one sub-chunk's code words as an fp16x2 subnormal operand.
//   q=4: w[0..3] hold the 32 nibbles;
//   q=2: w[0..1] hold the 32 2-bit codes;
//   q=3: w[0..1] hold the low 2-bit plane, w[2] the high bit of all 32
//        codes; the high bit is moved two places above its low field, so
//        the operand is the 3-bit code at the same bit position.
template <int Q>
__device__ __forceinline__ uint32_t unpack_pair(const uint32_t* w, int p) {
  if constexpr (Q == 4) {
    const uint32_t v = (p & 2) ? (w[p >> 2] >> 8) : w[p >> 2];
    return v & ((p & 1) ? 0x00F000F0u : 0x000F000Fu);
  } else {
    const int e = p & 7, pos = 2 * (e % 3);
    const uint32_t word = w[(p >> 3) & 1];
    const uint32_t v = e < 3 ? word : (e < 6 ? (word >> 6) : (word >> 12));
    const uint32_t lo = v & (0x00030003u << pos);
    if constexpr (Q == 2) {
      return lo;
    } else {
      // high bits of elements 16w+e and 16w+e+8 at bits e and 16+e
      const uint32_t hw = __byte_perm(w[2], 0u, (p >> 3) ? 0x4342u : 0x4140u);
      const int d = pos + 2 - e;
      const uint32_t hs = d >= 0 ? (hw << d) : (hw >> (-d));
      return lo | (hs & (0x00040004u << pos));
    }
  }
}

}  // namespace gv
}  // namespace sss
