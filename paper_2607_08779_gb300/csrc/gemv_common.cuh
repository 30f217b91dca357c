// gemv_common.cuh -- pieces of the batch-1 streaming GEMV (gemv_stream.cu):
// bounded mbarrier waits, the fp16-subnormal
// code unpack feeding mma.sync m16n8k16, and the staging of the activation
// vector in mma order with the per-sub-chunk sums of the Appendix B.3
// row-sum term.
#pragma once

#include <stdint.h>

#include "sss_internal.cuh"

namespace sss {
namespace gv {

constexpr uint64_t kWaitNs = 1000000000ull;

template <int Q>
struct SQ;
template <>
struct SQ<4> {
  // pairs per sub-chunk; 32-bit code words per (row, sub-chunk)
  static constexpr int NP = 16, NW = 4;
};
template <>
struct SQ<2> {
  static constexpr int NP = 16, NW = 2;
};
template <>
struct SQ<3> {
  static constexpr int NP = 32, NW = 3;
};

__device__ __forceinline__ uint32_t su32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t gtime() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void bar_init(uint64_t* b, uint32_t c) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(b)), "r"(c) : "memory");
}
__device__ __forceinline__ void bar_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(su32(b)) : "memory");
}
__device__ __forceinline__ void bar_expect(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(su32(b)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool bar_try(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(su32(b)), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded wait; false if it gave up (own limit, or *abort raised elsewhere)
__device__ __forceinline__ bool bar_wait(uint64_t* b, uint32_t parity, volatile int* abort) {
  if (bar_try(b, parity)) return true;
  const uint64_t t0 = gtime();
  for (uint32_t it = 1;; ++it) {
    if (bar_try(b, parity)) return true;
    if ((it & 255u) == 0) {
      if (*abort) return false;
      if (gtime() - t0 > kWaitNs) {
        *abort = 1;
        return false;
      }
    }
  }
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
__device__ __forceinline__ float2 lds64f(uint32_t addr) {
  float2 v;
  asm volatile("ld.shared.v2.f32 {%0,%1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr));
  return v;
}

// activation pair p of a 32-code sub-chunk: (element a, element b, multiplier)
template <int Q>
__device__ __forceinline__ void pair_desc(int p, int& ea, int& eb, float& mult) {
  if (Q == 4) {
    const int w = p >> 2, i = p & 3;
    ea = 8 * w + i;
    eb = ea + 4;
    mult = (i & 1) ? 0.0625f : 1.f;
  } else if (Q == 2 || p < 16) {
    const int w = p >> 3, e = p & 7;
    ea = 16 * w + e;
    eb = ea + 8;
    const int m3 = e % 3;
    mult = (m3 == 0) ? 1.f : (m3 == 1 ? 0.25f : 0.0625f);
  } else {
    const int j = p - 16;
    ea = j;
    eb = j + 16;
    mult = 4.f / static_cast<float>(1 << (j & 3));
  }
}

// pair p of a sub-chunk's words as an fp16x2 subnormal operand
template <int Q>
__device__ __forceinline__ uint32_t unpack_pair(const uint32_t* w, int p) {
  if constexpr (Q == 4) {
    const uint32_t v = (p & 2) ? (w[p >> 2] >> 8) : w[p >> 2];
    return v & ((p & 1) ? 0x00F000F0u : 0x000F000Fu);
  } else {
    if (Q == 2 || p < 16) {
      const int e = p & 7;
      const uint32_t word = w[(p >> 3) & 1];
      const uint32_t v = e < 3 ? word : (e < 6 ? (word >> 6) : (word >> 12));
      return v & (0x00030003u << (2 * (e % 3)));
    } else {
      const int j = p - 16;
      return (w[2] >> (4 * (j >> 2))) & (0x00010001u << (j & 3));
    }
  }
}

// Bytes of one 32-code sub-chunk's activations in shared memory, arranged
// as the mma B operand (NP fp16 pairs) plus 16 bytes of padding that spread
// the eight columns' rows over the banks.
template <int Q>
struct XLayout {
  static constexpr int XPITCH = SQ<Q>::NP * 4 + 16;
};

// Stage the bf16 activations x[0..32*nsc) in shared memory for the mma B
// operand: sub-chunk i (32 elements) becomes NP fp16 pairs in unpack order,
// each pre-divided by the power of two its code position carries, at
// xs + i*XPITCH; bias[i] = its sum times 2^-24 (min-max grid) or times
// -2^(q-1) * 2^-24 (symmetric grids).  Threads tid = 0..nthreads-1 share the
// work; the caller synchronises afterwards.
template <int Q, bool ASYM>
__device__ __forceinline__ void stage_x(const uint16_t* x, int nsc, unsigned char* xs, float* bias,
                                        int tid, int nthreads) {
  using SL = XLayout<Q>;
  constexpr int NP = SQ<Q>::NP;
  constexpr int HALF = 1 << (Q - 1);
  for (int i = tid; i < nsc; i += nthreads) {
    const uint4* src = reinterpret_cast<const uint4*>(x + static_cast<int64_t>(i) * 32);
    uint4 v[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) v[c] = __ldg(src + c);
    float xv[32];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const uint32_t wv[4] = {v[c].x, v[c].y, v[c].z, v[c].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        xv[8 * c + 2 * e] = __uint_as_float(wv[e] << 16);
        xv[8 * c + 2 * e + 1] = __uint_as_float(wv[e] & 0xFFFF0000u);
      }
    }
    float sum = 0.f;
#pragma unroll
    for (int e = 0; e < 32; ++e) sum += xv[e];
    uint32_t pr[NP];
#pragma unroll
    for (int p = 0; p < NP; ++p) {
      int ea, eb;
      float mult;
      pair_desc<Q>(p, ea, eb, mult);
      __half2 hv = __floats2half2_rn(xv[ea] * mult, xv[eb] * mult);
      pr[p] = *reinterpret_cast<uint32_t*>(&hv);
    }
    unsigned char* dst = xs + static_cast<size_t>(i) * SL::XPITCH;
#pragma unroll
    for (int c = 0; c < NP / 4; ++c)
      *reinterpret_cast<uint4*>(dst + 16 * c) = make_uint4(pr[4 * c], pr[4 * c + 1], pr[4 * c + 2], pr[4 * c + 3]);
    bias[i] = ASYM ? sum * 0x1p-24f : -static_cast<float>(HALF) * 0x1p-24f * sum;
  }
}

}  // namespace gv
}  // namespace sss
