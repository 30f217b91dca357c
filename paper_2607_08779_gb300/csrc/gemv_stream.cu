// gemv_stream.cu -- persistent, warp-specialised batch-1 decode GEMV over
// packed q-bit codes (sm_103a), the streaming path of sss_gemv and
// sss_gemv_multi.
//
// Same arithmetic as gemv.cu (Appendix B.3 expansion; codes unpacked as fp16
// subnormals into mma.sync m16n8k16 with one B column per 32-code
// sub-chunk; per-group scale and the row-sum term in fp32), organised for
// streaming bandwidth:
//
//  * persistent CTAs of 16 warps, one per SM, walking 16-row tiles of all
//    jobs (several weight matrices sharing one activation vector, e.g. a
//    fused q/k/v projection) round-robin;
//  * the 16 warps form groups of KW = 1..16 warps (chosen per launch to
//    balance the work); a group owns one tile at a time and its warps split
//    the tile's units (256 codes of every row) round-robin;
//  * every lane loads the exact bytes it will multiply (its two sub-chunks of
//    rows g and g+8, and their scales) straight into a ring of registers,
//    D-1 units ahead of use -- 512 threads keep ~100 KB per SM in flight.
//    (Measured on this GPU: the bulk-copy/TMA engine streams this pattern at
//    ~4 TB/s at most, plain loads from all warps at ~6.5 TB/s; staging the
//    codes through shared memory saturated the shared-memory instruction
//    queue.)  Shared memory holds only the activation operand;
//  * with KW > 1 a tile's partials meet in a double-buffered shared array
//    behind mbarriers and only the reducing warp waits; with KW = 1 a warp
//    owns whole tiles and writes y directly.
//
// The activation vector is staged once per CTA, after the grid-dependency
// wait of a programmatic dependent launch (weights may be prefetched before
// it only when the caller states they are not written upstream).  Every
// mbarrier wait is bounded; on expiry the kernel raises SSS_FLAG_TIMEOUT and
// winds down without further waits.
#include <cuda.h>

#include <stdint.h>
#include <string.h>

#include <algorithm>

#include "sss_internal.cuh"

namespace sss {
namespace {

constexpr int kWarps = 16;                // warps per CTA
constexpr int kThreads = kWarps * 32;
constexpr int kMaxJobs = 4;
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

struct StreamJob {
  const uint8_t* codes;
  const uint16_t* scales;
  const uint16_t* mins;
  float* y;
  int64_t n;
  int64_t tile0;  // first global tile index of this job
};

struct StreamArgs {
  StreamJob job[kMaxJobs];
  int njobs;
  const uint16_t* x;  // bf16 [k]
  int64_t k;
  int64_t ntiles;
  int lgkw;            // log2(warps per tile)
  int early_weights;   // prefetch weights before the grid-dependency wait
  uint32_t* status;
};

// Bytes of one 32-code sub-chunk's activations in shared memory, arranged
// as the mma B operand (NP fp16 pairs) plus 16 bytes of padding that spread
// the eight columns' rows over the banks.
template <int Q>
struct XLayout {
  static constexpr int XPITCH = SQ<Q>::NP * 4 + 16;
};

template <int Q, bool ASYM, int G, int D>
__global__ void __launch_bounds__(kThreads, 1) gemv_stream_kernel(const __grid_constant__ StreamArgs a) {
  using SL = XLayout<Q>;
  constexpr int NP = SQ<Q>::NP;
  constexpr int HALF = 1 << (Q - 1);
  constexpr int LGG = G == 32 ? 5 : (G == 64 ? 6 : 7);
  constexpr int R = 16;
  extern __shared__ __align__(128) unsigned char smem[];

  const int nsc = static_cast<int>(a.k / 32);  // 32-code sub-chunks per row
  const int nunits = nsc / 8;                  // units of 256 codes
  const int64_t nG = a.k / G;
  const int64_t row_bytes = a.k * Q / 8;
  const int lgkw = a.lgkw;
  const int KW = 1 << lgkw;                    // warps per tile
  const int ngrp = kWarps >> lgkw;             // tiles in flight per CTA

  // ---- shared memory carve-up ----
  unsigned char* xs = smem;                                                 // [nsc][XPITCH]
  float* bias = reinterpret_cast<float*>(xs + static_cast<size_t>(nsc) * SL::XPITCH);  // [nsc]
  unsigned char* zero = reinterpret_cast<unsigned char*>(bias + nsc);      // 128 B
  uint64_t* pready = reinterpret_cast<uint64_t*>(zero + 128);              // [kWarps][2]
  uint64_t* pfree = pready + 2 * kWarps;                                   // [kWarps][2]
  float* part = reinterpret_cast<float*>(pfree + 2 * kWarps);              // [kWarps][2][R]
  volatile int* abort = reinterpret_cast<volatile int*>(part + 2 * kWarps * R);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;
  const int grp = warp >> lgkw;        // this warp's group (one tile at a time)
  const int kw = warp & (KW - 1);      // its share of the tile's k-range

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2 * kWarps; ++i) {
      bar_init(&pready[i], KW * 8);  // the 8 quad leaders of every warp of a group
      bar_init(&pfree[i], 1);
    }
    *abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  for (int i = threadIdx.x; i < 32; i += blockDim.x) reinterpret_cast<uint32_t*>(zero)[i] = 0u;
  // allow the next kernel in the stream to be scheduled as SMs free up
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  // ---- this warp's stream: tiles t = (blockIdx.x * ngrp + grp) + i * (gridDim.x
  // * ngrp), i = 0, 1, ..., and in each tile the units u = kw, kw + KW, ... ----
  const int64_t tstride = static_cast<int64_t>(gridDim.x) * ngrp;
  const int64_t tfirst = static_cast<int64_t>(blockIdx.x) * ngrp + grp;
  const int64_t my_tiles = tfirst < a.ntiles ? (a.ntiles - tfirst + tstride - 1) / tstride : 0;
  const bool has_units = kw < nunits;

  // This warp's flat unit stream: unit k is unit u = kw + (k % upw) * KW of
  // its i = k / upw-th tile, upw = units per tile for this warp.
  const int upw = has_units ? (nunits - kw + KW - 1) >> lgkw : 0;
  const int64_t total = my_tiles * upw;

  // fetch cursor: tile index, unit, and that tile's row pointers
  int64_t fi = 0;
  int fu = kw;
  const uint8_t* frow[2] = {nullptr, nullptr};
  const uint16_t* fsrow[2] = {nullptr, nullptr};
  const uint16_t* fmrow[2] = {nullptr, nullptr};
  auto set_tile = [&](int64_t i) {
    if (i >= my_tiles) return;
    const int64_t t = tfirst + i * tstride;
    int j = 0;
    while (j + 1 < a.njobs && t >= a.job[j + 1].tile0) ++j;
    const StreamJob& jb = a.job[j];
    const int64_t row0 = (t - jb.tile0) * R;
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      int64_t r = row0 + gq + 8 * hh;
      if (r >= jb.n) r = jb.n - 1;  // a valid row; results past n are never stored
      frow[hh] = jb.codes + r * row_bytes;
      fsrow[hh] = jb.scales + r * nG;
      if constexpr (ASYM) fmrow[hh] = jb.mins + r * nG;
    }
  };
  // the registers of one unit: code words of (row half hh, column parity h),
  // and the aligned fp16 scale (min) pair of each row
  struct Regs {
    uint32_t w[2][2][4];
    uint32_t s[2], m[2];
  };
  auto fetch = [&](Regs& rg) {
    if (fi >= my_tiles) return;
    const int s0 = fu * 8 + 2 * tq;  // the lane's first sub-chunk (column 2tq)
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const uint8_t* rp = frow[hh];
      if constexpr (Q == 4) {  // sub-chunk s at byte 16s
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const uint4 v = __ldcs(reinterpret_cast<const uint4*>(rp + 16 * (s0 + h)));
          rg.w[hh][h][0] = v.x; rg.w[hh][h][1] = v.y; rg.w[hh][h][2] = v.z; rg.w[hh][h][3] = v.w;
        }
      } else if constexpr (Q == 2) {  // sub-chunks s0, s0+1 at bytes 8s: 16 contiguous bytes
        const uint4 v = __ldcs(reinterpret_cast<const uint4*>(rp + 8 * s0));
        rg.w[hh][0][0] = v.x; rg.w[hh][0][1] = v.y;
        rg.w[hh][1][0] = v.z; rg.w[hh][1][1] = v.w;
      } else {  // q=3: two low-plane words and one high-plane word per sub-chunk
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int e0 = (s0 + h) * 32;
          const int gbyte = (e0 >> LGG) * (3 * G / 8);
          const int sc = (e0 & (G - 1)) >> 5;
          const uint32_t* lo = reinterpret_cast<const uint32_t*>(rp + gbyte + 8 * sc);
          rg.w[hh][h][0] = __ldcs(lo);
          rg.w[hh][h][1] = __ldcs(lo + 1);
          rg.w[hh][h][2] = __ldcs(reinterpret_cast<const uint32_t*>(rp + gbyte + G / 4 + 4 * sc));
        }
      }
      const int gpair = ((s0 << 5) >> LGG) & ~1;
      rg.s[hh] = __ldcs(reinterpret_cast<const uint32_t*>(fsrow[hh] + gpair));
      if constexpr (ASYM) rg.m[hh] = __ldcs(reinterpret_cast<const uint32_t*>(fmrow[hh] + gpair));
    }
    fu += KW;
    if (fu >= nunits) {
      fu = kw;
      ++fi;
      set_tile(fi);
    }
  };

  Regs ring[D];
  set_tile(0);
  if (!a.early_weights) asm volatile("griddepcontrol.wait;" ::: "memory");
#pragma unroll
  for (int d = 0; d < D - 1; ++d)
    if (d < total) fetch(ring[d]);
  asm volatile("griddepcontrol.wait;" ::: "memory");  // x is produced upstream

  // ---- stage the activations in mma order, and per-sub-chunk sums ----
  for (int i = threadIdx.x; i < nsc; i += kThreads) {
    const uint4* src = reinterpret_cast<const uint4*>(a.x + static_cast<int64_t>(i) * 32);
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
  __syncthreads();

  bool ok = true;
  float acc[2] = {0.f, 0.f};
  int64_t ci = 0;   // tile of the unit being computed
  int cu = kw;      // the unit
  auto compute = [&](const Regs& rg) {
    const int u = cu;
    // h=0 mmas only write even columns and h=1 mmas odd ones: the lane's
    // column 2tq is in dh[0] and 2tq+1 in dh[1]
    float dh[2][4];
#pragma unroll
    for (int h = 0; h < 2; ++h) dh[h][0] = dh[h][1] = dh[h][2] = dh[h][3] = 0.f;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      // column gq of B carries sub-chunk u*8 + gq: active for this h iff it
      // is this lane's own sub-chunk (gq == 2tq + h); others read zeros
      const unsigned char* xp =
          (gq == 2 * tq + h) ? xs + static_cast<size_t>(u * 8 + gq) * SL::XPITCH : zero;
#pragma unroll
      for (int jm = 0; jm < NP / 2; jm += 2) {
        const uint4 bv = *reinterpret_cast<const uint4*>(xp + jm * 8);
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          const int p = 2 * (jm + jj);
          mma16816(dh[h], unpack_pair<Q>(rg.w[0][h], p), unpack_pair<Q>(rg.w[1][h], p),
                   unpack_pair<Q>(rg.w[0][h], p + 1), unpack_pair<Q>(rg.w[1][h], p + 1),
                   jj ? bv.z : bv.x, jj ? bv.w : bv.y);
        }
      }
    }
    // per-group scale (and min) of this lane's two columns
    const int s0 = u * 8 + 2 * tq;
    const int sel0 = ((s0 << 5) >> LGG) & 1, sel1 = (((s0 + 1) << 5) >> LGG) & 1;
    const float bb0 = bias[s0], bb1 = bias[s0 + 1];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const float2 sf = __half22float2(*reinterpret_cast<const __half2*>(&rg.s[hh]));
      const float s_0 = sel0 ? sf.y : sf.x;
      const float s_1 = sel1 ? sf.y : sf.x;
      const float d0 = dh[0][2 * hh], d1 = dh[1][2 * hh + 1];
      if constexpr (ASYM) {
        const float2 mf = __half22float2(*reinterpret_cast<const __half2*>(&rg.m[hh]));
        acc[hh] += s_0 * d0 + (sel0 ? mf.y : mf.x) * bb0 + s_1 * d1 + (sel1 ? mf.y : mf.x) * bb1;
      } else {
        acc[hh] += s_0 * (d0 + bb0) + s_1 * (d1 + bb1);
      }
    }
  };
  auto tile_end = [&](int64_t i) {
    const int64_t t = tfirst + i * tstride;
    int j = 0;
    while (j + 1 < a.njobs && t >= a.job[j + 1].tile0) ++j;
    const StreamJob& jb = a.job[j];
    const int64_t row0 = (t - jb.tile0) * R;
    float v[2];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      float x = acc[hh];
      x += __shfl_xor_sync(0xffffffffu, x, 1);
      x += __shfl_xor_sync(0xffffffffu, x, 2);
      v[hh] = x;
      acc[hh] = 0.f;
    }
    if (KW == 1) {
      if (tq == 0) {
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int64_t r = row0 + gq + 8 * hh;
          if (r < jb.n) jb.y[r] = v[hh] * 0x1p24f;
        }
      }
      return;
    }
    // the group's KW partials meet behind mbarriers; only the reducing warp
    // (kw == i % KW) waits for them
    const int b = static_cast<int>(i & 1);
    const uint32_t use = static_cast<uint32_t>(i >> 1) & 1u;
    float* pb = part + (static_cast<size_t>(grp) * 2 + b) * KW * R;
    uint64_t* rdy = &pready[grp * 2 + b];
    uint64_t* fre = &pfree[grp * 2 + b];
    if (tq == 0) {
      if (!bar_wait(fre, use ^ 1u, abort)) ok = false;
      pb[kw * R + gq] = v[0];
      pb[kw * R + gq + 8] = v[1];
      bar_arrive(rdy);
    }
    if (kw == static_cast<int>(i & (KW - 1))) {
      if (!bar_wait(rdy, use, abort)) ok = false;
      if (lane < R) {
        float sum = 0.f;
        for (int c = 0; c < KW; ++c) sum += pb[c * R + lane];
        const int64_t r = row0 + lane;
        if (r < jb.n && ok) jb.y[r] = sum * 0x1p24f;
      }
      __syncwarp();
      if (lane == 0) bar_arrive(fre);
    }
  };

  // warps without units still take part in every tile's reduction
  if (upw == 0) {
    for (int64_t i = 0; i < my_tiles; ++i) tile_end(i);
  }
  // the units, D at a time so the register ring is indexed at compile time;
  // unit k + D - 1 is loaded while unit k is computed
  for (int64_t k0 = 0; k0 < total; k0 += D) {
#pragma unroll
    for (int r = 0; r < D; ++r) {
      const int64_t k = k0 + r;
      if (k < total) {
        if (k + D - 1 < total) fetch(ring[(r + D - 1) % D]);
        compute(ring[r]);
        cu += KW;
        if (cu >= nunits) {
          tile_end(ci);
          cu = kw;
          ++ci;
        }
      }
    }
  }
  if (*abort && threadIdx.x == 0 && a.status != nullptr) atomicOr(a.status, SSS_FLAG_TIMEOUT);
}

template <int Q, bool ASYM>
size_t smem_bytes(int64_t k, int depth) {
  using SL = XLayout<Q>;
  const int64_t nsc = k / 32;
  // activations | sums | zeros | 4*kWarps barriers | partials | flag
  (void)depth;
  return static_cast<size_t>(nsc) * SL::XPITCH +
         4 * nsc + 128 + 8 * 4 * kWarps + 4 * 2 * kWarps * 16 + 16;
}

template <int Q, bool ASYM, int G, int D>
cudaError_t launch_d(StreamArgs& a, int grid, bool pdl, cudaStream_t stream) {
  const size_t smem = smem_bytes<Q, ASYM>(a.k, D);
  auto kern = gemv_stream_kernel<Q, ASYM, G, D>;
  cudaError_t e = ensure_smem(kern, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int Q, bool ASYM, int G>
cudaError_t launch_g(StreamArgs& a, int grid, bool pdl, cudaStream_t stream) {
  if (smem_bytes<Q, ASYM>(a.k, 0) > 227 * 1024) return cudaErrorNotSupported;
  return launch_d<Q, ASYM, G, (Q == 3 ? 3 : 4)>(a, grid, pdl, stream);
}

template <int Q, bool ASYM>
cudaError_t launch_q(const sss_qtensor_t* const* ts, StreamArgs& a, bool pdl,
                     cudaStream_t stream) {
  int64_t tiles = 0;
  for (int j = 0; j < a.njobs; ++j) {
    a.job[j].tile0 = tiles;
    tiles += (ts[j]->n + 15) / 16;
  }
  a.ntiles = tiles;
  // Warps per tile: the power of two that minimises the busiest warp's
  // units (rounds of tiles x units per warp per tile), preferring fewer
  // warps per tile (less reduction) on ties.
  const int sms = device_sm_count();
  const int64_t nunits = a.k / 256;
  int best = 0;
  int64_t best_cost = INT64_MAX;
  for (int lg = 0; lg <= 4; ++lg) {
    const int kwn = 1 << lg;
    if (kwn > 1 && kwn > nunits) break;
    const int64_t inflight = static_cast<int64_t>(sms) * (kWarps >> lg);
    const int64_t rounds = (tiles + inflight - 1) / inflight;
    const int64_t cost = rounds * ((nunits + kwn - 1) / kwn);
    if (cost < best_cost) {
      best_cost = cost;
      best = lg;
    }
  }
  a.lgkw = best;
  const int64_t per_cta = kWarps >> best;
  const int grid = static_cast<int>(std::max<int64_t>(
      1, std::min<int64_t>(sms, (tiles + per_cta - 1) / per_cta)));
  switch (ts[0]->group) {
    case 32: return launch_g<Q, ASYM, 32>(a, grid, pdl, stream);
    case 64: return launch_g<Q, ASYM, 64>(a, grid, pdl, stream);
    case 128: return launch_g<Q, ASYM, 128>(a, grid, pdl, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

bool gemv_stream_eligible(const sss_qtensor_t& t, const uint16_t* x) {
  auto al = [](const void* p, size_t b) { return (reinterpret_cast<uintptr_t>(p) % b) == 0; };
  if (t.k <= 0 || t.n <= 0) return false;
  if (t.k % 256 != 0) return false;             // whole 256-code units per row
  if ((t.k / t.group) % 2 != 0) return false;   // 4-byte scale pairs
  if (!al(t.codes, 16) || !al(t.scales, 4) || !al(x, 16)) return false;
  if (t.grid == SSS_GRID_ASYM && !al(t.mins, 4)) return false;
  // the staged activations and a 3-deep ring must fit in shared memory
  const int64_t nsc = t.k / 32;
  const int64_t xbytes = nsc * ((t.q == 3 ? 32 : 16) * 4 + 16 + 4);
  const int64_t slot = (2 * 2 * (t.q == 3 ? 3 : (t.q == 4 ? 4 : 2)) + 2 * (t.grid == SSS_GRID_ASYM ? 2 : 1)) * 128;
  return xbytes + 3 * kWarps * slot + 2048 <= 227 * 1024;
}

cudaError_t launch_gemv_stream(const sss_qtensor_t* const* ts, float* const* ys, int count,
                               const uint16_t* x, uint32_t flags, uint32_t* status,
                               cudaStream_t stream) {
  if (count < 1 || count > kMaxJobs) return cudaErrorInvalidValue;
  StreamArgs a;
  memset(&a, 0, sizeof a);
  a.njobs = count;
  a.x = x;
  a.k = ts[0]->k;
  a.early_weights = (flags & SSS_GEMV_WEIGHTS_READY) ? 1 : 0;
  a.status = status;
  for (int j = 0; j < count; ++j) {
    a.job[j].codes = ts[j]->codes;
    a.job[j].scales = ts[j]->scales;
    a.job[j].mins = ts[j]->mins;
    a.job[j].y = ys[j];
    a.job[j].n = ts[j]->n;
  }
  const bool pdl = (flags & SSS_GEMV_PDL) != 0;
  const bool asym = ts[0]->grid == SSS_GRID_ASYM;
  switch (ts[0]->q) {
    case 2: return asym ? launch_q<2, true>(ts, a, pdl, stream) : launch_q<2, false>(ts, a, pdl, stream);
    case 3: return asym ? launch_q<3, true>(ts, a, pdl, stream) : launch_q<3, false>(ts, a, pdl, stream);
    case 4: return asym ? launch_q<4, true>(ts, a, pdl, stream) : launch_q<4, false>(ts, a, pdl, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace sss
