// gemv_batch.cu -- decode GEMV for batches of 2..16 activation vectors over
// packed q-bit codes (sm_103a), the batched path of sss_gemv.
//
// y[b][r] = sum_k w^[r][k] x[b][k] with w^ the dequantised weight of
// eq:quantizer (Appendix B.3 product).  Unlike the batch-1 kernels, the
// batch fills the columns of the mma instead of sub-chunks, so the weight
// operand must already carry its scale:
//
//  * codes are unpacked in registers with the fp16 "magic number" form: the
//    code field OR-ed into the mantissa of 1024.0 is 1024 + u*2^p exactly
//    (p = the field's bit offset); one HSUB2 removes 1024 and the symmetric
//    offset 2^(q-1)*2^p, one HMUL2 applies the group scale (min-max grid:
//    HFMA2 with the scale and the min times 2^p).  The operand is
//    fp16(w^ * 2^p): the weight rounded once to fp16 (<= 2^-11 relative, as
//    in sss_gemm).  It fits fp16 while |w^| * 16 < 65520; a group whose
//    scale lets its codes pass that bound raises SSS_FLAG_RANGE (checked per
//    scale, conservatively: (|s| 2^(q-1), or |s| (2^q - 1) + |m|) * 16);
//  * x is staged per K slab in shared memory in mma-B order, pre-divided by
//    2^p, as fp16: 4 batch columns for batch 2..4, 8 for 5..8, 16 (two mma
//    column blocks) for 9..16, columns past the batch zero.  Each thread
//    loads four pieces of x before converting any, so staging costs about
//    one load latency;
//  * mma.sync m16n8k16: lane (g, t) feeds rows g and g+8 with codes of its
//    own two 32-code sub-chunks of each 256-code unit (the bytes it loads,
//    16-byte vector loads into a 2-deep register ring); the k order inside
//    an mma is free, and B holds x of batch row g at those codes (one
//    16-byte shared load per two mmas);
//  * persistent CTAs of 16 warps walk 16-row tiles; groups of KW warps share
//    a tile and split its units.  With KW > 1 each warp leaves its partial
//    of each tile in its own slot of a shared array, with no wait, and after
//    the slab the CTA sums each tile's partials in warp order; with KW = 1 a
//    warp writes y itself.  For each K slab the CTA stages x once and runs
//    all its tiles over it (later slabs add to y, in the same CTA, so the
//    result does not depend on timing).  The kernel has no data-dependent
//    waits, only CTA-wide barriers around the staging and the sums.
#include <cuda.h>

#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <type_traits>

#include "gemv_common.cuh"

namespace sss {
namespace {

using namespace gv;

constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
constexpr int kSmemMax = 227 * 1024;

struct BatchArgs {
  const uint8_t* codes;
  const uint16_t* scales;
  const uint16_t* mins;
  const uint16_t* x;  // bf16 [batch][k]
  float* y;           // [batch][n]
  int64_t n, k;
  int batch;
  int64_t ntiles;
  int lgkw;        // log2(warps per tile)
  int slab_units;  // units of 256 codes per x slab
  int rounds;      // tiles per warp group at most (the partial array's depth)
  uint32_t* status;
};

__device__ __forceinline__ uint32_t hsub2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
__device__ __forceinline__ uint32_t hmul2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}
__device__ __forceinline__ uint32_t hfma2(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t r;
  asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(c));
  return r;
}
__device__ __forceinline__ uint32_t f16x2_of(uint32_t h) { return h | (h << 16); }
// fp16 bits of 2^e times v (v an fp16 in the low half), exact for the
// normal range; computed as a multiply by a power of two
__device__ __forceinline__ uint32_t f16x2_scaled(uint32_t h, int e) {
  const uint32_t p2 = static_cast<uint32_t>((15 + e) << 10);  // fp16 2^e
  return hmul2(f16x2_of(h), f16x2_of(p2));
}

// Bit offset inside its 16-bit half of the field pair p of a sub-chunk after
// the unpack's word shift (as unpack_pair): q=4: 0 or 4; q=2/3: 0, 2 or 4.
template <int Q>
__device__ __forceinline__ constexpr int pair_pos(int p) {
  return Q == 4 ? ((p & 1) ? 4 : 0) : 2 * ((p & 7) % 3);
}

// pair p of one sub-chunk's code words as fp16x2 (1024 + u*2^pos)
template <int Q>
__device__ __forceinline__ uint32_t magic_pair(const uint32_t* w, int p) {
  return unpack_pair<Q>(w, p) | 0x64006400u;
}

// NBC = batch columns of the staged x: 4 (batch 2..4), 8 (5..8) or 16
// (9..16).  An mma covers 8 columns; with NBC = 4 only lanes 0..15 (columns
// 0..3) have entries of their own, and lanes 16..31 read those of lane - 16,
// so columns 4..7 repeat columns 0..3 and their results are dropped.
template <int NBC>
struct XShape {
  static constexpr int NBLK = NBC < 8 ? 1 : NBC / 8;  // mma column blocks
  static constexpr int LS = NBC < 8 ? 16 : 32;        // lanes with entries per block
  static constexpr int XU = 8 * NBLK * LS * 16;       // staged x bytes per unit
};

template <int Q, bool ASYM, int G, int NBC, int D>
__global__ void __launch_bounds__(kThreads, 1) gemv_batch_kernel(const __grid_constant__ BatchArgs a) {
  using XS = XShape<NBC>;
  constexpr int NBLK = XS::NBLK;
  constexpr int LS = XS::LS;
  constexpr int XU = XS::XU;
  constexpr int R = 16;
  constexpr int HALF = 1 << (Q - 1);
  constexpr int UB = 32 * Q;                // code bytes of one row in one unit
  constexpr int SPU = 256 / G;              // scales of one row in one unit
  extern __shared__ __align__(128) unsigned char smem[];

  const int nunits = static_cast<int>(a.k / 256);
  const int64_t nG = a.k / G;
  const int64_t row_bytes = a.k * Q / 8;
  const int lgkw = a.lgkw;
  const int KW = 1 << lgkw;
  const int ngrp = kWarps >> lgkw;
  const int SK = a.slab_units;
  const int nslabs = (nunits + SK - 1) / SK;

  // ---- shared memory: x slab [SK][8][NBLK][LS] x 16 B | row partials
  // [ngrp][rounds][KW][NBC][R] fp32 (KW > 1) ----
  unsigned char* xs = smem;
  float* part = reinterpret_cast<float*>(xs + static_cast<size_t>(SK) * XU);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;
  const int grp = warp >> lgkw;
  const int kw = warp & (KW - 1);
  const uint32_t xs_a = su32(xs);

  // Entries of batch columns past the batch are zero (staging never writes
  // them); this touches nothing produced upstream, so it precedes the
  // grid-dependency wait.
  if (a.batch < NBC) {
    const int entries = SK * 8 * NBLK * LS;
    for (int e = threadIdx.x; e < entries; e += kThreads) {
      const int col = 8 * ((e / LS) % NBLK) + ((e % LS) >> 2);
      if (col >= a.batch)
        asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" ::"r"(xs_a + 16u * e), "r"(0u)
                     : "memory");
    }
  }
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  const int64_t tstride = static_cast<int64_t>(gridDim.x) * ngrp;
  const int64_t tfirst = static_cast<int64_t>(grp) * gridDim.x + blockIdx.x;
  const int64_t my_tiles = tfirst < a.ntiles ? (a.ntiles - tfirst + tstride - 1) / tstride : 0;
  // this warp's units of slab s: s*SK + kw + r*KW < min((s+1)*SK, nunits)
  auto units_in = [&](int s) -> int {
    const int su = min(SK, nunits - s * SK);
    return kw < su ? (su - kw + KW - 1) >> lgkw : 0;
  };

  const int lane_c = Q == 4 ? 32 * tq : (Q == 2 ? 16 * tq : (G == 128 ? 48 * (tq >> 1) + 16 * (tq & 1) : 24 * tq));
  const int lane_s = G == 32 ? 2 * tq : (G == 64 ? tq : (tq >> 1));

  // ---- fetch cursor over (slab, tile, unit) ----
  int fs = 0;
  int64_t fi = 0;
  int fleft = 0;
  const uint8_t* cp[2] = {nullptr, nullptr};
  const uint16_t* sp[2] = {nullptr, nullptr};
  const uint16_t* mp[2] = {nullptr, nullptr};
  auto set_fetch = [&]() {
    // advance to the next (slab, tile) holding units of this warp
    while (fs < nslabs) {
      const int ups = units_in(fs);
      if (ups > 0 && fi < my_tiles) {
        const int64_t row0 = (tfirst + fi * tstride) * R;
        const int u0 = fs * SK + kw;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          int64_t r = row0 + gq + 8 * hh;
          if (r >= a.n) r = a.n - 1;  // a valid row; results past n are never stored
          cp[hh] = a.codes + r * row_bytes + static_cast<int64_t>(u0) * UB + lane_c;
          sp[hh] = a.scales + r * nG + static_cast<int64_t>(u0) * SPU + lane_s;
          if constexpr (ASYM) mp[hh] = a.mins + r * nG + static_cast<int64_t>(u0) * SPU + lane_s;
        }
        fleft = ups;
        return;
      }
      ++fs;
      fi = 0;
    }
  };
  struct Regs {
    uint32_t w[2][2][4];
    uint32_t s[2], m[2];
  };
  auto fetch = [&](Regs& rg) {
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const uint8_t* rp = cp[hh];
      if constexpr (Q == 4) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const uint4 v = __ldcs(reinterpret_cast<const uint4*>(rp + 16 * h));
          rg.w[hh][h][0] = v.x; rg.w[hh][h][1] = v.y; rg.w[hh][h][2] = v.z; rg.w[hh][h][3] = v.w;
        }
      } else if constexpr (Q == 2) {
        const uint4 v = __ldcs(reinterpret_cast<const uint4*>(rp));
        rg.w[hh][0][0] = v.x; rg.w[hh][0][1] = v.y;
        rg.w[hh][1][0] = v.z; rg.w[hh][1][1] = v.w;
      } else if constexpr (G == 128) {
        const uint4 lo = __ldcs(reinterpret_cast<const uint4*>(rp));
        const uint2 hi = __ldcs(reinterpret_cast<const uint2*>(rp + 32 - 8 * (tq & 1)));
        rg.w[hh][0][0] = lo.x; rg.w[hh][0][1] = lo.y; rg.w[hh][0][2] = hi.x;
        rg.w[hh][1][0] = lo.z; rg.w[hh][1][1] = lo.w; rg.w[hh][1][2] = hi.y;
      } else {
        const uint2 p0 = __ldcs(reinterpret_cast<const uint2*>(rp));
        const uint2 p1 = __ldcs(reinterpret_cast<const uint2*>(rp + 8));
        const uint2 p2 = __ldcs(reinterpret_cast<const uint2*>(rp + 16));
        if constexpr (G == 32) {
          rg.w[hh][0][0] = p0.x; rg.w[hh][0][1] = p0.y; rg.w[hh][0][2] = p1.x;
          rg.w[hh][1][0] = p1.y; rg.w[hh][1][1] = p2.x; rg.w[hh][1][2] = p2.y;
        } else {
          rg.w[hh][0][0] = p0.x; rg.w[hh][0][1] = p0.y; rg.w[hh][0][2] = p2.x;
          rg.w[hh][1][0] = p1.x; rg.w[hh][1][1] = p1.y; rg.w[hh][1][2] = p2.y;
        }
      }
      if constexpr (G == 32) {
        rg.s[hh] = __ldcs(reinterpret_cast<const uint32_t*>(sp[hh]));
        if constexpr (ASYM) rg.m[hh] = __ldcs(reinterpret_cast<const uint32_t*>(mp[hh]));
      } else {
        rg.s[hh] = __ldcs(reinterpret_cast<const unsigned short*>(sp[hh]));
        if constexpr (ASYM) rg.m[hh] = __ldcs(reinterpret_cast<const unsigned short*>(mp[hh]));
      }
      cp[hh] += UB * KW;
      sp[hh] += SPU * KW;
      if constexpr (ASYM) mp[hh] += SPU * KW;
    }
    if (--fleft == 0) {
      ++fi;
      if (fi >= my_tiles) {
        ++fs;
        fi = 0;
      }
      set_fetch();
    }
  };

  // total units of this warp over all slabs and tiles
  int total = 0;
  for (int s = 0; s < nslabs; ++s) total += static_cast<int>(my_tiles) * units_in(s);

  float acc[NBLK][4];
#pragma unroll
  for (int nb = 0; nb < NBLK; ++nb)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[nb][e] = 0.f;

  // Stage slab s: x[n][32*(8u + sc) + e] for the slab's units u, in mma-B
  // order: the 16 bytes at (u, j2, nb, lane = 4g + t) hold, for batch
  // column n = 8nb + g, the activation pairs 4j2 .. 4j2+3 of quad t (quad
  // t's sub-chunk 2t + (j2 >> 2), pairs (4j2) & 15 .. (4j2+3) & 15), each
  // element pre-divided by 2^p: the B operands of two consecutive mmas.  One
  // item is 16 elements (half a sub-chunk) of one batch row; consecutive
  // items run along k, and a thread loads U items before converting any of
  // them, so their loads are in flight together (U = 4 for the first slab,
  // staged before the weight ring fills; 2 for later slabs, while the
  // ring's registers are live).
  auto slab_items = [&](int s) { return min(SK, nunits - s * SK) * 16 * a.batch; };
  auto stage_load = [&](int s, int base, auto& v) {
    constexpr int U = sizeof(v) / sizeof(v[0]);
    const int items = slab_items(s), per_row = items / a.batch;
#pragma unroll
    for (int c = 0; c < U; ++c) {
      const int it = base + c * kThreads;
      if (it < items) {
        const int n = it / per_row, w = it - n * per_row;  // w = 2 * sub-chunk + half
        const uint4* src = reinterpret_cast<const uint4*>(
            a.x + static_cast<int64_t>(n) * a.k + static_cast<int64_t>(s) * SK * 256 + 16 * w);
        v[c][0] = __ldg(src);
        v[c][1] = __ldg(src + 1);
      }
    }
  };
  auto stage_put = [&](int s, int base, const auto& v) {
    constexpr int U = sizeof(v) / sizeof(v[0]);
    const int items = slab_items(s), per_row = items / a.batch;
#pragma unroll
    for (int c = 0; c < U; ++c) {
      const int it = base + c * kThreads;
      if (it < items) {
        const int n = it / per_row, w = it - n * per_row;
        const int hf = w & 1, scu = w >> 1;
        const int ul = scu >> 3, sc = scu & 7;
        float xv[16];
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
          const uint32_t wv[4] = {v[c][cc].x, v[c][cc].y, v[c][cc].z, v[c][cc].w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            xv[8 * cc + 2 * e] = __uint_as_float(wv[e] << 16);
            xv[8 * cc + 2 * e + 1] = __uint_as_float(wv[e] & 0xFFFF0000u);
          }
        }
        uint32_t pr[8];
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
          int ea, eb;
          float mult;
          pair_desc<Q>(jj, ea, eb, mult);  // pair 8hf + jj, offsets within this half
          __half2 hv = __floats2half2_rn(xv[ea] * mult, xv[eb] * mult);
          pr[jj] = *reinterpret_cast<uint32_t*>(&hv);
        }
        // pair P = 8hf + jj of sub-chunk sc = 2t + h is quad t's pair
        // 16h + P: entry j2 = 4h + 2hf + (jj >> 2), 8-byte slot (jj >> 1) & 1
        const int t = sc >> 1, h = sc & 1;
#pragma unroll
        for (int qd = 0; qd < 2; ++qd) {
          const int j2 = 4 * h + 2 * hf + qd;
          const uint32_t dst = xs_a + static_cast<uint32_t>(
              ul * XU + ((j2 * NBLK + (n >> 3)) * LS + 4 * (n & 7) + t) * 16);
          asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(dst), "r"(pr[4 * qd]),
                       "r"(pr[4 * qd + 1]), "r"(pr[4 * qd + 2]), "r"(pr[4 * qd + 3])
                       : "memory");
        }
      }
    }
  };
  auto stage_from = [&](auto u_tag, int s, int start) {
    constexpr int U = decltype(u_tag)::value;
    for (int base = start; base < slab_items(s); base += U * kThreads) {
      uint4 v[U][2];
      stage_load(s, base, v);
      stage_put(s, base, v);
    }
  };

  // Every global access follows the grid-dependency wait.  Slab 0 of x is
  // staged before the weight ring is filled: its loads return from L2 in
  // well under a microsecond, but the shared-memory stores of its
  // conversion would otherwise wait behind the ring's DRAM loads in the
  // SM's load/store queue.  The barrier comes before the ring's loads too,
  // so no warp waits for another warp's loads to be issued.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  stage_from(std::integral_constant<int, 4>{}, 0, threadIdx.x);
  __syncthreads();
  Regs ring[D];
  set_fetch();
#pragma unroll
  for (int d = 0; d < D; ++d)
    if (d < total) fetch(ring[d]);

  // constants of the operand formation
  uint32_t off[3];
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    // fp16x2 of 1024 + 2^(q-1)*4^i (symmetric) or 1024 (min-max)
    const float o = 1024.f + (ASYM ? 0.f : static_cast<float>(HALF << (2 * i)));
    __half2 hv = __floats2half2_rn(o, o);
    off[i] = *reinterpret_cast<uint32_t*>(&hv);
  }

  // fp16 range of the operand: symmetric grids keep the largest |s| bit
  // pattern of each half (fp16 magnitudes order as their bits), the min-max
  // grid tests each group
  uint32_t smax = 0u;
  bool big = false;
  const uint32_t xlane = static_cast<uint32_t>(lane & (LS - 1)) * 16u;
  auto compute = [&](const Regs& rg, int ul) {
    const uint32_t xu = xs_a + static_cast<uint32_t>(ul * XU) + xlane;
    if constexpr (!ASYM) smax = __vmaxu2(smax, __vmaxu2(rg.s[0] & 0x7FFF7FFFu, rg.s[1] & 0x7FFF7FFFu));
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      // the fp16 scale (and min) of sub-chunk 2tq + h for rows gq, gq + 8
      uint32_t S[2], M[2][3];
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const uint32_t sb = G == 32 ? ((rg.s[hh] >> (16 * h)) & 0xFFFFu) : (rg.s[hh] & 0xFFFFu);
        S[hh] = f16x2_of(sb);
        if constexpr (ASYM) {
          const float sa = fabsf(__half2float(__ushort_as_half(static_cast<unsigned short>(sb))));
          const uint32_t mb = G == 32 ? ((rg.m[hh] >> (16 * h)) & 0xFFFFu) : (rg.m[hh] & 0xFFFFu);
          const float ma = fabsf(__half2float(__ushort_as_half(static_cast<unsigned short>(mb))));
          big |= (sa * static_cast<float>(2 * HALF - 1) + ma) * 16.f >= 65520.f;
#pragma unroll
          for (int i = 0; i < 3; ++i) M[hh][i] = i == 0 ? f16x2_of(mb) : f16x2_scaled(mb, 2 * i);
        }
      }
      auto deq = [&](int hh, int p) -> uint32_t {
        const int i = pair_pos<Q>(p) >> 1;  // 0, 1 or 2 (pos 0, 2, 4)
        const uint32_t t = hsub2(magic_pair<Q>(rg.w[hh][h], p), off[i]);
        if constexpr (ASYM) return hfma2(t, S[hh], M[hh][i]);
        else return hmul2(t, S[hh]);
      };
#pragma unroll
      for (int jm = 0; jm < 8; jm += 2) {
        uint4 bv[NBLK];
#pragma unroll
        for (int nb = 0; nb < NBLK; ++nb)
          bv[nb] = lds128(xu + static_cast<uint32_t>((((4 * h + (jm >> 1)) * NBLK + nb) * LS) * 16));
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          const int p = 2 * (jm + jj);
          const uint32_t a0 = deq(0, p), a1 = deq(1, p), a2 = deq(0, p + 1), a3 = deq(1, p + 1);
#pragma unroll
          for (int nb = 0; nb < NBLK; ++nb)
            mma16816(acc[nb], a0, a1, a2, a3, jj ? bv[nb].z : bv[nb].x, jj ? bv[nb].w : bv[nb].y);
        }
      }
    }
  };

  // ---- tile end: y = sum (first slab) or y += sum (later slabs).  KW = 1:
  // the warp owns the tile and writes y itself; KW > 1: the warp leaves its
  // partial in its own slot, summed after the slab ----
  auto tile_end = [&](int s, int64_t i) {
    if (KW == 1) {
      const int64_t row0 = (tfirst + i * tstride) * R;
#pragma unroll
      for (int nb = 0; nb < NBLK; ++nb)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int64_t r = row0 + gq + 8 * (e >> 1);
          const int b = 8 * nb + 2 * tq + (e & 1);
          if (r < a.n && b < a.batch) {
            float* yp = a.y + static_cast<int64_t>(b) * a.n + r;
            *yp = (s == 0 ? 0.f : *yp) + acc[nb][e];
          }
          acc[nb][e] = 0.f;
        }
      return;
    }
    float* pb = part + ((static_cast<size_t>(grp) * a.rounds + i) * KW + kw) * (NBC * R);
#pragma unroll
    for (int nb = 0; nb < NBLK; ++nb)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int b = 8 * nb + 2 * tq + (e & 1);
        if (b < NBC) pb[b * R + gq + 8 * (e >> 1)] = acc[nb][e];
        acc[nb][e] = 0.f;
      }
  };
  // the slab's sums of every tile's KW partials, in warp order (warps with
  // no unit in the slab left no partial)
  auto slab_sums = [&](int s) {
    const int kwn = min(KW, min(SK, nunits - s * SK));
    const int per_grp = a.rounds * NBC * R;
    for (int idx = threadIdx.x; idx < ngrp * per_grp; idx += kThreads) {
      const int g = idx / per_grp, rem = idx - g * per_grp;
      const int i = rem / (NBC * R), b = (rem / R) % NBC, row = rem % R;
      if (b >= a.batch) continue;
      const int64_t t = (static_cast<int64_t>(i) * ngrp + g) * gridDim.x + blockIdx.x;
      if (t >= a.ntiles) continue;
      const int64_t r = t * R + row;
      if (r >= a.n) continue;
      const float* pb = part + (static_cast<size_t>(g) * a.rounds + i) * KW * (NBC * R) + b * R + row;
      float sum = 0.f;
      for (int c = 0; c < kwn; ++c) sum += pb[c * (NBC * R)];
      float* yp = a.y + static_cast<int64_t>(b) * a.n + r;
      *yp = (s == 0 ? 0.f : *yp) + sum;
    }
  };

  // the units: unit gk of this warp's stream is computed from ring slot
  // gk % D, which then takes unit gk + D (the switch keeps every slot's
  // index a compile-time constant, so the ring stays in registers)
  int gk = 0, slot = 0;
  auto step = [&](Regs& rg, int ul) {
    compute(rg, ul);
    if (gk + D < total) fetch(rg);
  };
  for (int s = 0; s < nslabs; ++s) {
    if (s > 0) {
      __syncthreads();  // every warp done with the previous slab and its sums
      stage_from(std::integral_constant<int, 2>{}, s, threadIdx.x);
      __syncthreads();
    }
    const int ups = units_in(s);
    for (int64_t i = 0; i < my_tiles; ++i) {
      for (int r = 0; r < ups; ++r, ++gk) {
        const int ul = kw + r * KW;  // unit within the slab
        switch (slot) {
          case 0: step(ring[0], ul); break;
          case 1: if constexpr (D > 1) step(ring[1], ul); break;
          case 2: if constexpr (D > 2) step(ring[2], ul); break;
          default: if constexpr (D > 3) step(ring[3], ul); break;
        }
        slot = slot + 1 == D ? 0 : slot + 1;
      }
      tile_end(s, i);
    }
    if (KW > 1) {
      __syncthreads();
      slab_sums(s);
    }
  }
  if constexpr (!ASYM) {
    // |s| * 2^(q-1) * 16 >= 65520 exactly when |s| >= the fp16 value that
    // 4095 / 2^(q-1) rounds up to
    const uint32_t m = max(smax & 0xFFFFu, smax >> 16);
    big = m >= static_cast<uint32_t>(__half_as_ushort(__float2half_ru(4095.f / HALF)));
  }
  if (__any_sync(0xffffffffu, big) && lane == 0 && a.status != nullptr)
    atomicOr(a.status, SSS_FLAG_RANGE);
}

// Register ring depth: units of weights in flight per warp.  Two: with
// three the unit loop, bound by instruction issue, ran no faster and the
// first loads took longer to issue.
constexpr int ring_depth(int, bool, int) { return 2; }

template <int NBC>
size_t batch_smem(int slab_units, int kw, int ngrp, int rounds) {
  return static_cast<size_t>(slab_units) * XShape<NBC>::XU +
         (kw > 1 ? static_cast<size_t>(ngrp) * rounds * kw * NBC * 16 * 4 : 0);
}

template <int Q, bool ASYM, int G, int NBC>
cudaError_t launch_b(const sss_qtensor_t& t, BatchArgs& a, cudaStream_t stream) {
  const int nunits = static_cast<int>(t.k / 256);
  const int64_t tiles = (t.n + 15) / 16;
  a.ntiles = tiles;
  const int sms = device_sm_count();
  const int grid = static_cast<int>(std::min<int64_t>(sms, tiles));
  const int64_t per_cta = (tiles + grid - 1) / grid;
  // Warps per tile KW and slab size: minimise the busiest warp's units
  // (rounds of the CTA's tiles x that warp's units over the slabs) plus two
  // units' worth per extra slab (a CTA-wide barrier and a re-stage of x),
  // preferring fewer warps per tile on ties; the slab is the largest that
  // fits beside the partial array.
  int best = -1, best_sk = 0;
  int64_t best_cost = INT64_MAX;
  for (int lg = 0; (1 << lg) <= kWarps; ++lg) {
    const int kwn = 1 << lg;
    if (kwn > 1 && kwn > nunits) break;
    const int ngrp = kWarps >> lg;
    const int64_t rounds = (per_cta + ngrp - 1) / ngrp;
    const size_t parts = batch_smem<NBC>(0, kwn, ngrp, static_cast<int>(std::min<int64_t>(rounds, 1 << 20)));
    if (parts + XShape<NBC>::XU > static_cast<size_t>(kSmemMax)) continue;
    const int sk = static_cast<int>(std::min<size_t>(nunits, (kSmemMax - parts) / XShape<NBC>::XU));
    const int nslabs = (nunits + sk - 1) / sk;
    int64_t units = 0;
    for (int s = 0; s < nslabs; ++s) units += (std::min(sk, nunits - s * sk) + kwn - 1) / kwn;
    const int64_t cost = rounds * units + 2 * (nslabs - 1);
    if (cost < best_cost) {
      best_cost = cost;
      best = lg;
      best_sk = sk;
    }
  }
  if (best < 0) return cudaErrorNotSupported;
  a.lgkw = best;
  a.slab_units = best_sk;
  a.rounds = static_cast<int>((per_cta + (kWarps >> best) - 1) / (kWarps >> best));
  const size_t smem = batch_smem<NBC>(best_sk, 1 << best, kWarps >> best, a.rounds);
  auto kern = gemv_batch_kernel<Q, ASYM, G, NBC, ring_depth(Q, ASYM, NBC)>;
  cudaError_t e = ensure_smem(kern, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int Q, bool ASYM, int G>
cudaError_t launch_bn(const sss_qtensor_t& t, BatchArgs& a, cudaStream_t stream) {
  if (a.batch <= 4) return launch_b<Q, ASYM, G, 4>(t, a, stream);
  if (a.batch <= 8) return launch_b<Q, ASYM, G, 8>(t, a, stream);
  return launch_b<Q, ASYM, G, 16>(t, a, stream);
}

template <int Q, bool ASYM>
cudaError_t launch_bg(const sss_qtensor_t& t, BatchArgs& a, cudaStream_t stream) {
  switch (t.group) {
    case 32: return launch_bn<Q, ASYM, 32>(t, a, stream);
    case 64: return launch_bn<Q, ASYM, 64>(t, a, stream);
    case 128: return launch_bn<Q, ASYM, 128>(t, a, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

bool gemv_batch_eligible(const sss_qtensor_t& t, const uint16_t* x, int batch, const float* y) {
  auto al = [](const void* p, size_t b) { return (reinterpret_cast<uintptr_t>(p) % b) == 0; };
  if (batch < 2 || batch > 16) return false;
  if (t.k <= 0 || t.n <= 0 || t.k % 256 != 0) return false;
  if (t.group != 32 && t.group != 64 && t.group != 128) return false;
  if ((t.k / t.group) % 2 != 0) return false;
  if (((t.n + 15) / 16) * (t.k / 256) >= (int64_t{1} << 29)) return false;
  if (!al(t.codes, 16) || !al(t.scales, 4) || !al(x, 16) || !al(y, 4)) return false;
  if (t.grid == SSS_GRID_ASYM && !al(t.mins, 4)) return false;
  return true;
}

cudaError_t launch_gemv_batch(const sss_qtensor_t& t, const uint16_t* x, int batch, float* y,
                              uint32_t* status, cudaStream_t stream) {
  BatchArgs a;
  memset(&a, 0, sizeof a);
  a.codes = t.codes;
  a.scales = t.scales;
  a.mins = t.mins;
  a.x = x;
  a.y = y;
  a.n = t.n;
  a.k = t.k;
  a.batch = batch;
  a.status = status;
  const bool asym = t.grid == SSS_GRID_ASYM;
  switch (t.q) {
    case 2: return asym ? launch_bg<2, true>(t, a, stream) : launch_bg<2, false>(t, a, stream);
    case 3: return asym ? launch_bg<3, true>(t, a, stream) : launch_bg<3, false>(t, a, stream);
    case 4: return asym ? launch_bg<4, true>(t, a, stream) : launch_bg<4, false>(t, a, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace sss
