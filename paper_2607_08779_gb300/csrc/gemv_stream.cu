// gemv_stream.cu -- persistent, warp-specialised batch-1 decode GEMV over
// packed q-bit codes (sm_103a), the streaming path of sss_gemv and
// sss_gemv_multi.
//
// Arithmetic (Appendix B.3 expansion): y = sum over groups of
// s * (sum u*x - 2^(q-1) * sum x) for the symmetric grids, s * sum u*x +
// m * sum x for the min-max grid, the integer part on the tensor cores:
// codes are masked in place into fp16 operands (u * 2^pos * 2^-24, exact)
// for mma.sync m16n8k16 with one B column per 32-code sub-chunk, and the
// activations are staged as fp16 with a power of two per sub-chunk that
// keeps them exact whatever their magnitude; scale, min and the row-sum
// term are applied per group in fp32.
//
// Organisation, for streaming bandwidth:
//  * persistent CTAs of 16 warps, one per SM, walking 16-row tiles of all
//    jobs (several weight matrices sharing one activation vector, e.g. a
//    fused q/k/v projection) round-robin;
//  * the 16 warps form groups of KW = 1..16 warps (chosen per launch to
//    balance the work); a group owns one tile at a time and its warps split
//    the tile's units (256 codes of every row) round-robin;
//  * every lane loads the exact bytes it will multiply (its two sub-chunks of
//    rows g and g+8, and their scales) straight into a D-slot ring of
//    registers; a slot is refilled as soon as its unit is multiplied, and
//    the whole ring is filled before the grid-dependency wait.  Shared
//    memory holds only the activation operand.
//  * with KW > 1 every warp leaves its row partials of each of its tiles in
//    its own slot of a shared array, with no wait; after the last unit the
//    CTA sums each tile's KW partials in warp order and stores y.  With
//    KW = 1 a warp owns whole tiles and writes y directly.
//
// The activation vector is staged once per CTA, after the grid-dependency
// wait of a programmatic dependent launch (weights may be prefetched before
// it only when the caller states they are not written upstream).  The
// kernel has no data-dependent waits: its only synchronisation is two
// CTA-wide barriers (after staging x, and before the final sums).
#include <cuda.h>

#include <stdint.h>
#include <string.h>

#include <algorithm>

#include "act_q8.cuh"
#include "gemv_common.cuh"

namespace sss {
namespace {

constexpr int kWarps = 16;                // warps per CTA
constexpr int kThreads = kWarps * 32;
constexpr int kMaxJobs = 4;
using namespace gv;

// ---------------------------------------------------------------------------
// Code fields as fp16 operands.  An fp16 bit pattern below 2048 (exponent
// field 0 or 1) has the value pattern * 2^-24, so a code masked in place at
// bit position pos of a 16-bit half (its top bit at most bit 10) is the
// operand u * 2^pos * 2^-24; the staged activation of that element carries
// 2^-pos.  Pair p of a 32-code sub-chunk holds elements ea (low half) and
// eb (high half):
//   q=4: p = 4w + i: elements 8w+i and 8w+i+4 at pos 0 (i even) or 4 (i odd),
//        nibble pairs 2 and 3 of each byte pair after one 8-bit shift;
//   q=2, q=3: p = 8w + e: elements 16w+e and 16w+e+8, whose 2-bit low fields
//        sit at bit 2e (e = 0..4) or, after one 10-bit shift, 2(e-5);
//        q=3 ORs the element's high-plane bit in at pos + 2.
// ---------------------------------------------------------------------------
template <int Q>
__device__ __forceinline__ void field_desc(int p, int& ea, int& eb, int& pos) {
  if (Q == 4) {
    const int w = p >> 2, i = p & 3;
    ea = 8 * w + i;
    eb = ea + 4;
    pos = (i & 1) ? 4 : 0;
  } else {
    const int w = p >> 3, e = p & 7;
    ea = 16 * w + e;
    eb = ea + 8;
    pos = e < 5 ? 2 * e : 2 * (e - 5);
  }
}

// the high-plane bits of elements 16w .. 16w+15 (w = word of the sub-chunk)
// spread to every other bit: element 16w+e at bit 2e (e < 8) and element
// 16w+8+e at bit 16+2e
__device__ __forceinline__ uint32_t spread_high(uint32_t hi_plane, int w) {
  uint32_t x = __byte_perm(hi_plane, 0u, w ? 0x4342u : 0x4140u);
  x = (x | (x << 4)) & 0x0F0F0F0Fu;
  x = (x | (x << 2)) & 0x33333333u;
  x = (x | (x << 1)) & 0x55555555u;
  return x;
}

// Operand of pair p.  w[0..3] (q=4), w[0..1] (q=2) or w[0..1] + the high
// plane w[2] (q=3) of one sub-chunk; hs[0..1] = spread_high of w[2] for q=3.
template <int Q>
__device__ __forceinline__ uint32_t field_pair(const uint32_t* w, const uint32_t* hs, int p) {
  if constexpr (Q == 4) {
    const uint32_t v = (p & 2) ? (w[p >> 2] >> 8) : w[p >> 2];
    return v & ((p & 1) ? 0x00F000F0u : 0x000F000Fu);
  } else {
    const int wi = (p >> 3) & 1, e = p & 7;
    const int pos = e < 5 ? 2 * e : 2 * (e - 5);
    const uint32_t v = e < 5 ? w[wi] : (w[wi] >> 10);
    const uint32_t lo = v & (0x00030003u << pos);
    if constexpr (Q == 2) {
      return lo;
    } else {
      // high bit of element e at 2e in hs; wanted at pos + 2
      const uint32_t h = e < 5 ? (hs[wi] << 2) : (hs[wi] >> 8);
      return lo | (h & (0x00040004u << pos));
    }
  }
}

// Stage the activations x[0 .. 32*nsc) for the mma B operand.  Sub-chunk i
// (32 elements, 64 bytes at xs + 64 i) holds its 16 fp16 pairs in pair
// order, element e as fl16(x_e * 2^(E_i - pos_e)): E_i is a power of two
// chosen per sub-chunk so that its largest |x| lands in [2^14, 2^15), which
// keeps every element exact in fp16 whatever the activations' magnitude.
// sbf[i] = {b_i, f_i}: f_i = 2^(24 - E_i) undoes both scalings in the
// epilogue, and b_i is the row-sum term of Appendix B.3 on the mma's scale:
// sum(x) * 2^(E_i - 24), times -2^(q-1) for the symmetric grids.  Two
// threads share a sub-chunk (16 elements each); threads tid = 0 ..
// nthreads-1 (nthreads even) share the work; the caller synchronises.
//
// With act_q8 the activations are first quantized to Q8_0 (act_q8.cuh; a
// sub-chunk is one Q8_0 block): the staged operand is the int8 code q
// (times 2^-pos, exact in fp16), f_i = fl16(d_i) * 2^24 and the row-sum
// term uses sum(q), so the mma's integer dot sum(u*q) is exact and the
// block scale meets the group scale in fp32 (the Appendix B.3 product on
// Q8_0 activations).  Non-finite or fp16-overflowing blocks set the status
// bits as sss_quantize_act_q8 does.
template <int Q, bool ASYM>
__device__ __forceinline__ void stage_x(const uint16_t* x, int nsc, uint32_t xs_a, float2* sbf,
                                        int tid, int nthreads, bool act_q8, uint32_t* status) {
  constexpr int HALF = 1 << (Q - 1);
  const int rounds = (2 * nsc + nthreads - 1) / nthreads;
  for (int r = 0; r < rounds; ++r) {
    const int t = tid + r * nthreads;
    const bool valid = t < 2 * nsc;
    const int i = t >> 1, hf = t & 1;
    float xv[16];
    if (valid) {
      const uint4* src = reinterpret_cast<const uint4*>(x + static_cast<int64_t>(i) * 32 + 16 * hf);
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const uint4 v = __ldg(src + c);
        const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          xv[8 * c + 2 * e] = __uint_as_float(wv[e] << 16);
          xv[8 * c + 2 * e + 1] = __uint_as_float(wv[e] & 0xFFFF0000u);
        }
      }
    } else {
#pragma unroll
      for (int e = 0; e < 16; ++e) xv[e] = 0.f;
    }
    float sum = 0.f, amax = 0.f;
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      sum += xv[e];
      amax = fmaxf(amax, fabsf(xv[e]));
    }
    sum += __shfl_xor_sync(0xffffffffu, sum, 1);
    amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 1));
    // E = 14 - floor(log2 amax), kept in [-100, 100] (0 for a zero sub-chunk)
    const int ex = static_cast<int>((__float_as_uint(amax) >> 23) & 0xFFu) - 127;
    int E = amax == 0.f ? 0 : max(-100, min(100, 14 - ex));
    float fq = 0.f;  // Q8_0: fl16(d) * 2^24
    if (act_q8) {
      unsigned bad = 0;
#pragma unroll
      for (int e = 0; e < 16; ++e) bad |= is_nonfinite(xv[e]);
      bad |= __shfl_xor_sync(0xffffffffu, bad, 1);
      unsigned flags = 0;
      uint16_t d16;
      const float d = q8_scale(amax, bad != 0, &d16, &flags);
      const float r = d != 0.f ? __frcp_rn(d) : 0.f;
      int qs = 0;
#pragma unroll
      for (int e = 0; e < 16; ++e) {
        const int qv = d != 0.f ? q8_code(xv[e], d, r) : 0;
        qs += qv;
        xv[e] = static_cast<float>(qv);
      }
      qs += __shfl_xor_sync(0xffffffffu, qs, 1);
      sum = static_cast<float>(qs);  // exact: |sum q| <= 32 * 127
      E = 0;
      fq = __half2float(__ushort_as_half(d16)) * 0x1p24f;
      if (valid && hf == 0 && flags != 0u && status != nullptr) atomicOr(status, flags);
    }
    if (valid) {
      uint32_t pr[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        // pair 8hf + j; both its elements lie in this half, at the same
        // offsets from the half's start for either half
        int ea, eb, pos;
        field_desc<Q>(j, ea, eb, pos);
        const float m = __int_as_float((127 + E - pos) << 23);  // 2^(E - pos)
        __half2 hv = __floats2half2_rn(xv[ea] * m, xv[eb] * m);
        pr[j] = *reinterpret_cast<uint32_t*>(&hv);
      }
      const uint32_t dst = xs_a + static_cast<uint32_t>(i * 64 + 32 * hf);
      asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(dst), "r"(pr[0]), "r"(pr[1]),
                   "r"(pr[2]), "r"(pr[3])
                   : "memory");
      asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(dst + 16u), "r"(pr[4]),
                   "r"(pr[5]), "r"(pr[6]), "r"(pr[7])
                   : "memory");
      if (hf == 0) {
        const float toE = __int_as_float((127 + E - 24) << 23);  // 2^(E - 24)
        const float b = sum * toE;
        const float f = act_q8 ? fq : __int_as_float((127 + 24 - E) << 23);  // 2^(24 - E)
        // min-max grid: b is the block's sum of activation values
        const float bsum = act_q8 ? fq * b : sum;
        sbf[i] = make_float2(ASYM ? bsum : -static_cast<float>(HALF) * b, f);
      }
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
  int act_q8;          // quantize the activations to Q8_0 while staging them
  int rounds;          // tiles per warp group at most (the partial array's depth)
  uint32_t* status;
};

template <int Q, bool ASYM, int G, int D>
__global__ void __launch_bounds__(kThreads, 1) gemv_stream_kernel(const __grid_constant__ StreamArgs a) {
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
  // staged activations [nsc][64 B] | two 64-byte zero blocks, the first 128
  // bytes past a 128-aligned offset (the B operand of lanes that carry no
  // data; see compute) | per-sub-chunk {b, f} | row partials (KW > 1)
  unsigned char* xs = smem;
  const uint32_t zoff = (static_cast<uint32_t>(nsc) * 64u + 127u) & ~127u;
  float2* sbf = reinterpret_cast<float2*>(xs + zoff + 128);              // [nsc]
  float* part = reinterpret_cast<float*>(sbf + nsc);                      // [ngrp][rounds][KW][R]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;
  const int grp = warp >> lgkw;        // this warp's group (one tile at a time)
  const int kw = warp & (KW - 1);      // its share of the tile's k-range

  if (threadIdx.x >= 32 && threadIdx.x < 64)
    reinterpret_cast<uint32_t*>(xs + zoff)[threadIdx.x - 32] = 0u;  // the zero blocks
  // allow the next kernel in the stream to be scheduled as SMs free up
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  // ---- this warp's stream: tiles t = (i * ngrp + grp) * gridDim.x + blockIdx.x,
  // i = 0, 1, ... (consecutive tiles go to different SMs, so every SM gets
  // within one tile of the same work), and in each tile the units u = kw,
  // kw + KW, ... ----
  const int64_t tstride = static_cast<int64_t>(gridDim.x) * ngrp;
  const int64_t tfirst = static_cast<int64_t>(grp) * gridDim.x + blockIdx.x;
  const int64_t my_tiles = tfirst < a.ntiles ? (a.ntiles - tfirst + tstride - 1) / tstride : 0;
  const bool has_units = kw < nunits;

  // This warp's flat unit stream: unit k is unit u = kw + (k % upw) * KW of
  // its i = k / upw-th tile, upw = units per tile for this warp (the host
  // keeps every count below 2^31).
  const int upw = has_units ? (nunits - kw + KW - 1) >> lgkw : 0;
  const int total = static_cast<int>(my_tiles) * upw;

  constexpr int UB = 32 * Q;    // code bytes of one row in one unit
  constexpr int SPU = 256 / G;  // scales of one row in one unit
  // the lane's byte offset in a unit's codes (sub-chunks 2tq, 2tq+1; q=3
  // addresses its planes per sub-chunk below) and its scale index in the
  // unit: the pair of groups 2tq, 2tq+1 for g=32, else its one group
  // q=3: the lane's two sub-chunks are 24 contiguous bytes at 24tq (g=32:
  // two groups [lo hi | lo hi]; g=64: one group [lo lo | hi hi]), or for
  // g=128 16 low-plane bytes at 48(tq>>1) + 16(tq&1) and 8 high-plane bytes
  // 32 bytes further on
  const int lane_c = Q == 4 ? 32 * tq : (Q == 2 ? 16 * tq : (G == 128 ? 48 * (tq >> 1) + 16 * (tq & 1) : 24 * tq));
  const int lane_s = G == 32 ? 2 * tq : (G == 64 ? tq : (tq >> 1));

  // the code/scale/min pointers of rows g and g+8 of this warp's i-th tile,
  // at its first unit
  auto tile_ptrs = [&](int64_t i, const uint8_t** c, const uint16_t** sc, const uint16_t** mn) {
    const int64_t t = tfirst + i * tstride;
    int j = 0;
    while (j + 1 < a.njobs && t >= a.job[j + 1].tile0) ++j;
    const StreamJob& jb = a.job[j];
    const int64_t row0 = (t - jb.tile0) * R;
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      int64_t r = row0 + gq + 8 * hh;
      if (r >= jb.n) r = jb.n - 1;  // a valid row; results past n are never stored
      c[hh] = jb.codes + r * row_bytes + kw * UB + lane_c;
      sc[hh] = jb.scales + r * nG + kw * SPU + lane_s;
      if constexpr (ASYM) mn[hh] = jb.mins + r * nG + kw * SPU + lane_s;
    }
  };
  // fetch cursor: the next unit to load into registers
  int64_t fi = 0;
  int fleft = 0;
  const uint8_t* cp[2] = {nullptr, nullptr};
  const uint16_t* sp[2] = {nullptr, nullptr};
  const uint16_t* mp[2] = {nullptr, nullptr};
  auto set_tile = [&](int64_t i) {
    if (i >= my_tiles) return;
    tile_ptrs(i, cp, sp, mp);
    fleft = upw;
  };
  // the registers of one unit: code words of (row half hh, column parity h),
  // and the fp16 scale (min) of each row: the pair of the lane's two groups
  // for g=32, else its one group in the low half
  struct Regs {
    uint32_t w[2][2][4];
    uint32_t s[2], m[2];
  };
  auto fetch = [&](Regs& rg) {
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const uint8_t* rp = cp[hh];
      if constexpr (Q == 4) {  // sub-chunk 2tq + h at byte 32tq + 16h
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const uint4 v = __ldcs(reinterpret_cast<const uint4*>(rp + 16 * h));
          rg.w[hh][h][0] = v.x; rg.w[hh][h][1] = v.y; rg.w[hh][h][2] = v.z; rg.w[hh][h][3] = v.w;
        }
      } else if constexpr (Q == 2) {  // sub-chunks 2tq, 2tq+1: 16 contiguous bytes
        const uint4 v = __ldcs(reinterpret_cast<const uint4*>(rp));
        rg.w[hh][0][0] = v.x; rg.w[hh][0][1] = v.y;
        rg.w[hh][1][0] = v.z; rg.w[hh][1][1] = v.w;
      } else if constexpr (G == 128) {  // q=3: [lo lo] (16 B) and [hi hi] (8 B)
        const uint4 lo = __ldcs(reinterpret_cast<const uint4*>(rp));
        const uint2 hi = __ldcs(reinterpret_cast<const uint2*>(rp + 32 - 8 * (tq & 1)));
        rg.w[hh][0][0] = lo.x; rg.w[hh][0][1] = lo.y; rg.w[hh][0][2] = hi.x;
        rg.w[hh][1][0] = lo.z; rg.w[hh][1][1] = lo.w; rg.w[hh][1][2] = hi.y;
      } else {  // q=3, g=32 / 64: 24 contiguous bytes
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
    if (--fleft == 0) set_tile(++fi);
  };

  Regs ring[D];
  set_tile(0);
  if (!a.early_weights) asm volatile("griddepcontrol.wait;" ::: "memory");
#pragma unroll
  for (int d = 0; d < D; ++d)
    if (d < total) fetch(ring[d]);
  asm volatile("griddepcontrol.wait;" ::: "memory");  // x is produced upstream

  // ---- stage the activations in mma order, and per-sub-chunk sums ----
  stage_x<Q, ASYM>(a.x, nsc, su32(xs), sbf, threadIdx.x, kThreads, a.act_q8 != 0, a.status);
  __syncthreads();

  float acc[2] = {0.f, 0.f};
  // Column gq of B carries sub-chunk 8u + gq of the unit in the mmas of
  // parity h = gq & 1, from the one lane of quad gq >> 1 whose own A rows
  // hold that sub-chunk (gq == 2tq + h); every other lane supplies zeros by
  // reading a zero block.  That leaves one data lane per quarter-warp, and
  // the zero block of each parity sits 64 bytes (mod 128) away from the data
  // lanes' banks, so the 16-byte loads are free of bank conflicts.
  const bool act0 = gq == 2 * tq, act1 = gq == 2 * tq + 1;
  const uint32_t xs_a = su32(xs), sbf_a = su32(sbf);
  const uint32_t z0 = xs_a + zoff + 64u, z1 = xs_a + zoff;  // zero blocks for h = 0, 1
  uint32_t xl = 0, bl = 0;
  int cleft = 0;
  int64_t ci = 0;
  auto start_tile = [&]() {
    xl = xs_a + static_cast<uint32_t>((kw * 8 + gq) * 64);
    bl = sbf_a + static_cast<uint32_t>((kw * 8 + 2 * tq) * 8);
    cleft = upw;
  };
  start_tile();
  auto compute = [&](const Regs& rg) {
    // h=0 mmas only write even columns and h=1 mmas odd ones: the lane's
    // column 2tq is in dh[0] and 2tq+1 in dh[1]
    float dh[2][4];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint32_t ba = h ? (act1 ? xl : z1) : (act0 ? xl : z0);
      uint32_t hs0[2] = {0u, 0u}, hs1[2] = {0u, 0u};
      if constexpr (Q == 3) {
        hs0[0] = spread_high(rg.w[0][h][2], 0);
        hs0[1] = spread_high(rg.w[0][h][2], 1);
        hs1[0] = spread_high(rg.w[1][h][2], 0);
        hs1[1] = spread_high(rg.w[1][h][2], 1);
      }
#pragma unroll
      for (int jm = 0; jm < NP / 2; jm += 2) {
        const uint4 bv = lds128(ba + 8u * static_cast<uint32_t>(jm));
#pragma unroll
        for (int jj = 0; jj < 2; ++jj) {
          const int p = 2 * (jm + jj);
          const uint32_t a0 = field_pair<Q>(rg.w[0][h], hs0, p);
          const uint32_t a1 = field_pair<Q>(rg.w[1][h], hs1, p);
          const uint32_t a2 = field_pair<Q>(rg.w[0][h], hs0, p + 1);
          const uint32_t a3 = field_pair<Q>(rg.w[1][h], hs1, p + 1);
          if (jm == 0 && jj == 0)
            mma16816_z(dh[h], a0, a1, a2, a3, bv.x, bv.y);
          else
            mma16816(dh[h], a0, a1, a2, a3, jj ? bv.z : bv.x, jj ? bv.w : bv.y);
        }
      }
    }
    // {b, f} of the lane's sub-chunks 8u + 2tq and 8u + 2tq + 1
    const uint4 bfv = lds128(bl);
    const float b0 = __uint_as_float(bfv.x), f0 = __uint_as_float(bfv.y);
    const float b1 = __uint_as_float(bfv.z), f1 = __uint_as_float(bfv.w);
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      float s_0, s_1, m_0 = 0.f, m_1 = 0.f;
      if constexpr (G == 32) {
        const float2 sf = __half22float2(*reinterpret_cast<const __half2*>(&rg.s[hh]));
        s_0 = sf.x;
        s_1 = sf.y;
        if constexpr (ASYM) {
          const float2 mf = __half22float2(*reinterpret_cast<const __half2*>(&rg.m[hh]));
          m_0 = mf.x;
          m_1 = mf.y;
        }
      } else {
        s_0 = s_1 = __half2float(__ushort_as_half(static_cast<unsigned short>(rg.s[hh])));
        if constexpr (ASYM) m_0 = m_1 = __half2float(__ushort_as_half(static_cast<unsigned short>(rg.m[hh])));
      }
      const float d0 = dh[0][2 * hh], d1 = dh[1][2 * hh + 1];
      if constexpr (ASYM) {
        acc[hh] += (s_0 * f0) * d0 + m_0 * b0 + (s_1 * f1) * d1 + m_1 * b1;
      } else {
        acc[hh] += (s_0 * f0) * (d0 + b0) + (s_1 * f1) * (d1 + b1);
      }
    }
    xl += static_cast<uint32_t>(8 * 64 * KW);
    bl += static_cast<uint32_t>(8 * 8 * KW);
  };
  // End of the compute cursor's tile i: the warp's two row partials (rows
  // gq and gq + 8, summed over the quad) go straight to y (KW = 1) or to the
  // warp's slot of the partial array (KW > 1), summed after the last unit.
  auto tile_end = [&](int64_t i) {
    float v[2];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      float x = acc[hh];
      x += __shfl_xor_sync(0xffffffffu, x, 1);
      x += __shfl_xor_sync(0xffffffffu, x, 2);
      v[hh] = x;
      acc[hh] = 0.f;
    }
    if (tq != 0) return;
    if (KW == 1) {
      const int64_t t = tfirst + i * tstride;
      int j = 0;
      while (j + 1 < a.njobs && t >= a.job[j + 1].tile0) ++j;
      const StreamJob& jb = a.job[j];
      const int64_t row0 = (t - jb.tile0) * R;
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const int64_t r = row0 + gq + 8 * hh;
        if (r < jb.n) jb.y[r] = v[hh];
      }
      return;
    }
    float* pb = part + ((static_cast<size_t>(grp) * a.rounds + i) * KW + kw) * R;
    pb[gq] = v[0];
    pb[gq + 8] = v[1];
  };

  // the units, D at a time so the register ring is indexed at compile time;
  // unit k + D - 1 is loaded while unit k is computed
  auto after_unit = [&]() {
    if (--cleft == 0) {
      tile_end(ci);
      ++ci;
      start_tile();
    }
  };
  // the units, D at a time so the register ring is indexed at compile time:
  // unit k is computed from slot k % D, which then takes unit k + D
  int k0 = 0;
  for (; k0 + 2 * D <= total; k0 += D) {  // every refill of these D units is in range
#pragma unroll
    for (int r = 0; r < D; ++r) {
      compute(ring[r]);
      fetch(ring[r]);
      after_unit();
    }
  }
  for (; k0 < total; k0 += D) {
#pragma unroll
    for (int r = 0; r < D; ++r) {
      const int k = k0 + r;
      if (k < total) {
        compute(ring[r]);
        if (k + D < total) fetch(ring[r]);
        after_unit();
      }
    }
  }
  if (KW == 1) return;
  // ---- the sums of the tiles' KW partials, in warp order (warps without
  // units left no partial) ----
  __syncthreads();
  const int kwn = KW < nunits ? KW : nunits;
  const int per_grp = a.rounds * R;
  for (int idx = threadIdx.x; idx < ngrp * per_grp; idx += kThreads) {
    const int g = idx / per_grp, i = (idx / R) % a.rounds, row = idx % R;
    const int64_t t = (static_cast<int64_t>(i) * ngrp + g) * gridDim.x + blockIdx.x;
    if (t >= a.ntiles) continue;
    int j = 0;
    while (j + 1 < a.njobs && t >= a.job[j + 1].tile0) ++j;
    const int64_t r = (t - a.job[j].tile0) * R + row;
    if (r >= a.job[j].n) continue;
    const float* pb = part + (static_cast<size_t>(g) * a.rounds + i) * KW * R + row;
    float sum = 0.f;
    for (int c = 0; c < kwn; ++c) sum += pb[c * R];
    a.job[j].y[r] = sum;
  }
}

// activations (rounded up to 128) | zero blocks | {b, f} | row partials
// (rounds x 1 KB when KW > 1)
size_t smem_bytes(int64_t k, int rounds = 0) {
  const int64_t nsc = k / 32;
  return static_cast<size_t>((nsc * 64 + 127) / 128 * 128 + 128 + 8 * nsc) +
         static_cast<size_t>(rounds) * kWarps * 16 * 4;
}
constexpr size_t kSmemMax = 227 * 1024;

template <int Q, bool ASYM, int G, int D>
cudaError_t launch_d(StreamArgs& a, int grid, bool pdl, cudaStream_t stream) {
  const size_t smem = smem_bytes(a.k, a.lgkw > 0 ? a.rounds : 0);
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
  if (smem_bytes(a.k, a.lgkw > 0 ? a.rounds : 0) > kSmemMax) return cudaErrorNotSupported;
  return launch_d<Q, ASYM, G, 2>(a, grid, pdl, stream);
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
  // One CTA per SM (fewer when there are fewer tiles); CTA c takes tiles
  // c, c + grid, ...  Warps per tile: the power of two that minimises the
  // busiest warp's units (rounds of that CTA's tiles x units per warp per
  // tile), preferring fewer warps per tile (less reduction) on ties, among
  // those whose partial array fits in shared memory (KW = 1 needs none).
  const int sms = device_sm_count();
  const int64_t nunits = a.k / 256;
  const int grid = static_cast<int>(std::min<int64_t>(sms, tiles));
  const int64_t per_cta = (tiles + grid - 1) / grid;
  int best = 0;
  int64_t best_cost = INT64_MAX;
  for (int lg = 0; (1 << lg) <= kWarps; ++lg) {
    const int kwn = 1 << lg;
    if (kwn > 1 && kwn > nunits) break;
    const int64_t ngrp = kWarps >> lg;
    const int64_t rounds = (per_cta + ngrp - 1) / ngrp;
    if (lg > 0 && smem_bytes(a.k, static_cast<int>(std::min<int64_t>(rounds, 1 << 20))) > kSmemMax)
      continue;
    const int64_t cost = rounds * ((nunits + kwn - 1) / kwn);
    if (cost < best_cost) {
      best_cost = cost;
      best = lg;
    }
  }
  a.lgkw = best;
  a.rounds = static_cast<int>((per_cta + (kWarps >> best) - 1) / (kWarps >> best));
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
  if (((t.n + 15) / 16) * (t.k / 256) >= (int64_t{1} << 29)) return false;  // 32-bit unit counts
  if ((t.k / t.group) % 2 != 0) return false;   // 4-byte scale pairs
  if (!al(t.codes, 16) || !al(t.scales, 4) || !al(x, 16)) return false;
  if (t.grid == SSS_GRID_ASYM && !al(t.mins, 4)) return false;
  // the staged activations must fit in shared memory
  return smem_bytes(t.k) <= 227 * 1024;
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
  a.act_q8 = (flags & SSS_GEMV_ACT_Q8) ? 1 : 0;
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
