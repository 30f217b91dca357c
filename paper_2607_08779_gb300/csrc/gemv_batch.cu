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
//    2^p, as fp16, one 8-column block per 8 batch rows (rows past the batch
//    are zero);
//  * mma.sync m16n8k16: lane (g, t) feeds rows g and g+8 with codes of its
//    own two 32-code sub-chunks of each 256-code unit (the bytes it loads,
//    16-byte vector loads into a 2-deep register ring); the k order inside
//    an mma is free, and B holds x of batch row g at those codes;
//  * persistent CTAs of 16 warps walk 16-row tiles; groups of KW warps share
//    a tile and split its units, their partials meeting in shared memory
//    behind bounded mbarrier waits.  For each K slab the CTA stages x once
//    and runs all its tiles over it (results of later slabs are added to y
//    by the same CTA).
#include <cuda.h>

#include <stdint.h>
#include <string.h>

#include <algorithm>

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
  int stall;       // test hook: the first tile's barrier stays one arrive short
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

template <int Q, bool ASYM, int G, int NBLK>
__global__ void __launch_bounds__(kThreads, 1) gemv_batch_kernel(const __grid_constant__ BatchArgs a) {
  constexpr int NBC = 8 * NBLK;             // batch columns (padded)
  constexpr int R = 16;
  constexpr int HALF = 1 << (Q - 1);
  constexpr int UB = 32 * Q;                // code bytes of one row in one unit
  constexpr int SPU = 256 / G;              // scales of one row in one unit
  constexpr int XU = 16 * 4 * NBC * 8;      // staged x bytes per unit
  extern __shared__ __align__(128) unsigned char smem[];

  const int nunits = static_cast<int>(a.k / 256);
  const int64_t nG = a.k / G;
  const int64_t row_bytes = a.k * Q / 8;
  const int lgkw = a.lgkw;
  const int KW = 1 << lgkw;
  const int ngrp = kWarps >> lgkw;
  const int SK = a.slab_units;
  const int nslabs = (nunits + SK - 1) / SK;

  // ---- shared memory: x slab | partials | barriers | flag ----
  unsigned char* xs = smem;                                      // [SK][16][NBLK][32 lanes] x 8 B
  float* part = reinterpret_cast<float*>(xs + static_cast<size_t>(SK) * XU);  // [ngrp][2][KW][R][NBC]
  uint64_t* pready = reinterpret_cast<uint64_t*>(part + 2 * kWarps * R * NBC);  // [kWarps][2]
  uint64_t* pfree = pready + 2 * kWarps;
  volatile int* abort = reinterpret_cast<volatile int*>(pfree + 2 * kWarps);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;
  const int grp = warp >> lgkw;
  const int kw = warp & (KW - 1);

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2 * kWarps; ++i) {
      bar_init(&pready[i], KW);  // every warp of a group, after its lanes wrote
      bar_init(&pfree[i], 1);
    }
    *abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
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

  Regs r0, r1;
  set_fetch();
  if (total > 0) fetch(r0);
  if (total > 1) fetch(r1);
  asm volatile("griddepcontrol.wait;" ::: "memory");  // x is produced upstream

  const uint32_t xs_a = su32(xs);
  bool ok = true;
  float acc[NBLK][4];
#pragma unroll
  for (int nb = 0; nb < NBLK; ++nb)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[nb][e] = 0.f;

  // Stage slab s: x[b][32*(8u + sc) + e] for the slab's units u, in mma-B
  // order: the 8 bytes at (u, j, nb, lane = 4g + t) hold, for batch column
  // n = 8nb + g, the activation pairs 2j and 2j+1 of quad t (quad t's
  // sub-chunk 2t + (j >> 3), pairs (2j) & 15 and (2j+1) & 15), each element
  // pre-divided by 2^p; a warp's B fragments of one mma are then 256
  // contiguous bytes.  One thread handles 16 elements (half a sub-chunk) of
  // one batch row.
  auto stage = [&](int s) {
    const int u0 = s * SK;
    const int su = min(SK, nunits - u0);
    const int items = su * 8 * NBC * 2;
    for (int it = threadIdx.x; it < items; it += kThreads) {
      const int hf = it & 1;
      const int n = (it >> 1) % NBC;
      const int scu = (it >> 1) / NBC;  // sub-chunk within the slab
      const int ul = scu >> 3, sc = scu & 7;
      uint32_t pr[8];
      if (n < a.batch) {
        const uint4* src = reinterpret_cast<const uint4*>(
            a.x + static_cast<int64_t>(n) * a.k + static_cast<int64_t>(u0 + ul) * 256 + 32 * sc + 16 * hf);
        float xv[16];
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
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
          int ea, eb;
          float mult;
          pair_desc<Q>(jj, ea, eb, mult);  // pair 8hf + jj, offsets within this half
          __half2 hv = __floats2half2_rn(xv[ea] * mult, xv[eb] * mult);
          pr[jj] = *reinterpret_cast<uint32_t*>(&hv);
        }
      } else {
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) pr[jj] = 0u;
      }
      // pair p = 8hf + jj of sub-chunk sc = 2t + h is quad t's pair
      // P = 16h + p, i.e. entry j = P >> 1, slot P & 1
      const int t = sc >> 1, h = sc & 1;
#pragma unroll
      for (int jj = 0; jj < 8; jj += 2) {
        const int j = 8 * h + 4 * hf + (jj >> 1);
        const uint32_t dst = xs_a + static_cast<uint32_t>(
            ul * XU + ((j * NBLK + (n >> 3)) * 32 + 4 * (n & 7) + t) * 8);
        asm volatile("st.shared.v2.u32 [%0], {%1,%2};" ::"r"(dst), "r"(pr[jj]), "r"(pr[jj + 1])
                     : "memory");
      }
    }
  };

  // constants of the operand formation
  uint32_t off[3];
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    // fp16x2 of 1024 + 2^(q-1)*4^i (symmetric) or 1024 (min-max)
    const float o = 1024.f + (ASYM ? 0.f : static_cast<float>(HALF << (2 * i)));
    __half2 hv = __floats2half2_rn(o, o);
    off[i] = *reinterpret_cast<uint32_t*>(&hv);
  }

  // a group of this thread's whose operand may leave the fp16 range
  bool big = false;
  auto compute = [&](const Regs& rg, int ul) {
    const uint32_t xu = xs_a + static_cast<uint32_t>(ul * XU);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      // the fp16 scale (and min) of sub-chunk 2tq + h for rows gq, gq + 8
      uint32_t S[2], M[2][3];
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        const uint32_t sb = G == 32 ? ((rg.s[hh] >> (16 * h)) & 0xFFFFu) : (rg.s[hh] & 0xFFFFu);
        S[hh] = f16x2_of(sb);
        const float sa = fabsf(__half2float(__ushort_as_half(static_cast<unsigned short>(sb))));
        if constexpr (!ASYM) big |= sa * static_cast<float>(HALF * 16) >= 65520.f;
        if constexpr (ASYM) {
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
      for (int jm = 0; jm < 8; ++jm) {
        const int p = 2 * jm;
        const int j = 8 * h + jm;
        const uint32_t a0 = deq(0, p), a1 = deq(1, p), a2 = deq(0, p + 1), a3 = deq(1, p + 1);
#pragma unroll
        for (int nb = 0; nb < NBLK; ++nb) {
          const float2 bv = lds64f(xu + static_cast<uint32_t>(((j * NBLK + nb) * 32 + lane) * 8));
          mma16816(acc[nb], a0, a1, a2, a3, __float_as_uint(bv.x), __float_as_uint(bv.y));
        }
      }
    }
  };

  // ---- tile end: the group's KW partials meet; y = sum (first slab) or
  // y += sum (later slabs) ----
  auto tile_end = [&](int s, int64_t i) {
    const int64_t row0 = (tfirst + i * tstride) * R;
    if (KW == 1) {
#pragma unroll
      for (int nb = 0; nb < NBLK; ++nb)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int64_t r = row0 + gq + 8 * (e >> 1);
          const int b = 8 * nb + 2 * tq + (e & 1);
          if (r < a.n && b < a.batch && ok) {
            float* yp = a.y + static_cast<int64_t>(b) * a.n + r;
            *yp = (s == 0 ? 0.f : *yp) + acc[nb][e];
          }
          acc[nb][e] = 0.f;
        }
      return;
    }
    const int bsel = static_cast<int>(i & 1);
    // the group's tiles alternate between two partial buffers; a buffer's
    // use count runs on over the slabs (each slab visits every tile once)
    const int64_t per_slab = bsel == 0 ? (my_tiles + 1) >> 1 : my_tiles >> 1;
    const uint32_t use = static_cast<uint32_t>(static_cast<int64_t>(s) * per_slab + (i >> 1)) & 1u;
    float* pb = part + (static_cast<size_t>(grp) * 2 + bsel) * KW * R * NBC;
    uint64_t* rdy = &pready[grp * 2 + bsel];
    uint64_t* fre = &pfree[grp * 2 + bsel];
    if (!bar_wait(fre, use ^ 1u, abort)) ok = false;
#pragma unroll
    for (int nb = 0; nb < NBLK; ++nb)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        pb[(kw * R + gq + 8 * (e >> 1)) * NBC + 8 * nb + 2 * tq + (e & 1)] = acc[nb][e];
        acc[nb][e] = 0.f;
      }
    __syncwarp();
    // (sss_test_set_stall: the last warp leaves the first tile's barrier one
    // arrive short, so its reducer's wait runs out)
    if (lane == 0 && !(a.stall && s == 0 && i == 0 && kw == KW - 1)) bar_arrive(rdy);
    if (kw == static_cast<int>(i & (KW - 1))) {
      if (!bar_wait(rdy, use, abort)) ok = false;
      for (int v = lane; v < R * NBC; v += 32) {
        const int rr = v / NBC, b = v % NBC;
        float sum = 0.f;
        for (int c = 0; c < KW; ++c) sum += pb[(c * R + rr) * NBC + b];
        const int64_t r = row0 + rr;
        if (r < a.n && b < a.batch && ok) {
          float* yp = a.y + static_cast<int64_t>(b) * a.n + r;
          *yp = (s == 0 ? 0.f : *yp) + sum;
        }
      }
      __syncwarp();
      if (lane == 0) bar_arrive(fre);
    }
  };

  int gk = 0;  // position in this warp's unit stream (register ring slot gk & 1)
  for (int s = 0; s < nslabs; ++s) {
    __syncthreads();  // barriers initialised / every warp done with the previous slab
    stage(s);
    __syncthreads();
    const int ups = units_in(s);
    for (int64_t i = 0; i < my_tiles; ++i) {
      for (int r = 0; r < ups; ++r, ++gk) {
        const int ul = kw + r * KW;  // unit within the slab
        if (gk & 1) {
          compute(r1, ul);
          if (gk + 2 < total) fetch(r1);
        } else {
          compute(r0, ul);
          if (gk + 2 < total) fetch(r0);
        }
      }
      tile_end(s, i);
    }
  }
  if (__any_sync(0xffffffffu, big) && lane == 0 && a.status != nullptr)
    atomicOr(a.status, SSS_FLAG_RANGE);
  if (*abort && threadIdx.x == 0 && a.status != nullptr) atomicOr(a.status, SSS_FLAG_TIMEOUT);
}

template <int NBLK>
size_t batch_smem(int slab_units) {
  return static_cast<size_t>(slab_units) * (16 * 4 * 8 * NBLK * 8) +
         static_cast<size_t>(2 * kWarps * 16 * 8 * NBLK) * 4 + 8 * 4 * kWarps + 16;
}

template <int Q, bool ASYM, int G, int NBLK>
cudaError_t launch_b(const sss_qtensor_t& t, BatchArgs& a, cudaStream_t stream) {
  const int nunits = static_cast<int>(t.k / 256);
  int sk = nunits;
  while (sk > 1 && batch_smem<NBLK>(sk) > static_cast<size_t>(kSmemMax)) sk = (sk + 1) / 2;
  if (batch_smem<NBLK>(sk) > static_cast<size_t>(kSmemMax)) return cudaErrorNotSupported;
  a.slab_units = sk;
  const size_t smem = batch_smem<NBLK>(sk);
  auto kern = gemv_batch_kernel<Q, ASYM, G, NBLK>;
  cudaError_t e = ensure_smem(kern, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int64_t tiles = (t.n + 15) / 16;
  a.ntiles = tiles;
  const int sms = device_sm_count();
  const int grid = static_cast<int>(std::min<int64_t>(sms, tiles));
  const int64_t per_cta = (tiles + grid - 1) / grid;
  int best = 0;
  int64_t best_cost = INT64_MAX;
  for (int lg = 0; (1 << lg) <= kWarps; ++lg) {
    const int kwn = 1 << lg;
    if (kwn > 1 && kwn > std::min(nunits, sk)) break;
    const int64_t ngrp = kWarps >> lg;
    const int64_t cost = ((per_cta + ngrp - 1) / ngrp) * ((nunits + kwn - 1) / kwn);
    if (cost < best_cost) {
      best_cost = cost;
      best = lg;
    }
  }
  a.lgkw = best;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int Q, bool ASYM, int G>
cudaError_t launch_bn(const sss_qtensor_t& t, BatchArgs& a, cudaStream_t stream) {
  return a.batch <= 8 ? launch_b<Q, ASYM, G, 1>(t, a, stream) : launch_b<Q, ASYM, G, 2>(t, a, stream);
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
  a.stall = (test_stall_mask() & SSS_TEST_STALL_GEMV_BATCH) ? 1 : 0;
  const bool asym = t.grid == SSS_GRID_ASYM;
  switch (t.q) {
    case 2: return asym ? launch_bg<2, true>(t, a, stream) : launch_bg<2, false>(t, a, stream);
    case 3: return asym ? launch_bg<3, true>(t, a, stream) : launch_bg<3, false>(t, a, stream);
    case 4: return asym ? launch_bg<4, true>(t, a, stream) : launch_bg<4, false>(t, a, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace sss
