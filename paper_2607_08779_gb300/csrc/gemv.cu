// gemv.cu -- decode GEMV over packed q-bit codes with fused dequantisation
// (sm_103a).
//
// y[b][r] = sum_groups s[r][j] * sum_{k in j} c[r][k] x[b][k]
//           (+ m[r][j] * sum_{k in j} x[b][k] for the min-max grid),
// the expansion of the quantized GEMM in Appendix B.3: the integer dot runs
// on the tensor cores, the per-group scale (and the asymmetric row-sum term)
// is applied to the fp32 group partial.
//
// Register unpack without bias.  A code u placed in the low 10 bits of an
// fp16 with a zero exponent field IS the fp16 subnormal u * 2^-24.  So one
// AND with a mask turns a 32-bit word of packed codes into an fp16x2 mma
// operand holding (u_a * 2^p * 2^-24, u_b * 2^p * 2^-24), where p is the bit
// offset of the field inside its 16-bit half.  The activation operand is
// pre-divided by 2^p (kept <= 16 so bf16 activations stay exact in fp16 for
// |x| >= 2^-10), so the product is exactly u*x*2^-24; the accumulator is
// rescaled by 2^24 at the end.  Symmetric codes are u = c + 2^(q-1); the
// bias is removed per group with the precomputed group sum of x.
//
// Operand pairing.  mma.m16n8k16: A is 16 rows x 16 k, lane (g, t) (g =
// lane/4, t = lane%4) supplies rows g and g+8 at k-slots {2t, 2t+1, 2t+8,
// 2t+9}; B is 16 k x 8 columns, the same lane supplies column g at those
// k-slots.  The k order inside an mma is free (x is permuted to match), so
// each lane feeds its k-slots from the codes of ITS OWN group, and column n
// of B carries the activations of group n only (zeros elsewhere): D[row][n]
// is then the dot of row with group n.  For batch 1 one warp step covers 8
// groups (lane t owns groups 2t and 2t+1, read as whole 16-byte chunks) and
// lane (g, t) ends up holding exactly the partials of its own two groups.
// For batch > 1 the same A is multiplied by each batch row in turn.
//
// Work split.  A CTA owns RT*16 rows; its warps interleave over 8-group
// steps of the CTA's k-range; the CTA's activations are staged once in
// shared memory in mma order.  When the row tiles alone cannot fill the
// GPU, KS CTAs of a thread-block cluster split k and the partials are
// reduced through distributed shared memory in rank order (deterministic,
// no workspace, no atomics).
#include <cooperative_groups.h>

#include <algorithm>

#include "sss_internal.cuh"

namespace cg = cooperative_groups;

namespace sss {
namespace {

constexpr int kMaxWarps = 4;
constexpr int kMaxKS = 8;

template <int Q>
struct QT;
template <>
struct QT<4> {
  static constexpr int NW = 4;   // 32-bit words per 32-code sub-chunk
  static constexpr int NP = 16;  // fp16x2 pairs per sub-chunk
};
template <>
struct QT<2> {
  static constexpr int NW = 2;
  static constexpr int NP = 16;
};
template <>
struct QT<3> {
  static constexpr int NW = 3;   // two low-plane words + one high-plane word
  static constexpr int NP = 32;  // 16 low pairs + 16 high pairs
};

// (element a, element b, multiplier) of activation pair p of a 32-code
// sub-chunk; the multiplier undoes the 2^p field offset (and carries the
// weight 4 of the q=3 high bit).
template <int Q>
__device__ __forceinline__ void pair_desc(int p, int& ea, int& eb, float& mult) {
  if constexpr (Q == 4) {
    const int w = p >> 2, i = p & 3;
    ea = 8 * w + i;
    eb = ea + 4;
    mult = (i & 1) ? 0.0625f : 1.f;
  } else if constexpr (Q == 2) {
    const int w = p >> 3, e = p & 7;
    ea = 16 * w + e;
    eb = ea + 8;
    const int m3 = e % 3;
    mult = (m3 == 0) ? 1.f : (m3 == 1 ? 0.25f : 0.0625f);
  } else {
    if (p < 16) {
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
}

// Pair p of one row's sub-chunk as an fp16x2 subnormal operand.
template <int Q>
__device__ __forceinline__ uint32_t unpack_pair(const uint32_t (&w)[QT<Q>::NW], int p) {
  if constexpr (Q == 4) {
    const uint32_t v = (p & 2) ? (w[p >> 2] >> 8) : w[p >> 2];
    return v & ((p & 1) ? 0x00F000F0u : 0x000F000Fu);
  } else {
    if (Q == 2 || p < 16) {
      const int e = p & 7;
      const uint32_t word = w[(p >> 3) & 1];
      const uint32_t v = e < 3 ? word : (e < 6 ? (word >> 6) : (word >> 12));
      const int m3 = e % 3;
      return v & (0x00030003u << (2 * m3));
    } else {
      const int j = p - 16;
      return (w[2] >> (4 * (j >> 2))) & (0x00010001u << (j & 3));
    }
  }
}

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                         uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Load the words of one 32-code sub-chunk (index sc) of group `grp` of the
// row whose codes start at `row`.  Zero when !valid.
template <int Q>
__device__ __forceinline__ void load_sub(const uint8_t* __restrict__ row, int grp,
                                         int sc, int G, bool valid,
                                         uint32_t (&w)[QT<Q>::NW]) {
  if constexpr (Q == 4) {
    uint4 v = make_uint4(0, 0, 0, 0);
    if (valid)
      v = __ldcs(reinterpret_cast<const uint4*>(row + static_cast<int64_t>(grp) * (G / 2) + sc * 16));
    w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
  } else if constexpr (Q == 2) {
    uint2 v = make_uint2(0, 0);
    if (valid)
      v = __ldcs(reinterpret_cast<const uint2*>(row + static_cast<int64_t>(grp) * (G / 4) + sc * 8));
    w[0] = v.x; w[1] = v.y;
  } else {
    w[0] = w[1] = w[2] = 0;
    if (valid) {
      const uint32_t* base = reinterpret_cast<const uint32_t*>(
          row + static_cast<int64_t>(grp) * (3 * G / 8));
      w[0] = __ldcs(base + 2 * sc);
      w[1] = __ldcs(base + 2 * sc + 1);
      w[2] = __ldcs(base + G / 16 + sc);
    }
  }
}

struct GemvArgs {
  const uint8_t* codes;
  const uint16_t* scales;
  const uint16_t* mins;
  const uint16_t* x;  // bf16 [batch][k]
  float* y;           // fp32 [batch][n]
  int64_t n, k;
  int G;
  int batch;
  int steps_per_cta;  // 8-group steps handled by one CTA
  int window_groups;  // groups staged in shared memory at once
};

// shared memory carve-up (bytes) for a window of `wg` groups
__host__ __device__ __forceinline__ int pitch_bytes(int q, int G) {
  return (G / 32) * (q == 3 ? 128 : 64) + 16;
}

// Registers of one work unit: the codes of one 32-code sub-chunk (sc) of the
// lane's two groups (h = 0, 1) for its RT x 2 rows, plus, for the first
// sub-chunk of a step, the fp16 scales (and mins) of those groups.
template <int Q, int RT>
struct Unit {
  uint32_t w[2][RT][2][QT<Q>::NW];
  uint32_t s[RT][2];  // two fp16: groups 2t and 2t+1 of the step
  uint32_t m[RT][2];
};

template <int Q, bool ASYM, int NB, int RT>
__global__ void __launch_bounds__(kMaxWarps * 32)
    gemv_kernel(const GemvArgs a) {
  constexpr int NP = QT<Q>::NP;
  constexpr int NW = QT<Q>::NW;
  constexpr int HALF = 1 << (Q - 1);
  extern __shared__ __align__(16) unsigned char smem[];

  const int G = a.G;
  const int SC = G / 32;  // 32-code sub-chunks per group
  const int pitch = pitch_bytes(Q, G);
  const int wg = a.window_groups;
  const int nwarps = blockDim.x >> 5;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;  // mma fragment coordinates
  const int64_t nG = a.k / G;

  // shared memory: [NB][wg][pitch] arranged activations | zero block |
  // [NB][wg] bias terms | [nwarps][NB][RT*16] warp partials | [NB][RT*16]
  unsigned char* xs = smem;
  unsigned char* zero = xs + static_cast<size_t>(NB) * wg * pitch;
  float* bias = reinterpret_cast<float*>(zero + 128);
  float* wpart = bias + NB * wg;
  float* cpart = wpart + nwarps * NB * RT * 16;

  const int64_t row0 = static_cast<int64_t>(blockIdx.x) * (RT * 16);
  const int64_t step_lo = static_cast<int64_t>(blockIdx.y) * a.steps_per_cta;
  const int64_t nsteps_total = (nG + 7) / 8;
  const int64_t step_hi = min(step_lo + a.steps_per_cta, nsteps_total);
  const int64_t row_bytes = a.k * Q / 8;

  // rows this lane feeds: tile tt, half hh -> row0 + 16*tt + gq + 8*hh
  const uint8_t* rowp[RT][2];
  const uint16_t* srow[RT][2];
  const uint16_t* mrow[RT][2];
  bool rowok[RT][2];
#pragma unroll
  for (int tt = 0; tt < RT; ++tt)
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const int64_t r = row0 + 16 * tt + gq + 8 * hh;
      rowok[tt][hh] = r < a.n;
      const int64_t rr = rowok[tt][hh] ? r : 0;
      rowp[tt][hh] = a.codes + rr * row_bytes;
      srow[tt][hh] = a.scales + rr * nG;
      mrow[tt][hh] = ASYM ? a.mins + rr * nG : nullptr;
    }

  // unit u of this warp in the window starting at step wstep:
  // step = wstep + warp + (u / SC) * nwarps, sc = u % SC
  auto load_unit = [&](Unit<Q, RT>& U, int64_t step, int sc) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int64_t grp = step * 8 + 2 * tq + h;
      const bool gok = grp < nG;
#pragma unroll
      for (int tt = 0; tt < RT; ++tt)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh)
          load_sub<Q>(rowp[tt][hh], static_cast<int>(grp), sc, G, gok && rowok[tt][hh],
                      U.w[h][tt][hh]);
    }
    if (sc == 0) {
      const int64_t g0 = step * 8 + 2 * tq;
#pragma unroll
      for (int tt = 0; tt < RT; ++tt)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          uint32_t lo = 0, hi = 0, mlo = 0, mhi = 0;
          if (rowok[tt][hh] && g0 < nG) {
            lo = __ldcs(srow[tt][hh] + g0);
            if constexpr (ASYM) mlo = __ldcs(mrow[tt][hh] + g0);
          }
          if (rowok[tt][hh] && g0 + 1 < nG) {
            hi = __ldcs(srow[tt][hh] + g0 + 1);
            if constexpr (ASYM) mhi = __ldcs(mrow[tt][hh] + g0 + 1);
          }
          U.s[tt][hh] = lo | (hi << 16);
          U.m[tt][hh] = mlo | (mhi << 16);
        }
    }
  };

  float acc[NB][RT][2];
#pragma unroll
  for (int b = 0; b < NB; ++b)
#pragma unroll
    for (int tt = 0; tt < RT; ++tt) acc[b][tt][0] = acc[b][tt][1] = 0.f;
  float d[NB][RT][4];
  uint32_t st[RT][2], mt[RT][2];  // scales of the step being accumulated

  for (int i = threadIdx.x; i < 32; i += blockDim.x) reinterpret_cast<uint32_t*>(zero)[i] = 0u;

  Unit<Q, RT> ua, ub;
  for (int64_t wstep = step_lo; wstep < step_hi; wstep += wg / 8) {
    const int64_t wgrp0 = wstep * 8;  // first group of the window
    const int64_t wsteps_end = min(step_hi, wstep + wg / 8);
    const int ngrp_win = static_cast<int>(min(static_cast<int64_t>(wg), nG - wgrp0));
    const int64_t my_steps =
        (wstep + warp < wsteps_end) ? (wsteps_end - (wstep + warp) + nwarps - 1) / nwarps : 0;
    const int nunits = static_cast<int>(my_steps) * SC;

    // the first unit's code loads go out before the activations are staged
    if (nunits > 0) load_unit(ua, wstep + warp, 0);

    __syncthreads();  // previous window fully consumed
    // ---- stage activations in mma order (one thread per batch row x group) ----
    for (int it = threadIdx.x; it < NB * ngrp_win; it += blockDim.x) {
      const int b = it / ngrp_win, gl = it - b * ngrp_win;
      unsigned char* dst = xs + (static_cast<size_t>(b) * wg + gl) * pitch;
      float sum = 0.f;
      for (int sc = 0; sc < SC; ++sc) {
        float xv[32];
        if (b < a.batch) {
          const uint4* src = reinterpret_cast<const uint4*>(
              a.x + static_cast<int64_t>(b) * a.k + (wgrp0 + gl) * G + sc * 32);
          uint4 v[4];
#pragma unroll
          for (int c = 0; c < 4; ++c) v[c] = __ldg(src + c);
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const uint32_t wv[4] = {v[c].x, v[c].y, v[c].z, v[c].w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              xv[8 * c + 2 * e] = __uint_as_float(wv[e] << 16);
              xv[8 * c + 2 * e + 1] = __uint_as_float(wv[e] & 0xFFFF0000u);
            }
          }
        } else {
#pragma unroll
          for (int e = 0; e < 32; ++e) xv[e] = 0.f;
        }
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
#pragma unroll
        for (int c = 0; c < NP / 4; ++c)
          *reinterpret_cast<uint4*>(dst + sc * NP * 4 + 16 * c) =
              make_uint4(pr[4 * c], pr[4 * c + 1], pr[4 * c + 2], pr[4 * c + 3]);
      }
      // symmetric: -2^(q-1) * 2^-24 * sum_g x; asymmetric: 2^-24 * sum_g x
      bias[b * wg + gl] = ASYM ? sum * 0x1p-24f : -static_cast<float>(HALF) * 0x1p-24f * sum;
    }
    __syncthreads();

    auto compute_unit = [&](const Unit<Q, RT>& U, int u) {
      const int64_t step = wstep + warp + static_cast<int64_t>(u / SC) * nwarps;
      const int sc = u % SC;
      const int gl0 = static_cast<int>(step * 8 - wgrp0);
      if (sc == 0) {
#pragma unroll
        for (int b = 0; b < NB; ++b)
#pragma unroll
          for (int tt = 0; tt < RT; ++tt) d[b][tt][0] = d[b][tt][1] = d[b][tt][2] = d[b][tt][3] = 0.f;
#pragma unroll
        for (int tt = 0; tt < RT; ++tt)
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            st[tt][hh] = U.s[tt][hh];
            mt[tt][hh] = U.m[tt][hh];
          }
      }
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        // column gq of B carries group step*8 + gq; it is this lane's own
        // group for h iff gq == 2*tq + h.  Other lanes read zeros.
        const bool active = (gq == 2 * tq + h) && (step * 8 + gq < nG);
        const unsigned char* xp0 =
            active ? xs + static_cast<size_t>(gl0 + gq) * pitch + sc * NP * 4 : zero;
        const size_t bstride = active ? static_cast<size_t>(wg) * pitch : 0;
#pragma unroll
        for (int j = 0; j < NP / 2; j += 2) {  // two mmas per 16-byte B load
          uint32_t A[2][RT][4];
#pragma unroll
          for (int jj = 0; jj < 2; ++jj) {
            const int p = 2 * (j + jj);
#pragma unroll
            for (int tt = 0; tt < RT; ++tt) {
              A[jj][tt][0] = unpack_pair<Q>(U.w[h][tt][0], p);      // row g,   k 2t..
              A[jj][tt][1] = unpack_pair<Q>(U.w[h][tt][1], p);      // row g+8, k 2t..
              A[jj][tt][2] = unpack_pair<Q>(U.w[h][tt][0], p + 1);  // row g,   k 2t+8..
              A[jj][tt][3] = unpack_pair<Q>(U.w[h][tt][1], p + 1);  // row g+8, k 2t+8..
            }
          }
#pragma unroll
          for (int b = 0; b < NB; ++b) {
            const uint4 bv = *reinterpret_cast<const uint4*>(xp0 + b * bstride + j * 8);
#pragma unroll
            for (int tt = 0; tt < RT; ++tt) {
              mma16816(d[b][tt], A[0][tt][0], A[0][tt][1], A[0][tt][2], A[0][tt][3], bv.x, bv.y);
              mma16816(d[b][tt], A[1][tt][0], A[1][tt][1], A[1][tt][2], A[1][tt][3], bv.z, bv.w);
            }
          }
        }
      }
      if (sc == SC - 1) {
        // per-group scale (and min): lane holds columns 2tq, 2tq+1 = its groups
        const int gl = gl0 + 2 * tq;
        const bool ok0 = step * 8 + 2 * tq < nG, ok1 = step * 8 + 2 * tq + 1 < nG;
#pragma unroll
        for (int tt = 0; tt < RT; ++tt)
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const __half2 s2 = *reinterpret_cast<const __half2*>(&st[tt][hh]);
            const float2 sf = __half22float2(s2);
            float2 mf = make_float2(0.f, 0.f);
            if constexpr (ASYM) mf = __half22float2(*reinterpret_cast<const __half2*>(&mt[tt][hh]));
#pragma unroll
            for (int b = 0; b < NB; ++b) {
              const float b0v = ok0 ? bias[b * wg + gl] : 0.f;
              const float b1v = ok1 ? bias[b * wg + gl + 1] : 0.f;
              const float d0 = d[b][tt][2 * hh], d1 = d[b][tt][2 * hh + 1];
              if constexpr (ASYM) {
                acc[b][tt][hh] += sf.x * d0 + mf.x * b0v + sf.y * d1 + mf.y * b1v;
              } else {
                acc[b][tt][hh] += sf.x * (d0 + b0v) + sf.y * (d1 + b1v);
              }
            }
          }
      }
    };

    // ---- ping-pong over this warp's units: loads run one unit ahead ----
    auto unit_step = [&](int64_t uu) { return wstep + warp + (uu / SC) * nwarps; };
    for (int u = 0; u < nunits; u += 2) {
      if (u + 1 < nunits) load_unit(ub, unit_step(u + 1), (u + 1) % SC);
      compute_unit(ua, u);
      if (u + 1 < nunits) {
        if (u + 2 < nunits) load_unit(ua, unit_step(u + 2), (u + 2) % SC);
        compute_unit(ub, u + 1);
      }
    }
  }

  // ---- reduce: the 4 lanes of a quad, then the CTA's warps, then the cluster ----
#pragma unroll
  for (int b = 0; b < NB; ++b)
#pragma unroll
    for (int tt = 0; tt < RT; ++tt)
#pragma unroll
      for (int hh = 0; hh < 2; ++hh) {
        float v = acc[b][tt][hh];
        v += __shfl_xor_sync(0xffffffffu, v, 1);
        v += __shfl_xor_sync(0xffffffffu, v, 2);
        if (tq == 0) wpart[(warp * NB + b) * (RT * 16) + 16 * tt + gq + 8 * hh] = v;
      }
  __syncthreads();
  for (int i = threadIdx.x; i < NB * RT * 16; i += blockDim.x) {
    float v = 0.f;
    for (int wv = 0; wv < nwarps; ++wv) v += wpart[wv * NB * RT * 16 + i];
    cpart[i] = v;
  }
  cg::cluster_group cluster = cg::this_cluster();
  const unsigned ks = cluster.num_blocks();
  if (ks > 1) {
    cluster.sync();
    if (cluster.block_rank() == 0) {
      for (int i = threadIdx.x; i < NB * RT * 16; i += blockDim.x) {
        float v = 0.f;
        for (unsigned rk = 0; rk < ks; ++rk) v += cluster.map_shared_rank(cpart, rk)[i];
        cpart[i] = v;
      }
    }
    cluster.sync();
    if (cluster.block_rank() != 0) return;
  } else {
    __syncthreads();
  }
  for (int i = threadIdx.x; i < NB * RT * 16; i += blockDim.x) {
    const int b = i / (RT * 16), rl = i - b * RT * 16;
    const int64_t r = row0 + rl;
    if (b < a.batch && r < a.n) a.y[static_cast<int64_t>(b) * a.n + r] = cpart[i] * 0x1p24f;
  }
}

struct Plan {
  int rt, nb, ks, warps, steps_per_cta, window_groups;
  int64_t row_tiles;
  size_t smem;
};

Plan make_plan(const sss_qtensor_t& t, int batch) {
  Plan p{};
  p.nb = batch <= 1 ? 1 : (batch <= 2 ? 2 : (batch <= 4 ? 4 : (batch <= 8 ? 8 : 16)));
  p.rt = (p.nb == 1) ? 2 : 1;
  const int64_t nG = t.k / t.group;
  const int64_t nsteps = (nG + 7) / 8;
  p.row_tiles = (t.n + p.rt * 16 - 1) / (p.rt * 16);
  const int sms = device_sm_count();
  int ks = static_cast<int>((2 * static_cast<int64_t>(sms) + p.row_tiles - 1) /
                            (p.row_tiles > 0 ? p.row_tiles : 1));
  ks = std::max(1, std::min<int>(ks, kMaxKS));
  ks = static_cast<int>(std::min<int64_t>(ks, std::max<int64_t>(1, nsteps)));
  p.steps_per_cta = static_cast<int>((nsteps + ks - 1) / std::max(1, ks));
  if (p.steps_per_cta < 1) p.steps_per_cta = 1;
  p.ks = static_cast<int>((nsteps + p.steps_per_cta - 1) / p.steps_per_cta);
  if (p.ks < 1) p.ks = 1;
  p.warps = std::max(1, std::min(kMaxWarps, p.steps_per_cta));
  const int pitch = pitch_bytes(t.q, t.group);
  // stage as much of the CTA's k-range as fits in ~48 KB, in whole steps
  int win = static_cast<int>((48 * 1024) / (static_cast<int64_t>(p.nb) * pitch)) / 8 * 8;
  win = std::max(8, win);
  p.window_groups = static_cast<int>(std::min<int64_t>(win, static_cast<int64_t>(p.steps_per_cta) * 8));
  p.smem = static_cast<size_t>(p.nb) * p.window_groups * pitch + 128 +
           sizeof(float) * (static_cast<size_t>(p.nb) * p.window_groups +
                            static_cast<size_t>(p.warps) * p.nb * p.rt * 16 +
                            static_cast<size_t>(p.nb) * p.rt * 16);
  return p;
}

template <int Q, bool ASYM, int NB, int RT>
cudaError_t run(const sss_qtensor_t& t, const uint16_t* x, int batch, float* y,
                const Plan& p, cudaStream_t stream) {
  auto kern = gemv_kernel<Q, ASYM, NB, RT>;
  cudaError_t e = ensure_smem(kern, static_cast<int>(p.smem));
  if (e != cudaSuccess) return e;
  GemvArgs a;
  a.codes = t.codes;
  a.scales = t.scales;
  a.mins = t.mins;
  a.x = x;
  a.y = y;
  a.n = t.n;
  a.k = t.k;
  a.G = t.group;
  a.batch = batch;
  a.steps_per_cta = p.steps_per_cta;
  a.window_groups = p.window_groups;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(p.row_tiles), static_cast<unsigned>(p.ks), 1);
  cfg.blockDim = dim3(32 * p.warps, 1, 1);
  cfg.dynamicSmemBytes = p.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = static_cast<unsigned>(p.ks);
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int Q, bool ASYM>
cudaError_t dispatch_nb(const sss_qtensor_t& t, const uint16_t* x, int batch,
                        float* y, const Plan& p, cudaStream_t stream) {
  switch (p.nb) {
    case 1: return run<Q, ASYM, 1, 2>(t, x, batch, y, p, stream);
    case 2: return run<Q, ASYM, 2, 1>(t, x, batch, y, p, stream);
    case 4: return run<Q, ASYM, 4, 1>(t, x, batch, y, p, stream);
    case 8: return run<Q, ASYM, 8, 1>(t, x, batch, y, p, stream);
    case 16: return run<Q, ASYM, 16, 1>(t, x, batch, y, p, stream);
  }
  return cudaErrorInvalidValue;
}

template <int Q>
cudaError_t dispatch_grid(const sss_qtensor_t& t, const uint16_t* x, int batch,
                          float* y, const Plan& p, cudaStream_t stream) {
  if (t.grid == SSS_GRID_ASYM) return dispatch_nb<Q, true>(t, x, batch, y, p, stream);
  return dispatch_nb<Q, false>(t, x, batch, y, p, stream);
}

}  // namespace

size_t gemv_workspace_bytes(const sss_qtensor_t&, int) { return 0; }

cudaError_t launch_gemv(const sss_qtensor_t& t, const uint16_t* x, int batch,
                        float* y, void* /*workspace*/, cudaStream_t stream) {
  if (t.n == 0 || batch == 0) return cudaSuccess;
  const Plan p = make_plan(t, batch);
  switch (t.q) {
    case 2: return dispatch_grid<2>(t, x, batch, y, p, stream);
    case 3: return dispatch_grid<3>(t, x, batch, y, p, stream);
    case 4: return dispatch_grid<4>(t, x, batch, y, p, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace sss
