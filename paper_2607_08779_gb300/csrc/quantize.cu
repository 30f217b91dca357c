// quantize.cu -- group-wise q-bit weight quantizer and dequantizer for
// sm_103a.
//
// Quantizer (direct casting, Appendix C.1): per group of G weights along k,
//   M = ||w||_inf, alpha = M / 2^(q-1)                          (eq:absmax)
//   gamma = -sign(w_i*) for the signed grid, +1 otherwise       (eq:sign_rule)
//   c = clip(RNE(w / (gamma*alpha)), A_q), u = c + 2^(q-1)      (eq:quantizer)
// or, for the min-max grid, s = (max-min)/(2^q-1) and u = clip(RNE((w-min)/s))
// (eq:minmax).  The rounding is that of the EXACT quotient (ties to even):
// the kernel rounds w * RN(1/s) to an integer and, when that product lies
// within 2^-18 of a half-integer, decides the side with the exact residual
// w - h*s of one fused multiply-add (a single rounding keeps the residual's
// sign exact).  Away from a half-integer the product's error (<= 2^-20 for
// |w/s| < 16) cannot change the rounded value.
//
// Memory layout: the fp32 weights and the outputs are flat arrays of groups
// (group G at element G*G_SIZE), so the kernel is a grid-stride sweep over
// groups.  G/32 lanes own a group, each lane a run of 32 weights (eight
// 16-byte streaming loads); the group max/min of more than one lane are
// butterfly shuffles.  Each lane packs its 32 codes into one vector store;
// lane 0 of the group stores the fp16 scale (and min, and clip counts).
// All per-weight arithmetic is on the full-rate FP32/integer pipes (no
// conversion instructions).  HBM-bound: 4 bytes read and q/8 + 2/G (+2/G)
// bytes written per weight.
#include <math.h>

#include <algorithm>

#include "rne.cuh"
#include "sss_internal.cuh"

namespace sss {
namespace {

// ---------------------------------------------------------------------------
// Quantizer: persistent CTAs, one per SM.  One thread streams the fp32
// weights into a ring of shared-memory stages with 1-D bulk copies (32 KB,
// 8192 weights each), so the HBM read keeps ~190 KB per SM in flight
// without holding registers; two sets of eight warps take alternate stages.
// A stage holds 256 runs of 32 consecutive weights; lane sl of a set owns
// run sl (one run per group for G = 32, G/32 runs per group otherwise).
// The lane reads its run's eight 16-byte chunks starting at chunk sl & 7 and
// wrapping, which puts the eight lanes of every quarter-warp on distinct
// banks; the packed codes are rotated back into element order before the
// store.
// ---------------------------------------------------------------------------

constexpr int kQChunk = 8192;                            // weights per stage
constexpr int kQStages = 6;
constexpr int kQSetWarps = 8;                            // warps of one consumer set
constexpr int kQThreads = 32 * (1 + 2 * kQSetWarps);     // producer warp + two sets
constexpr int kQSmem = kQStages * kQChunk * 4 + 2 * kQStages * 8 + 16;
constexpr uint64_t kQWaitNs = 1000000000ull;             // bounded waits: 1 s

__device__ __forceinline__ uint32_t q_su32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ bool q_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// bounded wait on a phase parity; false when it gave up (its own limit, or
// *abort raised by another role)
__device__ __forceinline__ bool q_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
  if (q_try(bar, parity)) return true;
  uint64_t t0;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  for (uint32_t it = 1;; ++it) {
    if (q_try(bar, parity)) return true;
    if ((it & 255u) == 0) {
      if (*abort) return false;
      uint64_t t;
      asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
      if (t - t0 > kQWaitNs) {
        *abort = 1;
        return false;
      }
    }
  }
}

// rotate the 64-bit value (hi:lo) left by n bits (0 <= n < 64)
__device__ __forceinline__ void rotl64(uint32_t& lo, uint32_t& hi, int n) {
  uint32_t a = lo, b = hi;
  if (n & 32) {
    a = hi;
    b = lo;
  }
  lo = __funnelshift_l(b, a, n & 31);
  hi = __funnelshift_l(a, b, n & 31);
}

// Pack the run's 32 codes and store them.  u[4j + e] is element
// 4 * ((j + r) & 7) + e of the run (the chunk order the lane read in);
// lg = the run's index within its group.
template <int Q, int G>
__device__ __forceinline__ void store_run(uint8_t* __restrict__ codes, int64_t grp, int lg, int r,
                                          const int (&u)[32]) {
  if constexpr (Q == 4) {
    // chunk c's four nibbles belong at bits 16c..16c+15: pack by slot, then
    // rotate the 128-bit value left by 16r
    uint32_t P[4];
#pragma unroll
    for (int wd = 0; wd < 4; ++wd) {
      uint32_t v = 0;
#pragma unroll
      for (int e = 0; e < 8; ++e) v |= static_cast<uint32_t>(u[8 * wd + e]) << (4 * e);
      P[wd] = v;
    }
    if (r & 1) {
      const uint32_t p0 = P[0], p1 = P[1], p2 = P[2], p3 = P[3];
      P[0] = __funnelshift_l(p3, p0, 16);
      P[1] = __funnelshift_l(p0, p1, 16);
      P[2] = __funnelshift_l(p1, p2, 16);
      P[3] = __funnelshift_l(p2, p3, 16);
    }
    const bool w1 = (r & 2) != 0, w2 = (r & 4) != 0;  // rotate by one word, by two words
    const uint32_t t0 = w1 ? P[3] : P[0], t1 = w1 ? P[0] : P[1];
    const uint32_t t2 = w1 ? P[1] : P[2], t3 = w1 ? P[2] : P[3];
    const uint4 out = make_uint4(w2 ? t2 : t0, w2 ? t3 : t1, w2 ? t0 : t2, w2 ? t1 : t3);
    reinterpret_cast<uint4*>(codes + grp * (G / 2))[lg] = out;
  } else if constexpr (Q == 2) {
    uint32_t lo = 0, hi = 0;
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      lo |= static_cast<uint32_t>(u[e]) << (2 * e);
      hi |= static_cast<uint32_t>(u[16 + e]) << (2 * e);
    }
    rotl64(lo, hi, 8 * r);
    reinterpret_cast<uint2*>(codes + grp * (G / 4))[lg] = make_uint2(lo, hi);
  } else {  // low 2-bit plane (q=2 layout), then the high-bit plane
    uint32_t l0 = 0, l1 = 0, hi = 0;
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      l0 |= static_cast<uint32_t>(u[e] & 3) << (2 * e);
      l1 |= static_cast<uint32_t>(u[16 + e] & 3) << (2 * e);
    }
#pragma unroll
    for (int e = 0; e < 32; ++e) hi |= static_cast<uint32_t>(u[e] >> 2) << e;
    rotl64(l0, l1, 8 * r);
    hi = __funnelshift_l(hi, hi, 4 * r);
    uint32_t* base = reinterpret_cast<uint32_t*>(codes + grp * (3 * G / 8));
    base[2 * lg] = l0;
    base[2 * lg + 1] = l1;
    base[G / 16 + lg] = hi;
  }
}

// Quantize one run of 32 weights (x[4j + e] = element 4*((j + r) & 7) + e,
// run index gr in the flat weight array) together with the other runs of
// its group (the L = G/32 consecutive lanes of the warp): group max / min,
// scale, codes, packing, scale / min / clip-count stores.  Every lane of
// the warp calls it (valid = false for lanes past the last run).  wat(e)
// re-reads x[e] as it was passed in (the rare exact-tie decisions use it,
// so x need not stay live in registers).
template <int Q, int GRID, int G, bool STATS, class Wat>
__device__ __forceinline__ void quantize_run(float (&x)[32], Wat wat, int r, bool valid, int64_t gr,
                                             uint8_t* __restrict__ codes,
                                             uint16_t* __restrict__ scales,
                                             uint16_t* __restrict__ mins,
                                             uint8_t* __restrict__ clip,
                                             uint32_t* __restrict__ status) {
  constexpr int L = G / 32;  // lanes (runs) per group
  constexpr int HALF = 1 << (Q - 1);
  constexpr int UMAX = (1 << Q) - 1;
  constexpr int OFF = (GRID == SSS_GRID_ASYM) ? 0 : HALF;
  const int64_t grp = gr / L;
  const int lg = static_cast<int>(gr % L);
  // max with NaN propagation: a NaN anywhere makes mx NaN, an infinity
  // makes mx or mn infinite, so the run is non-finite iff they are
  float mx = x[0], mn = x[0];
#pragma unroll
  for (int e = 0; e < 32; ++e) {
    asm("max.NaN.f32 %0, %0, %1;" : "+f"(mx) : "f"(x[e]));
    mn = fminf(mn, x[e]);
  }
  unsigned bad = (is_nonfinite(mx) || is_nonfinite(mn)) ? 1u : 0u;
#pragma unroll
  for (int o = L / 2; o >= 1; o >>= 1) {
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    bad |= __shfl_xor_sync(0xffffffffu, bad, o);
  }
  unsigned flags = bad ? SSS_FLAG_NONFINITE : 0u;
  int u[32];
  int n_self = 0, n_other = 0;
  uint16_t s16, m16 = 0;
  if constexpr (GRID != SSS_GRID_ASYM) {
    // M = ||w||_inf; gamma* = -sign(w_i*): the outlier is positive iff
    // max w > -min w (a tie keeps gamma = +1).
    const float M = fmaxf(mx, -mn);
    const float gamma = (GRID == SSS_GRID_SIGNED_SYM && mx > -mn) ? -1.f : 1.f;
    const float alpha = __fmul_rn(M, 1.0f / HALF);  // M * 2^-(q-1), exact unless subnormal
    // an alpha that underflows to zero (M <= 2^(q-151)) leaves no scale
    // s != 0: such a group is quantized like an all-zero group
    const bool zero = (alpha == 0.f) || bad;
    const float s = zero ? 0.f : gamma * alpha;
    if (zero) {
#pragma unroll
      for (int e = 0; e < 32; ++e) u[e] = HALF;
    } else {
      float ss = s, sig = 1.f;
      // alpha is an exact power-of-two scaling of M unless it is
      // subnormal; then |w/s| may exceed 2^(q-1) slightly and both ends
      // clip (otherwise c_pre >= -2^(q-1) and only +2^(q-1) leaves A_q)
      const bool lo_clip = M < 0x1p-96f || M > 0x1p+96f;
      if (lo_clip) {  // keep 1/s normal: scale w and s by 2^+-64
        sig = (M < 1.f) ? 0x1p+64f : 0x1p-64f;
        ss = __fmul_rn(s, sig);
#pragma unroll
        for (int e = 0; e < 32; ++e) x[e] = __fmul_rn(x[e], sig);
      }
      const float rc = __frcp_rn(ss);
      // c_pre + 2^(q-1); w * 1 is w, so the re-read matches x in both cases
      codes_of<OFF>(x, ss, rc, u, [&](int e) { return __fmul_rn(wat(e), sig); });
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        if constexpr (STATS) {
          n_self += (u[e] == 2 * HALF);  // c_pre == +2^(q-1): in C_gamma
          n_other += (u[e] == 0);        // c_pre == -2^(q-1): in C_-gamma
        }
        u[e] = min(u[e], UMAX);
      }
      if (lo_clip) {
#pragma unroll
        for (int e = 0; e < 32; ++e) u[e] = max(u[e], 0);
      }
    }
    s16 = __half_as_ushort(__float2half_rn(s));
  } else {
    mn = __fadd_rn(mn, 0.f);  // a zero minimum is stored as +0
    mx = __fadd_rn(mx, 0.f);
    bool zero = (mx == mn) || bad;
    float s = 0.f;
    if (!zero) {
      s = __fdiv_rn(__fsub_rn(mx, mn), static_cast<float>(UMAX));
      if (is_nonfinite(s)) {
        flags |= SSS_FLAG_RANGE;
        zero = true;
      } else if (s == 0.f) {
        zero = true;
      }
    }
    if (zero) {
#pragma unroll
      for (int e = 0; e < 32; ++e) u[e] = 0;
    } else {
      float ss = s, sig = 1.f;
      if (s < 0x1p-96f || s > 0x1p+96f) {
        sig = (s < 1.f) ? 0x1p+64f : 0x1p-64f;
        ss = __fmul_rn(s, sig);
      }
      const float rc = __frcp_rn(ss);
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        x[e] = __fsub_rn(x[e], mn);  // fl32(w - min) >= 0
        if (sig != 1.f) x[e] = __fmul_rn(x[e], sig);
      }
      codes_of<0>(x, ss, rc, u, [&](int e) {
        const float d = __fsub_rn(wat(e), mn);
        return sig != 1.f ? __fmul_rn(d, sig) : d;
      });
#pragma unroll
      for (int e = 0; e < 32; ++e) u[e] = min(u[e], UMAX);
    }
    s16 = __half_as_ushort(__float2half_rn(s));  // inf when the step overflowed
    m16 = __half_as_ushort(__float2half_rn(mn));
    if ((m16 & 0x7fffu) == 0x7c00u) flags |= SSS_FLAG_RANGE;
  }
  if ((s16 & 0x7fffu) == 0x7c00u) flags |= SSS_FLAG_RANGE;
  if (valid) store_run<Q, G>(codes, grp, lg, r, u);
  if constexpr (STATS) {
#pragma unroll
    for (int o = L / 2; o >= 1; o >>= 1) {
      n_self += __shfl_xor_sync(0xffffffffu, n_self, o);
      n_other += __shfl_xor_sync(0xffffffffu, n_other, o);
    }
  }
  if (valid && lg == 0) {
    scales[grp] = s16;
    if constexpr (GRID == SSS_GRID_ASYM) mins[grp] = m16;
    if constexpr (STATS) {
      clip[2 * grp] = static_cast<uint8_t>(n_self);
      clip[2 * grp + 1] = static_cast<uint8_t>(n_other);
    }
    if (flags != 0u && status != nullptr) atomicOr(status, flags);
  }
}

template <int Q, int GRID, int G, bool STATS>
__global__ void __launch_bounds__(kQThreads, 1)
    quantize_kernel(const float* __restrict__ w, int64_t nweights, uint8_t* __restrict__ codes,
                    uint16_t* __restrict__ scales, uint16_t* __restrict__ mins,
                    uint8_t* __restrict__ clip, uint32_t* __restrict__ status) {
  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kQStages * kQChunk * 4);
  uint64_t* empty = full + kQStages;
  volatile int* abort = reinterpret_cast<volatile int*>(empty + kQStages);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t nchunks = (nweights + kQChunk - 1) / kQChunk;
  // this CTA's chunks: blockIdx.x + i * gridDim.x, i = 0 .. my - 1
  const int64_t my =
      blockIdx.x < nchunks ? (nchunks - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kQStages; ++s) {
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(q_su32(&full[s])) : "memory");
      asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(q_su32(&empty[s])),
                   "r"(kQSetWarps)
                   : "memory");
    }
    *abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // Launched as a programmatic dependent launch: the set-up above may run
  // while the preceding kernel drains; no global memory is touched before
  // that kernel has completed.  The next kernel may be scheduled at once
  // (it, in turn, waits for this one before it reads what this writes).
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  __syncthreads();

  if (warp == 0) {
    // ---------------- producer: bulk copies into the ring ----------------
    if (lane == 0) {
      int64_t issued = 0;
      for (int64_t i = 0; i < my; ++i) {
        const int s = static_cast<int>(i % kQStages);
        const uint32_t ph = static_cast<uint32_t>(i / kQStages) & 1u;
        if (!q_wait(q_su32(&empty[s]), ph ^ 1u, abort)) break;
        const int64_t w0 = (blockIdx.x + i * gridDim.x) * static_cast<int64_t>(kQChunk);
        const uint32_t bytes =
            static_cast<uint32_t>((nweights - w0 < kQChunk ? nweights - w0 : kQChunk) * 4);
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(
                         q_su32(&full[s])),
                     "r"(bytes)
                     : "memory");
        asm volatile(
            "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, "
            "[%3];" ::"r"(q_su32(smem + s * kQChunk * 4)),
            "l"(w + w0), "r"(bytes), "r"(q_su32(&full[s]))
            : "memory");
        issued = i + 1;
      }
      if (*abort) {  // copies still in flight must land before the CTA exits
        int drain = 0;
        for (int64_t i = issued > kQStages ? issued - kQStages : 0; i < issued; ++i)
          (void)q_wait(q_su32(&full[i % kQStages]), static_cast<uint32_t>(i / kQStages) & 1u,
                       &drain);
      }
    }
  } else {
    // ---------------- consumers: set `set` takes local chunks i = set, set + 2, ... --------
    const int set = (warp - 1) / kQSetWarps;
    const int sl = ((warp - 1) % kQSetWarps) * 32 + lane;  // run within the chunk
    const int r = sl & 7;                                  // first chunk this lane reads
    for (int64_t i = set; i < my; i += 2) {
      const int s = static_cast<int>(i % kQStages);
      if (!q_wait(q_su32(&full[s]), static_cast<uint32_t>(i / kQStages) & 1u, abort)) break;
      const int64_t w0 = (blockIdx.x + i * gridDim.x) * static_cast<int64_t>(kQChunk);
      const int64_t nrun = (nweights - w0 < kQChunk ? nweights - w0 : kQChunk) / 32;
      const bool valid = sl < nrun;
      float x[32];
      const uint32_t run_a = q_su32(smem + s * kQChunk * 4 + sl * 128);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (valid)
          asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];"
                       : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                       : "r"(run_a + 16u * static_cast<uint32_t>((j + r) & 7)));
        x[4 * j] = v.x; x[4 * j + 1] = v.y; x[4 * j + 2] = v.z; x[4 * j + 3] = v.w;
      }
      // the stage is released after the run is quantized: the rare exact
      // tie decisions re-read their weights from it
      quantize_run<Q, GRID, G, STATS>(
          x,
          [&](int e) {
            float v = 0.f;
            if (valid)
              asm volatile("ld.shared.f32 %0, [%1];"
                           : "=f"(v)
                           : "r"(run_a + 16u * static_cast<uint32_t>(((e >> 2) + r) & 7) +
                                 4u * static_cast<uint32_t>(e & 3)));
            return v;
          },
          r, valid, w0 / 32 + sl, codes, scales, mins, clip, status);
      __syncwarp();
      if (lane == 0)
        asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(q_su32(&empty[s]))
                     : "memory");
    }
  }
  __syncthreads();
  if (*abort && threadIdx.x == 0 && status != nullptr) atomicOr(status, SSS_FLAG_TIMEOUT);
}

// ---------------------------------------------------------------------------
// Normalized Hadamard rotation of the weights (Sec. 5 "Composition with PTQ
// methods"; Appendix C: mergeable rotations folded into the weights, grids
// computed on the rotated weights).  The transform of a block of b values
// (b a power of two) is the in-place fast Walsh-Hadamard transform in IEEE
// fp32 -- strides h = 1, 2, ..., b/2, butterflies (a, c) -> (a + c, a - c)
// -- then every value times norm = the fp32 nearest to 1/sqrt(b).  The
// butterflies of one stage are independent, so any assignment of them to
// threads gives the same bits as the sequential loop.
// A CTA takes 8192 values at a time into shared memory: 8192/b blocks of a
// row (input side), or b rows of 8192/b columns (output side).
// ---------------------------------------------------------------------------

constexpr int kRotChunk = 8192;
constexpr int kRotThreads = 256;

// log2(b) butterfly stages over the chunk in shared memory, stride h acting
// on element index bits; `col` = values per row of the tile (1 for the
// input side: a block is contiguous; C for the output side, where the
// block runs down a column of a [b][C] tile)
__device__ __forceinline__ void fwht_chunk(float* s, int b, int col) {
  const int half = kRotChunk / 2;
  for (int h = 1; h < b; h <<= 1) {
    const int hs = h * col;  // element distance of the butterfly pair
    for (int beta = threadIdx.x; beta < half; beta += kRotThreads) {
      // butterfly beta: the pair's lower element has bit log2(hs) clear
      const int j = ((beta / hs) * 2 * hs) + (beta % hs);
      const float a = s[j], c = s[j + hs];
      s[j] = __fadd_rn(a, c);
      s[j + hs] = __fsub_rn(a, c);
    }
    __syncthreads();
  }
}

// input side: out[r][c0 .. c0+b) = H_b w[r][c0 .. c0+b) / sqrt(b)
__global__ void __launch_bounds__(kRotThreads)
    hadamard_rows_kernel(const float* __restrict__ w, float* __restrict__ out, int64_t nweights,
                         int b, float norm) {
  __shared__ __align__(16) float s[kRotChunk];
  const int64_t nchunks = (nweights + kRotChunk - 1) / kRotChunk;
  for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const int64_t w0 = c * kRotChunk;
    const int nv = static_cast<int>(nweights - w0 < kRotChunk ? nweights - w0 : kRotChunk);
    for (int i = threadIdx.x; i < kRotChunk / 4; i += kRotThreads)
      reinterpret_cast<float4*>(s)[i] =
          4 * i < nv ? __ldcs(reinterpret_cast<const float4*>(w + w0) + i)
                     : make_float4(0.f, 0.f, 0.f, 0.f);
    __syncthreads();
    fwht_chunk(s, b, 1);
    for (int i = threadIdx.x; i < nv / 4; i += kRotThreads) {
      float4 v = reinterpret_cast<float4*>(s)[i];
      v.x = __fmul_rn(v.x, norm); v.y = __fmul_rn(v.y, norm);
      v.z = __fmul_rn(v.z, norm); v.w = __fmul_rn(v.w, norm);
      reinterpret_cast<float4*>(out + w0)[i] = v;
    }
    __syncthreads();
  }
}

// output side: for every column, out[r0 .. r0+b)[c] = H_b w[r0 .. r0+b)[c] / sqrt(b);
// a tile is b rows x C = 8192/b columns (16-byte accesses when C >= 4)
__global__ void __launch_bounds__(kRotThreads)
    hadamard_cols_kernel(const float* __restrict__ w, float* __restrict__ out, int64_t n,
                         int64_t k, int b, float norm) {
  __shared__ __align__(16) float s[kRotChunk];
  const int C = kRotChunk / b;
  const int vec = C >= 4 ? 4 : 1;
  const int64_t tiles_c = k / C, tiles = (n / b) * tiles_c;
  for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    const int64_t r0 = (t / tiles_c) * b, c0 = (t % tiles_c) * C;
    for (int i = threadIdx.x; i < kRotChunk / vec; i += kRotThreads) {
      const int e = vec * i, r = e / C, cc = e % C;
      const float* src = w + (r0 + r) * k + c0 + cc;
      if (vec == 4)
        reinterpret_cast<float4*>(s)[i] = __ldcs(reinterpret_cast<const float4*>(src));
      else
        s[e] = __ldcs(src);
    }
    __syncthreads();
    fwht_chunk(s, b, C);
    for (int i = threadIdx.x; i < kRotChunk / vec; i += kRotThreads) {
      const int e = vec * i, r = e / C, cc = e % C;
      float* dst = out + (r0 + r) * k + c0 + cc;
      if (vec == 4) {
        float4 v = reinterpret_cast<float4*>(s)[i];
        v.x = __fmul_rn(v.x, norm); v.y = __fmul_rn(v.y, norm);
        v.z = __fmul_rn(v.z, norm); v.w = __fmul_rn(v.w, norm);
        reinterpret_cast<float4*>(dst)[0] = v;
      } else {
        dst[0] = __fmul_rn(s[e], norm);
      }
    }
    __syncthreads();
  }
}

// The input-side rotation fused into the quantizer: each 8192-value chunk
// is rotated in shared memory and quantized from there (the rotated fp32
// weights never reach HBM).  Thread t owns run t of the chunk and reads it
// in the rotated chunk order of the ring quantizer.
template <int Q, int GRID, int G, bool STATS>
__global__ void __launch_bounds__(kRotThreads)
    rotate_quantize_kernel(const float* __restrict__ w, int64_t nweights, int b, float norm,
                           uint8_t* __restrict__ codes, uint16_t* __restrict__ scales,
                           uint16_t* __restrict__ mins, uint8_t* __restrict__ clip,
                           uint32_t* __restrict__ status) {
  __shared__ __align__(16) float s[kRotChunk];
  const int64_t nchunks = (nweights + kRotChunk - 1) / kRotChunk;
  const int sl = threadIdx.x, r = sl & 7;
  for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const int64_t w0 = c * kRotChunk;
    const int nv = static_cast<int>(nweights - w0 < kRotChunk ? nweights - w0 : kRotChunk);
    for (int i = threadIdx.x; i < kRotChunk / 4; i += kRotThreads)
      reinterpret_cast<float4*>(s)[i] =
          4 * i < nv ? __ldcs(reinterpret_cast<const float4*>(w + w0) + i)
                     : make_float4(0.f, 0.f, 0.f, 0.f);
    __syncthreads();
    fwht_chunk(s, b, 1);
    const bool valid = 32 * sl < nv;
    float x[32];
    const float4* run = reinterpret_cast<const float4*>(s + 32 * sl);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float4 v = run[(j + r) & 7];
      x[4 * j] = __fmul_rn(v.x, norm); x[4 * j + 1] = __fmul_rn(v.y, norm);
      x[4 * j + 2] = __fmul_rn(v.z, norm); x[4 * j + 3] = __fmul_rn(v.w, norm);
    }
    quantize_run<Q, GRID, G, STATS>(
        x,
        [&](int e) {
          return __fmul_rn(reinterpret_cast<const float*>(run)[4 * (((e >> 2) + r) & 7) + (e & 3)],
                           norm);
        },
        r, valid, w0 / 32 + sl, codes, scales, mins, clip, status);
    __syncthreads();  // the chunk is read: the next one may overwrite it
  }
}

// ---------------------------------------------------------------------------
// Dequantizer: w^ = f16(s)*c (exact in fp32) or fl32(fl32(f16(s)*u) + f16(m)).
// One thread per 8 consecutive weights of a group.
// ---------------------------------------------------------------------------

template <int Q>
__device__ __forceinline__ void load_codes8(const uint8_t* __restrict__ codes,
                                            int64_t group, int j, int G,
                                            int (&u)[8]) {
  if constexpr (Q == 4) {
    const uint32_t b = *reinterpret_cast<const uint32_t*>(codes + group * (G / 2) + j / 2);
#pragma unroll
    for (int e = 0; e < 8; ++e) u[e] = (b >> (4 * e)) & 0xf;
  } else if constexpr (Q == 2) {
    const uint16_t b = *reinterpret_cast<const uint16_t*>(codes + group * (G / 4) + j / 4);
#pragma unroll
    for (int e = 0; e < 8; ++e) u[e] = (b >> (2 * e)) & 0x3;
  } else {
    const uint8_t* base = codes + group * (3 * G / 8);
    const uint16_t lo = *reinterpret_cast<const uint16_t*>(base + j / 4);
    const uint8_t hi = base[G / 4 + j / 8];
#pragma unroll
    for (int e = 0; e < 8; ++e) u[e] = ((lo >> (2 * e)) & 0x3) | (((hi >> e) & 1) << 2);
  }
}

template <int Q, int GRID, int OUT>
__global__ void __launch_bounds__(256)
    dequantize_kernel(const uint8_t* __restrict__ codes,
                      const uint16_t* __restrict__ scales,
                      const uint16_t* __restrict__ mins, int64_t nvec, int G,
                      void* __restrict__ out) {
  constexpr int HALF = 1 << (Q - 1);
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
       i < nvec; i += stride) {
    const int64_t e0 = i * 8;
    const int64_t group = e0 / G;
    const int j = static_cast<int>(e0 - group * G);
    int u[8];
    load_codes8<Q>(codes, group, j, G, u);
    const float s = __half2float(__ushort_as_half(scales[group]));
    float v[8];
    if constexpr (GRID == SSS_GRID_ASYM) {
      const float m = __half2float(__ushort_as_half(mins[group]));
#pragma unroll
      for (int e = 0; e < 8; ++e)
        v[e] = __fadd_rn(__fmul_rn(s, static_cast<float>(u[e])), m);
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = __fmul_rn(s, static_cast<float>(u[e] - HALF));
    }
    if constexpr (OUT == SSS_OUT_F32) {
      float4* o = reinterpret_cast<float4*>(static_cast<float*>(out) + e0);
      o[0] = make_float4(v[0], v[1], v[2], v[3]);
      o[1] = make_float4(v[4], v[5], v[6], v[7]);
    } else if constexpr (OUT == SSS_OUT_F16) {
      __half2 h[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) h[e] = __floats2half2_rn(v[2 * e], v[2 * e + 1]);
      *reinterpret_cast<uint4*>(static_cast<__half*>(out) + e0) =
          *reinterpret_cast<uint4*>(h);
    } else {
      __nv_bfloat162 h[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) h[e] = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
      *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(out) + e0) =
          *reinterpret_cast<uint4*>(h);
    }
  }
}

int grid_for(int64_t work_items, int threads, int per_sm) {
  const int64_t want = (work_items + threads - 1) / threads;
  const int64_t cap = static_cast<int64_t>(device_sm_count()) * per_sm;
  return static_cast<int>(want < cap ? (want < 1 ? 1 : want) : cap);
}

template <int Q, int GRID, int G, bool STATS>
cudaError_t quantize_launch(const float* w, const sss_qtensor_t& t, uint8_t* clip,
                            uint32_t* status, cudaStream_t stream) {
  auto kern = quantize_kernel<Q, GRID, G, STATS>;
  cudaError_t e = ensure_smem(kern, kQSmem);
  if (e != cudaSuccess) return e;
  const int64_t nweights = t.n * t.k;
  const int64_t nchunks = (nweights + kQChunk - 1) / kQChunk;
  const int grid = static_cast<int>(std::min<int64_t>(device_sm_count(), nchunks));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid), 1, 1);
  cfg.blockDim = dim3(kQThreads, 1, 1);
  cfg.dynamicSmemBytes = kQSmem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, w, nweights, t.codes, t.scales, t.mins, clip, status);
}

template <int Q, int GRID, int G>
cudaError_t quantize_dispatch(const float* w, const sss_qtensor_t& t,
                              uint8_t* clip, uint32_t* status,
                              cudaStream_t stream) {
  if (clip != nullptr) return quantize_launch<Q, GRID, G, true>(w, t, clip, status, stream);
  return quantize_launch<Q, GRID, G, false>(w, t, clip, status, stream);
}

template <int Q, int GRID>
cudaError_t quantize_dispatch_g(const float* w, const sss_qtensor_t& t,
                                uint8_t* clip, uint32_t* status,
                                cudaStream_t stream) {
  switch (t.group) {
    case 32: return quantize_dispatch<Q, GRID, 32>(w, t, clip, status, stream);
    case 64: return quantize_dispatch<Q, GRID, 64>(w, t, clip, status, stream);
    case 128: return quantize_dispatch<Q, GRID, 128>(w, t, clip, status, stream);
  }
  return cudaErrorInvalidValue;
}

template <int Q>
cudaError_t quantize_dispatch_grid(const float* w, const sss_qtensor_t& t,
                                   uint8_t* clip, uint32_t* status,
                                   cudaStream_t stream) {
  switch (t.grid) {
    case SSS_GRID_UNSIGNED_SYM:
      return quantize_dispatch_g<Q, SSS_GRID_UNSIGNED_SYM>(w, t, clip, status, stream);
    case SSS_GRID_SIGNED_SYM:
      return quantize_dispatch_g<Q, SSS_GRID_SIGNED_SYM>(w, t, clip, status, stream);
    case SSS_GRID_ASYM:
      return quantize_dispatch_g<Q, SSS_GRID_ASYM>(w, t, clip, status, stream);
  }
  return cudaErrorInvalidValue;
}

template <int Q, int GRID>
cudaError_t dequant_dispatch_out(const sss_qtensor_t& t, void* out, int dtype,
                                 cudaStream_t stream) {
  const int64_t nvec = t.n * t.k / 8;
  const int grid = grid_for(nvec, 256, 16);
  switch (dtype) {
    case SSS_OUT_F32:
      dequantize_kernel<Q, GRID, SSS_OUT_F32><<<grid, 256, 0, stream>>>(
          t.codes, t.scales, t.mins, nvec, t.group, out);
      break;
    case SSS_OUT_F16:
      dequantize_kernel<Q, GRID, SSS_OUT_F16><<<grid, 256, 0, stream>>>(
          t.codes, t.scales, t.mins, nvec, t.group, out);
      break;
    case SSS_OUT_BF16:
      dequantize_kernel<Q, GRID, SSS_OUT_BF16><<<grid, 256, 0, stream>>>(
          t.codes, t.scales, t.mins, nvec, t.group, out);
      break;
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

template <int Q>
cudaError_t dequant_dispatch_grid(const sss_qtensor_t& t, void* out, int dtype,
                                  cudaStream_t stream) {
  if (t.grid == SSS_GRID_ASYM)
    return dequant_dispatch_out<Q, SSS_GRID_ASYM>(t, out, dtype, stream);
  return dequant_dispatch_out<Q, SSS_GRID_SIGNED_SYM>(t, out, dtype, stream);
}

template <int Q, int GRID, int G>
cudaError_t rotq_dispatch(const float* w, int b, float norm, const sss_qtensor_t& t,
                          uint8_t* clip, uint32_t* status, cudaStream_t stream) {
  const int64_t nweights = t.n * t.k;
  const int64_t nchunks = (nweights + kRotChunk - 1) / kRotChunk;
  const int grid = static_cast<int>(std::min<int64_t>(device_sm_count() * 8, nchunks));
  if (clip != nullptr)
    rotate_quantize_kernel<Q, GRID, G, true><<<grid, kRotThreads, 0, stream>>>(
        w, nweights, b, norm, t.codes, t.scales, t.mins, clip, status);
  else
    rotate_quantize_kernel<Q, GRID, G, false><<<grid, kRotThreads, 0, stream>>>(
        w, nweights, b, norm, t.codes, t.scales, t.mins, clip, status);
  return cudaGetLastError();
}

template <int Q, int GRID>
cudaError_t rotq_g(const float* w, int b, float norm, const sss_qtensor_t& t, uint8_t* clip,
                   uint32_t* status, cudaStream_t stream) {
  switch (t.group) {
    case 32: return rotq_dispatch<Q, GRID, 32>(w, b, norm, t, clip, status, stream);
    case 64: return rotq_dispatch<Q, GRID, 64>(w, b, norm, t, clip, status, stream);
    case 128: return rotq_dispatch<Q, GRID, 128>(w, b, norm, t, clip, status, stream);
  }
  return cudaErrorInvalidValue;
}

template <int Q>
cudaError_t rotq_grid(const float* w, int b, float norm, const sss_qtensor_t& t, uint8_t* clip,
                      uint32_t* status, cudaStream_t stream) {
  switch (t.grid) {
    case SSS_GRID_UNSIGNED_SYM:
      return rotq_g<Q, SSS_GRID_UNSIGNED_SYM>(w, b, norm, t, clip, status, stream);
    case SSS_GRID_SIGNED_SYM:
      return rotq_g<Q, SSS_GRID_SIGNED_SYM>(w, b, norm, t, clip, status, stream);
    case SSS_GRID_ASYM:
      return rotq_g<Q, SSS_GRID_ASYM>(w, b, norm, t, clip, status, stream);
  }
  return cudaErrorInvalidValue;
}

// the fp32 nearest to 1/sqrt(b)
float hadamard_norm(int b) { return static_cast<float>(1.0 / sqrt(static_cast<double>(b))); }

}  // namespace

cudaError_t launch_hadamard(const float* w, float* out, int64_t n, int64_t k, int b, int side,
                            cudaStream_t stream) {
  const int sms = device_sm_count();
  if (side == 0) {
    const int64_t nchunks = (n * k + kRotChunk - 1) / kRotChunk;
    const int grid = static_cast<int>(std::min<int64_t>(sms * 8, nchunks));
    hadamard_rows_kernel<<<grid, kRotThreads, 0, stream>>>(w, out, n * k, b, hadamard_norm(b));
  } else {
    const int64_t tiles = (n / b) * (k / (kRotChunk / b));
    const int grid = static_cast<int>(std::min<int64_t>(sms * 8, tiles));
    hadamard_cols_kernel<<<grid, kRotThreads, 0, stream>>>(w, out, n, k, b, hadamard_norm(b));
  }
  return cudaGetLastError();
}

cudaError_t launch_quantize_rotated(const float* w, int b, const sss_qtensor_t& t, uint8_t* clip,
                                    uint32_t* status, cudaStream_t stream) {
  const float norm = hadamard_norm(b);
  switch (t.q) {
    case 2: return rotq_grid<2>(w, b, norm, t, clip, status, stream);
    case 3: return rotq_grid<3>(w, b, norm, t, clip, status, stream);
    case 4: return rotq_grid<4>(w, b, norm, t, clip, status, stream);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_quantize(const float* w, const sss_qtensor_t& t,
                            uint8_t* clip, uint32_t* status,
                            cudaStream_t stream) {
  switch (t.q) {
    case 2: return quantize_dispatch_grid<2>(w, t, clip, status, stream);
    case 3: return quantize_dispatch_grid<3>(w, t, clip, status, stream);
    case 4: return quantize_dispatch_grid<4>(w, t, clip, status, stream);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_dequantize(const sss_qtensor_t& t, void* out, int dtype,
                              cudaStream_t stream) {
  switch (t.q) {
    case 2: return dequant_dispatch_grid<2>(t, out, dtype, stream);
    case 3: return dequant_dispatch_grid<3>(t, out, dtype, stream);
    case 4: return dequant_dispatch_grid<4>(t, out, dtype, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace sss
