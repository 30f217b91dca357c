// lsq.cu -- sss_quantize_lsq: symmetric-grid quantization with every
// group's scale refined by LSQ steps (Sec. 5 "Composition with learned
// rotations and grid parameters"; Appendix C: LSQ with s != 0 for the
// signed formats, s > 0 for the conventional ones).  The paper learns the
// scales through the model loss on calibration data; this path is the
// data-free reading on each group's own reconstruction loss
// L(s) = sum (s c_i - w_i)^2:
//   s_0 = the signed absmax scale gamma* alpha (or alpha > 0);
//   per step, in IEEE fp32 without fused multiply-add:
//     v_i = w_i / s,  c_i = clip(rint(v_i), -2^(q-1), 2^(q-1) - 1),
//     d_i = c_i - v_i inside the range, the clip value outside (LSQ's
//           straight-through estimate of dw^_i / ds),
//     t_i = (2 (s c_i - w_i)) d_i,  G = pairwise sum of t over the group
//           (t_i <- t_i + t_{i+h}, h = g/2, ..., 1),
//     s <- s - step * G, step = lr / sqrt(g (2^(q-1) - 1)) (LSQ's gradient
//           scale), keeping the sign of s (a step that would cross or reach
//           zero halves s instead);
//   then the codes of the refined scale by the quantizer's exact-quotient
//   rounding, packed in the library's layout, with the fp16 scale.
// One warp per group: lane l holds elements l + 32 e, so the in-lane
// levels of the pairwise sum come first and the last five are butterfly
// shuffles -- the order above, bit for bit.
#include <math.h>

#include <algorithm>

#include "rne.cuh"
#include "sss_internal.cuh"

namespace sss {
namespace {

constexpr int kLsqThreads = 256;

template <int Q, bool SIGNED, int G>
__global__ void __launch_bounds__(kLsqThreads)
    lsq_kernel(const float* __restrict__ w, int64_t ngroups, int steps, float step,
               uint8_t* __restrict__ codes, uint16_t* __restrict__ scales,
               uint32_t* __restrict__ status) {
  constexpr int E = G / 32;  // elements per lane
  constexpr int HALF = 1 << (Q - 1);
  constexpr float QN = -static_cast<float>(HALF), QP = static_cast<float>(HALF - 1);
  const int lane = threadIdx.x & 31;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (kLsqThreads / 32);
  for (int64_t grp = static_cast<int64_t>(blockIdx.x) * (kLsqThreads / 32) + (threadIdx.x >> 5);
       grp < ngroups; grp += warps) {  // warp-uniform
    float x[E];
#pragma unroll
    for (int e = 0; e < E; ++e) x[e] = __ldcs(w + grp * G + lane + 32 * e);
    // the (signed) absmax scale, as the quantizer forms it
    float mx = x[0], mn = x[0];
    unsigned bad = 0;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      mx = fmaxf(mx, x[e]);
      mn = fminf(mn, x[e]);
      bad |= is_nonfinite(x[e]);
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
      bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
    const float M = fmaxf(mx, -mn);
    const float gamma = (SIGNED && mx > -mn) ? -1.f : 1.f;
    const float alpha = __fmul_rn(M, 1.0f / HALF);
    const bool zero = (alpha == 0.f) || bad;
    float s = zero ? 0.f : gamma * alpha;
    // ---- LSQ steps ----
    if (!zero) {
      for (int it = 0; it < steps; ++it) {
        float t[E];
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const float v = __fdiv_rn(x[e], s);
          float c, d;
          if (v <= QN) {
            c = QN;
            d = QN;
          } else if (v >= QP) {
            c = QP;
            d = QP;
          } else {
            c = fminf(fmaxf(rintf(v), QN), QP);
            d = __fsub_rn(c, v);
          }
          const float err = __fsub_rn(__fmul_rn(s, c), x[e]);
          t[e] = __fmul_rn(__fmul_rn(2.f, err), d);
        }
#pragma unroll
        for (int h = E / 2; h >= 1; h >>= 1)
#pragma unroll
          for (int e = 0; e < h; ++e) t[e] = __fadd_rn(t[e], t[e + h]);
        float gsum = t[0];
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) gsum = __fadd_rn(gsum, __shfl_xor_sync(0xffffffffu, gsum, o));
        float sn = __fsub_rn(s, __fmul_rn(step, gsum));
        if (__fmul_rn(sn, s) <= 0.f) sn = __fmul_rn(s, 0.5f);
        s = sn;
      }
    }
    // ---- codes of the refined scale (exact-quotient rounding) ----
    int u[E];
    if (zero) {
#pragma unroll
      for (int e = 0; e < E; ++e) u[e] = HALF;
    } else {
      float ss = s, sig = 1.f;
      const float as = fabsf(s) * static_cast<float>(HALF);  // about ||w||_inf
      if (as < 0x1p-96f || as > 0x1p+96f) {  // keep 1/s normal: scale w and s by 2^+-64
        sig = (as < 1.f) ? 0x1p+64f : 0x1p-64f;
        ss = __fmul_rn(s, sig);
      }
      const float r = __frcp_rn(ss);
#pragma unroll
      for (int e = 0; e < E; ++e) {
        const int up = code_of<HALF>(sig == 1.f ? x[e] : __fmul_rn(x[e], sig), ss, r);
        u[e] = max(0, min(up, 2 * HALF - 1));
      }
    }
    const uint16_t s16 = __half_as_ushort(__float2half_rn(s));
    // ---- pack: element l + 32 e is code l of run e of the group ----
#pragma unroll
    for (int e = 0; e < E; ++e) {
      if constexpr (Q == 4) {  // run e: 4 words, word l/8 holds codes 8(l/8) .. +7
        uint32_t v = static_cast<uint32_t>(u[e]) << (4 * (lane & 7));
#pragma unroll
        for (int o = 1; o < 8; o <<= 1) v |= __shfl_xor_sync(0xffffffffu, v, o);
        if ((lane & 7) == 0)
          reinterpret_cast<uint32_t*>(codes + grp * (G / 2) + 16 * e)[lane >> 3] = v;
      } else if constexpr (Q == 2) {  // run e: 2 words, word l/16 holds codes 16(l/16) .. +15
        uint32_t v = static_cast<uint32_t>(u[e]) << (2 * (lane & 15));
#pragma unroll
        for (int o = 1; o < 16; o <<= 1) v |= __shfl_xor_sync(0xffffffffu, v, o);
        if ((lane & 15) == 0)
          reinterpret_cast<uint32_t*>(codes + grp * (G / 4) + 8 * e)[lane >> 4] = v;
      } else {  // q = 3: run e's low-plane words 2e, 2e+1; high-plane word G/16 + e
        uint32_t v = static_cast<uint32_t>(u[e] & 3) << (2 * (lane & 15));
#pragma unroll
        for (int o = 1; o < 16; o <<= 1) v |= __shfl_xor_sync(0xffffffffu, v, o);
        const uint32_t hi = __ballot_sync(0xffffffffu, (u[e] >> 2) & 1);
        uint32_t* base = reinterpret_cast<uint32_t*>(codes + grp * (3 * G / 8));
        if ((lane & 15) == 0) base[2 * e + (lane >> 4)] = v;
        if (lane == 0) base[G / 16 + e] = hi;
      }
    }
    if (lane == 0) {
      scales[grp] = s16;
      unsigned flags = bad ? SSS_FLAG_NONFINITE : 0u;
      if ((s16 & 0x7fffu) == 0x7c00u) flags |= SSS_FLAG_RANGE;
      if (flags != 0u && status != nullptr) atomicOr(status, flags);
    }
  }
}

template <int Q, bool SIGNED>
cudaError_t lsq_g(const float* w, const sss_qtensor_t& t, int steps, float step,
                  uint32_t* status, cudaStream_t stream) {
  const int64_t ngroups = t.n * (t.k / t.group);
  const int64_t want = (ngroups + kLsqThreads / 32 - 1) / (kLsqThreads / 32);
  const int grid = static_cast<int>(
      std::max<int64_t>(1, std::min<int64_t>(want, static_cast<int64_t>(device_sm_count()) * 8)));
  switch (t.group) {
    case 32:
      lsq_kernel<Q, SIGNED, 32><<<grid, kLsqThreads, 0, stream>>>(w, ngroups, steps, step, t.codes,
                                                                  t.scales, status);
      break;
    case 64:
      lsq_kernel<Q, SIGNED, 64><<<grid, kLsqThreads, 0, stream>>>(w, ngroups, steps, step, t.codes,
                                                                  t.scales, status);
      break;
    case 128:
      lsq_kernel<Q, SIGNED, 128><<<grid, kLsqThreads, 0, stream>>>(w, ngroups, steps, step,
                                                                   t.codes, t.scales, status);
      break;
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_quantize_lsq(const float* w, const sss_qtensor_t& t, int steps, float lr,
                                uint32_t* status, cudaStream_t stream) {
  // LSQ's gradient scale 1/sqrt(g (2^(q-1) - 1)), times the rate, in fp32
  const float gscale = static_cast<float>(
      1.0 / sqrt(static_cast<double>(t.group) * static_cast<double>((1 << (t.q - 1)) - 1)));
  const float step = lr * gscale;
  const bool sgn = t.grid == SSS_GRID_SIGNED_SYM;
  switch (t.q) {
    case 2: return sgn ? lsq_g<2, true>(w, t, steps, step, status, stream)
                       : lsq_g<2, false>(w, t, steps, step, status, stream);
    case 3: return sgn ? lsq_g<3, true>(w, t, steps, step, status, stream)
                       : lsq_g<3, false>(w, t, steps, step, status, stream);
    case 4: return sgn ? lsq_g<4, true>(w, t, steps, step, status, stream)
                       : lsq_g<4, false>(w, t, steps, step, status, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace sss
