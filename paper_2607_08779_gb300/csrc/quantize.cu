// quantize.cu -- group-wise q-bit weight quantizer and dequantizer for
// sm_103a.
//
// Quantizer (direct casting, Appendix C.1): per group of G weights along k,
//   M = ||w||_inf, alpha = M / 2^(q-1)                          (eq:absmax)
//   gamma = -sign(w_i*) for the signed grid, +1 otherwise       (eq:sign_rule)
//   c = clip(RNE(w / (gamma*alpha)), A_q), u = c + 2^(q-1)      (eq:quantizer)
// or, for the min-max grid, s = (max-min)/(2^q-1) and u = clip(RNE((w-min)/s))
// (eq:minmax).  The rounding is that of the EXACT quotient (ties to even):
// the kernel multiplies by the correctly rounded reciprocal of s and, when
// the product lies within 2^-17 of a half-integer, decides the side with the
// exact residual w - h*s of one fused multiply-add (a single rounding keeps
// the residual's sign exact).  Away from a half-integer the product's error
// (< 2^-19 for |w/s| < 16) cannot change the rounded value.
//
// Memory layout: the fp32 weights and the outputs are flat arrays of groups
// (group G at element G*G_SIZE), so the kernel is a grid-stride sweep over
// groups.  G/4 lanes own a group, each lane one 16-byte vector of 4 weights
// (a streaming load); the group max/min are butterfly shuffles over those
// lanes.  Each lane packs its 4 codes and stores them; lane 0 of the group
// stores the fp16 scale (and min, and clip counts).  HBM-bound: 4 bytes read
// and q/8 + 2/G (+2/G) bytes written per weight.
#include "sss_internal.cuh"

namespace sss {
namespace {

constexpr int kQuantThreads = 256;
constexpr int kQuantUnroll = 4;

// RNE of the exact quotient w/s given r = RN(1/s).  See the file comment.
__device__ __forceinline__ int rne_quotient(float w, float s, float r) {
  const float f = __fmul_rn(w, r);
  const float fl = floorf(f);
  const float h = __fadd_rn(fl, 0.5f);
  float c = rintf(f);
  if (fabsf(__fsub_rn(f, h)) <= 0x1p-17f) {
    const float e = __fmaf_rn(-h, s, w);     // w - h*s, one rounding
    const float side = (s > 0.f) ? e : -e;   // sign of (w/s - h)
    if (side > 0.f) {
      c = __fadd_rn(fl, 1.f);
    } else if (side < 0.f) {
      c = fl;
    } else {                                  // exact tie: to even
      c = (static_cast<int>(fl) & 1) ? __fadd_rn(fl, 1.f) : fl;
    }
  }
  return static_cast<int>(c);
}

template <int Q>
__device__ __forceinline__ void store_codes(uint8_t* __restrict__ codes,
                                            int64_t group, int lg, int G,
                                            const int (&u)[4], bool valid) {
  if constexpr (Q == 4) {
    const uint16_t v = static_cast<uint16_t>(u[0] | (u[1] << 4) | (u[2] << 8) |
                                             (u[3] << 12));
    if (valid)
      reinterpret_cast<uint16_t*>(codes + group * (G / 2))[lg] = v;
  } else if constexpr (Q == 2) {
    const uint8_t v =
        static_cast<uint8_t>(u[0] | (u[1] << 2) | (u[2] << 4) | (u[3] << 6));
    if (valid) codes[group * (G / 4) + lg] = v;
  } else {  // Q == 3: low 2-bit plane (q=2 layout), then the high-bit plane
    const uint8_t lo = static_cast<uint8_t>((u[0] & 3) | ((u[1] & 3) << 2) |
                                            ((u[2] & 3) << 4) |
                                            ((u[3] & 3) << 6));
    const unsigned hi = static_cast<unsigned>((u[0] >> 2) | ((u[1] >> 2) << 1) |
                                              ((u[2] >> 2) << 2) |
                                              ((u[3] >> 2) << 3));
    const unsigned hi_next = __shfl_down_sync(0xffffffffu, hi, 1);
    uint8_t* base = codes + group * (3 * G / 8);
    if (valid) {
      base[lg] = lo;
      if ((lg & 1) == 0) base[G / 4 + (lg >> 1)] = static_cast<uint8_t>(hi | (hi_next << 4));
    }
  }
}

template <int Q, int GRID, int G>
__global__ void __launch_bounds__(kQuantThreads)
    quantize_kernel(const float* __restrict__ w, int64_t ngroups,
                    uint8_t* __restrict__ codes, uint16_t* __restrict__ scales,
                    uint16_t* __restrict__ mins, uint8_t* __restrict__ clip,
                    uint32_t* __restrict__ status) {
  constexpr int L = G / 4;      // lanes per group
  constexpr int GPW = 32 / L;   // groups per warp per sweep
  constexpr int HALF = 1 << (Q - 1);
  constexpr int UMAX = (1 << Q) - 1;
  const int lane = threadIdx.x & 31;
  const int lg = lane % L;
  const int64_t slot =
      ((static_cast<int64_t>(blockIdx.x) * kQuantThreads + threadIdx.x) >> 5) * GPW +
      lane / L;
  const int64_t nslots = (static_cast<int64_t>(gridDim.x) * kQuantThreads >> 5) * GPW;

  for (int64_t g0 = slot; g0 - lane / L < ngroups; g0 += nslots * kQuantUnroll) {
    float4 v[kQuantUnroll];
#pragma unroll
    for (int t = 0; t < kQuantUnroll; ++t) {
      const int64_t grp = g0 + t * nslots;
      if (grp < ngroups)
        v[t] = __ldcs(reinterpret_cast<const float4*>(w + grp * G) + lg);
      else
        v[t] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int t = 0; t < kQuantUnroll; ++t) {
      const int64_t grp = g0 + t * nslots;
      const bool valid = grp < ngroups;
      float x[4] = {v[t].x, v[t].y, v[t].z, v[t].w};
      float mx = fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3]));
      float mn = fminf(fminf(x[0], x[1]), fminf(x[2], x[3]));
      unsigned bad = is_nonfinite(x[0]) | is_nonfinite(x[1]) |
                     is_nonfinite(x[2]) | is_nonfinite(x[3]);
#pragma unroll
      for (int o = L / 2; o >= 1; o >>= 1) {
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
        bad |= __shfl_xor_sync(0xffffffffu, bad, o);
      }
      unsigned flags = bad ? SSS_FLAG_NONFINITE : 0u;
      int u[4];
      int n_self = 0, n_other = 0;
      uint16_t s16, m16 = 0;
      if constexpr (GRID != SSS_GRID_ASYM) {
        // M = ||w||_inf; gamma* = -sign(w_i*): the outlier is positive iff
        // max w > -min w (a tie keeps gamma = +1).
        const float M = fmaxf(mx, -mn);
        const bool zero = (M == 0.f) || bad;
        const float gamma = (GRID == SSS_GRID_SIGNED_SYM && mx > -mn) ? -1.f : 1.f;
        const float alpha = __fmul_rn(M, 1.0f / HALF);  // M * 2^-(q-1)
        const float s = zero ? 0.f : gamma * alpha;
        float ss = s, sig = 1.f;
        if (!zero && (M < 0x1p-96f || M > 0x1p+96f)) {  // keep 1/s normal
          sig = (M < 1.f) ? 0x1p+64f : 0x1p-64f;
          ss = __fmul_rn(s, sig);
        }
        const float r = __frcp_rn(ss);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          int cp = 0;
          if (!zero) {
            const float xv = (sig == 1.f) ? x[e] : __fmul_rn(x[e], sig);
            cp = rne_quotient(xv, ss, r);
          }
          n_self += (cp == HALF);
          n_other += (cp == -HALF);
          const int c = min(max(cp, -HALF), HALF - 1);
          u[e] = c + HALF;
        }
        s16 = __half_as_ushort(__float2half_rn(s));
      } else {
        if (mn == 0.f) mn = 0.f;  // a zero minimum is stored as +0
        if (mx == 0.f) mx = 0.f;
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
        float ss = s, sig = 1.f;
        if (!zero && (s < 0x1p-96f || s > 0x1p+96f)) {
          sig = (s < 1.f) ? 0x1p+64f : 0x1p-64f;
          ss = __fmul_rn(s, sig);
        }
        const float r = zero ? 0.f : __frcp_rn(ss);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          int cp = 0;
          if (!zero) {
            float d = __fsub_rn(x[e], mn);
            if (sig != 1.f) d = __fmul_rn(d, sig);
            cp = rne_quotient(d, ss, r);
          }
          u[e] = min(max(cp, 0), UMAX);
        }
        s16 = __half_as_ushort(__float2half_rn(s));  // inf when the step overflowed
        m16 = __half_as_ushort(__float2half_rn(mn));
        if ((m16 & 0x7fffu) == 0x7c00u) flags |= SSS_FLAG_RANGE;
      }
      if ((s16 & 0x7fffu) == 0x7c00u) flags |= SSS_FLAG_RANGE;
      store_codes<Q>(codes, grp, lg, G, u, valid);
      if (clip != nullptr) {
#pragma unroll
        for (int o = L / 2; o >= 1; o >>= 1) {
          n_self += __shfl_xor_sync(0xffffffffu, n_self, o);
          n_other += __shfl_xor_sync(0xffffffffu, n_other, o);
        }
      }
      if (valid && lg == 0) {
        scales[grp] = s16;
        if constexpr (GRID == SSS_GRID_ASYM) mins[grp] = m16;
        if (clip != nullptr) {
          clip[2 * grp] = static_cast<uint8_t>(n_self);
          clip[2 * grp + 1] = static_cast<uint8_t>(n_other);
        }
        if (flags != 0u && status != nullptr) atomicOr(status, flags);
      }
    }
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

template <int Q, int GRID, int G>
cudaError_t quantize_dispatch(const float* w, const sss_qtensor_t& t,
                              uint8_t* clip, uint32_t* status,
                              cudaStream_t stream) {
  const int64_t ngroups = t.n * (t.k / G);
  constexpr int lanes = G / 4;
  const int64_t threads_needed = (ngroups * lanes + kQuantUnroll - 1) / kQuantUnroll;
  const int grid = grid_for(threads_needed, kQuantThreads, 8);
  quantize_kernel<Q, GRID, G><<<grid, kQuantThreads, 0, stream>>>(
      w, ngroups, t.codes, t.scales, t.mins, clip, status);
  return cudaGetLastError();
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

}  // namespace

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
