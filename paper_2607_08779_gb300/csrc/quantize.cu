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
#include "sss_internal.cuh"

namespace sss {
namespace {

constexpr int kQuantThreads = 256;

// 1.5 * 2^23: adding it to |v| < 2^22 rounds v to an integer (ties to even)
// held in the low mantissa bits.
constexpr float kMagic = 12582912.0f;

// Stored code u = RNE(w / s) + OFF of the EXACT quotient, given r = RN(1/s)
// (OFF = 2^(q-1) for the symmetric grids, 0 for the min-max grid; OFF is
// even, so the parity of the rounded sum is that of the code).  One FMA
// rounds w*r straight to an integer; a second FMA gives the remainder
// w*r - c.  Only when that remainder is within 2^-18 of +-1/2 can the exact
// quotient fall on the other side of the half-integer h (|w*r - w/s| <=
// 16 * 2^-24 here), and then the sign of the single-rounding residual
// w - h*s decides it exactly; a zero residual is an exact tie -> even.
template <int OFF>
__device__ __forceinline__ int code_of(float w, float s, float r) {
  constexpr float MAGIC = kMagic + static_cast<float>(OFF);
  const float t = __fmaf_rn(w, r, MAGIC);
  float c = __fsub_rn(t, MAGIC);
  int u = __float_as_int(t) - __float_as_int(kMagic);
  const float dd = __fmaf_rn(w, r, -c);  // w*r - c
  if (fabsf(__fsub_rn(fabsf(dd), 0.5f)) <= 0x1p-18f) {
    const float h = __fadd_rn(c, copysignf(0.5f, dd));   // the half-integer at stake
    const float e = __fmaf_rn(-h, s, w);                  // w - h*s, one rounding
    const float side = (s > 0.f) ? e : -e;                // sign of (w/s - h)
    const float lo = __fsub_rn(h, 0.5f), hi = __fadd_rn(h, 0.5f);
    float cc;
    if (side > 0.f) {
      cc = hi;
    } else if (side < 0.f) {
      cc = lo;
    } else {  // exact tie: to even
      cc = (static_cast<int>(lo) & 1) ? hi : lo;
    }
    u += static_cast<int>(__fsub_rn(cc, c));
  }
  return u;
}

// Pack 32 codes (element e of this lane's run at index e) and store them.
template <int Q, int G>
__device__ __forceinline__ void store_codes32(uint8_t* __restrict__ codes, int64_t group,
                                              int lg, const int (&u)[32]) {
  if constexpr (Q == 4) {
    uint32_t wv[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      uint32_t v = 0;
#pragma unroll
      for (int e = 0; e < 8; ++e) v |= static_cast<uint32_t>(u[8 * i + e]) << (4 * e);
      wv[i] = v;
    }
    reinterpret_cast<uint4*>(codes + group * (G / 2))[lg] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  } else if constexpr (Q == 2) {
    uint32_t wv[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      uint32_t v = 0;
#pragma unroll
      for (int e = 0; e < 16; ++e) v |= static_cast<uint32_t>(u[16 * i + e]) << (2 * e);
      wv[i] = v;
    }
    reinterpret_cast<uint2*>(codes + group * (G / 4))[lg] = make_uint2(wv[0], wv[1]);
  } else {  // low 2-bit plane (q=2 layout), then the high-bit plane
    uint32_t lo[2], hi = 0;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      uint32_t v = 0;
#pragma unroll
      for (int e = 0; e < 16; ++e) v |= static_cast<uint32_t>(u[16 * i + e] & 3) << (2 * e);
      lo[i] = v;
    }
#pragma unroll
    for (int e = 0; e < 32; ++e) hi |= static_cast<uint32_t>(u[e] >> 2) << e;
    uint32_t* base = reinterpret_cast<uint32_t*>(codes + group * (3 * G / 8));
    base[2 * lg] = lo[0];
    base[2 * lg + 1] = lo[1];
    base[G / 16 + lg] = hi;
  }
}

template <int Q, int GRID, int G, bool STATS>
__global__ void __launch_bounds__(kQuantThreads)
    quantize_kernel(const float* __restrict__ w, int64_t ngroups,
                    uint8_t* __restrict__ codes, uint16_t* __restrict__ scales,
                    uint16_t* __restrict__ mins, uint8_t* __restrict__ clip,
                    uint32_t* __restrict__ status) {
  constexpr int L = G / 32;     // lanes per group, 32 weights each
  constexpr int GPW = 32 / L;   // groups per warp per sweep
  constexpr int HALF = 1 << (Q - 1);
  constexpr int UMAX = (1 << Q) - 1;
  constexpr int OFF = (GRID == SSS_GRID_ASYM) ? 0 : HALF;
  const int lane = threadIdx.x & 31;
  const int lg = lane % L;
  const int64_t slot =
      ((static_cast<int64_t>(blockIdx.x) * kQuantThreads + threadIdx.x) >> 5) * GPW + lane / L;
  const int64_t nslots = (static_cast<int64_t>(gridDim.x) * kQuantThreads >> 5) * GPW;

  for (int64_t grp = slot; grp - lane / L < ngroups; grp += nslots) {  // warp-uniform
    const bool valid = grp < ngroups;
    float x[32];
    {
      const float4* src = reinterpret_cast<const float4*>(w + (valid ? grp : 0) * G) + lg * 8;
      float4 v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = valid ? __ldcs(src + i) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        x[4 * i] = v[i].x; x[4 * i + 1] = v[i].y; x[4 * i + 2] = v[i].z; x[4 * i + 3] = v[i].w;
      }
    }
    float mx = x[0], mn = x[0], sum = 0.f;
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      mx = fmaxf(mx, x[e]);
      mn = fminf(mn, x[e]);
      sum += x[e];  // NaN/Inf anywhere -> non-finite sum (checked exactly below)
    }
    unsigned bad = 0;
    if (is_nonfinite(sum)) {
#pragma unroll
      for (int e = 0; e < 32; ++e) bad |= is_nonfinite(x[e]);
    }
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
        float ss = s;
        // alpha is an exact power-of-two scaling of M unless it is
        // subnormal; then |w/s| may exceed 2^(q-1) slightly and both ends clip
        int lo_clip = 0x80000000;
        if (M < 0x1p-96f || M > 0x1p+96f) {  // keep 1/s normal: scale w and s by 2^+-64
          const float sig = (M < 1.f) ? 0x1p+64f : 0x1p-64f;
          ss = __fmul_rn(s, sig);
#pragma unroll
          for (int e = 0; e < 32; ++e) x[e] = __fmul_rn(x[e], sig);
          lo_clip = 0;
        }
        const float r = __frcp_rn(ss);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int up = code_of<OFF>(x[e], ss, r);  // c_pre + 2^(q-1)
          if constexpr (STATS) {
            n_self += (up == 2 * HALF);  // c_pre == +2^(q-1): in C_gamma
            n_other += (up == 0);        // c_pre == -2^(q-1): in C_-gamma
          }
          u[e] = max(min(up, UMAX), lo_clip);  // normally only +2^(q-1) leaves A_q
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
        const float r = __frcp_rn(ss);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          float d = __fsub_rn(x[e], mn);  // fl32(w - min) >= 0
          if (sig != 1.f) d = __fmul_rn(d, sig);
          u[e] = min(code_of<0>(d, ss, r), UMAX);
        }
      }
      s16 = __half_as_ushort(__float2half_rn(s));  // inf when the step overflowed
      m16 = __half_as_ushort(__float2half_rn(mn));
      if ((m16 & 0x7fffu) == 0x7c00u) flags |= SSS_FLAG_RANGE;
    }
    if ((s16 & 0x7fffu) == 0x7c00u) flags |= SSS_FLAG_RANGE;
    if (valid) store_codes32<Q, G>(codes, grp, lg, u);
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
  constexpr int lanes = G / 32;
  const int grid = grid_for(ngroups * lanes, kQuantThreads, 8);
  if (clip != nullptr)
    quantize_kernel<Q, GRID, G, true><<<grid, kQuantThreads, 0, stream>>>(
        w, ngroups, t.codes, t.scales, t.mins, clip, status);
  else
    quantize_kernel<Q, GRID, G, false><<<grid, kQuantThreads, 0, stream>>>(
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
