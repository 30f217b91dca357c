// diag.cu -- sss_sign_diagnostics: the cardinality margin and the realised
// l2 gain of the signed absmax sign rule on every weight group (Sec. 4,
// rem:cardinality-margin and fig:theory-diagnostics).
//
// For a group w with signed-absmax sign gamma* (eq:sign_rule) and
// alpha = ||w||_inf / 2^(q-1):
//   margin m = |C_-gamma*| - |C_gamma*|   (def:clipped-set: the coordinates
//            whose unclipped code RNE(w / (gamma* alpha)) is -2^(q-1),
//            resp. +2^(q-1))
//   gain   g = ||w - Q_-gamma*(w)||^2 - ||w - Q_gamma*(w)||^2,
// with the dequantised weights of the stored fp16 scale, as the formats
// deploy them.  Round-to-nearest-even of the exact quotient is odd, so the
// two signs give opposite unclipped codes and their clipped codes differ
// only on C_gamma* and C_-gamma*, where w^+ - w^- = -s16.  Hence
//   g = -s16 * [ sum over C_gamma*  of (2 w - s16 (2^q - 1))
//              + sum over C_-gamma* of (2 w + s16 (2^q - 1)) ],
// whose terms are exact in fp64 (a few tens of significant bits at the
// scale of s16), so g is computed exactly.  Groups with NaN/Inf are
// skipped (SSS_FLAG_NONFINITE); all-zero groups have m = 0, g = 0.
//
// The per-element arithmetic (group max, sign, scale, exact-quotient
// rounding) is the quantizer's; the kernel reads the fp32 weights once
// (HBM-bound) and writes 2 + 8 bytes per group.
#include <algorithm>

#include "rne.cuh"
#include "sss_internal.cuh"

namespace sss {
namespace {

constexpr int kDiagThreads = 256;

template <int Q, int G>
__global__ void __launch_bounds__(kDiagThreads)
    diag_kernel(const float* __restrict__ w, int64_t nruns, int16_t* __restrict__ margin,
                double* __restrict__ gain, unsigned long long* __restrict__ hist,
                uint32_t* __restrict__ status) {
  constexpr int L = G / 32;  // lanes (runs of 32 weights) per group
  constexpr int HALF = 1 << (Q - 1);
  constexpr int NB = 2 * G + 1;  // margin values -G .. G
  __shared__ unsigned long long sh[NB * 3];
  for (int i = threadIdx.x; i < NB * 3; i += blockDim.x) sh[i] = 0ull;
  __syncthreads();

  const int lane = threadIdx.x & 31;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x; base < nruns;
       base += stride) {  // warp-uniform: every lane joins the shuffles
    const int64_t run = base + threadIdx.x;
    const bool valid = run < nruns;
    float x[32];
    {
      const float4* src = reinterpret_cast<const float4*>(w + (valid ? run : 0) * 32);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float4 v = valid ? __ldcs(src + i) : make_float4(0.f, 0.f, 0.f, 0.f);
        x[4 * i] = v.x; x[4 * i + 1] = v.y; x[4 * i + 2] = v.z; x[4 * i + 3] = v.w;
      }
    }
    float mx = x[0], mn = x[0];
    unsigned bad = 0;
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      mx = fmaxf(mx, x[e]);
      mn = fminf(mn, x[e]);
      bad |= is_nonfinite(x[e]);
    }
#pragma unroll
    for (int o = L / 2; o >= 1; o >>= 1) {
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
      bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
    // the signed absmax grid, as the quantizer forms it
    const float M = fmaxf(mx, -mn);
    const float gamma = (mx > -mn) ? -1.f : 1.f;
    const float alpha = __fmul_rn(M, 1.0f / HALF);
    const bool zero = (alpha == 0.f) || bad;
    const float s = zero ? 0.f : gamma * alpha;
    const double s16 = static_cast<double>(__half2float(__float2half_rn(s)));
    const double span = static_cast<double>((1 << Q) - 1) * s16;  // s16 (2^q - 1)
    int n_self = 0, n_other = 0;
    double acc = 0.0;
    if (!zero) {
      float ss = s, sig = 1.f;
      if (M < 0x1p-96f || M > 0x1p+96f) {  // keep 1/s normal, as the quantizer does
        sig = (M < 1.f) ? 0x1p+64f : 0x1p-64f;
        ss = __fmul_rn(s, sig);
      }
      const float r = __frcp_rn(ss);
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        const int up = code_of<HALF>(sig == 1.f ? x[e] : __fmul_rn(x[e], sig), ss, r);
        if (up == 2 * HALF) {  // C_gamma*
          ++n_self;
          acc += 2.0 * static_cast<double>(x[e]) - span;
        } else if (up == 0) {  // C_-gamma*
          ++n_other;
          acc += 2.0 * static_cast<double>(x[e]) + span;
        }
      }
    }
#pragma unroll
    for (int o = L / 2; o >= 1; o >>= 1) {
      n_self += __shfl_xor_sync(0xffffffffu, n_self, o);
      n_other += __shfl_xor_sync(0xffffffffu, n_other, o);
      acc += __shfl_xor_sync(0xffffffffu, acc, o);
    }
    if (valid && (lane % L) == 0) {
      const int64_t grp = run / L;
      if (bad) {
        if (status != nullptr) atomicOr(status, SSS_FLAG_NONFINITE);
      } else {
        const int m = n_other - n_self;
        const double g = (n_self + n_other) ? -s16 * acc : 0.0;
        if (margin != nullptr) margin[grp] = static_cast<int16_t>(m);
        if (gain != nullptr) gain[grp] = g;
        const int col = g < 0.0 ? 0 : (g == 0.0 ? 1 : 2);
        atomicAdd(&sh[(m + G) * 3 + col], 1ull);
      }
    }
  }
  __syncthreads();
  if (hist != nullptr)
    for (int i = threadIdx.x; i < NB * 3; i += blockDim.x)
      if (sh[i] != 0ull) atomicAdd(&hist[i], sh[i]);
}

template <int Q, int G>
cudaError_t diag_launch(const float* w, int64_t n, int64_t k, int16_t* margin, double* gain,
                        unsigned long long* hist, uint32_t* status, cudaStream_t stream) {
  const int64_t nruns = n * k / 32;
  const int64_t want = (nruns + kDiagThreads - 1) / kDiagThreads;
  const int grid = static_cast<int>(
      std::max<int64_t>(1, std::min<int64_t>(want, static_cast<int64_t>(device_sm_count()) * 8)));
  diag_kernel<Q, G><<<grid, kDiagThreads, 0, stream>>>(w, nruns, margin, gain, hist, status);
  return cudaGetLastError();
}

template <int Q>
cudaError_t diag_g(const float* w, int64_t n, int64_t k, int g, int16_t* margin, double* gain,
                   unsigned long long* hist, uint32_t* status, cudaStream_t stream) {
  switch (g) {
    case 32: return diag_launch<Q, 32>(w, n, k, margin, gain, hist, status, stream);
    case 64: return diag_launch<Q, 64>(w, n, k, margin, gain, hist, status, stream);
    case 128: return diag_launch<Q, 128>(w, n, k, margin, gain, hist, status, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_sign_diagnostics(const float* w, int64_t n, int64_t k, int q, int g,
                                    int16_t* margin, double* gain, unsigned long long* hist,
                                    uint32_t* status, cudaStream_t stream) {
  switch (q) {
    case 2: return diag_g<2>(w, n, k, g, margin, gain, hist, status, stream);
    case 3: return diag_g<3>(w, n, k, g, margin, gain, hist, status, stream);
    case 4: return diag_g<4>(w, n, k, g, margin, gain, hist, status, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace sss
