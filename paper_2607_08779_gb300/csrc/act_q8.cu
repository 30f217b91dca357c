// act_q8.cu -- sss_quantize_act_q8: bf16 activations [rows][k] to Q8_0
// (int8 codes, one fp16 scale per block of 32), see act_q8.cuh.
//
// Four lanes share a block, eight activations each (one 16-byte load); the
// block max and the non-finite flag are two butterfly shuffles.  HBM-bound:
// 2 bytes read and 1 + 2/32 bytes written per activation.
#include <algorithm>

#include "act_q8.cuh"

namespace sss {
namespace {

__global__ void __launch_bounds__(256)
    act_q8_kernel(const uint16_t* __restrict__ x, int64_t nvec, int8_t* __restrict__ q,
                  uint16_t* __restrict__ d, uint32_t* __restrict__ status) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  // warp-uniform trip count: every lane takes part in the shuffles
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x; base < nvec; base += stride) {
    const int64_t i = base + threadIdx.x;  // this lane's 8 activations: i*8 .. i*8+7
    const bool valid = i < nvec;
    float v[8];
    const uint4 raw = valid ? __ldcs(reinterpret_cast<const uint4*>(x) + i) : make_uint4(0, 0, 0, 0);
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[2 * e] = __uint_as_float(w[e] << 16);
      v[2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
    }
    float amax = 0.f;
    unsigned bad = 0;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      amax = fmaxf(amax, fabsf(v[e]));
      bad |= is_nonfinite(v[e]);
    }
#pragma unroll
    for (int o = 1; o <= 2; o <<= 1) {
      amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
      bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
    unsigned flags = 0;
    uint16_t d16;
    const float dd = q8_scale(amax, bad != 0, &d16, &flags);
    uint32_t packed[2] = {0u, 0u};
    if (dd != 0.f) {
      const float r = __frcp_rn(dd);
#pragma unroll
      for (int e = 0; e < 8; ++e)
        packed[e >> 2] |= (static_cast<uint32_t>(q8_code(v[e], dd, r)) & 0xFFu) << (8 * (e & 3));
    }
    if (valid) {
      reinterpret_cast<uint2*>(q)[i] = make_uint2(packed[0], packed[1]);
      if ((threadIdx.x & 3) == 0) {
        d[i >> 2] = d16;
        if (flags != 0u && status != nullptr) atomicOr(status, flags);
      }
    }
  }
}

// The GEMM's activation operand from Q8_0: fl16(fl16(d) * q) per element
// (the tensor cores take fp16; the product of the fp16 scale and the int8
// code is rounded once).
__global__ void __launch_bounds__(256)
    act_q8_f16_kernel(const uint16_t* __restrict__ x, int64_t nvec, __half* __restrict__ out,
                      uint32_t* __restrict__ status) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x; base < nvec; base += stride) {
    const int64_t i = base + threadIdx.x;
    const bool valid = i < nvec;
    float v[8];
    const uint4 raw = valid ? __ldcs(reinterpret_cast<const uint4*>(x) + i) : make_uint4(0, 0, 0, 0);
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[2 * e] = __uint_as_float(w[e] << 16);
      v[2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
    }
    float amax = 0.f;
    unsigned bad = 0;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      amax = fmaxf(amax, fabsf(v[e]));
      bad |= is_nonfinite(v[e]);
    }
#pragma unroll
    for (int o = 1; o <= 2; o <<= 1) {
      amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
      bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
    unsigned flags = 0;
    uint16_t d16;
    const float dd = q8_scale(amax, bad != 0, &d16, &flags);
    const float df = __half2float(__ushort_as_half(d16));
    uint32_t o[4] = {0u, 0u, 0u, 0u};
    if (dd != 0.f) {
      const float r = __frcp_rn(dd);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a = df * static_cast<float>(q8_code(v[2 * e], dd, r));
        const float b = df * static_cast<float>(q8_code(v[2 * e + 1], dd, r));
        __half2 hv = __floats2half2_rn(a, b);
        o[e] = *reinterpret_cast<uint32_t*>(&hv);
      }
    }
    if (valid) {
      reinterpret_cast<uint4*>(out)[i] = make_uint4(o[0], o[1], o[2], o[3]);
      if ((threadIdx.x & 3) == 0 && flags != 0u && status != nullptr) atomicOr(status, flags);
    }
  }
}

}  // namespace

cudaError_t launch_act_q8_f16(const uint16_t* x, int64_t rows, int64_t k, __half* out,
                              uint32_t* status, cudaStream_t stream) {
  const int64_t nvec = rows * k / 8;
  const int64_t want = (nvec + 255) / 256;
  const int grid = static_cast<int>(
      std::max<int64_t>(1, std::min<int64_t>(want, static_cast<int64_t>(device_sm_count()) * 8)));
  act_q8_f16_kernel<<<grid, 256, 0, stream>>>(x, nvec, out, status);
  return cudaGetLastError();
}

cudaError_t launch_act_q8(const uint16_t* x, int64_t rows, int64_t k, int8_t* q, uint16_t* d,
                          uint32_t* status, cudaStream_t stream) {
  const int64_t nvec = rows * k / 8;
  const int64_t want = (nvec + 255) / 256;
  const int grid = static_cast<int>(
      std::max<int64_t>(1, std::min<int64_t>(want, static_cast<int64_t>(device_sm_count()) * 8)));
  act_q8_kernel<<<grid, 256, 0, stream>>>(x, nvec, q, d, status);
  return cudaGetLastError();
}

}  // namespace sss
