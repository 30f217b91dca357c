// sss_internal.cuh -- declarations shared by the CUDA translation units of
// the library (not installed; the public interface is include/sss.h).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "sss.h"

namespace sss {

// Number of SMs of the current device (queried once per device).
int device_sm_count();

// cuTensorMapEncodeTiled, resolved through the runtime's driver entry point
// (the library does not link libcuda); nullptr if unavailable.
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();

// Launchers.  Arguments are validated by the C ABI before these run.
cudaError_t launch_quantize(const float* w, const sss_qtensor_t& t,
                            uint8_t* clip_counts, uint32_t* status,
                            cudaStream_t stream);
cudaError_t launch_dequantize(const sss_qtensor_t& t, void* out, int out_dtype,
                              cudaStream_t stream);

size_t gemv_workspace_bytes(const sss_qtensor_t& t, int batch);
cudaError_t launch_gemv(const sss_qtensor_t& t, const uint16_t* x, int batch,
                        float* y, void* workspace, cudaStream_t stream);

bool gemv_stream_eligible(const sss_qtensor_t& t, const uint16_t* x);
cudaError_t launch_gemv_stream(const sss_qtensor_t* const* ts, float* const* ys, int count,
                               const uint16_t* x, uint32_t flags, uint32_t* status,
                               cudaStream_t stream);

bool gemv_batch_eligible(const sss_qtensor_t& t, const uint16_t* x, int batch, const float* y);
cudaError_t launch_gemv_batch(const sss_qtensor_t& t, const uint16_t* x, int batch, float* y,
                              uint32_t* status, cudaStream_t stream);

// matrices of one sss_gemm_multi call (sharing X)
constexpr int kMaxGemmJobs = 4;
size_t gemm_workspace_bytes(const sss_qtensor_t& t, int64_t m);
size_t gemm_multi_workspace_bytes(const sss_qtensor_t* const* ts, int count, int64_t m);
size_t gemm_workspace_min_bytes(const sss_qtensor_t& t, int64_t m);
cudaError_t launch_gemm(const sss_qtensor_t& t, const uint16_t* x, int64_t m,
                        float* y, void* workspace, size_t ws_bytes, uint32_t* status,
                        cudaStream_t stream, bool act_q8 = false);
cudaError_t launch_gemm_multi(const sss_qtensor_t* const* ts, float* const* ys, int count,
                              const uint16_t* x, int64_t m, void* workspace, size_t ws_bytes,
                              uint32_t* status, cudaStream_t stream, bool act_q8);

cudaError_t launch_act_q8(const uint16_t* x, int64_t rows, int64_t k, int8_t* q, uint16_t* d,
                          uint32_t* status, cudaStream_t stream);
cudaError_t launch_act_q8_f16(const uint16_t* x, int64_t rows, int64_t k, __half* out,
                              uint32_t* status, cudaStream_t stream);

cudaError_t launch_hadamard(const float* w, float* out, int64_t n, int64_t k, int b, int side,
                            cudaStream_t stream);
cudaError_t launch_quantize_rotated(const float* w, int b, const sss_qtensor_t& t, uint8_t* clip,
                                    uint32_t* status, cudaStream_t stream);

cudaError_t launch_quantize_lsq(const float* w, const sss_qtensor_t& t, int steps, float lr,
                                uint32_t* status, cudaStream_t stream);

cudaError_t launch_sign_diagnostics(const float* w, int64_t n, int64_t k, int q, int g,
                                    int16_t* margin, double* gain, unsigned long long* hist,
                                    uint32_t* status, cudaStream_t stream);

// The kernel families whose next launches skip one barrier arrive
// (sss_test_set_stall; 0 in normal use).
uint32_t test_stall_mask();

// Record a message for sss_last_error() on this thread.
void set_error_message(const char* msg);

// Raise a kernel's dynamic shared-memory limit once per (kernel, device)
// (the call is not stream-ordered; doing it once keeps launches cheap and
// capturable in CUDA graphs).
cudaError_t ensure_smem_impl(const void* kernel, int bytes);
template <typename K>
cudaError_t ensure_smem(K kernel, int bytes) {
  return ensure_smem_impl(reinterpret_cast<const void*>(kernel), bytes);
}

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------

__device__ __forceinline__ bool is_nonfinite(float v) {
  return (__float_as_uint(v) & 0x7f800000u) == 0x7f800000u;
}

}  // namespace sss
