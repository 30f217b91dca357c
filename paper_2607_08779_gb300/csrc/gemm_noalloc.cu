// gemm_noalloc.cu -- sss_gemm_noalloc: the prefill GEMM with its scratch
// (the fp16 copy of the activations) in a static device array instead of a
// caller-provided workspace.
//
// Callers that cannot hand the library a workspace use it: a plain C host
// without a device allocator, or a serving loop that must not call
// cudaMalloc between requests (it synchronises the device and can fail
// under memory pressure).  The array lives in this translation unit's
// module, so with lazy module loading it takes device memory only once this
// entry point is first used.
#include <mutex>
#include <stdio.h>

#include "sss_internal.cuh"

namespace {

constexpr size_t kScratchBytes = size_t{32} << 20;  // 32 MiB: m * k * 2 bytes of fp16 X
constexpr int kMaxDevices = 64;

// Each call writes the fp16 copy of X (and any split-K partial tiles)
// before reading them, and zeroes the split counters it uses first.
static __device__ __align__(256) unsigned char g_gemm_scratch[kScratchBytes];

std::mutex g_mu;
void* g_ptr[kMaxDevices] = {};

// The scratch's device address for the current device, looked up once per
// device (with that device current); nullptr and the CUDA error on failure.
void* scratch_ptr(cudaError_t* err) {
  int dev = 0;
  *err = cudaGetDevice(&dev);
  if (*err != cudaSuccess) return nullptr;
  if (dev < 0 || dev >= kMaxDevices) {
    *err = cudaErrorInvalidDevice;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_ptr[dev] == nullptr) {
    void* p = nullptr;
    *err = cudaGetSymbolAddress(&p, g_gemm_scratch);
    if (*err != cudaSuccess) return nullptr;
    g_ptr[dev] = p;
  }
  return g_ptr[dev];
}

}  // namespace

extern "C" {

size_t sss_gemm_noalloc_max_scratch_bytes(void) { return kScratchBytes; }

sss_status_t sss_gemm_noalloc(const sss_qtensor_t* qt, const uint16_t* x_bf16, int64_t m,
                              float* y, uint32_t* dev_status, void* stream) {
  if (qt == nullptr) return SSS_E_ARG;
  // sss_gemm itself rejects m outside 0..2^24 with SSS_E_ARG; a larger m
  // must not reach the size check below as a wrapped byte count
  if (m < 0 || m > (int64_t{1} << 24)) return SSS_E_ARG;
  // the fp16 copy of X must fit (the call also keeps split-K partial tiles
  // in the array when they fit beside it)
  const size_t need = sss_workspace_bytes(qt, m, SSS_OP_GEMM) == 0
                          ? 0
                          : sss::gemm_workspace_min_bytes(*qt, m);
  if (need > kScratchBytes) {
    sss::set_error_message("sss_gemm_noalloc: the fp16 copy of X needs more than the "
                           "32 MiB static scratch (m * k * 2 bytes > 33554432)");
    return SSS_E_WORKSPACE;
  }
  cudaError_t err = cudaSuccess;
  void* ws = scratch_ptr(&err);
  if (ws == nullptr) {
    char msg[200];
    snprintf(msg, sizeof msg,
             "sss_gemm_noalloc: cudaGetSymbolAddress of the static scratch failed: %s (%d)",
             cudaGetErrorString(err), static_cast<int>(err));
    sss::set_error_message(msg);
    return SSS_E_CUDA;
  }
  return sss_gemm(qt, x_bf16, m, y, ws, kScratchBytes, dev_status, stream);
}

}  // extern "C"
