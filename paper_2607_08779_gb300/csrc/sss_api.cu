// sss_api.cu -- the C ABI declared in include/sss.h: synchronous argument
// validation, dispatch to the kernels' launchers, and error mapping.  No
// entry point allocates device memory.
#include <atomic>
#include <map>
#include <mutex>
#include <utility>
#include <stdio.h>
#include <string.h>

#include "sss_internal.cuh"

namespace sss {

namespace {
thread_local char g_last_error[256] = "";

void set_error(const char* what, cudaError_t e) {
  snprintf(g_last_error, sizeof g_last_error, "%s: %s (%d)", what,
           cudaGetErrorString(e), static_cast<int>(e));
}

// largest n or k a tensor may have, and the most tokens of one sss_gemm:
// keeps every size product of the launchers far inside int64/size_t and the
// GEMM's token-tile grid dimension inside its 65535 limit
constexpr int64_t kMaxDim = int64_t{1} << 31;
constexpr int64_t kMaxTokens = int64_t{1} << 24;

bool aligned(const void* p, size_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

sss_status_t check_tensor(const sss_qtensor_t* t) {
  if (t == nullptr) return SSS_E_ARG;
  if (t->q < 2 || t->q > 4) return SSS_E_ARG;
  if (t->group != 32 && t->group != 64 && t->group != 128) return SSS_E_ARG;
  if (t->grid < SSS_GRID_UNSIGNED_SYM || t->grid > SSS_GRID_ASYM) return SSS_E_ARG;
  if (t->reserved != 0) return SSS_E_ARG;
  if (t->n < 0 || t->k < 0) return SSS_E_ARG;
  if (t->n > kMaxDim || t->k > kMaxDim) return SSS_E_ARG;
  if (t->k % t->group != 0) return SSS_E_ARG;
  if (t->n > 0 && t->k > 0) {
    if (t->codes == nullptr || t->scales == nullptr) return SSS_E_ARG;
    if (t->grid == SSS_GRID_ASYM && t->mins == nullptr) return SSS_E_ARG;
  }
  return SSS_OK;
}

sss_status_t finish(const char* what, cudaError_t e) {
  if (e == cudaSuccess) return SSS_OK;
  if (e == cudaErrorNotSupported) {
    set_error(what, e);
    return SSS_E_UNSUPPORTED;
  }
  set_error(what, e);
  return SSS_E_CUDA;
}

}  // namespace

cudaError_t ensure_smem_impl(const void* kernel, int bytes) {
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, int> configured;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  int& have = configured[std::make_pair(kernel, dev)];
  if (have >= bytes) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) have = bytes;
  return e;
}

EncodeTiledFn tensor_map_encoder() {
  static std::once_flag once;
  static EncodeTiledFn fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

int device_sm_count() {
  static std::mutex mu;
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0)
      v = 148;
    cache[dev] = v;
  }
  return cache[dev];
}

namespace {
std::atomic<uint32_t> g_test_stall{0};
}  // namespace

uint32_t test_stall_mask() { return g_test_stall.load(std::memory_order_relaxed); }

void set_error_message(const char* msg) {
  snprintf(g_last_error, sizeof g_last_error, "%s", msg);
}

}  // namespace sss

using namespace sss;

extern "C" {

size_t sss_codes_bytes(int64_t n, int64_t k, int32_t q) {
  if (n < 0 || k < 0 || q < 2 || q > 4) return 0;
  return static_cast<size_t>(n) * static_cast<size_t>(k) * static_cast<size_t>(q) / 8;
}

const char* sss_status_string(sss_status_t s) {
  switch (s) {
    case SSS_OK: return "SSS_OK";
    case SSS_E_ARG: return "SSS_E_ARG: invalid argument";
    case SSS_E_UNSUPPORTED: return "SSS_E_UNSUPPORTED: unsupported combination";
    case SSS_E_ALIGN: return "SSS_E_ALIGN: misaligned pointer";
    case SSS_E_CUDA: return "SSS_E_CUDA: CUDA error";
    case SSS_E_WORKSPACE: return "SSS_E_WORKSPACE: workspace too small";
  }
  return "unknown sss_status_t";
}

const char* sss_last_error(void) { return g_last_error; }

void sss_test_set_stall(uint32_t mask) {
  g_test_stall.store(mask & (SSS_TEST_STALL_GEMV | SSS_TEST_STALL_GEMV_BATCH | SSS_TEST_STALL_GEMM),
                     std::memory_order_relaxed);
}

sss_status_t sss_quantize(const float* w, const sss_qtensor_t* out,
                          uint8_t* clip_counts, uint32_t* dev_status,
                          void* stream) {
  sss_status_t st = check_tensor(out);
  if (st != SSS_OK) return st;
  if (out->n == 0 || out->k == 0) return SSS_OK;
  if (w == nullptr) return SSS_E_ARG;
  if (!aligned(w, 16)) return SSS_E_ALIGN;
  if (!aligned(out->scales, 2) || (out->mins && !aligned(out->mins, 2))) return SSS_E_ALIGN;
  if (!aligned(out->codes, 16)) return SSS_E_ALIGN;
  if (dev_status && !aligned(dev_status, 4)) return SSS_E_ALIGN;
  return finish("sss_quantize",
                launch_quantize(w, *out, clip_counts, dev_status,
                                static_cast<cudaStream_t>(stream)));
}

sss_status_t sss_dequantize(const sss_qtensor_t* qt, void* out, int32_t out_dtype,
                            void* stream) {
  sss_status_t st = check_tensor(qt);
  if (st != SSS_OK) return st;
  if (out_dtype < SSS_OUT_F32 || out_dtype > SSS_OUT_BF16) return SSS_E_ARG;
  if (qt->n == 0 || qt->k == 0) return SSS_OK;
  if (out == nullptr) return SSS_E_ARG;
  if (!aligned(out, 16)) return SSS_E_ALIGN;
  if (!aligned(qt->codes, 4) || !aligned(qt->scales, 2) || (qt->mins && !aligned(qt->mins, 2)))
    return SSS_E_ALIGN;
  return finish("sss_dequantize",
                launch_dequantize(*qt, out, out_dtype, static_cast<cudaStream_t>(stream)));
}

size_t sss_workspace_bytes(const sss_qtensor_t* qt, int64_t m_or_batch, int32_t op) {
  if (check_tensor(qt) != SSS_OK || m_or_batch < 0) return 0;
  if (op == SSS_OP_GEMV) return gemv_workspace_bytes(*qt, static_cast<int>(m_or_batch));
  if (op == SSS_OP_GEMM) return gemm_workspace_bytes(*qt, m_or_batch);
  return 0;
}

sss_status_t sss_gemv(const sss_qtensor_t* qt, const uint16_t* x_bf16, int32_t batch,
                      float* y, void* workspace, size_t ws_bytes,
                      uint32_t* dev_status, void* stream) {
  sss_status_t st = check_tensor(qt);
  if (st != SSS_OK) return st;
  if (batch < 1 || batch > 16) return SSS_E_ARG;
  if (qt->n == 0) return SSS_OK;
  if (x_bf16 == nullptr || y == nullptr) return SSS_E_ARG;
  if (qt->k > 0 && (!aligned(qt->codes, 16) || !aligned(x_bf16, 16) ||
                    !aligned(qt->scales, 2) || (qt->mins && !aligned(qt->mins, 2))))
    return SSS_E_ALIGN;
  if (!aligned(y, 4)) return SSS_E_ALIGN;
  const size_t need = gemv_workspace_bytes(*qt, batch);
  if (need > 0 && (workspace == nullptr || ws_bytes < need)) return SSS_E_WORKSPACE;
  if (qt->k == 0) {  // empty reduction: y = 0
    return finish("sss_gemv",
                  cudaMemsetAsync(y, 0, sizeof(float) * static_cast<size_t>(batch) * qt->n,
                                  static_cast<cudaStream_t>(stream)));
  }
  // batch 1: the streaming kernel; batch 2..16: the batched kernel (fp16
  // weight operand); shapes neither takes (k not a multiple of 256,
  // unaligned buffers): the general kernel
  if (batch == 1 && gemv_stream_eligible(*qt, x_bf16)) {
    const sss_qtensor_t* one[1] = {qt};
    float* yy[1] = {y};
    return finish("sss_gemv", launch_gemv_stream(one, yy, 1, x_bf16, 0u, dev_status,
                                                 static_cast<cudaStream_t>(stream)));
  }
  if (batch >= 2 && gemv_batch_eligible(*qt, x_bf16, batch, y)) {
    return finish("sss_gemv", launch_gemv_batch(*qt, x_bf16, batch, y, dev_status,
                                                static_cast<cudaStream_t>(stream)));
  }
  return finish("sss_gemv", launch_gemv(*qt, x_bf16, batch, y, workspace,
                                        static_cast<cudaStream_t>(stream)));
}

sss_status_t sss_gemv_multi(const sss_qtensor_t* const* qts, float* const* ys, int32_t count,
                            const uint16_t* x_bf16, uint32_t flags, uint32_t* dev_status,
                            void* stream) {
  if (qts == nullptr || ys == nullptr || count < 1 || count > 4) return SSS_E_ARG;
  if ((flags & ~(SSS_GEMV_PDL | SSS_GEMV_WEIGHTS_READY | SSS_GEMV_ACT_Q8)) != 0) return SSS_E_ARG;
  bool stream_ok = true;
  for (int j = 0; j < count; ++j) {
    sss_status_t st = check_tensor(qts[j]);
    if (st != SSS_OK) return st;
    const sss_qtensor_t& t = *qts[j];
    const sss_qtensor_t& t0 = *qts[0];
    if (t.k != t0.k || t.q != t0.q || t.group != t0.group || t.grid != t0.grid) return SSS_E_ARG;
    if (t.n > 0 && ys[j] == nullptr) return SSS_E_ARG;
    if (ys[j] != nullptr && !aligned(ys[j], 4)) return SSS_E_ALIGN;
    if (t.n > 0 && !gemv_stream_eligible(t, x_bf16)) stream_ok = false;
    if (t.n == 0) stream_ok = false;
  }
  if (x_bf16 == nullptr) return SSS_E_ARG;
  if (dev_status && !aligned(dev_status, 4)) return SSS_E_ALIGN;
  if (stream_ok && qts[0]->k > 0) {
    return finish("sss_gemv_multi", launch_gemv_stream(qts, ys, count, x_bf16, flags, dev_status,
                                                       static_cast<cudaStream_t>(stream)));
  }
  // the general kernels take bf16 activations only
  if (flags & SSS_GEMV_ACT_Q8) return SSS_E_UNSUPPORTED;
  for (int j = 0; j < count; ++j) {
    sss_status_t st = sss_gemv(qts[j], x_bf16, 1, ys[j], nullptr, 0, dev_status, stream);
    if (st != SSS_OK) return st;
  }
  return SSS_OK;
}

namespace {
sss_status_t gemm_common(const char* name, const sss_qtensor_t* qt, const uint16_t* x_bf16,
                         int64_t m, float* y, void* workspace, size_t ws_bytes,
                         uint32_t* dev_status, void* stream, bool act_q8) {
  sss_status_t st = check_tensor(qt);
  if (st != SSS_OK) return st;
  if (m < 0 || m > kMaxTokens) return SSS_E_ARG;
  if (m == 0 || qt->n == 0) return SSS_OK;
  if (x_bf16 == nullptr || y == nullptr) return SSS_E_ARG;
  if (qt->k % 64 != 0) return SSS_E_UNSUPPORTED;
  if (qt->n % 4 != 0) return SSS_E_UNSUPPORTED;
  if (!aligned(qt->codes, 16) || !aligned(x_bf16, 16) || !aligned(y, 16) ||
      !aligned(qt->scales, 2) || (qt->mins && !aligned(qt->mins, 2)))
    return SSS_E_ALIGN;
  if (dev_status && !aligned(dev_status, 4)) return SSS_E_ALIGN;
  // the fp16 copy of X must fit; a workspace of sss_workspace_bytes also
  // holds the split-K partial tiles, which the call then uses where they help
  const size_t need = gemm_workspace_min_bytes(*qt, m);
  if (need > 0 && (workspace == nullptr || ws_bytes < need)) return SSS_E_WORKSPACE;
  if (workspace != nullptr && !aligned(workspace, 16)) return SSS_E_ALIGN;
  if (qt->k == 0) {
    return finish(name, cudaMemsetAsync(y, 0, sizeof(float) * static_cast<size_t>(m) * qt->n,
                                        static_cast<cudaStream_t>(stream)));
  }
  return finish(name, launch_gemm(*qt, x_bf16, m, y, workspace, ws_bytes, dev_status,
                                  static_cast<cudaStream_t>(stream), act_q8));
}
}  // namespace

sss_status_t sss_gemm(const sss_qtensor_t* qt, const uint16_t* x_bf16, int64_t m,
                      float* y, void* workspace, size_t ws_bytes,
                      uint32_t* dev_status, void* stream) {
  return gemm_common("sss_gemm", qt, x_bf16, m, y, workspace, ws_bytes, dev_status, stream,
                     false);
}

namespace {
// the matrices of one sss_gemm_multi call: valid, alike in k, q, group and
// grid, each with n % 4 == 0 and aligned buffers; the ones with rows kept
sss_status_t gemm_multi_jobs(const sss_qtensor_t* const* qts, float* const* ys, int32_t count,
                             const sss_qtensor_t** keep, float** keep_y, int* kept) {
  if (qts == nullptr || count < 1 || count > kMaxGemmJobs) return SSS_E_ARG;
  *kept = 0;
  for (int j = 0; j < count; ++j) {
    sss_status_t st = check_tensor(qts[j]);
    if (st != SSS_OK) return st;
    const sss_qtensor_t& t = *qts[j];
    const sss_qtensor_t& t0 = *qts[0];
    if (t.k != t0.k || t.q != t0.q || t.group != t0.group || t.grid != t0.grid) return SSS_E_ARG;
    if (t.n == 0) continue;
    if (keep_y != nullptr) {
      if (ys == nullptr || ys[j] == nullptr) return SSS_E_ARG;
      if (t.k > 0 && t.n % 4 != 0) return SSS_E_UNSUPPORTED;
      if (!aligned(ys[j], 16)) return SSS_E_ALIGN;
      if (t.k > 0 && (!aligned(t.codes, 16) || !aligned(t.scales, 2) ||
                      (t.mins && !aligned(t.mins, 2))))
        return SSS_E_ALIGN;
      keep_y[*kept] = ys[j];
    }
    keep[(*kept)++] = qts[j];
  }
  return SSS_OK;
}
}  // namespace

size_t sss_gemm_multi_workspace_bytes(const sss_qtensor_t* const* qts, int32_t count,
                                      int64_t m) {
  const sss_qtensor_t* keep[kMaxGemmJobs];
  int kept = 0;
  if (m < 0 || gemm_multi_jobs(qts, nullptr, count, keep, nullptr, &kept) != SSS_OK) return 0;
  if (kept == 0 || m == 0) return 0;
  return gemm_multi_workspace_bytes(keep, kept, m);
}

sss_status_t sss_gemm_multi(const sss_qtensor_t* const* qts, float* const* ys, int32_t count,
                            const uint16_t* x_bf16, int64_t m, void* workspace, size_t ws_bytes,
                            uint32_t* dev_status, void* stream) {
  const sss_qtensor_t* keep[kMaxGemmJobs];
  float* keep_y[kMaxGemmJobs];
  int kept = 0;
  sss_status_t st = gemm_multi_jobs(qts, ys, count, keep, keep_y, &kept);
  if (st != SSS_OK) return st;
  if (m < 0 || m > kMaxTokens) return SSS_E_ARG;
  if (m == 0 || kept == 0) return SSS_OK;
  if (x_bf16 == nullptr) return SSS_E_ARG;
  const int64_t k = keep[0]->k;
  if (k % 64 != 0) return SSS_E_UNSUPPORTED;
  if (!aligned(x_bf16, 16)) return SSS_E_ALIGN;
  if (dev_status && !aligned(dev_status, 4)) return SSS_E_ALIGN;
  const size_t need = gemm_workspace_min_bytes(*keep[0], m);
  if (need > 0 && (workspace == nullptr || ws_bytes < need)) return SSS_E_WORKSPACE;
  if (workspace != nullptr && !aligned(workspace, 16)) return SSS_E_ALIGN;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (k == 0) {
    for (int j = 0; j < kept; ++j) {
      const cudaError_t e =
          cudaMemsetAsync(keep_y[j], 0, sizeof(float) * static_cast<size_t>(m) * keep[j]->n, s);
      if (e != cudaSuccess) return finish("sss_gemm_multi", e);
    }
    return SSS_OK;
  }
  return finish("sss_gemm_multi", launch_gemm_multi(keep, keep_y, kept, x_bf16, m, workspace,
                                                    ws_bytes, dev_status, s, false));
}

sss_status_t sss_gemm_q8(const sss_qtensor_t* qt, const uint16_t* x_bf16, int64_t m,
                         float* y, void* workspace, size_t ws_bytes,
                         uint32_t* dev_status, void* stream) {
  if (qt != nullptr && qt->k % 32 != 0) return SSS_E_ARG;
  return gemm_common("sss_gemm_q8", qt, x_bf16, m, y, workspace, ws_bytes, dev_status, stream,
                     true);
}

namespace {
bool pow2_block(int64_t b) { return b >= 2 && b <= 8192 && (b & (b - 1)) == 0; }
}  // namespace

sss_status_t sss_hadamard(const float* w, float* out, int64_t n, int64_t k, int32_t block,
                          int32_t side, void* stream) {
  if (n < 0 || k < 0 || n > kMaxDim || k > kMaxDim || !pow2_block(block)) return SSS_E_ARG;
  if (side != SSS_ROTATE_INPUT && side != SSS_ROTATE_OUTPUT) return SSS_E_ARG;
  if (side == SSS_ROTATE_INPUT && (k % block != 0 || k % 4 != 0)) return SSS_E_ARG;
  if (side == SSS_ROTATE_OUTPUT && (n % block != 0 || k % (8192 / block) != 0)) return SSS_E_ARG;
  if (n == 0 || k == 0) return SSS_OK;
  if (w == nullptr || out == nullptr) return SSS_E_ARG;
  if (!aligned(w, 16) || !aligned(out, 16)) return SSS_E_ALIGN;
  return finish("sss_hadamard", launch_hadamard(w, out, n, k, block, side,
                                                static_cast<cudaStream_t>(stream)));
}

sss_status_t sss_quantize_rotated(const float* w, int32_t block, const sss_qtensor_t* out,
                                  uint8_t* clip_counts, uint32_t* dev_status, void* stream) {
  sss_status_t st = check_tensor(out);
  if (st != SSS_OK) return st;
  if (!pow2_block(block) || out->k % block != 0) return SSS_E_ARG;
  if (out->n == 0 || out->k == 0) return SSS_OK;
  if (w == nullptr) return SSS_E_ARG;
  if (!aligned(w, 16) || !aligned(out->codes, 16) || !aligned(out->scales, 2) ||
      (out->mins && !aligned(out->mins, 2)) || (dev_status && !aligned(dev_status, 4)))
    return SSS_E_ALIGN;
  return finish("sss_quantize_rotated",
                launch_quantize_rotated(w, block, *out, clip_counts, dev_status,
                                        static_cast<cudaStream_t>(stream)));
}

sss_status_t sss_quantize_lsq(const float* w, const sss_qtensor_t* out, int32_t steps,
                              float lr, uint32_t* dev_status, void* stream) {
  sss_status_t st = check_tensor(out);
  if (st != SSS_OK) return st;
  if (out->grid == SSS_GRID_ASYM) return SSS_E_UNSUPPORTED;
  if (steps < 0 || !(lr >= 0.f) || !(lr < 1e30f)) return SSS_E_ARG;
  if (out->n == 0 || out->k == 0) return SSS_OK;
  if (w == nullptr) return SSS_E_ARG;
  if (!aligned(w, 4) || !aligned(out->codes, 4) || !aligned(out->scales, 2) ||
      (dev_status && !aligned(dev_status, 4)))
    return SSS_E_ALIGN;
  return finish("sss_quantize_lsq", launch_quantize_lsq(w, *out, steps, lr, dev_status,
                                                        static_cast<cudaStream_t>(stream)));
}

sss_status_t sss_sign_diagnostics(const float* w, int64_t n, int64_t k, int32_t q,
                                  int32_t group, int16_t* margin, double* gain,
                                  uint64_t* hist, uint32_t* dev_status, void* stream) {
  if (n < 0 || k < 0 || n > kMaxDim || k > kMaxDim) return SSS_E_ARG;
  if (q < 2 || q > 4) return SSS_E_ARG;
  if (group != 32 && group != 64 && group != 128) return SSS_E_ARG;
  if (k % group != 0) return SSS_E_ARG;
  if (n == 0 || k == 0) return SSS_OK;
  if (w == nullptr) return SSS_E_ARG;
  if (!aligned(w, 16) || (margin && !aligned(margin, 2)) || (gain && !aligned(gain, 8)) ||
      (hist && !aligned(hist, 8)) || (dev_status && !aligned(dev_status, 4)))
    return SSS_E_ALIGN;
  return finish("sss_sign_diagnostics",
                launch_sign_diagnostics(w, n, k, q, group, margin, gain,
                                        reinterpret_cast<unsigned long long*>(hist), dev_status,
                                        static_cast<cudaStream_t>(stream)));
}

sss_status_t sss_quantize_act_q8(const uint16_t* x_bf16, int64_t rows, int64_t k, int8_t* q,
                                 uint16_t* d, uint32_t* dev_status, void* stream) {
  if (rows < 0 || k < 0 || rows > kMaxDim || k > kMaxDim || k % 32 != 0) return SSS_E_ARG;
  if (rows == 0 || k == 0) return SSS_OK;
  if (x_bf16 == nullptr || q == nullptr || d == nullptr) return SSS_E_ARG;
  if (!aligned(x_bf16, 16) || !aligned(q, 8) || !aligned(d, 2)) return SSS_E_ALIGN;
  if (dev_status && !aligned(dev_status, 4)) return SSS_E_ALIGN;
  return finish("sss_quantize_act_q8",
                launch_act_q8(x_bf16, rows, k, q, d, dev_status, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
