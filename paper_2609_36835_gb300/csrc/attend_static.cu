// arckv_attend_static: compact attention with no caller workspace and no
// allocation at call time.  Its scratch is one file-scope __device__ array
// that the CUDA module loader places in every context that loads this
// library; the array stays resident until the process exits.
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "kernels.h"

namespace {

// the scratch layout of arckv_attend (attend_layout: status word, logits,
// operand triples, partial outputs), in floats
constexpr size_t kStaticScratchFloats = ARCKV_ATTEND_STATIC_MAX_FLOATS;

__device__ __align__(256) float g_attend_scratch[kStaticScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
float* g_scratch_addr[kMaxDevices];        // per device, filled by the first call on that device
unsigned long long g_scratch_ctx[kMaxDevices];   // id of the context the address belongs to

PFN_cuCtxGetCurrent_v4000 g_ctx_current = nullptr;
PFN_cuCtxGetId_v12000 g_ctx_id = nullptr;
std::once_flag g_ctx_once;

// Id of the current CUDA context (unique for the life of the process), or 0
// when the driver does not report one or no context is current yet (the
// address is then looked up again on the next call).  A reset of the device's primary
// context (cudaDeviceReset) makes a new context with a new id, in which the
// array has to be looked up again.
unsigned long long current_context_id() {
  std::call_once(g_ctx_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fn, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_ctx_current = (PFN_cuCtxGetCurrent_v4000)fn;
    fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_ctx_id = (PFN_cuCtxGetId_v12000)fn;
  });
  if (!g_ctx_current || !g_ctx_id) return 0;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (g_ctx_current(&ctx) != CUDA_SUCCESS || !ctx || g_ctx_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// The symbol's device address, looked up with the device current the first
// time a call runs on that device (and again after a reset of its context).
// In host code `g_attend_scratch` names a host-side shadow, never the device
// memory, so kernels only ever receive this looked-up address.
arckv_status scratch_for_current_device(float** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return ARCKV_ERR_CUDA;
  const unsigned long long ctx = current_context_id();
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_addr[dev] || g_scratch_ctx[dev] != ctx) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_attend_scratch) != cudaSuccess || !p) return ARCKV_ERR_CUDA;
    g_scratch_addr[dev] = (float*)p;
    g_scratch_ctx[dev] = ctx;
  }
  *out = g_scratch_addr[dev];
  return ARCKV_OK;
}

}  // namespace

extern "C" {

size_t arckv_attend_static_floats(int32_t H_kv, int32_t n, int32_t t, int32_t d) {
  if (H_kv < 1 || n < 1 || t < 1 || d != 128) return 0;
  const size_t bytes = arckv_attend_workspace_bytes(H_kv, n, t, d);   // the workspace layout of arckv_attend
  return bytes == 0 ? 0 : (bytes + 3) / 4;
}

arckv_status arckv_attend_static(int32_t H_kv, int32_t n, int32_t t, int32_t d, float logit_scale, const void* Q,
                                 const float* C_k, const float* beta, const float* C_v, float* O, void* stream) {
  if (d != 128) return ARCKV_ERR_UNSUPPORTED;
  const size_t need = arckv_attend_static_floats(H_kv, n, t, d);
  if (need == 0) return ARCKV_ERR_SHAPE;
  if (need > kStaticScratchFloats) return ARCKV_ERR_WORKSPACE;
  if (!Q || !C_k || !beta || !C_v || !O) return ARCKV_ERR_INVALID_ARG;
  if (!(logit_scale >= 0.f) || !isfinite(logit_scale)) return ARCKV_ERR_INVALID_ARG;
  float* base = nullptr;
  arckv_status s = scratch_for_current_device(&base);
  if (s != ARCKV_OK) return s;
  cudaStream_t st = (cudaStream_t)stream;
  arckv::DevStatus* stt = (arckv::DevStatus*)base;
  const float scale = logit_scale > 0.f ? logit_scale : 1.0f / sqrtf((float)d);
  cudaGetLastError();
  // the array keeps the previous call's contents: the status word must start at
  // zero (every other scratch region is written before it is read)
  if (cudaMemsetAsync(stt, 0, sizeof(arckv::DevStatus), st) != cudaSuccess) return ARCKV_ERR_CUDA;
  if (arckv::launch_attend(H_kv, n, t, scale, (const arckv::bf16*)Q, C_k, beta, C_v, O, (char*)base, stt, st) < 0)
    return ARCKV_ERR_CUDA;
  arckv::launch_check_finite(O, (long long)H_kv * n * d, stt, st);
  if (cudaGetLastError() != cudaSuccess) return ARCKV_ERR_CUDA;
  unsigned int code = 0;
  if (cudaMemcpyAsync(&code, stt, sizeof(code), cudaMemcpyDeviceToHost, st) != cudaSuccess) return ARCKV_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return ARCKV_ERR_CUDA;
  return (arckv_status)code;
}

}  // extern "C"
