// dmoe_router_no_alloc: the router of dmoe_router for callers that cannot allocate device
// memory (for example code that runs where cudaMalloc is forbidden or unavailable: inside
// an allocator callback, a plugin host that owns all device memory, or a real-time loop
// that must never touch the allocator). Its scratch lives in a fixed-size array in the
// library's own device memory instead of a caller workspace.
//
// The array is a file-scope __device__ variable: every GPU that loads the library keeps it
// for the life of the process. Host code cannot pass the array's name to a kernel (on the
// host it only names a stand-in, not a device address), so the device address is looked
// up once per device with cudaGetSymbolAddress, with that device current, and cached.
// The array's first bytes are the fault record of the router kernels (the first region of
// the workspace layout, at offset 0 for every shape); dmoe_router_no_alloc_device_error
// reads and clears it.
#include <mutex>
#include <stdio.h>

#include "dmoe_internal.cuh"

namespace dmoe {
namespace {

constexpr size_t kRouterStaticScratchBytes = (size_t)4 << 20;  // 4 MiB
constexpr int kMaxDevices = 64;

__device__ __align__(256) uint8_t g_router_scratch[kRouterStaticScratchBytes];

std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_router_scratch on the current device (looked up on first use).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_router_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

bool ok16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace dmoe

using namespace dmoe;

extern "C" dmoe_status dmoe_router_no_alloc(const dmoe_layer_desc* desc, const void* x,
                                            const float* w_r, const float* bias,
                                            int32_t* topk_idx, float* topk_gate,
                                            int32_t* coreset, int32_t* coreset_size,
                                            float* probs, void* stream) {
  size_t ws_total = 0;
  dmoe_status st = dmoe_workspace_size(desc, &ws_total);  // validates the desc
  if (st != DMOE_OK) return st;
  if (x == nullptr || w_r == nullptr || topk_idx == nullptr || topk_gate == nullptr ||
      !ok16(x) || !ok16(w_r) || !ok16(topk_idx) || !ok16(topk_gate) ||
      (bias != nullptr && !ok16(bias)) || (probs != nullptr && !ok16(probs)) ||
      (coreset != nullptr && !ok16(coreset)) ||
      (coreset_size != nullptr && !ok16(coreset_size)))
    return DMOE_ERR_INVALID_ARG;

  // The router uses the leading regions of the workspace plan: the fault record, the stage
  // counters, the partial logits, the scores, the masked scores and the top-k candidates;
  // the next region starts at tk_idx.
  const Workspace plan = plan_workspace(*desc);
  const size_t need = plan.tk_idx;
  if (need > kRouterStaticScratchBytes) {
    char msg[160];
    snprintf(msg, sizeof(msg),
             "dmoe_router_no_alloc: this shape needs %zu bytes of scratch, more than the "
             "%zu-byte static buffer",
             need, kRouterStaticScratchBytes);
    set_last_error_text(msg);
    return DMOE_ERR_UNSUPPORTED;
  }
  void* scratch = nullptr;
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) {
    set_last_error(e);
    return DMOE_ERR_CUDA;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The fault record is not cleared here: as in a caller workspace, a recorded fault stays
  // until dmoe_router_no_alloc_device_error reads it (the array starts zero-filled when the
  // library is loaded).
  uint8_t* base = static_cast<uint8_t*>(scratch);
  RouterArgs a{};
  a.x = static_cast<const __nv_bfloat16*>(x);
  a.w_r = w_r;
  a.bias = bias;
  a.logits_part = reinterpret_cast<float*>(base + plan.logits_part);
  a.probs = probs != nullptr ? probs : reinterpret_cast<float*>(base + plan.probs);
  a.probs_requested = probs != nullptr;
  a.probs_hat = reinterpret_cast<float*>(base + plan.probs_hat);
  a.cand = reinterpret_cast<uint2*>(base + plan.cand);
  a.topk_idx = topk_idx;
  a.topk_gate = topk_gate;
  a.coreset = coreset;
  a.coreset_size = coreset_size;
  a.T = desc->n_blocks * desc->block_size;
  a.d = desc->d_model;
  a.E = desc->n_experts;
  a.k = desc->top_k;
  a.kb = mask_top_k(*desc);
  a.B = desc->block_size;
  a.n_blocks = desc->n_blocks;
  a.mode = desc->mode;
  a.splits = plan.router_splits;
  a.top_p = desc->top_p;
  a.err = reinterpret_cast<DevErrRecord*>(base + plan.err);
  e = launch_router(a, nullptr, reinterpret_cast<int32_t*>(base + plan.tickets), s);
  if (e != cudaSuccess) {
    set_last_error(e);
    return DMOE_ERR_CUDA;
  }
  return DMOE_OK;
}

extern "C" dmoe_status dmoe_router_no_alloc_device_error(void* stream, int32_t* info) {
  void* scratch = nullptr;
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) {
    set_last_error(e);
    return DMOE_ERR_CUDA;
  }
  // the fault record heads the workspace layout: the same reader as for a caller workspace
  static_assert(sizeof(DevErrRecord) <= 256, "the fault record is the first region");
  return dmoe_get_device_error(scratch, stream, info);
}

extern "C" dmoe_status dmoe_no_alloc_scratch(void** device_ptr, size_t* bytes) {
  if (device_ptr == nullptr || bytes == nullptr) return DMOE_ERR_INVALID_ARG;
  void* scratch = nullptr;
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) {
    set_last_error(e);
    return DMOE_ERR_CUDA;
  }
  *device_ptr = scratch;
  *bytes = kRouterStaticScratchBytes;
  return DMOE_OK;
}
