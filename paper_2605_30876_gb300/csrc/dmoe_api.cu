// C-ABI entry points of libdmoe: argument checks, workspace carve-up and kernel launches.
// Nothing here allocates device memory or synchronises, except dmoe_get_device_error.
#include <stdio.h>
#include <string.h>

#include <mutex>
#include <unordered_map>

#include "dmoe_internal.cuh"

namespace dmoe {

namespace {
thread_local char g_last_error[256] = "";

// Workspaces whose W_r parts were written by dmoe_router_prepare, with the W_r they hold.
std::mutex g_prep_mu;
std::unordered_map<const void*, const void*> g_prep;

// Does `ws` hold the parts of `w_r`? If not, the split this call makes writes w_r's parts
// there, so an earlier preparation of the workspace no longer holds.
bool parts_prepared(const void* ws, const void* w_r) {
  std::lock_guard<std::mutex> lock(g_prep_mu);
  auto it = g_prep.find(ws);
  if (it == g_prep.end()) return false;
  if (it->second == w_r) return true;
  g_prep.erase(it);
  return false;
}

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Router logits kernel choice: 0 = the fused decode-size launch (logits written directly);
// otherwise the split of the tiled kernel's d-reduction: enough CTAs to spread the W_r read
// (about 128 tiles), a divisor of d/32, at most 32 partial sums.
int router_splits(const dmoe_layer_desc& d) {
  if (route_cluster_ok(d.n_blocks * d.block_size, d.d_model, d.n_experts)) return 0;
  if (route_cluster_logits_ok(d.d_model, d.n_experts)) return 1;   // one [T, E] logits array
  const int tiles = ((d.n_experts + 63) / 64) * ((d.n_blocks * d.block_size + 31) / 32);
  int target = 128 / tiles;
  if (target < 1) target = 1;
  if (target > 32) target = 32;
  const int kch = d.d_model / 32;
  int best = 1;
  for (int s = 1; s <= target; ++s)
    if (kch % s == 0) best = s;
  return best;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
}  // namespace

namespace {
struct ProfSlot {
  cudaEvent_t begin = nullptr, end = nullptr;
};
thread_local ProfSlot g_prof[DMOE_KERNEL_COUNT];
}  // namespace

// Inside a stream capture the event becomes an external record node of the graph (recorded
// at every replay); outside, a plain record.
void prof_record(cudaEvent_t ev, cudaStream_t s) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cs) != cudaSuccess) cudaGetLastError();
  if (cs == cudaStreamCaptureStatusActive)
    cudaEventRecordWithFlags(ev, s, cudaEventRecordExternal);
  else
    cudaEventRecord(ev, s);
}
void prof_begin(int kernel, cudaStream_t s) {
  if (g_prof[kernel].begin != nullptr) prof_record(g_prof[kernel].begin, s);
}
void prof_end(int kernel, cudaStream_t s) {
  if (g_prof[kernel].end != nullptr) prof_record(g_prof[kernel].end, s);
}
bool prof_serial(int kernel) { return g_prof[kernel].begin != nullptr; }

void set_last_error(cudaError_t e) {
  snprintf(g_last_error, sizeof(g_last_error), "%s: %s", cudaGetErrorName(e),
           cudaGetErrorString(e));
}

void set_last_error_text(const char* msg) {
  snprintf(g_last_error, sizeof(g_last_error), "%s", msg);
}

int device_sm_count() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (dev >= 0 && dev < 64 && cache[dev] > 0) return cache[dev];
  int n = 1;
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  if (dev >= 0 && dev < 64) cache[dev] = n;
  return n;
}

Workspace plan_workspace(const dmoe_layer_desc& d) {
  Workspace w{};
  const size_t T = (size_t)d.n_blocks * d.block_size, E = d.n_experts, k = d.top_k;
  const size_t dm = d.d_model, I = d.d_ff, Is = d.d_ff_shared;
  w.router_splits = router_splits(d);
  const bool tc = !route_cluster_ok((int)T, (int)dm, (int)E) &&
                  router_tc_ok((int)T, (int)dm, (int)E);
  w.tc_splits = tc ? router_tc_splits((int)T, (int)dm) : 0;
  w.n_max = expert_n_max(d);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + (bytes == 0 ? 1 : bytes), 256);
    return o;
  };
  w.err = take(sizeof(DevErrRecord));
  w.tickets = take(sizeof(int32_t) * kRouteTickets);
  w.n_unique = take(sizeof(int32_t));
  w.logits_part = take(sizeof(float) * (w.router_splits == 0 ? 1 : w.router_splits) * T * E);
  w.probs = take(sizeof(float) * T * E);
  w.probs_hat = take(sizeof(float) * T * E);
  w.cand = take(sizeof(uint2) * T * ((E + 31) / 32) * (size_t)mask_top_k(d));
  w.tk_idx = take(sizeof(int32_t) * T * k);
  w.tk_gate = take(sizeof(float) * T * k);
  w.unique_ids = take(sizeof(int32_t) * E);
  w.offsets = take(sizeof(int32_t) * (E + 1));
  w.rows = take(sizeof(int32_t) * T * k);
  w.pos = take(sizeof(int32_t) * T * k);
  w.xperm = take(2 * T * k * dm);
  w.h = take(2 * T * k * I);
  w.hs = take(2 * T * Is);
  // gate/up tile counters, then (block top-k on the general path) the rows copied per
  // (group, token tile)
  w.h_ready = take(sizeof(int32_t) * 2 * experts_ready_counters((int)T, (int)E, w.n_max));
  w.yslot = take(sizeof(float) * T * k * dm);
  w.yshared = take(sizeof(float) * T * dm);
  const bool dec = experts_decode_ok((int)T, (int)dm, (int)I, (int)Is);
  w.hdense = take(dec ? 2 * (E + 1) * (size_t)((T + 15) / 16 * 16) * (I > Is ? I : Is) : 0);
  w.spec = take(dec || d.mode == DMOE_ROUTE_BLOCK
                    ? sizeof(uint32_t) * d.n_blocks *
                          (spec_words((int)k) > kSpecMaskWords ? spec_words((int)k)
                                                               : kSpecMaskWords)
                    : 0);
  const size_t nchunks = (T + 31) / 32;
  w.disp_bits = take(sizeof(uint32_t) * nchunks * E);
  w.disp_base = take(sizeof(int32_t) * nchunks * E);
  w.disp_off = take(sizeof(int32_t) * E);
  w.w_parts_bytes = tc ? router_tc_parts_bytes((int)dm, (int)E) : 0;
  w.w_parts = take(w.w_parts_bytes);
  w.tc_part = take(sizeof(float) * (size_t)w.tc_splits * T * E);
  w.total = off;
  return w;
}

}  // namespace dmoe

using namespace dmoe;

namespace {

dmoe_status check_desc(const dmoe_layer_desc* d) {
  if (d == nullptr) return DMOE_ERR_INVALID_ARG;
  const long T = (long)d->n_blocks * d->block_size;
  if (d->d_model <= 0 || d->n_experts <= 0 || d->top_k <= 0 || d->d_ff <= 0 ||
      d->d_ff_shared < 0 || d->block_size <= 0 || d->n_blocks <= 0)
    return DMOE_ERR_INVALID_ARG;
  if (d->mode != DMOE_ROUTE_TOKEN && d->mode != DMOE_ROUTE_BLOCK) return DMOE_ERR_INVALID_ARG;
  if (!(d->top_p == d->top_p) || d->top_p < 0.f) return DMOE_ERR_INVALID_ARG;  // NaN or < 0
  if (d->top_k > d->n_experts) return DMOE_ERR_INVALID_ARG;
  if (d->block_top_k < 0 || (d->block_top_k > 0 && d->block_top_k < d->top_k) ||
      d->block_top_k > d->n_experts)
    return DMOE_ERR_INVALID_ARG;
  if (d->block_top_k > kMaxTopK) return DMOE_ERR_UNSUPPORTED;
  if (d->top_k > kMaxTopK || d->n_experts > kMaxExperts || d->n_experts % 8 != 0)
    return DMOE_ERR_UNSUPPORTED;
  if (d->d_model % 128 != 0 || d->d_model > kMaxDModel) return DMOE_ERR_UNSUPPORTED;
  if (d->d_ff % kTileM != 0 || d->d_ff > kMaxFF) return DMOE_ERR_UNSUPPORTED;
  if (d->d_ff_shared % kTileM != 0 || d->d_ff_shared > kMaxFF) return DMOE_ERR_UNSUPPORTED;
  if (T > kMaxTokens) return DMOE_ERR_UNSUPPORTED;
  return DMOE_OK;
}

dmoe_status check_ws(const dmoe_layer_desc* d, void* ws, size_t ws_bytes, Workspace* plan) {
  *plan = plan_workspace(*d);
  if (ws == nullptr || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return DMOE_ERR_INVALID_ARG;
  if (ws_bytes < plan->total) return DMOE_ERR_WORKSPACE;
  return DMOE_OK;
}

template <class T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<uint8_t*>(ws) + off);
}

void set_dispatch_scratch(DispatchArgs* a, void* ws, const Workspace& plan) {
  a->bits = at<uint32_t>(ws, plan.disp_bits);
  a->base = at<int32_t>(ws, plan.disp_base);
  a->off = at<int32_t>(ws, plan.disp_off);
  a->ticket = at<int32_t>(ws, plan.tickets) + kDispatchTicket;
}

dmoe_status cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return DMOE_OK;
  set_last_error(e);
  return DMOE_ERR_CUDA;
}

bool all_aligned(std::initializer_list<const void*> ptrs) {
  for (const void* p : ptrs)
    if (p == nullptr || (reinterpret_cast<uintptr_t>(p) & 15u) != 0) return false;
  return true;
}

dmoe_status run_router(const dmoe_layer_desc* desc, const void* x, const float* w_r,
                       const float* bias, int32_t* topk_idx, float* topk_gate, int32_t* coreset,
                       int32_t* coreset_size, float* probs, void* ws, const Workspace& plan,
                       cudaStream_t s, const L2Prefetch& shared_pf = L2Prefetch(),
                       const DispatchArgs* dsp = nullptr, uint32_t* spec_words = nullptr,
                       int32_t* ready_clear = nullptr, int n_ready_clear = 0,
                       bool spec_mask = false) {
  RouterArgs a{};
  a.spec_words = spec_words;
  a.spec_mask = spec_mask;
  a.ready_clear = ready_clear;
  a.n_ready_clear = n_ready_clear;
  a.x = static_cast<const __nv_bfloat16*>(x);
  a.w_r = w_r;
  a.bias = bias;
  a.logits_part = at<float>(ws, plan.logits_part);
  a.probs = probs != nullptr ? probs : at<float>(ws, plan.probs);
  a.probs_requested = probs != nullptr;
  a.probs_hat = at<float>(ws, plan.probs_hat);
  a.cand = at<uint2>(ws, plan.cand);
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
  a.err = at<DevErrRecord>(ws, plan.err);
  a.shared_pf = shared_pf;
  a.w_parts = plan.w_parts_bytes > 0 ? at<__nv_bfloat16>(ws, plan.w_parts) : nullptr;
  a.parts_ready = a.w_parts != nullptr && parts_prepared(ws, w_r);
  a.tc_splits = plan.tc_splits;
  a.tc_part = plan.tc_splits > 0 ? at<float>(ws, plan.tc_part) : nullptr;
  return cuda_status(launch_router(a, dsp, at<int32_t>(ws, plan.tickets), s));
}

dmoe_status run_dispatch(const dmoe_layer_desc* desc, const int32_t* topk_idx, int32_t* n_unique,
                         int32_t* unique_ids, int32_t* offsets, int32_t* rows, int32_t* pos,
                         void* ws, const Workspace& plan, cudaStream_t s) {
  DispatchArgs a{};
  a.topk_idx = topk_idx;
  a.n_unique = n_unique;
  a.unique_ids = unique_ids;
  a.offsets = offsets;
  a.rows = rows;
  a.pos = pos;
  a.T = desc->n_blocks * desc->block_size;
  a.E = desc->n_experts;
  a.k = desc->top_k;
  a.err = at<DevErrRecord>(ws, plan.err);
  set_dispatch_scratch(&a, ws, plan);
  return cuda_status(launch_dispatch(a, s));
}

dmoe_status run_experts(const dmoe_layer_desc* desc, const void* x, const void* w_gate,
                        const void* w_up, const void* w_down, const void* ws_gate,
                        const void* ws_up, const void* ws_down, const float* topk_gate,
                        const int32_t* n_unique, const int32_t* unique_ids,
                        const int32_t* offsets, const int32_t* rows, const int32_t* pos,
                        void* y, void* ws, const Workspace& plan, cudaStream_t s,
                        bool shared_prefetched = false, uint32_t* spec_words = nullptr,
                        bool gathered = false, int32_t* topk_idx = nullptr,
                        int32_t* pos_out = nullptr, int32_t* n_unique_out = nullptr,
                        int32_t* unique_ids_out = nullptr, bool spec_mask = false) {
  ExpertArgs a{};
  a.spec_mask = spec_mask;
  a.topk_idx = topk_idx;
  a.pos_out = pos_out;
  a.n_unique_out = n_unique_out;
  a.unique_ids_out = unique_ids_out;
  a.prefetch_shared = !shared_prefetched;
  a.gathered = gathered;
  a.spec_words = spec_words;
  a.spec_blocks = desc->n_blocks;
  a.x = static_cast<const __nv_bfloat16*>(x);
  a.w_gate = w_gate;
  a.w_up = w_up;
  a.w_down = w_down;
  a.ws_gate = ws_gate;
  a.ws_up = ws_up;
  a.ws_down = ws_down;
  a.topk_gate = topk_gate;
  a.n_unique = n_unique;
  a.unique_ids = unique_ids;
  a.offsets = offsets;
  a.rows = rows;
  a.pos = pos;
  a.y = static_cast<__nv_bfloat16*>(y);
  a.xperm = at<__nv_bfloat16>(ws, plan.xperm);
  a.h = at<__nv_bfloat16>(ws, plan.h);
  a.hs = at<__nv_bfloat16>(ws, plan.hs);
  a.yslot = at<float>(ws, plan.yslot);
  a.h_ready = at<int32_t>(ws, plan.h_ready);
  a.hdense = at<__nv_bfloat16>(ws, plan.hdense);
  a.tickets = at<int32_t>(ws, plan.tickets);
  a.yshared = at<float>(ws, plan.yshared);
  a.err = at<DevErrRecord>(ws, plan.err);
  a.T = desc->n_blocks * desc->block_size;
  a.d = desc->d_model;
  a.E = desc->n_experts;
  a.k = desc->top_k;
  a.I = desc->d_ff;
  a.Is = desc->d_ff_shared;
  a.n_max = plan.n_max;
  if (experts_decode_ok(a.T, a.d, a.I, a.Is)) return cuda_status(launch_experts_decode(a, s));
  return cuda_status(launch_experts(a, s));
}

}  // namespace

extern "C" {

dmoe_status dmoe_workspace_size(const dmoe_layer_desc* desc, size_t* bytes) {
  if (bytes == nullptr) return DMOE_ERR_INVALID_ARG;
  const dmoe_status st = check_desc(desc);
  if (st != DMOE_OK) return st;
  *bytes = plan_workspace(*desc).total;
  return DMOE_OK;
}

dmoe_status dmoe_router(const dmoe_layer_desc* desc, const void* x, const float* w_r,
                        const float* bias, int32_t* topk_idx, float* topk_gate,
                        int32_t* coreset, int32_t* coreset_size, float* probs,
                        void* workspace, size_t workspace_bytes, void* stream) {
  dmoe_status st = check_desc(desc);
  if (st != DMOE_OK) return st;
  if (!all_aligned({x, w_r, topk_idx, topk_gate})) return DMOE_ERR_INVALID_ARG;
  if ((bias != nullptr && !aligned16(bias)) || (probs != nullptr && !aligned16(probs)) ||
      (coreset != nullptr && !aligned16(coreset)) ||
      (coreset_size != nullptr && !aligned16(coreset_size)))
    return DMOE_ERR_INVALID_ARG;
  Workspace plan;
  st = check_ws(desc, workspace, workspace_bytes, &plan);
  if (st != DMOE_OK) return st;
  return run_router(desc, x, w_r, bias, topk_idx, topk_gate, coreset, coreset_size, probs,
                    workspace, plan, static_cast<cudaStream_t>(stream));
}

dmoe_status dmoe_router_prepare(const dmoe_layer_desc* desc, const float* w_r, void* workspace,
                                size_t workspace_bytes, void* stream) {
  dmoe_status st = check_desc(desc);
  if (st != DMOE_OK) return st;
  if (!all_aligned({w_r})) return DMOE_ERR_INVALID_ARG;
  Workspace plan;
  st = check_ws(desc, workspace, workspace_bytes, &plan);
  if (st != DMOE_OK) return st;
  {
    std::lock_guard<std::mutex> lock(g_prep_mu);
    g_prep.erase(workspace);
  }
  if (plan.w_parts_bytes == 0) return DMOE_OK;   // this shape's router reads W_r itself
  const cudaError_t e = launch_router_wsplit(w_r, at<__nv_bfloat16>(workspace, plan.w_parts),
                                             desc->d_model, desc->n_experts,
                                             static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_status(e);
  std::lock_guard<std::mutex> lock(g_prep_mu);
  g_prep[workspace] = w_r;
  return DMOE_OK;
}

dmoe_status dmoe_dispatch(const dmoe_layer_desc* desc, const int32_t* topk_idx,
                          int32_t* n_unique, int32_t* unique_ids, int32_t* offsets,
                          int32_t* rows, int32_t* pos, void* workspace, size_t workspace_bytes,
                          void* stream) {
  dmoe_status st = check_desc(desc);
  if (st != DMOE_OK) return st;
  if (!all_aligned({topk_idx, n_unique, unique_ids, offsets, rows, pos}))
    return DMOE_ERR_INVALID_ARG;
  Workspace plan;
  st = check_ws(desc, workspace, workspace_bytes, &plan);
  if (st != DMOE_OK) return st;
  return run_dispatch(desc, topk_idx, n_unique, unique_ids, offsets, rows, pos, workspace, plan,
                      static_cast<cudaStream_t>(stream));
}

dmoe_status dmoe_moe_forward(const dmoe_layer_desc* desc, const void* x, const void* w_gate,
                             const void* w_up, const void* w_down, const void* ws_gate,
                             const void* ws_up, const void* ws_down, const float* topk_gate,
                             const int32_t* n_unique, const int32_t* unique_ids,
                             const int32_t* offsets, const int32_t* rows, const int32_t* pos,
                             void* y, void* workspace, size_t workspace_bytes, void* stream) {
  dmoe_status st = check_desc(desc);
  if (st != DMOE_OK) return st;
  if (!all_aligned({x, w_gate, w_up, w_down, topk_gate, n_unique, unique_ids, offsets, rows,
                    pos, y}))
    return DMOE_ERR_INVALID_ARG;
  if (desc->d_ff_shared > 0 && !all_aligned({ws_gate, ws_up, ws_down})) return DMOE_ERR_INVALID_ARG;
  Workspace plan;
  st = check_ws(desc, workspace, workspace_bytes, &plan);
  if (st != DMOE_OK) return st;
  return run_experts(desc, x, w_gate, w_up, w_down, ws_gate, ws_up, ws_down, topk_gate, n_unique,
                     unique_ids, offsets, rows, pos, y, workspace, plan,
                     static_cast<cudaStream_t>(stream));
}

dmoe_status dmoe_layer_forward(const dmoe_layer_desc* desc, const void* x, const float* w_r,
                               const float* bias, const void* w_gate, const void* w_up,
                               const void* w_down, const void* ws_gate, const void* ws_up,
                               const void* ws_down, void* y, int32_t* topk_idx,
                               float* topk_gate, int32_t* n_unique, int32_t* unique_ids,
                               void* workspace, size_t workspace_bytes, void* stream) {
  dmoe_status st = check_desc(desc);
  if (st != DMOE_OK) return st;
  if (!all_aligned({x, w_r, w_gate, w_up, w_down, y})) return DMOE_ERR_INVALID_ARG;
  if (desc->d_ff_shared > 0 && !all_aligned({ws_gate, ws_up, ws_down})) return DMOE_ERR_INVALID_ARG;
  if ((bias != nullptr && !aligned16(bias)) || (topk_idx != nullptr && !aligned16(topk_idx)) ||
      (topk_gate != nullptr && !aligned16(topk_gate)) ||
      (n_unique != nullptr && !aligned16(n_unique)) ||
      (unique_ids != nullptr && !aligned16(unique_ids)))
    return DMOE_ERR_INVALID_ARG;
  Workspace plan;
  st = check_ws(desc, workspace, workspace_bytes, &plan);
  if (st != DMOE_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int32_t* idx = topk_idx != nullptr ? topk_idx : at<int32_t>(workspace, plan.tk_idx);
  float* gate = topk_gate != nullptr ? topk_gate : at<float>(workspace, plan.tk_gate);
  int32_t* nu = n_unique != nullptr ? n_unique : at<int32_t>(workspace, plan.n_unique);
  int32_t* uid = unique_ids != nullptr ? unique_ids : at<int32_t>(workspace, plan.unique_ids);
  int32_t* offs = at<int32_t>(workspace, plan.offsets);
  int32_t* rows = at<int32_t>(workspace, plan.rows);
  int32_t* pos = at<int32_t>(workspace, plan.pos);
  // In the fused call the shared expert's weights start streaming into L2 with the router.
  L2Prefetch shared_pf;
  if (desc->d_ff_shared > 0) {
    shared_pf.ptr[0] = ws_gate;
    shared_pf.ptr[1] = ws_up;
    shared_pf.ptr[2] = ws_down;
    shared_pf.bytes = (int64_t)desc->d_ff_shared * desc->d_model * 2;
  }
  DispatchArgs dsp{};
  dsp.topk_idx = idx;
  dsp.n_unique = nu;
  dsp.unique_ids = uid;
  dsp.offsets = offs;
  dsp.rows = rows;
  dsp.pos = pos;
  dsp.T = desc->n_blocks * desc->block_size;
  dsp.E = desc->n_experts;
  dsp.k = desc->top_k;
  dsp.err = at<DevErrRecord>(workspace, plan.err);
  set_dispatch_scratch(&dsp, workspace, plan);
  const int T_all = desc->n_blocks * desc->block_size;
  // general path: the dispatch placement also writes x in dispatch order and clears the
  // expert launch's tile counters (no gather launch); with block top-k the expert launch
  // does the dispatch itself (spec_general)
  const bool general = !route_cluster_ok(T_all, desc->d_model, desc->n_experts) &&
                       !experts_decode_ok(T_all, desc->d_model, desc->d_ff, desc->d_ff_shared);
  const bool spec_general = general && experts_spec_ok(*desc, plan.n_max);
  const bool gathered = general && !spec_general;
  if (gathered) {
    dsp.x = static_cast<const __nv_bfloat16*>(x);
    dsp.xperm = at<__nv_bfloat16>(workspace, plan.xperm);
    dsp.d = desc->d_model;
    dsp.zero = at<int32_t>(workspace, plan.h_ready);
    dsp.n_zero = experts_ready_counters(T_all, desc->n_experts, plan.n_max);
  }
  // block routing through the decode-size launches: the expert launch starts streaming on
  // the early-published coresets, before the routing launch ends. With block top-k (every
  // token keeps the whole coreset) their union is the unique set, published as ids. With
  // fewer experts per token than the coreset holds, or p <= 0.6 over blocks of 32 or more
  // tokens, the union contains the unique set and is seldom larger (most members are kept
  // by some token of the block): published as masks, and the down epilogue takes each
  // group's rows from the dispatch once it is complete. Larger p or smaller blocks leave
  // many members unkept: streaming them cost more than the early start saved.
  const int T = desc->n_blocks * desc->block_size;
  uint32_t* spec_w = nullptr;
  bool spec_mask = false;
  if (desc->mode == DMOE_ROUTE_BLOCK && route_cluster_ok(T, desc->d_model, desc->n_experts) &&
      experts_decode_ok(T, desc->d_model, desc->d_ff, desc->d_ff_shared)) {
    const bool ids = desc->top_p <= 0.f && mask_top_k(*desc) == desc->top_k;
    const bool masks = (desc->top_p <= 0.f && !ids) ||
                       (desc->top_p > 0.f && desc->top_p <= 0.6f && desc->block_size >= 32);
    if (ids || masks) {
      spec_w = at<uint32_t>(workspace, plan.spec);
      spec_mask = masks;
    }
  }
  if (spec_general) {
    spec_w = at<uint32_t>(workspace, plan.spec);
    st = run_router(desc, x, w_r, bias, idx, gate, nullptr, nullptr, nullptr, workspace, plan, s,
                    shared_pf, nullptr, spec_w, at<int32_t>(workspace, plan.h_ready),
                    2 * experts_ready_counters(T, desc->n_experts, plan.n_max));
    if (st != DMOE_OK) return st;
    return run_experts(desc, x, w_gate, w_up, w_down, ws_gate, ws_up, ws_down, gate, nu, uid,
                       offs, rows, pos, y, workspace, plan, s, /*shared_prefetched=*/true, spec_w,
                       false, idx, pos, nu, uid);
  }
  st = run_router(desc, x, w_r, bias, idx, gate, nullptr, nullptr, nullptr, workspace, plan, s,
                  shared_pf, &dsp, spec_w, nullptr, 0, spec_mask);
  if (st != DMOE_OK) return st;
  return run_experts(desc, x, w_gate, w_up, w_down, ws_gate, ws_up, ws_down, gate, nu, uid, offs,
                     rows, pos, y, workspace, plan, s, /*shared_prefetched=*/true, spec_w,
                     gathered, nullptr, nullptr, nullptr, nullptr, spec_mask);
}

dmoe_status dmoe_get_device_error(void* workspace, void* stream, int32_t* info) {
  if (workspace == nullptr) return DMOE_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_status(e);
  DevErrRecord rec{};
  e = cudaMemcpy(&rec, workspace, sizeof(rec), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_status(e);
  if (info != nullptr) {
    info[0] = rec.code;
    info[1] = rec.where;
    info[2] = rec.value;
    info[3] = 0;
  }
  if (rec.code == kErrNone) return DMOE_OK;
  e = cudaMemset(workspace, 0, sizeof(rec));
  if (e != cudaSuccess) return cuda_status(e);
  return rec.code == kErrTimeout ? DMOE_ERR_TIMEOUT : DMOE_ERR_DEVICE;
}

dmoe_status dmoe_set_debug_hold(void* workspace, int32_t hold, void* stream) {
  if (workspace == nullptr || hold < 0) return DMOE_ERR_INVALID_ARG;
  // the fault record heads the workspace; its last word is the hold
  static_assert(offsetof(DevErrRecord, hold) == 12, "record layout");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(s);
  if (e == cudaSuccess)
    e = cudaMemcpy(static_cast<uint8_t*>(workspace) + offsetof(DevErrRecord, hold), &hold,
                   sizeof(hold), cudaMemcpyHostToDevice);
  return cuda_status(e);
}

dmoe_status dmoe_set_profile_events(int32_t kernel, void* ev_begin, void* ev_end) {
  if (kernel < 0 || kernel >= DMOE_KERNEL_COUNT) return DMOE_ERR_INVALID_ARG;
  g_prof[kernel].begin = static_cast<cudaEvent_t>(ev_begin);
  g_prof[kernel].end = static_cast<cudaEvent_t>(ev_end);
  return DMOE_OK;
}

const char* dmoe_status_string(dmoe_status status) {
  switch (status) {
    case DMOE_OK: return "DMOE_OK";
    case DMOE_ERR_INVALID_ARG: return "DMOE_ERR_INVALID_ARG: invalid argument";
    case DMOE_ERR_UNSUPPORTED: return "DMOE_ERR_UNSUPPORTED: shape outside this build's limits";
    case DMOE_ERR_WORKSPACE: return "DMOE_ERR_WORKSPACE: workspace too small";
    case DMOE_ERR_CUDA: return "DMOE_ERR_CUDA: CUDA call or launch failed";
    case DMOE_ERR_DEVICE: return "DMOE_ERR_DEVICE: a kernel recorded a fault";
    case DMOE_ERR_TIMEOUT: return "DMOE_ERR_TIMEOUT: a kernel's bounded wait ran out";
  }
  return "unknown dmoe_status";
}

const char* dmoe_last_error_message(void) { return g_last_error; }

int32_t dmoe_abi_version(void) { return DMOE_ABI_VERSION; }

int32_t dmoe_layer_forward_launches(const dmoe_layer_desc* desc) {
  if (check_desc(desc) != DMOE_OK) return -1;
  const int T = desc->n_blocks * desc->block_size;
  int n = 0;
  if (route_cluster_ok(T, desc->d_model, desc->n_experts)) {
    n += 1;                                                   // routing with the dispatch
  } else {
    n += 2;                                                   // logits, softmax / top-k
    n += router_tc_ok(T, desc->d_model, desc->n_experts) ? 1 : 0;   // the split of W_r
    n += desc->mode == DMOE_ROUTE_BLOCK ? 1 : 0;              // Algorithm 1
    n += 2;                                                   // dispatch: count, place
  }
  // experts and combine; the general experts' gather is a launch of its own only after the
  // fused routing launch (otherwise the dispatch placement does it); with block top-k on the
  // general path the expert launch does the dispatch (no dispatch launches)
  const bool dec = experts_decode_ok(T, desc->d_model, desc->d_ff, desc->d_ff_shared);
  const bool cluster = route_cluster_ok(T, desc->d_model, desc->n_experts);
  if (!cluster && !dec && experts_spec_ok(*desc, expert_n_max(*desc))) n -= 2;
  n += (!dec && cluster) ? 3 : 2;
  return n;
}

}  // extern "C"
