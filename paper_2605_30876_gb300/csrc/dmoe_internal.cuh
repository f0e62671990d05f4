// Internal declarations shared by the CUDA translation units of libdmoe (not installed).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/dmoe.h"

namespace dmoe {

// ---------------------------------------------------------------------------------------
// limits of this build (mirrored in include/dmoe.h)
// ---------------------------------------------------------------------------------------
constexpr int kMaxExperts = 256;
constexpr int kMaxTopK = 16;
constexpr int kMaxTokens = 4096;
constexpr int kMaxDModel = 16384;
constexpr int kMaxFF = 8192;
constexpr int kTileM = 128;        // MMA M (weight rows per tile)
constexpr int kTileK = 64;         // K elements per pipeline stage (128 B of bf16)
constexpr int kMaxPersistentCtas = 320;

// ---------------------------------------------------------------------------------------
// device fault record, at the head of the workspace
// ---------------------------------------------------------------------------------------
enum DevErr : int32_t {
  kErrNone = 0,
  kErrTimeout = 1,        // a bounded mbarrier wait ran out
  kErrExpertId = 2,       // an expert id outside [0, E)
  kErrDupExpert = 3,      // the same expert twice in one token's list
  kErrBadDispatch = 4,    // dispatch data inconsistent (counts, offsets)
};
enum DevWhere : int32_t {
  kAtRouter = 1, kAtBlockRoute = 2, kAtDispatch = 3, kAtGateUp = 4, kAtDown = 5,
  kAtCombine = 6, kAtGather = 7,
};
constexpr int kRouteTickets = 256;
constexpr int kRouteClusterCtas = 8;   // CTAs per cluster of the decode-size routing launch
struct DevErrRecord {
  int32_t code;
  int32_t where;
  int32_t value;
  int32_t hold;   // diagnostic (normally 0): see dmoe_set_debug_hold
};

__device__ __forceinline__ void record_error(DevErrRecord* rec, int code, int where, int value) {
  if (atomicCAS(&rec->code, 0, code) == 0) {
    rec->where = where;
    rec->value = value;
  }
}

// ---------------------------------------------------------------------------------------
// workspace layout (byte offsets from the workspace base; every region 256-B aligned)
// ---------------------------------------------------------------------------------------
struct Workspace {
  size_t err;          // DevErrRecord
  size_t tickets;      // int32 [kRouteTickets]: stage counters of the routing launch (zero between calls)
  size_t n_unique;     // int32 [1]  (used when the caller does not supply one)
  size_t logits_part;  // fp32 [router_splits, T, E]
  size_t probs;        // fp32 [T, E]
  size_t probs_hat;    // fp32 [T, E]   TopKMask(s_i, k)
  size_t cand;         // uint2 [T, ceil(E/32), k]: decode-size routing, each 32-expert group's
                       // k best (order key, id) per token
  size_t tk_idx;       // int32 [T, k] routed experts (when the caller does not supply)
  size_t tk_gate;      // fp32 [T, k]
  size_t unique_ids;   // int32 [E]
  size_t offsets;      // int32 [E + 1]
  size_t rows;         // int32 [T*k]
  size_t pos;          // int32 [T*k]
  size_t xperm;        // bf16 [T*k, d]   x gathered in dispatch order
  size_t h;            // bf16 [T*k, I]   SwiGLU intermediate of the routed experts
  size_t hs;           // bf16 [T, I_s]   shared-expert intermediate
  size_t h_ready;      // int32 [(E+1) * token tiles]: published gate/up tiles
  size_t yslot;        // [T*k, d] expert outputs per (token, slot): fp32 (decode-size path)
                       // or bf16 (general path); sized for fp32
  size_t yshared;      // [T, d], the same element type
  size_t hdense;       // bf16 [(E+1) * n_pad, max(I, I_s)]: H per group over all tokens
  size_t spec;         // int32 [n_blocks, k]: the coreset of every block (block top-k call)
                       // (decode-size forwards only)
  size_t disp_bits;    // u32 [ceil(T/32), E]: dispatch, token bitmap per (32-token chunk, expert)
  size_t disp_base;    // int32 [ceil(T/32), E]: dispatch, pairs of the expert in earlier chunks
  size_t disp_off;     // int32 [E]: dispatch, first row of every expert (all experts)
  size_t w_parts;      // bf16 [3E, d]: split of W_r for the tcgen05 router (large forwards)
  size_t w_parts_bytes;
  size_t tc_part;      // fp32 [tc_splits, T, E]: the tcgen05 router's partial logits
  size_t total;
  int router_splits;
  int tc_splits;       // slices of d of the tcgen05 router logits (0: not used)
  int n_max;           // token tile (MMA N) of the expert GEMMs
};

// Token tile (MMA N) of the general expert kernel: every group's rows are covered by tiles
// of n_max rows (a tile of at most half of that loads a half-height box). Each tile streams
// the group's weights through its SM again, so the tile is as wide as the forward allows:
// 128 rows, or 256 in block mode with blocks of 16 or more tokens at 1024 or more tokens
// (every unique expert then takes whole blocks, hundreds of rows; one K box per stage keeps
// four stages in shared memory).
inline int expert_n_max(const dmoe_layer_desc& d) {
  const int T = d.n_blocks * d.block_size;
  const int cap = (d.mode == DMOE_ROUTE_BLOCK && d.block_size >= 16 && T >= 1024) ? 256 : 128;
  int n = ((T + 15) / 16) * 16;
  return n > cap ? cap : (n < 16 ? 16 : n);
}

Workspace plan_workspace(const dmoe_layer_desc& d);

// The k of Algorithm 1's TopKMask and coreset floor: block_top_k in block mode when set,
// else the per-token k.
inline int mask_top_k(const dmoe_layer_desc& d) {
  return (d.mode == DMOE_ROUTE_BLOCK && d.block_top_k > 0) ? d.block_top_k : d.top_k;
}

// ---------------------------------------------------------------------------------------
// launchers (each defined in its own translation unit)
// ---------------------------------------------------------------------------------------
// Weights to pull into L2 ahead of their use (bulk L2 prefetch; all null = none): three
// matrices of `bytes` each per expert, expert e at ptr[m] + e * bytes.
struct L2Prefetch {
  const void* ptr[3] = {nullptr, nullptr, nullptr};
  int64_t bytes = 0;
};

__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
constexpr int64_t kPrefetchChunk = 64 * 1024;

// Issues chunk `c` (of `per_expert * 3 * n` chunks) of the prefetch list: matrix-major, then
// expert (by position in `ids`, or 0..n-1 when ids is null), then chunk within the matrix.
__device__ __forceinline__ void l2_prefetch_chunk(const L2Prefetch& pf, const int32_t* ids,
                                                  int n, int c) {
  const int64_t per = (pf.bytes + kPrefetchChunk - 1) / kPrefetchChunk;
  const int64_t per_mat = per * n;
  const int m = (int)(c / per_mat);
  const int64_t r = c - m * per_mat;
  const int u = (int)(r / per);
  const int64_t off = (r - (int64_t)u * per) * kPrefetchChunk;
  const int e = ids != nullptr ? ids[u] : u;
  const int64_t len = pf.bytes - off < kPrefetchChunk ? pf.bytes - off : kPrefetchChunk;
  if (m < 3 && pf.ptr[m] != nullptr && len > 0)
    prefetch_l2_bulk(static_cast<const uint8_t*>(pf.ptr[m]) + (int64_t)e * pf.bytes + off,
                     (uint32_t)len);
}

// Spreads the chunks of one expert's three matrices over `nctas` CTAs (call from one thread).
__device__ __forceinline__ void issue_shared_prefetch(const L2Prefetch& pf, int cta, int nctas) {
  if (pf.bytes > 0) {
    const int per = (int)((pf.bytes + kPrefetchChunk - 1) / kPrefetchChunk);
    for (int c = cta; c < 3 * per; c += nctas) l2_prefetch_chunk(pf, nullptr, 1, c);
  }
}

struct RouterArgs {
  const __nv_bfloat16* x;
  const float* w_r;
  const float* bias;
  float* logits_part;
  float* probs;        // [T, E]
  float* probs_hat;    // [T, E] (block mode)
  uint2* cand;         // [T, ceil(E/32), kb] (decode-size routing)
  int32_t* topk_idx;   // [T, k] final routing
  float* topk_gate;    // [T, k]
  int32_t* coreset;    // [n_blocks, E] or null
  int32_t* coreset_size;
  int T, d, E, k, B, n_blocks, mode, splits;
  int kb;              // k of TopKMask and of the coreset floor (block mode; k >= this k)
  float top_p;
  DevErrRecord* err;
  L2Prefetch shared_pf;   // the shared expert's weights (one "expert")
  bool probs_requested;   // the caller wants the scores in `probs`
  __nv_bfloat16* w_parts; // [3E, d]: the bf16 split of W_r for the tcgen05 router, or null
                          // (then the mma.sync / FFMA logits run)
  int tc_splits;          // slices of d of the tcgen05 logits
  float* tc_part;         // [tc_splits, T, E]: their partial sums
  bool parts_ready;       // w_parts already holds this W_r's split (dmoe_router_prepare)
  // block top-k (p <= 0) in the fused decode-size call: every block's coreset, which is
  // then the block's routing, is published early here: spec_words(k) words per block, three
  // ids and a marker byte each, one 32-bit store per word (a word reads as zero until it is
  // complete; zero between calls); nullptr otherwise
  uint32_t* spec_words;
  // spec_words hold every block's coreset as a mask instead (block routing with p > 0, or
  // fewer experts per token than the coreset holds: the coresets' union then contains the
  // unique experts): kSpecMaskWords words per block, the 256-bit member mask, then a marker
  // stored with release semantics after it
  bool spec_mask;
  // with spec_words on the general path: the gate/up tile counters of the expert launch that
  // follows, cleared by the block routing launch before it lets that launch start (the
  // dispatch launches, which clear them otherwise, do not run then)
  int32_t* ready_clear;
  int n_ready_clear;
};

struct DispatchArgs {
  const int32_t* topk_idx;
  int32_t* n_unique;
  int32_t* unique_ids;
  int32_t* offsets;
  int32_t* rows;
  int32_t* pos;
  int T, E, k;
  DevErrRecord* err;
  // scratch of the multi-CTA dispatch (Workspace::disp_*) and its ticket (zero between calls)
  uint32_t* bits;
  int32_t* base;
  int32_t* off;
  int32_t* ticket;
  // optional (the fused layer call of the general path): the placement also copies x's
  // rows into dispatch order (xperm [T*k, d]) and clears zero[0 .. n_zero) (the expert
  // launch's tile counters), so that the expert launch needs no gather launch
  const __nv_bfloat16* x;
  __nv_bfloat16* xperm;
  int d;
  int32_t* zero;
  int n_zero;
};
// ticket index (in Workspace::tickets) of the dispatch launch
constexpr int kDispatchTicket = 1;
cudaError_t launch_dispatch(const DispatchArgs& a, cudaStream_t s);

// Routing of one forward. With `dsp` set, the dispatch is computed too (inside the fused
// decode-size launch, or by launch_dispatch otherwise). `tickets` is a workspace array of
// kRouteTickets ints that is zero between calls.
cudaError_t launch_router(const RouterArgs& a, const DispatchArgs* dsp, int32_t* tickets,
                          cudaStream_t s);
bool route_cluster_ok(int T, int d, int E);
// The logits stage of that launch alone, over tiles of 64 tokens (any T): logits + bias
// into a.logits_part [T, E] (no split).
bool route_cluster_logits_ok(int d, int E);
cudaError_t launch_logits_cluster(const RouterArgs& a, cudaStream_t s);
// The logits of a large forward on tcgen05 (router_logits_tc.cu): the split of W_r into
// a.w_parts, then the products over `splits` slices of d into a.tc_part [splits, T, E]
// (router_softmax_kernel adds them in order, with the bias). Needs T >= 128, d % 64 == 0,
// E % 32 == 0; router_tc_splits gives the split.
bool router_tc_ok(int T, int d, int E);
int router_tc_splits(int T, int d);
size_t router_tc_parts_bytes(int d, int E);
cudaError_t launch_router_tc(const RouterArgs& a, int splits, cudaStream_t s);
// The split of W_r into its three bf16 parts (the first launch of launch_router_tc).
cudaError_t launch_router_wsplit(const float* w_r, __nv_bfloat16* parts, int d, int E,
                                 cudaStream_t s);
cudaError_t launch_route_cluster(const RouterArgs& a, const DispatchArgs* dsp, int32_t* tickets,
                                 cudaStream_t s);

struct ExpertArgs {
  // inputs
  const __nv_bfloat16* x;
  const void* w_gate; const void* w_up; const void* w_down;
  const void* ws_gate; const void* ws_up; const void* ws_down;
  const float* topk_gate;
  const int32_t* n_unique; const int32_t* unique_ids; const int32_t* offsets;
  const int32_t* rows; const int32_t* pos;
  __nv_bfloat16* y;
  // workspace
  __nv_bfloat16* xperm; __nv_bfloat16* h; __nv_bfloat16* hs;
  void* yslot; void* yshared;   // fp32 (decode-size path) or bf16 (general path) rows
  int32_t* h_ready;
  __nv_bfloat16* hdense;  // decode-size path: H per group over all tokens
  int32_t* tickets;       // kRouteTickets ints, zero between calls
  DevErrRecord* err;
  bool prefetch_shared;   // the shared expert's weights were not prefetched by the router
  bool gathered;          // xperm is written and the tile counters cleared (by the dispatch)
  // decode-size path, block top-k: the unique experts are the union of the published
  // coresets (RouterArgs::spec_words), known before the routing launch ends; nullptr
  // otherwise
  uint32_t* spec_words;
  int spec_blocks;
  bool spec_mask;         // the words are coreset masks (RouterArgs::spec_mask)
  // general path with spec_words (block top-k): the expert launch writes the dispatch's
  // outputs from the published coresets and the routing's topk_idx
  const int32_t* topk_idx;
  int32_t* pos_out;
  int32_t* n_unique_out;
  int32_t* unique_ids_out;
  // shape
  int T, d, E, k, I, Is, n_max;
};
cudaError_t launch_experts(const ExpertArgs& a, cudaStream_t s);
int experts_ready_counters(int T, int E, int n_max);
// Block top-k on the general path (every token keeps its block's whole coreset): the expert
// launch plans from the coresets the block routing launch publishes, reads the token rows
// from x block by block and writes the dispatch's outputs, so that no dispatch launch runs.
bool experts_spec_ok(const dmoe_layer_desc& d, int n_max);
// gate-weighted combine of the expert rows into y (the last launch of both expert paths);
// it also clears zero[0 .. n_zero) and zero2[0 .. n_zero2) once the launch before it has
// ended. meta_early: the slot indices and gates may be read before that launch ends (they
// were complete before it released the combine)
// rows_bf16: the rows per (token, slot) and the shared rows are bf16 (general path), else fp32
cudaError_t launch_combine(const ExpertArgs& a, cudaStream_t s, int32_t* zero = nullptr,
                           int n_zero = 0, uint32_t* zero2 = nullptr, int n_zero2 = 0,
                           bool meta_early = false, bool rows_bf16 = false);

// Words of one block's published coreset (three 8-bit ids and a marker byte per word).
__host__ __device__ inline int spec_words(int k) { return (k + 2) / 3; }
// words per block of a published coreset mask: the member mask, then the marker
constexpr int kSpecMaskWords = kMaxExperts / 32 + 1;
// Decode-sized forwards (T <= 64): one persistent launch over gate/up and down tiles of
// every group, all tokens at once (no gather), then the combine.
bool experts_decode_ok(int T, int d, int I, int Is);
cudaError_t launch_experts_decode(const ExpertArgs& a, cudaStream_t s);

// profiling events (dmoe_set_profile_events), per host thread
void prof_begin(int kernel, cudaStream_t s);
void prof_end(int kernel, cudaStream_t s);
// events are set for `kernel` on this host thread: its launch is made without programmatic
// dependent launch, so that the events bracket its own execution only
bool prof_serial(int kernel);

// Programmatic dependent launch: a kernel launched with `pdl` set may start while the
// previous kernel on the stream is still running; it must call pdl_wait() before reading
// anything that kernel writes. pdl_launch_dependents() lets the next kernel start early.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Cluster launch (clusters of cluster_x CTAs along x), optionally as a programmatic
// dependent launch (see pdl_wait).
template <typename... KArgs, typename... Args>
cudaError_t launch_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                           cudaStream_t s, int cluster_x, bool pdl, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster_x;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch_ex(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                      cudaStream_t s, bool pdl, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// host helpers
int device_sm_count();
void set_last_error(cudaError_t e);
void set_last_error_text(const char* msg);

}  // namespace dmoe
