/*
 * dmoe.h — C ABI of the block-routed MoE-layer forward of dMoE
 * ("dLLMs with Learnable Block Experts", arXiv 2605.30876) on one GB300 (sm_103a).
 *
 * The layer: a router scores every token over the |E| routed experts (§4.2,
 * s_i = Router(t_i)); Algorithm 1 (§4.2) aggregates the token scores of each diffusion
 * block, keeps a top-p coreset of experts and routes every token to its k best experts
 * inside that coreset; the selected experts run as SwiGLU FFNs, an optional shared expert
 * runs on every token, and the outputs are combined with the gate weights. Token-level
 * routing (the "Original" baseline of §5.1) is kept as a mode.
 *
 * Conventions for every call below
 *  - All tensor pointers are DEVICE pointers of the current CUDA device unless marked
 *    "host". The caller owns all memory; the library never allocates, frees or
 *    synchronises on the forward path (dmoe_get_device_error is the one call that syncs).
 *  - Layouts are dense row-major, the last index fastest. bf16 tensors are passed as
 *    `const void*` (IEEE bfloat16 bit patterns); every tensor base must be 16-byte aligned.
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream). All
 *    work is enqueued asynchronously on it, in order; calls on one workspace must not
 *    overlap on the GPU.
 *  - Outputs are fully overwritten (no need to zero them).
 *  - Argument errors are detected on the host before anything is launched and return
 *    DMOE_ERR_INVALID_ARG / DMOE_ERR_UNSUPPORTED / DMOE_ERR_WORKSPACE; launch failures
 *    return DMOE_ERR_CUDA (dmoe_last_error_message() has the CUDA text). Faults detected
 *    on the device (an expert id out of range, a pipeline wait that timed out) never
 *    trap: the kernels record a code in the workspace and exit; dmoe_get_device_error()
 *    reads and clears it.
 *  - Notation: T = n_blocks * block_size tokens, d = d_model, E = n_experts, k = top_k,
 *    I = d_ff, I_s = d_ff_shared.
 */
#ifndef DMOE_H_
#define DMOE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DMOE_ABI_VERSION 2

typedef enum {
  DMOE_OK = 0,
  DMOE_ERR_INVALID_ARG = 1,   /* null pointer, bad size, misaligned pointer           */
  DMOE_ERR_UNSUPPORTED = 2,   /* valid but outside what this build implements         */
  DMOE_ERR_WORKSPACE = 3,     /* workspace smaller than dmoe_workspace_size()         */
  DMOE_ERR_CUDA = 4,          /* a CUDA runtime/driver call or a launch failed        */
  DMOE_ERR_DEVICE = 5,        /* a kernel recorded a fault (see dmoe_get_device_error) */
  DMOE_ERR_TIMEOUT = 6        /* a kernel's bounded wait ran out                      */
} dmoe_status;

typedef enum {
  DMOE_ROUTE_TOKEN = 0,       /* R_i = TopK(s_i, k): the token-level baseline (§5.1)  */
  DMOE_ROUTE_BLOCK = 1        /* Algorithm 1 (§4.2) per diffusion block               */
} dmoe_route_mode;

/* Shape and routing parameters of one MoE-layer forward (plain data, host memory).
 * Limits of this build: 1 <= k <= 16, k <= E <= 256, E % 8 == 0; d % 128 == 0,
 * block_top_k = 0 or k <= block_top_k <= min(E, 16);
 * 128 <= d <= 16384; I % 128 == 0 and I_s % 128 == 0 (I_s may be 0), I, I_s <= 8192;
 * 1 <= T <= 4096; block_size >= 1. */
typedef struct {
  int32_t d_model;        /* d                                                       */
  int32_t n_experts;      /* |E| routed experts                                      */
  int32_t top_k;          /* k experts per token                                     */
  int32_t d_ff;           /* I, intermediate size of a routed SwiGLU expert          */
  int32_t d_ff_shared;    /* I_s of the shared expert, 0 = no shared expert          */
  int32_t block_size;     /* B, tokens per diffusion block                           */
  int32_t n_blocks;       /* blocks in this forward (one per sequence), T = n_blocks*B */
  int32_t mode;           /* dmoe_route_mode                                         */
  float top_p;            /* block mode: coreset threshold p. The coreset is the
                             shortest prefix of the experts sorted by normalised block
                             score whose running sum reaches p, extended to at least
                             block_top_k entries; p <= 0 gives exactly block_top_k (block
                             top-k), p >= 1 every
                             expert with a nonzero block score. Ignored in token mode. */
  int32_t block_top_k;    /* block mode: the k of Algorithm 1's TopKMask (the per-token
                             contribution to the block score) and of the coreset floor;
                             0 means top_k. A value above top_k keeps Algorithm 1's
                             coreset but lets every token use only the top_k best members
                             of it by its own score (the "fewer experts for each token"
                             direction of App. A); then top_k <= block_top_k <= min(E, 16).
                             Ignored in token mode. */
} dmoe_layer_desc;

/* Bytes of device workspace needed by every call below for this shape (host only; no
 * CUDA call). One workspace sized for the desc serves all calls on that desc. A workspace
 * must be zero-filled once before its first use; every call leaves it reusable. */
dmoe_status dmoe_workspace_size(const dmoe_layer_desc* desc, size_t* bytes /* host */);

/* Router and routing — §4.2 (s_i = Router(t_i); S_block = aggregation of the s_i;
 * C = Top-P(S~_block, p)) and Algorithm 1 (TopKMask, sum, Normalize, TopP,
 * MaskOutside, TopK), or token-level TopK in DMOE_ROUTE_TOKEN mode.
 *   x        bf16 [T, d]     token representations t_i (tokens of block b are rows
 *                            b*B .. b*B+B-1)
 *   w_r      fp32 [d, E]     router weight
 *   bias     fp32 [E]        router bias, or NULL for none
 *   topk_idx int32 [T, k]    out: R_i, expert ids by descending s_i (ties: lower id)
 *   topk_gate fp32 [T, k]    out: g_ij = s_i[R_ij] / sum_j s_i[R_ij]
 *   coreset  int32 [n_blocks, E] out or NULL: coreset ids of each block sorted by
 *                            normalised block score (ties: lower id), -1 past its size
 *   coreset_size int32 [n_blocks] out or NULL (in token mode the coreset rows are all -1
 *                            and the sizes 0)
 *   probs    fp32 [T, E]     out or NULL: the router scores s_i (softmax of the logits)
 * The router runs in fp32: logits = x W_r + b, softmax, all decisions on fp32 values. */
dmoe_status dmoe_router(const dmoe_layer_desc* desc, const void* x, const float* w_r,
                        const float* bias, int32_t* topk_idx, float* topk_gate,
                        int32_t* coreset, int32_t* coreset_size, float* probs,
                        void* workspace, size_t workspace_bytes, void* stream);

/* Router weight preparation (optional, once per W_r, like a weight layout conversion at
 * load time). Forwards of more than 64 tokens compute the fp32 router logits of §4.2 on
 * the tensor cores from an exact three-part bf16 split of W_r (hi + mid + lo = w to 2^-27),
 * which every router or layer call otherwise writes into the workspace first. This call
 * writes that split into the workspace and remembers on the host that the workspace holds
 * it for this w_r pointer; router and layer calls on the workspace with the same w_r then
 * skip the split. Call it again after changing W_r in place. A call with another w_r
 * splits that one, and the workspace then no longer holds this one's split. A no-op for
 * shapes whose router reads W_r directly.
 *   w_r      fp32 [d, E]     device, router weight (read)
 *   workspace                as for dmoe_router; stream: the CUDA stream of the split */
dmoe_status dmoe_router_prepare(const dmoe_layer_desc* desc, const float* w_r, void* workspace,
                                size_t workspace_bytes, void* stream);

/* Dispatch: the unique experts of one forward (the "unique expert count" of §3 and §5)
 * and the expert -> (token, slot) lists, computed on the device without a host round-trip.
 *   topk_idx   int32 [T, k]   routed experts (e.g. from dmoe_router); every id must be in
 *                             [0, E) and distinct within a token, else the device flag is
 *                             set (DMOE_ERR_DEVICE) and the outputs are unspecified
 *   n_unique   int32 [1]      out: U
 *   unique_ids int32 [E]      out: the U ids ascending, then -1
 *   offsets    int32 [E + 1]  out: offsets[u] .. offsets[u+1] is the slice of `rows` of
 *                             the u-th unique expert; offsets[u] = T*k for u >= U
 *   rows       int32 [T * k]  out: t*k + slot, ordered by (expert, token)
 *   pos        int32 [T * k]  out: pos[t*k + slot] = r such that rows[r] = t*k + slot */
dmoe_status dmoe_dispatch(const dmoe_layer_desc* desc, const int32_t* topk_idx,
                          int32_t* n_unique, int32_t* unique_ids, int32_t* offsets,
                          int32_t* rows, int32_t* pos,
                          void* workspace, size_t workspace_bytes, void* stream);

/* Expert execution ("MoE includes routing and expert execution", §3): for every token t,
 *   y_t = sum_j g_tj * W_down[R_tj] (silu(W_gate[R_tj] x_t) * (W_up[R_tj] x_t))
 *         + W_sd (silu(W_sg x_t) * (W_su x_t))            (shared expert, if I_s > 0)
 * as a grouped GEMM over the unique experts only: each unique expert's bf16 weights are
 * streamed from HBM once per forward (tcgen05 MMA, fp32 accumulation; the SwiGLU
 * intermediate is rounded to bf16; the combine is fp32, y is rounded to bf16).
 *   x          bf16 [T, d]
 *   w_gate     bf16 [E, I, d];  w_up bf16 [E, I, d];  w_down bf16 [E, d, I]
 *   ws_gate    bf16 [I_s, d];   ws_up bf16 [I_s, d];  ws_down bf16 [d, I_s]  (NULL if I_s == 0)
 *   topk_gate  fp32 [T, k]      gates g (as from dmoe_router)
 *   n_unique, unique_ids, offsets, rows, pos: as written by dmoe_dispatch
 *   y          bf16 [T, d]      out */
dmoe_status dmoe_moe_forward(const dmoe_layer_desc* desc, const void* x,
                             const void* w_gate, const void* w_up, const void* w_down,
                             const void* ws_gate, const void* ws_up, const void* ws_down,
                             const float* topk_gate, const int32_t* n_unique,
                             const int32_t* unique_ids, const int32_t* offsets,
                             const int32_t* rows, const int32_t* pos, void* y,
                             void* workspace, size_t workspace_bytes, void* stream);

/* The whole layer: dmoe_router + dmoe_dispatch + dmoe_moe_forward on `stream` with every
 * intermediate in the workspace and no host round-trip. The optional outputs (NULL to
 * skip) receive the routing: topk_idx [T,k], topk_gate [T,k], n_unique [1],
 * unique_ids [E]. Arguments otherwise as above. */
dmoe_status dmoe_layer_forward(const dmoe_layer_desc* desc, const void* x,
                               const float* w_r, const float* bias,
                               const void* w_gate, const void* w_up, const void* w_down,
                               const void* ws_gate, const void* ws_up, const void* ws_down,
                               void* y, int32_t* topk_idx, float* topk_gate,
                               int32_t* n_unique, int32_t* unique_ids,
                               void* workspace, size_t workspace_bytes, void* stream);

/* Number of kernel launches one dmoe_layer_forward call makes for `desc` (the decode-size
 * path: routing 1, experts 1, combine 1), counting the split of W_r where the router uses
 * it: a call on a workspace that dmoe_router_prepare prepared for its W_r makes one launch
 * fewer then. Returns -1 for an invalid or unsupported desc. Host-only, no GPU needed. */
int32_t dmoe_layer_forward_launches(const dmoe_layer_desc* desc);

/* Kernels of the forward, for dmoe_set_profile_events. */
typedef enum {
  DMOE_KERNEL_ROUTER = 0,     /* router logits, softmax/top-k and Algorithm 1 kernels */
  DMOE_KERNEL_DISPATCH = 1,   /* unique experts and expert -> token lists            */
  DMOE_KERNEL_GATHER = 2,     /* x rows in dispatch order                            */
  DMOE_KERNEL_EXPERTS = 3,    /* grouped gate/up GEMM + SwiGLU and down GEMM         */
  DMOE_KERNEL_COMBINE = 4,    /* gate-weighted sum over slots + shared expert -> y   */
  DMOE_KERNEL_COUNT = 5
} dmoe_kernel_id;

/* Profiling aid, not part of the method: while set, every launch of `kernel` made by a
 * call on this host thread records `ev_begin` just before it and `ev_end` just after it on
 * the call's stream (cudaEvent_t handles passed as void*, created with timing enabled;
 * recorded as external events, so they also work inside a CUDA-graph capture). The expert
 * launch is then made without programmatic dependent launch: it starts once the launch
 * before it has ended, so that the events bracket its own execution (not an early start
 * spent waiting for the routing). Passing NULL for both clears the setting. Returns
 * DMOE_ERR_INVALID_ARG for an unknown kernel. */
dmoe_status dmoe_set_profile_events(int32_t kernel, void* ev_begin, void* ev_end);

/* dmoe_router for callers that cannot allocate device memory. The paper has no
 * counterpart: this is a deployment convenience. Some callers may not call cudaMalloc (or
 * any allocator) at all: code running inside an allocator or memory-pool callback, a host
 * framework or plugin that owns every device allocation itself, or a latency-critical loop
 * that must never enter the allocator. This call takes no workspace: its scratch (partial
 * logits, scores, the fault record) lives in a fixed 4 MiB array in the library's own
 * device memory, which every GPU that loads the library holds until the process exits.
 * The caller still passes every input and output, exactly as for dmoe_router, and the
 * results are the same.
 *  - The call allocates nothing and frees nothing (no cudaMalloc/cudaFree, no allocating
 *    library routine). The scratch it needs is the leading part of the workspace layout,
 *    each region rounded up to 256 bytes: the fault record and the stage counters (1.3 KB),
 *    the partial logits (T*E fp32, times the router's split of d when d is not a multiple
 *    of 256), the scores and the masked scores (T*E fp32 each) and the top-k candidates
 *    (T * ceil(E/32) * k_mask * 8 bytes, k_mask = block_top_k or k). With E = 256 and
 *    k = 8 that is about 3.6 KB per token: at most 1169 tokens. Larger shapes return
 *    DMOE_ERR_UNSUPPORTED, with the sizes in dmoe_last_error_message().
 *  - The first call on each device looks up the array's device address (with that device
 *    current) and caches it; make that first call before any CUDA-graph stream capture.
 *    A device reset (cudaDeviceReset) reloads the library's device code at a new address:
 *    do not call this entry point on that device again in the same process.
 *  - All calls share the one array and it keeps the previous call's contents: the stage
 *    counters return to zero at the end of every call, and everything else a call reads it
 *    has written first. A fault a kernel records (a bounded wait that ran out) stays in the
 *    array until dmoe_router_no_alloc_device_error reads and clears it.
 *    Calls whose executions overlap on the GPU (two streams, or two host threads) race on
 *    the array and give wrong results: serialise them.
 * Arguments, layouts and errors otherwise as for dmoe_router. */
dmoe_status dmoe_router_no_alloc(const dmoe_layer_desc* desc, const void* x, const float* w_r,
                                 const float* bias, int32_t* topk_idx, float* topk_gate,
                                 int32_t* coreset, int32_t* coreset_size, float* probs,
                                 void* stream);

/* The fault record of dmoe_router_no_alloc on the current device: synchronises `stream`,
 * then reads and clears it. Returns and fills `info` (host, 4 int32, or NULL) as
 * dmoe_get_device_error does for a workspace. */
dmoe_status dmoe_router_no_alloc_device_error(void* stream, int32_t* info);

/* Device address and size (host outputs) of the static scratch array of
 * dmoe_router_no_alloc on the current device, looked up as that call does. For inspection
 * and tests: the array starts with the same fault record as a workspace, so any call given
 * it as a workspace shares it with dmoe_router_no_alloc (and the serialisation rule above
 * applies). */
dmoe_status dmoe_no_alloc_scratch(void** device_ptr, size_t* bytes);

/* Synchronises `stream`, then reads and clears the fault code the kernels recorded in
 * `workspace`. Returns DMOE_OK if none, DMOE_ERR_TIMEOUT for a bounded wait that ran out,
 * DMOE_ERR_DEVICE for any other recorded fault, DMOE_ERR_CUDA if the sync failed.
 * `info` (host, 4 int32, or NULL) receives {code, where, value, 0}. */
dmoe_status dmoe_get_device_error(void* workspace, void* stream, int32_t* info);

/* Diagnostic, not part of the method: makes a bounded wait of the expert launch run out,
 * so that the timeout path can be tested without any fault on the GPU. While `hold` is
 * nonzero, every down tile of the decode-size expert launch (at most 64 tokens) of a call
 * on `workspace` waits for `hold` more gate/up tiles of its group than exist; its wait runs
 * out after 1 s, the launch records DMOE_ERR_TIMEOUT in the workspace and unwinds (no trap),
 * and that call's outputs are unspecified. dmoe_get_device_error, which reads the fault,
 * clears the hold with it; a hold of 0 clears it too. The hold is the last 32-bit word of
 * the fault record at the head of the workspace. Synchronises `stream`, then writes it with
 * a blocking copy. DMOE_ERR_INVALID_ARG for a null workspace or a negative hold. */
dmoe_status dmoe_set_debug_hold(void* workspace, int32_t hold, void* stream);

/* Static description of a status code (host). */
const char* dmoe_status_string(dmoe_status status);

/* Text of the last CUDA error seen by a call on this host thread ("" if none). */
const char* dmoe_last_error_message(void);

/* DMOE_ABI_VERSION of the loaded library. */
int32_t dmoe_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* DMOE_H_ */
