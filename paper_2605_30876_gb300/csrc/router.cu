// Router and block-level routing kernels (§4.2 and Algorithm 1 of arXiv 2605.30876).
//
// Decode-sized batches take the single cluster launch of route_cluster.cu. Larger batches
// use one kernel per step:
//   logits                 the split of W_r and tcgen05 tiles of 128 tokens x E experts over
//                          slices of d (router_logits_tc.cu); where its shape rules do not
//                          hold, the
//                          logits stage of the cluster launch over 64-token tiles (mma.sync,
//                          the same exact split of W_r), else router_logits_kernel (fp32
//                          FFMA, 32 x 64 tiles, optional split over d)
//   router_softmax_kernel  one warp per token: sum the partials in split order, + b,
//                          softmax, top-k
//   block_route_kernel     one CTA per diffusion block: Algorithm 1 (routing_device.cuh)
//
// Every reduction runs in a fixed order, so the routing is identical from run to run.
#include <math.h>

#ifdef DMOE_TRACE
#include <stdint.h>
// Debug builds: per-CTA phase stamps of the block routing kernel (%globaltimer, ns)
__device__ uint64_t g_brtrace[64 * 32];
#define DMOE_STAMP(st)                                                               \
  do {                                                                               \
    if (threadIdx.x == 0 && blockIdx.x < 64) {                                       \
      uint64_t t_;                                                                   \
      asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                         \
      g_brtrace[blockIdx.x * 32 + (st)] = t_;                                        \
    }                                                                                \
  } while (0)
#endif
#include "block_reduce.cuh"
#include "dmoe_internal.cuh"
#include "routing_device.cuh"
#include "trace_log.cuh"

namespace dmoe {
namespace {

constexpr int kRtTok = 32;   // tokens per logits tile (tiled kernel)
constexpr int kRtExp = 64;   // experts per logits tile
constexpr int kRtK = 32;     // d per smem step

// part[split, t, e] = sum over d in split's chunk of x[t, d] * w_r[d, e]  (fp32, d ascending)
__global__ void __launch_bounds__(256)
router_logits_kernel(const __nv_bfloat16* __restrict__ x, const float* __restrict__ w_r,
                     float* __restrict__ part, int T, int d, int E, int dchunk, L2Prefetch pf) {
  __shared__ float xs[kRtK][kRtTok + 1];
  __shared__ __align__(16) float wsm[kRtK][kRtExp];
  const int e0 = blockIdx.x * kRtExp, t0 = blockIdx.y * kRtTok, split = blockIdx.z;
  const int dbeg = split * dchunk, dend = dbeg + dchunk;
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  pdl_launch_dependents();
  pdl_wait();
  if (tid == 0)
    issue_shared_prefetch(pf, (blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x,
                          gridDim.x * gridDim.y * gridDim.z);
  float acc[2][4];
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int k0 = dbeg; k0 < dend; k0 += kRtK) {
    {  // x tile: 32 tokens x 32 d, 4 bf16 per thread, stored transposed
      const int tt = tid >> 3, kk = (tid & 7) * 4, t = t0 + tt;
      float v0 = 0.f, v1 = 0.f, v2 = 0.f, v3 = 0.f;
      if (t < T) {
        const uint2 raw = *reinterpret_cast<const uint2*>(x + (size_t)t * d + k0 + kk);
        const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&raw.x);
        const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&raw.y);
        v0 = __low2float(a); v1 = __high2float(a); v2 = __low2float(b); v3 = __high2float(b);
      }
      xs[kk + 0][tt] = v0; xs[kk + 1][tt] = v1; xs[kk + 2][tt] = v2; xs[kk + 3][tt] = v3;
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {  // W_r tile: 32 d x 64 experts
      const int kk = (tid >> 4) + h * 16, e = e0 + (tid & 15) * 4;
      float4 w = make_float4(0.f, 0.f, 0.f, 0.f);
      if (e < E) w = *reinterpret_cast<const float4*>(w_r + (size_t)(k0 + kk) * E + e);
      *reinterpret_cast<float4*>(&wsm[kk][(tid & 15) * 4]) = w;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kRtK; ++kk) {
      const float a0 = xs[kk][ty * 2], a1 = xs[kk][ty * 2 + 1];
      const float4 w = *reinterpret_cast<const float4*>(&wsm[kk][tx * 4]);
      acc[0][0] = fmaf(a0, w.x, acc[0][0]); acc[0][1] = fmaf(a0, w.y, acc[0][1]);
      acc[0][2] = fmaf(a0, w.z, acc[0][2]); acc[0][3] = fmaf(a0, w.w, acc[0][3]);
      acc[1][0] = fmaf(a1, w.x, acc[1][0]); acc[1][1] = fmaf(a1, w.y, acc[1][1]);
      acc[1][2] = fmaf(a1, w.z, acc[1][2]); acc[1][3] = fmaf(a1, w.w, acc[1][3]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int t = t0 + ty * 2 + i, e = e0 + tx * 4;
    if (t < T && e < E)
      *reinterpret_cast<float4*>(part + ((size_t)split * T + t) * E + e) =
          make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
  }
}

// Eight tokens per CTA, one warp each. k is the TopKMask width in block mode and the
// routed k in token mode.
__global__ void __launch_bounds__(256)
router_softmax_kernel(const float* __restrict__ part, int splits, const float* __restrict__ bias,
                      float* __restrict__ probs, float* __restrict__ probs_hat,
                      int32_t* __restrict__ topk_idx, float* __restrict__ topk_gate,
                      int T, int E, int k, int mode) {
  pdl_wait();
  pdl_launch_dependents();   // after the wait: a waiting dependent would share the SMs
  KLOG(5, 0);
  const int t = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (t >= T) return;
  token_route_warp(part + (size_t)t * E, splits, (size_t)T * E, bias, E, k, mode,
                   probs + (size_t)t * E, probs_hat + (size_t)t * E, topk_idx + (size_t)t * k,
                   topk_gate + (size_t)t * k);
  KLOG(5, 1);
}

__global__ void __launch_bounds__(256)
block_route_kernel(const float* __restrict__ probs, const float* __restrict__ probs_hat,
                   int E, int kb, int k, int B, float top_p,
                   int32_t* __restrict__ topk_idx, float* __restrict__ topk_gate,
                   int32_t* __restrict__ coreset, int32_t* __restrict__ coreset_size,
                   uint32_t* __restrict__ spec, int32_t* __restrict__ ready, int n_ready) {
  pdl_wait();
  if (spec != nullptr) {
    // the expert launch that follows polls this block's coreset words and counts on its
    // gate/up tile counters being zero: both are cleared, and made visible, before this CTA
    // lets it start (the previous call has ended: the wait above)
    if ((int)threadIdx.x < spec_words(k)) spec[(size_t)blockIdx.x * spec_words(k) + threadIdx.x] = 0u;
    if (blockIdx.x == 0)
      for (int i = threadIdx.x; i < n_ready; i += blockDim.x) ready[i] = 0;
    __threadfence();
    __syncthreads();
  }
  pdl_launch_dependents();   // after the wait: a waiting dependent would share the SMs
  KLOG(6, 0);
  DMOE_STAMP(0);
  block_route_cta(blockIdx.x, probs, probs_hat, E, kb, k, B, top_p, topk_idx, topk_gate, coreset,
                  coreset_size, spec);
  KLOG(6, 1);
}

}  // namespace

cudaError_t launch_router(const RouterArgs& a, const DispatchArgs* dsp, int32_t* tickets,
                          cudaStream_t s) {
  prof_begin(DMOE_KERNEL_ROUTER, s);
  cudaError_t e;
  if (route_cluster_ok(a.T, a.d, a.E)) {
    e = launch_route_cluster(a, dsp, tickets, s);
    if (e != cudaSuccess) return e;
  } else {
    // logits (+ bias): on tcgen05 when the shape allows it (after the split of W_r), else
    // on mma.sync in the cluster launch's logits stage, else the FFMA tiles with partial
    // sums over a split of d; then softmax and top-k
    const bool tc = a.w_parts != nullptr && a.tc_part != nullptr && a.tc_splits > 0 &&
                    router_tc_ok(a.T, a.d, a.E);
    const bool cl = !tc && route_cluster_logits_ok(a.d, a.E);
    if (tc) {
      e = launch_router_tc(a, a.tc_splits, s);
      if (e != cudaSuccess) return e;
    } else if (cl) {
      e = launch_logits_cluster(a, s);
      if (e != cudaSuccess) return e;
    } else {
      const int dchunk = a.d / a.splits;
      dim3 g1((a.E + kRtExp - 1) / kRtExp, (a.T + kRtTok - 1) / kRtTok, a.splits);
      router_logits_kernel<<<g1, 256, 0, s>>>(a.x, a.w_r, a.logits_part, a.T, a.d, a.E, dchunk,
                                              a.shared_pf);
    }
    // partial sums over slices of d (tc: tc_splits, FFMA: splits, + bias) or one [T, E]
    // array of logits with the bias in (cl)
    e = launch_ex(router_softmax_kernel, dim3((a.T + 7) / 8), dim3(256), 0, s, true,
                  tc ? a.tc_part : a.logits_part, tc ? a.tc_splits : (cl ? 1 : a.splits),
                  cl ? nullptr : a.bias,
                  a.probs, a.probs_hat, a.topk_idx, a.topk_gate, a.T, a.E, a.kb, a.mode);
    if (e != cudaSuccess) return e;
    if (a.mode == DMOE_ROUTE_BLOCK) {
      e = launch_ex(block_route_kernel, dim3(a.n_blocks), dim3(256), 0, s, true, a.probs,
                    a.probs_hat, a.E, a.kb, a.k, a.B, a.top_p, a.topk_idx, a.topk_gate, a.coreset,
                    a.coreset_size, a.spec_words, a.ready_clear, a.n_ready_clear);
      if (e != cudaSuccess) return e;
    } else {
      if (a.coreset != nullptr)
        e = cudaMemsetAsync(a.coreset, 0xff, sizeof(int32_t) * (size_t)a.n_blocks * a.E, s);
      if (e == cudaSuccess && a.coreset_size != nullptr)
        e = cudaMemsetAsync(a.coreset_size, 0, sizeof(int32_t) * (size_t)a.n_blocks, s);
      if (e != cudaSuccess) return e;
    }
    if (dsp != nullptr) {
      e = launch_dispatch(*dsp, s);
      if (e != cudaSuccess) return e;
    }
  }
  prof_end(DMOE_KERNEL_ROUTER, s);
  return cudaGetLastError();
}

}  // namespace dmoe

#ifdef DMOE_TRACE
DMOE_KLOG_EXPORT(dmoe_debug_klog_routerg)
extern "C" int dmoe_debug_brtrace(void* host) {
  return (int)cudaMemcpyFromSymbol(host, g_brtrace, sizeof(g_brtrace));
}
#endif
