// Router and block-level routing kernels (§4.2 and Algorithm 1 of arXiv 2605.30876).
//
//   router_logits_kernel   logits = x W_r, fp32 FFMA, split over d into partial sums
//   router_softmax_kernel  sum the partials in split order, + b, softmax, per-token TopK;
//                          token mode: gates; block mode: TopKMask(s_i, k)
//   block_route_kernel     one CTA per diffusion block: S_block = sum of the masked scores,
//                          Normalize (L1), sort, Top-P with the k floor, then MaskOutside +
//                          TopK per token and the gate renormalisation
//
// Every reduction runs in a fixed order, so the routing is identical from run to run.
#include <math.h>

#include "block_reduce.cuh"
#include "dmoe_internal.cuh"

namespace dmoe {
namespace {

constexpr int kRtTok = 32;   // tokens per logits tile
constexpr int kRtExp = 64;   // experts per logits tile
constexpr int kRtK = 32;     // d per smem step

// part[split, t, e] = sum over d in split's chunk of x[t, d] * w_r[d, e]  (fp32, d ascending)
__global__ void __launch_bounds__(256)
router_logits_kernel(const __nv_bfloat16* __restrict__ x, const float* __restrict__ w_r,
                     float* __restrict__ part, int T, int d, int E, int dchunk) {
  __shared__ float xs[kRtK][kRtTok + 1];
  __shared__ __align__(16) float wsm[kRtK][kRtExp];
  const int e0 = blockIdx.x * kRtExp, t0 = blockIdx.y * kRtTok, split = blockIdx.z;
  const int dbeg = split * dchunk, dend = dbeg + dchunk;
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
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

// One CTA per token, thread e = expert e (E <= 256).
__global__ void __launch_bounds__(256)
router_softmax_kernel(const float* __restrict__ part, int splits, const float* __restrict__ bias,
                      float* __restrict__ probs, float* __restrict__ probs_hat,
                      int32_t* __restrict__ topk_idx, float* __restrict__ topk_gate,
                      int T, int E, int k, int mode) {
  __shared__ float sv[kMaxExperts];
  __shared__ float topv[kMaxTopK];
  __shared__ float scratch[32];
  const int t = blockIdx.x, e = threadIdx.x;
  float logit = -INFINITY;
  if (e < E) {
    float acc = 0.f;
    for (int s = 0; s < splits; ++s) acc += part[((size_t)s * T + t) * E + e];
    if (bias != nullptr) acc += bias[e];
    logit = acc;
  }
  const float mx = block_max(logit, scratch);
  const float ex = (e < E) ? expf(logit - mx) : 0.f;
  const float sum = block_sum(ex, scratch);
  const float s = ex / sum;
  if (e < E) {
    probs[(size_t)t * E + e] = s;
    sv[e] = s;
  }
  __syncthreads();
  int rank = 0;
  if (e < E) {
    for (int j = 0; j < E; ++j) {
      const float v = sv[j];
      rank += (v > s) || (v == s && j < e);
    }
  }
  const bool sel = (e < E) && rank < k;
  if (mode == DMOE_ROUTE_BLOCK) {
    if (e < E) probs_hat[(size_t)t * E + e] = sel ? s : 0.f;
  } else {
    if (sel) topv[rank] = s;
    __syncthreads();
    if (sel) {
      float tot = 0.f;
      for (int j = 0; j < k; ++j) tot += topv[j];
      topk_idx[(size_t)t * k + rank] = e;
      topk_gate[(size_t)t * k + rank] = s / tot;
    }
  }
}

// One CTA per diffusion block (Algorithm 1), 256 threads.
__global__ void __launch_bounds__(256)
block_route_kernel(const float* __restrict__ probs, const float* __restrict__ probs_hat,
                   int E, int k, int B, float top_p,
                   int32_t* __restrict__ topk_idx, float* __restrict__ topk_gate,
                   int32_t* __restrict__ coreset, int32_t* __restrict__ coreset_size) {
  __shared__ float st_s[kMaxExperts];
  __shared__ float sorted_v[kMaxExperts];
  __shared__ int order[kMaxExperts];
  __shared__ float wv[8][kMaxExperts];
  __shared__ float wsel_v[8][kMaxTopK];
  __shared__ int wsel_e[8][kMaxTopK];
  __shared__ float fscr[32];
  __shared__ int iscr[32];
  const int b = blockIdx.x, tid = threadIdx.x;
  const int t0 = b * B;
  const bool live = tid < E;

  // S_block = sum over the block's tokens (ascending) of TopKMask(s_i, k)
  float S = 0.f;
  if (live)
    for (int i = 0; i < B; ++i) S += probs_hat[(size_t)(t0 + i) * E + tid];
  // Normalize: L1
  const float tot = block_sum(S, fscr);
  const float st = live ? S / tot : 0.f;
  if (live) st_s[tid] = st;
  __syncthreads();
  // sort descending, ties -> lower expert id
  if (live) {
    int rank = 0;
    for (int j = 0; j < E; ++j) {
      const float v = st_s[j];
      rank += (v > st) || (v == st && j < tid);
    }
    order[rank] = tid;
    sorted_v[rank] = st;
  }
  __syncthreads();
  // Top-P over the sorted order: running sum, thread r = sorted position r
  const float v = live ? sorted_v[tid] : 0.f;
  const float cum = block_inclusive_scan(v, fscr);
  const int nnz = block_sum_i((live && v > 0.f) ? 1 : 0, iscr);
  int m;
  if (top_p >= 1.f) {
    m = nnz;
  } else {
    const int first = block_min_i((live && cum >= top_p) ? tid : 0x7fffffff, iscr);
    m = (first == 0x7fffffff) ? nnz : first + 1;
    m = min(m, nnz);
  }
  const int size = max(m, k);
  if (coreset != nullptr && live) coreset[(size_t)b * E + tid] = (tid < size) ? order[tid] : -1;
  if (coreset_size != nullptr && tid == 0) coreset_size[b] = size;

  // MaskOutside + TopK for every token of the block (one warp per token)
  const int warp = tid >> 5, lane = tid & 31;
  for (int i = warp; i < B; i += 8) {
    const int t = t0 + i;
    for (int c = lane; c < size; c += 32) wv[warp][c] = probs[(size_t)t * E + order[c]];
    __syncwarp();
    for (int c = lane; c < size; c += 32) {
      const float cv = wv[warp][c];
      const int ce = order[c];
      int r = 0;
      for (int j = 0; j < size; ++j) {
        const float vj = wv[warp][j];
        r += (vj > cv) || (vj == cv && order[j] < ce);
      }
      if (r < k) {
        wsel_v[warp][r] = cv;
        wsel_e[warp][r] = ce;
      }
    }
    __syncwarp();
    if (lane < k) {
      float g = 0.f;
      for (int j = 0; j < k; ++j) g += wsel_v[warp][j];
      topk_idx[(size_t)t * k + lane] = wsel_e[warp][lane];
      topk_gate[(size_t)t * k + lane] = wsel_v[warp][lane] / g;
    }
    __syncwarp();
  }
}

}  // namespace

cudaError_t launch_router(const RouterArgs& a, cudaStream_t s) {
  const int dchunk = a.d / a.splits;
  prof_begin(DMOE_KERNEL_ROUTER, s);
  dim3 g1((a.E + kRtExp - 1) / kRtExp, (a.T + kRtTok - 1) / kRtTok, a.splits);
  router_logits_kernel<<<g1, 256, 0, s>>>(a.x, a.w_r, a.logits_part, a.T, a.d, a.E, dchunk);
  router_softmax_kernel<<<a.T, 256, 0, s>>>(a.logits_part, a.splits, a.bias, a.probs,
                                            a.probs_hat, a.topk_idx, a.topk_gate, a.T, a.E,
                                            a.k, a.mode);
  if (a.mode == DMOE_ROUTE_BLOCK) {
    block_route_kernel<<<a.n_blocks, 256, 0, s>>>(a.probs, a.probs_hat, a.E, a.k, a.B,
                                                  a.top_p, a.topk_idx, a.topk_gate,
                                                  a.coreset, a.coreset_size);
  } else {
    cudaError_t e = cudaSuccess;
    if (a.coreset != nullptr)
      e = cudaMemsetAsync(a.coreset, 0xff, sizeof(int32_t) * (size_t)a.n_blocks * a.E, s);
    if (e == cudaSuccess && a.coreset_size != nullptr)
      e = cudaMemsetAsync(a.coreset_size, 0, sizeof(int32_t) * (size_t)a.n_blocks, s);
    if (e != cudaSuccess) return e;
  }
  prof_end(DMOE_KERNEL_ROUTER, s);
  return cudaGetLastError();
}

}  // namespace dmoe
