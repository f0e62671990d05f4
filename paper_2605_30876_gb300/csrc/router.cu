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
  pdl_launch_dependents();
  pdl_wait();
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

// Logits of 8 tokens x 16 experts over the full d, for small token counts (no partial
// sums): x and W_r slices are staged in shared memory by cp.async in 512-wide d chunks
// (double-buffered); warp w reduces d sub-range w of every chunk, lane l owns token l/4 and
// experts 4*(l%4)..+3; the 8 warp partials are added in warp order at the end.
constexpr int kSmTok = 8, kSmExp = 16, kSmChunk = 512, kSmXPad = 8;

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(n)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_le1() {
  asm volatile("cp.async.wait_group 1;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}

__global__ void __launch_bounds__(256)
router_logits_small_kernel(const __nv_bfloat16* __restrict__ x, const float* __restrict__ w_r,
                           float* __restrict__ logits, int T, int d, int E) {
  extern __shared__ __align__(16) uint8_t lsm[];
  // per buffer: W [kSmChunk][kSmExp] fp32, then x [kSmTok][kSmChunk + kSmXPad] bf16
  constexpr int kWBytes = kSmChunk * kSmExp * 4;
  constexpr int kXStride = kSmChunk + kSmXPad;
  constexpr int kBufBytes = kWBytes + kSmTok * kXStride * 2;
  const int e0 = blockIdx.x * kSmExp, t0 = blockIdx.y * kSmTok;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tl = lane >> 2, el = (lane & 3) * 4;
  const int nchunks = d / kSmChunk;
  pdl_launch_dependents();
  pdl_wait();

  auto stage = [&](int c, int buf) {
    float* ws = reinterpret_cast<float*>(lsm + buf * kBufBytes);
    __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(lsm + buf * kBufBytes + kWBytes);
    const int dbase = c * kSmChunk;
    // W: kSmChunk rows x 64 B = 4 x 16 B per row
    for (int i = tid; i < kSmChunk * 4; i += 256) {
      const int r = i >> 2, q = i & 3;
      const int e = e0 + q * 4;
      const bool ok = e < E;
      cp_async16(ws + r * kSmExp + q * 4, w_r + (size_t)(dbase + r) * E + (ok ? e : 0), ok);
    }
    // x: kSmTok rows x kSmChunk bf16 = 64 x 16 B per row
    for (int i = tid; i < kSmTok * (kSmChunk / 8); i += 256) {
      const int r = i / (kSmChunk / 8), q = i % (kSmChunk / 8);
      const int t = t0 + r;
      const bool ok = t < T;
      cp_async16(xs + r * kXStride + q * 8, x + (size_t)(ok ? t : 0) * d + dbase + q * 8, ok);
    }
    cp_async_commit();
  };

  float acc0 = 0.f, acc1 = 0.f, acc2 = 0.f, acc3 = 0.f;
  stage(0, 0);
  for (int c = 0; c < nchunks; ++c) {
    const int buf = c & 1;
    if (c + 1 < nchunks) {
      stage(c + 1, buf ^ 1);
      cp_async_wait_le1();
    } else {
      cp_async_wait_all();
    }
    __syncthreads();
    const float* ws = reinterpret_cast<const float*>(lsm + buf * kBufBytes);
    const __nv_bfloat16* xs =
        reinterpret_cast<const __nv_bfloat16*>(lsm + buf * kBufBytes + kWBytes);
    const int dl0 = warp * (kSmChunk / 8);
#pragma unroll 8
    for (int j = 0; j < kSmChunk / 8; ++j) {
      const int dl = dl0 + j;
      const float xv = __bfloat162float(xs[tl * kXStride + dl]);
      const float4 w = *reinterpret_cast<const float4*>(ws + dl * kSmExp + el);
      acc0 = fmaf(xv, w.x, acc0);
      acc1 = fmaf(xv, w.y, acc1);
      acc2 = fmaf(xv, w.z, acc2);
      acc3 = fmaf(xv, w.w, acc3);
    }
    __syncthreads();
  }
  // cross-warp sum in warp order
  float* red = reinterpret_cast<float*>(lsm);  // [8 warps][kSmTok][kSmExp]
  red[(warp * kSmTok + tl) * kSmExp + el + 0] = acc0;
  red[(warp * kSmTok + tl) * kSmExp + el + 1] = acc1;
  red[(warp * kSmTok + tl) * kSmExp + el + 2] = acc2;
  red[(warp * kSmTok + tl) * kSmExp + el + 3] = acc3;
  __syncthreads();
  if (tid < kSmTok * kSmExp) {
    const int t = tid / kSmExp, e = tid % kSmExp;
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) v += red[(w * kSmTok + t) * kSmExp + e];
    if (t0 + t < T && e0 + e < E) logits[(size_t)(t0 + t) * E + e0 + e] = v;
  }
}

size_t router_small_smem() {
  return 2 * ((size_t)kSmChunk * kSmExp * 4 + (size_t)kSmTok * (kSmChunk + kSmXPad) * 2);
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
  pdl_launch_dependents();
  pdl_wait();
  float logit = -INFINITY;
  if (e < E) {
    float acc = 0.f;
#pragma unroll 4
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
  pdl_launch_dependents();
  pdl_wait();

  // S_block = sum over the block's tokens (ascending) of TopKMask(s_i, k)
  float S = 0.f;
  if (live) {
#pragma unroll 8
    for (int i = 0; i < B; ++i) S += probs_hat[(size_t)(t0 + i) * E + tid];
  }
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
  prof_begin(DMOE_KERNEL_ROUTER, s);
  if (a.splits == 0) {
    // small token count: full-d tiles of 8 tokens x 16 experts, logits written directly
    static int attr_dev_mask = 0;
    int dev = 0;
    cudaGetDevice(&dev);
    const size_t smem = router_small_smem();
    if (dev < 31 && !(attr_dev_mask & (1 << dev))) {
      cudaError_t e = cudaFuncSetAttribute(router_logits_small_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)smem);
      if (e != cudaSuccess) return e;
      attr_dev_mask |= 1 << dev;
    }
    dim3 g0((a.E + kSmExp - 1) / kSmExp, (a.T + kSmTok - 1) / kSmTok);
    router_logits_small_kernel<<<g0, 256, smem, s>>>(a.x, a.w_r, a.logits_part, a.T, a.d, a.E);
  } else {
    const int dchunk = a.d / a.splits;
    dim3 g1((a.E + kRtExp - 1) / kRtExp, (a.T + kRtTok - 1) / kRtTok, a.splits);
    router_logits_kernel<<<g1, 256, 0, s>>>(a.x, a.w_r, a.logits_part, a.T, a.d, a.E, dchunk);
  }
  const int nsum = a.splits == 0 ? 1 : a.splits;
  cudaError_t le = launch_ex(router_softmax_kernel, dim3(a.T), dim3(256), 0, s, true,
                             a.logits_part, nsum, a.bias, a.probs, a.probs_hat, a.topk_idx,
                             a.topk_gate, a.T, a.E, a.k, a.mode);
  if (le != cudaSuccess) return le;
  if (a.mode == DMOE_ROUTE_BLOCK) {
    le = launch_ex(block_route_kernel, dim3(a.n_blocks), dim3(256), 0, s, true, a.probs,
                   a.probs_hat, a.E, a.k, a.B, a.top_p, a.topk_idx, a.topk_gate, a.coreset,
                   a.coreset_size);
    if (le != cudaSuccess) return le;
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
