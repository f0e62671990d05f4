// Router and block-level routing kernels (§4.2 and Algorithm 1 of arXiv 2605.30876).
//
// Decode-sized batches (T <= 128 tokens, d a multiple of 512) take one launch:
//   route_fused_kernel   every CTA computes a logits tile (8 tokens x 16 experts, full d,
//                        fp32 FFMA); the last CTA to finish (atomic ticket) then computes,
//                        for every token, the softmax and the top-k (token mode: the gates;
//                        block mode: TopKMask), runs Algorithm 1 for every block and, in the
//                        fused layer call, the dispatch of the forward.
// Larger batches use one kernel per step:
//   router_logits_kernel   logits = x W_r, fp32 FFMA, 32 x 64 tiles, optional split over d
//   router_softmax_kernel  one warp per token: sum the partials in split order, + b,
//                          softmax, top-k
//   block_route_kernel     one CTA per diffusion block: S_block = sum of the masked scores,
//                          Normalize (L1), sort, Top-P with the k floor, then MaskOutside +
//                          TopK per token and the gate renormalisation
//
// Every reduction runs in a fixed order, so the routing is identical from run to run.
#include <math.h>

#include "block_reduce.cuh"
#include "dispatch_impl.cuh"
#include "dmoe_internal.cuh"

namespace dmoe {
namespace {

constexpr int kRtTok = 32;   // tokens per logits tile (tiled kernel)
constexpr int kRtExp = 64;   // experts per logits tile
constexpr int kRtK = 32;     // d per smem step
constexpr int kSmTok = 8, kSmExp = 16, kSmChunk = 512, kSmXPad = 8, kSmBufs = 4;
constexpr int kFusedMaxTokens = 128;

__device__ __forceinline__ void issue_shared_prefetch(const L2Prefetch& pf, int cta, int nctas) {
  if (pf.bytes > 0) {  // start streaming the shared expert while the router runs
    const int per = (int)((pf.bytes + kPrefetchChunk - 1) / kPrefetchChunk);
    for (int c = cta; c < 3 * per; c += nctas) l2_prefetch_chunk(pf, nullptr, 1, c);
  }
}

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

// ---------------------------------------------------------------- small-T logits tile
__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(src), "r"(n)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
// waits until at most `n` (0..3) committed groups are still pending
__device__ __forceinline__ void cp_async_wait_n(int n) {
  switch (n) {
    case 0: asm volatile("cp.async.wait_group 0;" ::: "memory"); break;
    case 1: asm volatile("cp.async.wait_group 1;" ::: "memory"); break;
    case 2: asm volatile("cp.async.wait_group 2;" ::: "memory"); break;
    default: asm volatile("cp.async.wait_group 3;" ::: "memory"); break;
  }
}

constexpr int kSmWBytes = kSmChunk * kSmExp * 4;
constexpr int kSmXStride = kSmChunk + kSmXPad;
constexpr int kSmBufBytes = kSmWBytes + kSmTok * kSmXStride * 2;

// Logits of tokens t0..t0+7 x experts e0..e0+15 over the full d (no partial sums): x and W_r
// slices staged in shared memory by cp.async in 512-wide d chunks (a ring of four
// buffers, so up to four chunks are in flight); warp w reduces d sub-range w of every
// chunk, lane l owns token l/4 and experts 4*(l%4)..+3; the 8 warp partials are added in
// warp order. 256 threads; `lsm` holds kSmBufs * kSmBufBytes bytes.
__device__ void logits_tile_small(const __nv_bfloat16* __restrict__ x,
                                  const float* __restrict__ w_r, float* __restrict__ logits,
                                  int T, int d, int E, int e0, int t0, uint8_t* lsm) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tl = lane >> 2, el = (lane & 3) * 4;
  const int nchunks = d / kSmChunk;

  auto stage = [&](int c) {
    const int buf = c % kSmBufs;
    float* ws = reinterpret_cast<float*>(lsm + buf * kSmBufBytes);
    __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(lsm + buf * kSmBufBytes + kSmWBytes);
    const int dbase = c * kSmChunk;
    for (int i = tid; i < kSmChunk * 4; i += 256) {      // W: rows of 64 B = 4 x 16 B
      const int r = i >> 2, q = i & 3;
      const int e = e0 + q * 4;
      const bool ok = e < E;
      cp_async16(ws + r * kSmExp + q * 4, w_r + (size_t)(dbase + r) * E + (ok ? e : 0), ok);
    }
    for (int i = tid; i < kSmTok * (kSmChunk / 8); i += 256) {  // x: 64 x 16 B per row
      const int r = i / (kSmChunk / 8), q = i % (kSmChunk / 8);
      const int t = t0 + r;
      const bool ok = t < T;
      cp_async16(xs + r * kSmXStride + q * 8, x + (size_t)(ok ? t : 0) * d + dbase + q * 8, ok);
    }
    cp_async_commit();
  };

  float acc0 = 0.f, acc1 = 0.f, acc2 = 0.f, acc3 = 0.f;
  const int pre = nchunks < kSmBufs ? nchunks : kSmBufs;
  for (int c = 0; c < pre; ++c) stage(c);
  for (int c = 0; c < nchunks; ++c) {
    const int ahead = (nchunks - 1 - c) < (kSmBufs - 1) ? (nchunks - 1 - c) : (kSmBufs - 1);
    cp_async_wait_n(ahead);
    __syncthreads();
    const int buf = c % kSmBufs;
    const float* ws = reinterpret_cast<const float*>(lsm + buf * kSmBufBytes);
    const __nv_bfloat16* xs =
        reinterpret_cast<const __nv_bfloat16*>(lsm + buf * kSmBufBytes + kSmWBytes);
    const int dl0 = warp * (kSmChunk / 8);
#pragma unroll 8
    for (int j = 0; j < kSmChunk / 8; ++j) {
      const int dl = dl0 + j;
      const float xv = __bfloat162float(xs[tl * kSmXStride + dl]);
      const float4 w = *reinterpret_cast<const float4*>(ws + dl * kSmExp + el);
      acc0 = fmaf(xv, w.x, acc0);
      acc1 = fmaf(xv, w.y, acc1);
      acc2 = fmaf(xv, w.z, acc2);
      acc3 = fmaf(xv, w.w, acc3);
    }
    __syncthreads();
    if (c + kSmBufs < nchunks) stage(c + kSmBufs);
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

size_t router_small_smem() { return (size_t)kSmBufs * kSmBufBytes; }

// ---------------------------------------------------------------- one token, one warp
// Router scores and top-k of one token by one warp (E <= 256; lane holds experts lane + 32j).
// logit(e) = sum over `nsum` partial rows (stride `pstride`) in order, + bias[e].
// Writes the scores to prow; block mode: TopKMask(s, k) to hrow; token mode: the k experts
// by descending score (ties: lower id) and their renormalised gates.
__device__ void token_route_warp(const float* lrow, int nsum, size_t pstride,
                                 const float* __restrict__ bias, int E, int k, int mode,
                                 float* prow, float* hrow, int32_t* idx_out, float* gate_out) {
  constexpr int J = kMaxExperts / 32;
  const int lane = threadIdx.x & 31;
  float v[J];
#pragma unroll
  for (int j = 0; j < J; ++j) {
    const int e = lane + 32 * j;
    float a = -INFINITY;
    if (e < E) {
      a = 0.f;
      for (int s = 0; s < nsum; ++s) a += __ldcg(lrow + (size_t)s * pstride + e);
      if (bias != nullptr) a += bias[e];
    }
    v[j] = a;
  }
  float m = v[0];
#pragma unroll
  for (int j = 1; j < J; ++j) m = fmaxf(m, v[j]);
  m = warp_max(m);
  float sum = 0.f;
#pragma unroll
  for (int j = 0; j < J; ++j) {
    v[j] = (lane + 32 * j < E) ? expf(v[j] - m) : 0.f;
    sum += v[j];
  }
  sum = warp_sum(sum);
#pragma unroll
  for (int j = 0; j < J; ++j) {
    v[j] = v[j] / sum;
    if (lane + 32 * j < E) prow[lane + 32 * j] = v[j];
  }
  // top-k: k rounds of a warp arg-max (score descending, expert id ascending)
  uint32_t taken = 0;
  int my_idx = 0;
  float my_val = 0.f;
  for (int r = 0; r < k; ++r) {
    float bv = -1.f;
    int bi = 0x7fffffff;
#pragma unroll
    for (int j = 0; j < J; ++j) {
      const int e = lane + 32 * j;
      if (e < E && !((taken >> j) & 1u) && (v[j] > bv || (v[j] == bv && e < bi))) {
        bv = v[j];
        bi = e;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (ov > bv || (ov == bv && oi < bi)) {
        bv = ov;
        bi = oi;
      }
    }
    if ((bi & 31) == lane) taken |= 1u << (bi >> 5);
    if (lane == r) {
      my_idx = bi;
      my_val = bv;
    }
  }
  if (mode == DMOE_ROUTE_BLOCK) {
#pragma unroll
    for (int j = 0; j < J; ++j)
      if (lane + 32 * j < E) hrow[lane + 32 * j] = ((taken >> j) & 1u) ? v[j] : 0.f;
  } else {
    float tot = 0.f;
    for (int r = 0; r < k; ++r) tot += __shfl_sync(0xffffffffu, my_val, r);
    if (lane < k) {
      idx_out[lane] = my_idx;
      gate_out[lane] = my_val / tot;
    }
  }
}

// Eight tokens per CTA, one warp each.
__global__ void __launch_bounds__(256)
router_softmax_kernel(const float* __restrict__ part, int splits, const float* __restrict__ bias,
                      float* __restrict__ probs, float* __restrict__ probs_hat,
                      int32_t* __restrict__ topk_idx, float* __restrict__ topk_gate,
                      int T, int E, int k, int mode) {
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (t >= T) return;
  token_route_warp(part + (size_t)t * E, splits, (size_t)T * E, bias, E, k, mode,
                   probs + (size_t)t * E, probs_hat + (size_t)t * E, topk_idx + (size_t)t * k,
                   topk_gate + (size_t)t * k);
}

// ---------------------------------------------------------------- Algorithm 1, one block
// Algorithm 1 for block b by a CTA of 256 threads (thread = expert for the block-level
// steps, one warp per token for MaskOutside + TopK).
__device__ void block_route_cta(int b, const float* probs, const float* probs_hat, int E, int k,
                                int B, float top_p, int32_t* __restrict__ topk_idx,
                                float* __restrict__ topk_gate, int32_t* __restrict__ coreset,
                                int32_t* __restrict__ coreset_size) {
  __shared__ float st_s[kMaxExperts];
  __shared__ float sorted_v[kMaxExperts];
  __shared__ int order[kMaxExperts];
  __shared__ float wv[8][kMaxExperts];
  __shared__ float wsel_v[8][kMaxTopK];
  __shared__ int wsel_e[8][kMaxTopK];
  __shared__ float fscr[32];
  __shared__ int iscr[32];
  const int tid = threadIdx.x;
  const int t0 = b * B;
  const bool live = tid < E;

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
  __syncthreads();
}

__global__ void __launch_bounds__(256)
block_route_kernel(const float* __restrict__ probs, const float* __restrict__ probs_hat,
                   int E, int k, int B, float top_p,
                   int32_t* __restrict__ topk_idx, float* __restrict__ topk_gate,
                   int32_t* __restrict__ coreset, int32_t* __restrict__ coreset_size) {
  pdl_launch_dependents();
  pdl_wait();
  block_route_cta(blockIdx.x, probs, probs_hat, E, k, B, top_p, topk_idx, topk_gate, coreset,
                  coreset_size);
}

// ---------------------------------------------------------------- fused decode path
struct FusedArgs {
  RouterArgs r;
  DispatchArgs dsp;   // dsp.n_unique == nullptr: no dispatch in this launch
  int32_t* ticket;
};

__global__ void __launch_bounds__(256)
route_fused_kernel(const FusedArgs f) {
  extern __shared__ __align__(16) uint8_t lsm[];
  __shared__ int s_last;
  __shared__ uint32_t s_bits[(kFusedMaxTokens / 32) * kMaxExperts];
  __shared__ uint16_t s_base[(kFusedMaxTokens / 32) * kMaxExperts];
  const RouterArgs& a = f.r;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int nctas = gridDim.x * gridDim.y;
  const int cta = blockIdx.y * gridDim.x + blockIdx.x;
  pdl_launch_dependents();
  pdl_wait();
  if (tid == 0) issue_shared_prefetch(a.shared_pf, cta, nctas);
  logits_tile_small(a.x, a.w_r, a.logits_part, a.T, a.d, a.E, blockIdx.x * kSmExp,
                    blockIdx.y * kSmTok, lsm);
  // the last CTA to finish its tile routes the whole forward
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(f.ticket, 1) == nctas - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int t = warp; t < a.T; t += 8)
    token_route_warp(a.logits_part + (size_t)t * a.E, 1, 0, a.bias, a.E, a.k, a.mode,
                     a.probs + (size_t)t * a.E, a.probs_hat + (size_t)t * a.E,
                     a.topk_idx + (size_t)t * a.k, a.topk_gate + (size_t)t * a.k);
  __syncthreads();
  if (a.mode == DMOE_ROUTE_BLOCK) {
    for (int b = 0; b < a.n_blocks; ++b)
      block_route_cta(b, a.probs, a.probs_hat, a.E, a.k, a.B, a.top_p, a.topk_idx,
                      a.topk_gate, a.coreset, a.coreset_size);
  } else {
    if (a.coreset != nullptr)
      for (int i = tid; i < a.n_blocks * a.E; i += blockDim.x) a.coreset[i] = -1;
    if (a.coreset_size != nullptr)
      for (int i = tid; i < a.n_blocks; i += blockDim.x) a.coreset_size[i] = 0;
    __syncthreads();
  }
  if (f.dsp.n_unique != nullptr)
    dispatch_cta(f.dsp.topk_idx, a.T, a.E, a.k, f.dsp.n_unique, f.dsp.unique_ids,
                 f.dsp.offsets, f.dsp.rows, f.dsp.pos, f.dsp.err, s_bits, s_base);
  if (tid == 0) *f.ticket = 0;  // ready for the next call
}

template <class K>
cudaError_t set_smem_once(K kernel, int bytes, int* mask) {
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 31 && (*mask & (1 << dev))) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && dev < 31) *mask |= 1 << dev;
  return e;
}

}  // namespace

bool router_fused_ok(int T, int d) { return T <= kFusedMaxTokens && d % kSmChunk == 0; }

cudaError_t launch_router(const RouterArgs& a, const DispatchArgs* dsp, int32_t* ticket,
                          cudaStream_t s) {
  prof_begin(DMOE_KERNEL_ROUTER, s);
  cudaError_t e;
  if (router_fused_ok(a.T, a.d)) {
    static int mask = 0;
    const size_t smem = router_small_smem();
    e = set_smem_once(route_fused_kernel, (int)smem, &mask);
    if (e != cudaSuccess) return e;
    FusedArgs f{};
    f.r = a;
    if (dsp != nullptr) f.dsp = *dsp;
    f.ticket = ticket;
    dim3 g((a.E + kSmExp - 1) / kSmExp, (a.T + kSmTok - 1) / kSmTok);
    e = launch_ex(route_fused_kernel, g, dim3(256), smem, s, false, f);
    if (e != cudaSuccess) return e;
  } else {
    const int dchunk = a.d / a.splits;
    dim3 g1((a.E + kRtExp - 1) / kRtExp, (a.T + kRtTok - 1) / kRtTok, a.splits);
    router_logits_kernel<<<g1, 256, 0, s>>>(a.x, a.w_r, a.logits_part, a.T, a.d, a.E, dchunk,
                                            a.shared_pf);
    e = launch_ex(router_softmax_kernel, dim3((a.T + 7) / 8), dim3(256), 0, s, true,
                  a.logits_part, a.splits, a.bias, a.probs, a.probs_hat, a.topk_idx,
                  a.topk_gate, a.T, a.E, a.k, a.mode);
    if (e != cudaSuccess) return e;
    if (a.mode == DMOE_ROUTE_BLOCK) {
      e = launch_ex(block_route_kernel, dim3(a.n_blocks), dim3(256), 0, s, true, a.probs,
                    a.probs_hat, a.E, a.k, a.B, a.top_p, a.topk_idx, a.topk_gate, a.coreset,
                    a.coreset_size);
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
