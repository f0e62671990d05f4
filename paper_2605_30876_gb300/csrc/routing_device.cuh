// Per-token and per-block routing steps shared by the routing kernels (§4.2 and
// Algorithm 1 of arXiv 2605.30876): the router scores and top-k of one token by one warp,
// and Algorithm 1 for one diffusion block by one CTA of 256 threads.
#pragma once

#include <math.h>

#include "block_reduce.cuh"
#include "dmoe_internal.cuh"

namespace dmoe {

// ---------------------------------------------------------------- one token, one warp
// Order-preserving 32-bit key of a float (larger float -> larger unsigned key).
__device__ __forceinline__ uint32_t order_key(float f) {
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float key_value(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// Candidate lists for the warp top-k: each lane holds 8 (key, id) pairs, kept sorted best
// first (larger key, then smaller id); key 0 marks an empty slot.
struct Cand8 {
  uint32_t key[8];
  uint32_t id[8];
};

__device__ __forceinline__ void cand_cx(Cand8& c, int a, int b) {
  // compare-exchange: slot a must hold the better of the two
  const bool swap = c.key[b] > c.key[a] || (c.key[b] == c.key[a] && c.id[b] < c.id[a]);
  const uint32_t ka = c.key[a], ia = c.id[a];
  c.key[a] = swap ? c.key[b] : ka;
  c.id[a] = swap ? c.id[b] : ia;
  c.key[b] = swap ? ka : c.key[b];
  c.id[b] = swap ? ia : c.id[b];
}

// Batcher odd-even merge sort of the 8 slots (19 compare-exchanges, 6 layers).
__device__ __forceinline__ void cand_sort(Cand8& c) {
  cand_cx(c, 0, 1); cand_cx(c, 2, 3); cand_cx(c, 4, 5); cand_cx(c, 6, 7);
  cand_cx(c, 0, 2); cand_cx(c, 1, 3); cand_cx(c, 4, 6); cand_cx(c, 5, 7);
  cand_cx(c, 1, 2); cand_cx(c, 5, 6);
  cand_cx(c, 0, 4); cand_cx(c, 1, 5); cand_cx(c, 2, 6); cand_cx(c, 3, 7);
  cand_cx(c, 2, 4); cand_cx(c, 3, 5);
  cand_cx(c, 1, 2); cand_cx(c, 3, 4); cand_cx(c, 5, 6);
}

// One selection round over the warp's sorted lists: the best remaining (key, id) of the
// warp by two single-instruction reductions; the lane that held it drops it.
__device__ __forceinline__ void cand_pop(Cand8& c, uint32_t& kmax, uint32_t& imin) {
  kmax = __reduce_max_sync(0xffffffffu, c.key[0]);
  imin = __reduce_min_sync(0xffffffffu, c.key[0] == kmax ? c.id[0] : 0xffffffffu);
  if (c.key[0] == kmax && c.id[0] == imin) {
#pragma unroll
    for (int j = 0; j < 7; ++j) {
      c.key[j] = c.key[j + 1];
      c.id[j] = c.id[j + 1];
    }
    c.key[7] = 0;
    c.id[7] = 0xffffffffu;
  }
}

// Warp top-k by descending value, ties to the lower id. Lane l holds candidates j < 8 with
// values v[j] (>= 0), ids id[j] and a validity mask. After the call lane r < k holds the
// r-th selection (my_id, my_val).
__device__ __forceinline__ void warp_topk(const float (&v)[8], const int (&id)[8], uint32_t valid,
                                          int k, int& my_id, float& my_val) {
  const int lane = threadIdx.x & 31;
  Cand8 c;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const bool ok = (valid >> j) & 1u;
    c.key[j] = ok ? order_key(v[j]) : 0u;
    c.id[j] = ok ? (uint32_t)id[j] : 0xffffffffu;
  }
  cand_sort(c);
  my_id = -1;
  my_val = 0.f;
  for (int r = 0; r < k; ++r) {
    uint32_t kmax, imin;
    cand_pop(c, kmax, imin);
    if (lane == r) {
      my_id = (int)imin;
      my_val = key_value(kmax);
    }
  }
}

// Router scores and top-k of one token by one warp (E <= 256; lane holds experts lane + 32j).
// logit(e) = sum over `nsum` partial rows (stride `pstride`) in order, + bias[e].
// Writes the scores to prow; block mode: TopKMask(s, k) to hrow; token mode: the k experts
// by descending score (ties: lower id) and their renormalised gates.
__device__ inline void token_route_warp(const float* lrow, int nsum, size_t pstride,
                                 const float* __restrict__ bias, int E, int k, int mode,
                                 float* prow, float* hrow, int32_t* idx_out, float* gate_out) {
  constexpr int J = kMaxExperts / 32;
  const int lane = threadIdx.x & 31;
  float v[J];
  int id[J];
  uint32_t valid = 0;
#pragma unroll
  for (int j = 0; j < J; ++j) {
    const int e = lane + 32 * j;
    id[j] = e;
    float a = -INFINITY;
    if (e < E) {
      valid |= 1u << j;
      a = 0.f;
      for (int s = 0; s < nsum; ++s) a += lrow[(size_t)s * pstride + e];
      if (bias != nullptr) a += bias[e];
    }
    v[j] = a;
  }
  uint32_t mk = 0;
#pragma unroll
  for (int j = 0; j < J; ++j)
    if ((valid >> j) & 1u) mk = max(mk, order_key(v[j]));
  const float m = key_value(__reduce_max_sync(0xffffffffu, mk));
  float sum = 0.f;
#pragma unroll
  for (int j = 0; j < J; ++j) {
    v[j] = ((valid >> j) & 1u) ? expf(v[j] - m) : 0.f;
    sum += v[j];
  }
  sum = warp_sum(sum);
#pragma unroll
  for (int j = 0; j < J; ++j) {
    v[j] = v[j] / sum;
    if ((valid >> j) & 1u) prow[lane + 32 * j] = v[j];
  }
  int my_idx;
  float my_val;
  warp_topk(v, id, valid, k, my_idx, my_val);
  if (mode == DMOE_ROUTE_BLOCK) {
    // TopKMask: zeros, then the k selected scores (expert e lives in lane e % 32)
#pragma unroll
    for (int j = 0; j < J; ++j)
      if ((valid >> j) & 1u) hrow[lane + 32 * j] = 0.f;
    __syncwarp();
    if (lane < k) hrow[my_idx] = my_val;
  } else {
    float tot = 0.f;
    for (int r = 0; r < k; ++r) tot += __shfl_sync(0xffffffffu, my_val, r);
    if (lane < k) {
      idx_out[lane] = my_idx;
      gate_out[lane] = my_val / tot;
    }
  }
}

// ---------------------------------------------------------------- Algorithm 1, one block
// Algorithm 1 for block b by a CTA of 256 threads (thread = expert for the block-level
// steps, one warp per token for MaskOutside + TopK).
__device__ inline void block_route_cta(int b, const float* probs, const float* probs_hat, int E, int k,
                                int B, float top_p, int32_t* __restrict__ topk_idx,
                                float* __restrict__ topk_gate, int32_t* __restrict__ coreset,
                                int32_t* __restrict__ coreset_size) {
  __shared__ __align__(16) float st_s[kMaxExperts];
  __shared__ int order[kMaxExperts];
  __shared__ int s_size;
  __shared__ float fscr[32];
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
  // Sort + Top-P + floor by one warp: the experts are taken in sorted order (S~ descending,
  // ties to the lower id) while the running fp32 sum is accumulated in that order; the
  // p rule stops at the first running sum >= p (p >= 1: at the last nonzero entry), the
  // floor then continues to k entries.
  if (tid < 32) {
    Cand8 c;
    int nz = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int e = tid + 32 * j;
      const bool ok = e < E;
      const float x = ok ? st_s[e] : 0.f;
      c.key[j] = ok ? order_key(x) : 0u;
      c.id[j] = ok ? (uint32_t)e : 0xffffffffu;
      nz += (ok && x > 0.f) ? 1 : 0;
    }
    const int nnz = __reduce_add_sync(0xffffffffu, nz);
    cand_sort(c);
    float cum = 0.f;
    int m = (top_p >= 1.f) ? nnz : -1;
    int cnt = 0;
    for (;;) {
      const int target = (m < 0) ? E : max(m, k);
      if (cnt >= target) break;
      uint32_t kmax, imin;
      cand_pop(c, kmax, imin);
      if (tid == 0) order[cnt] = (int)imin;
      cum += key_value(kmax);
      ++cnt;
      if (m < 0 && (cum >= top_p || cnt >= nnz)) m = min(cnt, nnz);
    }
    if (tid == 0) s_size = max(m, k);
  }
  __syncthreads();
  const int size = s_size;
  if (coreset != nullptr && live) coreset[(size_t)b * E + tid] = (tid < size) ? order[tid] : -1;
  if (coreset_size != nullptr && tid == 0) coreset_size[b] = size;

  // MaskOutside + TopK for every token of the block (one warp per token): lane l holds the
  // coreset members at sorted positions l + 32j
  const int warp = tid >> 5, lane = tid & 31;
  for (int i = warp; i < B; i += 8) {
    const int t = t0 + i;
    float cv[8];
    int ce[8];
    uint32_t valid = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int c = lane + 32 * j;
      ce[j] = 0;
      cv[j] = 0.f;
      if (c < size) {
        valid |= 1u << j;
        ce[j] = order[c];
        cv[j] = probs[(size_t)t * E + ce[j]];
      }
    }
    int my_e;
    float my_v;
    warp_topk(cv, ce, valid, k, my_e, my_v);
    float g = 0.f;
    for (int r = 0; r < k; ++r) g += __shfl_sync(0xffffffffu, my_v, r);
    if (lane < k) {
      topk_idx[(size_t)t * k + lane] = my_e;
      topk_gate[(size_t)t * k + lane] = my_v / g;
    }
  }
  __syncthreads();
}

}  // namespace dmoe
