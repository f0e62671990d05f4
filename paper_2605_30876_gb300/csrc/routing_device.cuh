// Per-token and per-block routing steps shared by the routing kernels (§4.2 and
// Algorithm 1 of arXiv 2605.30876): the router scores and top-k of one token by one warp,
// and Algorithm 1 for one diffusion block by one CTA of 256 threads.
#pragma once

#ifndef DMOE_STAMP
#define DMOE_STAMP(st) ((void)0)
#endif

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

// Softmax over one token's experts held by a warp (lane holds experts lane + 32j; invalid
// slots are -inf on entry and 0 on exit): exp(v - max) * (1 / sum), fp32, the sum in a fixed
// order (exp by the hardware exponential: a few ulp, far inside the routing tolerance).
__device__ __forceinline__ void warp_softmax8(float (&v)[kMaxExperts / 32], uint32_t valid) {
  constexpr int J = kMaxExperts / 32;
  float mx = -INFINITY;
#pragma unroll
  for (int j = 0; j < J; ++j)
    if ((valid >> j) & 1u) mx = fmaxf(mx, v[j]);
  const float m = key_value(__reduce_max_sync(0xffffffffu, order_key(mx)));
  float sum = 0.f;
#pragma unroll
  for (int j = 0; j < J; ++j) {
    v[j] = ((valid >> j) & 1u) ? __expf(v[j] - m) : 0.f;
    sum += v[j];
  }
  const float inv = 1.f / warp_sum(sum);
#pragma unroll
  for (int j = 0; j < J; ++j) v[j] *= inv;
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
    v[j] = 0.f;
    if (e < E) valid |= 1u << j;
  }
  // partial rows outermost, eight at a time: their 8 J loads go out together; the sum keeps
  // the row order
  for (int s0 = 0; s0 < nsum; s0 += 8) {
    float l[8][J];
#pragma unroll
    for (int q = 0; q < 8; ++q)
#pragma unroll
      for (int j = 0; j < J; ++j)
        l[q][j] = (s0 + q < nsum && ((valid >> j) & 1u))
                      ? lrow[(size_t)(s0 + q) * pstride + lane + 32 * j]
                      : 0.f;
#pragma unroll
    for (int q = 0; q < 8; ++q)
      if (s0 + q < nsum)
#pragma unroll
        for (int j = 0; j < J; ++j) v[j] += l[q][j];
  }
#pragma unroll
  for (int j = 0; j < J; ++j) {
    if ((valid >> j) & 1u) {
      if (bias != nullptr) v[j] += bias[lane + 32 * j];
    } else {
      v[j] = -INFINITY;
    }
  }
  warp_softmax8(v, valid);
#pragma unroll
  for (int j = 0; j < J; ++j)
    if ((valid >> j) & 1u) prow[lane + 32 * j] = v[j];
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

// A block's coreset for the expert launch, by one warp: the 256-bit member mask (relaxed
// stores), then the marker word with release semantics, so that a reader that acquires a
// nonzero marker sees the whole mask.
__device__ inline void publish_coreset_mask(uint32_t* __restrict__ words, const int* order,
                                            int size) {
  const int lane = threadIdx.x & 31;
  uint32_t m[kMaxExperts / 32];
#pragma unroll
  for (int w = 0; w < kMaxExperts / 32; ++w) m[w] = 0u;
  for (int i = lane; i < size; i += 32) {
    const int e = order[i];
#pragma unroll
    for (int w = 0; w < kMaxExperts / 32; ++w)
      if ((e >> 5) == w) m[w] |= 1u << (e & 31);
  }
  uint32_t mine = 0u;
#pragma unroll
  for (int w = 0; w < kMaxExperts / 32; ++w) {
    const uint32_t all = __reduce_or_sync(0xffffffffu, m[w]);
    if (lane == w) mine = all;
  }
  if (lane < kMaxExperts / 32)
    asm volatile("st.relaxed.gpu.global.u32 [%0], %1;" ::"l"(words + lane), "r"(mine) : "memory");
  __syncwarp();
  if (lane == 0)
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(words + kMaxExperts / 32), "r"(1u)
                 : "memory");
}

// ---------------------------------------------------------------- Algorithm 1, one block
// Algorithm 1 for one block of B tokens by a CTA of 256 threads. The block's rows come
// through accessors, so the same steps serve rows in global memory and rows spread over the
// shared memory of a cluster:
//   hat(i, e)   TopKMask(s_i, k)[e] of the block's i-th token
//   prob(i, e)  s_i[e]
//   out(i, r, e, g)  the r-th selection of token i: expert e with gate g

// Aggregate, Normalize, Sort, Top-P and the k floor (thread = expert). Leaves the coreset in
// order[0, size) (S~ descending, ties to the lower id) and returns size; writes the coreset
// outputs when given. `order` is a shared array of kMaxExperts entries.
//
// Top-P accumulates the sorted values in order in fp32 and stops at the first running sum
// >= p (p >= 1: at the last nonzero entry); the floor extends the coreset to k entries
// (zero entries in id order). For p <= 0 (block top-k) the coreset is the k largest sums,
// taken by one warp without the normalisation. For 0 < p < 1 every warp sorts its 32
// entries by rank, then one warp merges the sorted lists by a tournament over their heads
// until both rules are met; for p >= 1 every nonzero S~ counts the nonzero entries that
// beat it (larger, or equal with a lower id), all in parallel. Needs blockDim.x ==
// kMaxExperts.
template <class HatFn>
__device__ inline int block_coreset_steps(int E, int k, int B, float top_p, HatFn hat, int* order,
                                          int32_t* __restrict__ coreset,
                                          int32_t* __restrict__ coreset_size,
                                          uint32_t* __restrict__ spec = nullptr,
                                          const float* rows = nullptr, int row_stride = 0) {
  __shared__ __align__(16) float st_s[kMaxExperts];
  __shared__ uint2 nz_kid[kMaxExperts];   // nonzero entries: (order key, id), ids ascending
  __shared__ int wcnt[2][8];
  __shared__ int s_size;
  __shared__ float fscr[32];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool live = tid < E;

  // S_block = sum over the block's tokens of TopKMask(s_i, k). With the rows given as an
  // array (16-byte aligned, B and E multiples of 4): thread t sums experts 4 (t mod 64) ..
  // + 3 over the t / 64-th quarter of the tokens (ascending, 16-byte loads), and the four
  // quarter sums of an expert are added in order; else every thread sums its expert over
  // all tokens in ascending order, 32 rows fetched at a time so that their loads overlap
  float S = 0.f;
  if (rows != nullptr && B % 4 == 0 && E % 4 == 0 && B >= 8) {
    __shared__ __align__(16) float qsum[4][kMaxExperts];
    const int eq = 4 * (tid & 63), rq = tid >> 6, nq = B / 4;
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
    if (eq < E) {
      const float* r0 = rows + (size_t)(rq * nq) * row_stride + eq;
      for (int i0 = 0; i0 < nq; i0 += 8) {
        float4 h[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (i0 + u < nq) h[u] = *reinterpret_cast<const float4*>(r0 + (size_t)(i0 + u) * row_stride);
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (i0 + u < nq) {
            a.x += h[u].x;
            a.y += h[u].y;
            a.z += h[u].z;
            a.w += h[u].w;
          }
      }
    }
    *reinterpret_cast<float4*>(&qsum[rq][eq]) = a;
    __syncthreads();
    if (live) S = ((qsum[0][tid] + qsum[1][tid]) + qsum[2][tid]) + qsum[3][tid];
  } else if (live) {
    for (int i0 = 0; i0 < B; i0 += 32) {
      float h[32];
#pragma unroll
      for (int u = 0; u < 32; ++u) h[u] = (i0 + u < B) ? hat(i0 + u, tid) : 0.f;
#pragma unroll
      for (int u = 0; u < 32; ++u)
        if (i0 + u < B) S += h[u];
    }
  }
  DMOE_STAMP(22);
  if (top_p <= 0.f) {
    // p <= 0 (block top-k): Top-P stops at the first entry and the floor extends the coreset
    // to the k best. S~ = S / sum(S) has the order of S (exactly so, where the fp32 division
    // would round two sums to one value), so the k best sums are taken directly: warp 0
    // holds all E sums, eight per lane, and selects them by a sort and k reductions.
    st_s[tid] = live ? S : 0.f;
    __syncthreads();
    if (warp == 0) {
      float v[8];
      int id[8];
      uint32_t valid = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int e = lane + 32 * j;
        id[j] = e;
        v[j] = e < E ? st_s[e] : 0.f;
        if (e < E) valid |= 1u << j;
      }
      int my_e;
      float my_v;
      warp_topk(v, id, valid, k, my_e, my_v);
      if (lane < k) order[lane] = my_e;
      if (spec != nullptr) {
        // block top-k: the coreset (the k best, best first) is every token's routing; it is
        // published for the expert launch at once, three 8-bit ids and a marker byte per
        // word, one relaxed store per word (a word reads as zero until it is complete)
        uint32_t w = 1u << 24;
#pragma unroll
        for (int j = 0; j < 3; ++j) {
          const int src = 3 * lane + j;
          const int ej = __shfl_sync(0xffffffffu, my_e, src & 31);
          if (src < k) w |= (uint32_t)ej << (8 * j);
        }
        if (lane < spec_words(k))
          asm volatile("st.relaxed.gpu.global.u32 [%0], %1;" ::"l"(spec + lane), "r"(w) : "memory");
      }
    }
    __syncthreads();
    if (coreset != nullptr && live) coreset[tid] = (tid < k) ? order[tid] : -1;
    if (coreset_size != nullptr && tid == 0) coreset_size[0] = k;
    __syncthreads();   // st_s and order are rewritten by a later block of the same CTA
    return k;
  }
  // Normalize: L1
  const float tot = block_sum(S, fscr);
  DMOE_STAMP(19);
  const float st = live ? S / tot : 0.f;
  if (top_p < 1.f) {
    // p < 1: the coreset is a short sorted prefix. Each warp sorts its 32 entries by their
    // ranks (larger key, then lower id); warp 0 then takes the entries in sorted order by a
    // tournament over the heads of the eight lists (lane w holds list w's head; each round
    // the best head by two single-instruction reductions, and its list advances) and keeps
    // the running sum. Padding entries (id >= E) have key 0 and are never reached.
    __shared__ uint32_t wkey[kMaxExperts];
    __shared__ uint2 wl[kMaxExperts];   // list of warp w: wl[32 w .. 32 w + 31], best first
    const uint32_t key = live ? order_key(st) : 0u;
    wkey[tid] = key;
    const uint32_t bnz = __ballot_sync(0xffffffffu, live && st > 0.f);
    if (lane == 0) wcnt[0][warp] = __popc(bnz);
    __syncwarp();
    int r = 0;
#pragma unroll 8
    for (int j = 0; j < 32; ++j) {
      const uint32_t kj = wkey[warp * 32 + j];
      r += (kj > key || (kj == key && j < lane)) ? 1 : 0;
    }
    wl[warp * 32 + r] = make_uint2(key, (uint32_t)tid);
    __syncthreads();
    if (warp == 0) {
      const int nw = (int)(blockDim.x >> 5);
      const int nnz = __reduce_add_sync(0xffffffffu, lane < nw ? wcnt[0][lane] : 0);
      int h = 0;
      uint2 hd = lane < nw ? wl[lane * 32] : make_uint2(0u, 0xffffffffu);
      float cum = 0.f;
      int m = -1, cnt = 0;
      for (;;) {
        const int target = (m < 0) ? E : max(m, k);
        if (cnt >= target) break;
        const uint32_t kmax = __reduce_max_sync(0xffffffffu, hd.x);
        const uint32_t imin = __reduce_min_sync(0xffffffffu, hd.x == kmax ? hd.y : 0xffffffffu);
        if (lane == 0) order[cnt] = (int)imin;
        cum += key_value(kmax);
        ++cnt;
        if (m < 0 && (cum >= top_p || cnt >= nnz)) m = min(cnt, nnz);
        if (hd.y == imin) {   // ids are unique: only the winner's list advances
          ++h;
          hd = h < 32 ? wl[lane * 32 + h] : make_uint2(0u, 0xffffffffu);
        }
      }
      if (lane == 0) s_size = max(m, k);
    }
    __syncthreads();
    const int size = s_size;
    if (coreset != nullptr && live) coreset[tid] = (tid < size) ? order[tid] : -1;
    if (coreset_size != nullptr && tid == 0) coreset_size[0] = size;
    __syncthreads();   // st_s and order are rewritten by a later block of the same CTA
    return size;
  }
  // p >= 1: every nonzero entry is in; sort them by ranks in parallel.
  // compact the nonzero entries (and count the zero ones), in id order
  const bool nz = live && st > 0.f;
  const bool z = live && !nz;
  const uint32_t bnz = __ballot_sync(0xffffffffu, nz), bz = __ballot_sync(0xffffffffu, z);
  __syncthreads();   // wcnt and the lists are rewritten by a later block of the same CTA
  if (lane == 0) {
    wcnt[0][warp] = __popc(bnz);
    wcnt[1][warp] = __popc(bz);
  }
  __syncthreads();
  int pnz = __popc(bnz & ((1u << lane) - 1u)), pz = __popc(bz & ((1u << lane) - 1u)), nnz = 0, nzero = 0;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
    if (w < warp) {
      pnz += wcnt[0][w];
      pz += wcnt[1][w];
    }
    nnz += wcnt[0][w];
    nzero += wcnt[1][w];
  }
  if (nz) nz_kid[pnz] = make_uint2(order_key(st), (uint32_t)tid);
  __syncthreads();
  DMOE_STAMP(20);
  // ranks of the nonzero entries -> sorted positions; zero entries after them by id
  if (nz) {
    const uint32_t key = order_key(st);
    int r = 0;
#pragma unroll 8
    for (int j = 0; j < nnz; ++j) {
      const uint2 kj = nz_kid[j];
      r += (kj.x > key || (kj.x == key && kj.y < (uint32_t)tid)) ? 1 : 0;
    }
    order[r] = tid;
    st_s[r] = st;
  }
  if (z) order[nnz + pz] = tid;
  __syncthreads();
  DMOE_STAMP(21);
  if (tid == 0) {
    int m = nnz;
    if (top_p < 1.f) {
      float cum = 0.f;
      for (int r = 0; r < nnz; ++r) {
        cum += st_s[r];
        if (cum >= top_p) {
          m = r + 1;
          break;
        }
      }
    }
    s_size = max(m, k);
  }
  __syncthreads();
  const int size = s_size;
  (void)nzero;
  if (coreset != nullptr && live) coreset[tid] = (tid < size) ? order[tid] : -1;
  if (coreset_size != nullptr && tid == 0) coreset_size[0] = size;
  return size;
}

// MaskOutside + TopK for every token of the block, one warp per token: lane l holds the
// coreset members at sorted positions l + 32j; the k best by descending score (ties: lower
// id), gates renormalised over the k in that order.
template <class ProbFn, class OutFn>
__device__ inline void mask_topk_warps(int k, int B, int size, const int* order, ProbFn prob,
                                       OutFn out) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = (int)(blockDim.x >> 5);
  if (size <= 32) {
    // one member per lane: k rounds of a tournament (larger score, ties to the lower id),
    // run for four of the warp's tokens at once (their reductions are independent, so they
    // overlap); the scores of those tokens are loaded before the first round
    const int e = lane < size ? order[lane] : -1;
    constexpr int kTok = 4;
    for (int i0 = warp; i0 < B; i0 += kTok * nw) {
      uint32_t key[kTok];
#pragma unroll
      for (int u = 0; u < kTok; ++u) {
        const int i = i0 + u * nw;
        key[u] = (i < B && e >= 0) ? order_key(prob(i, e)) : 0u;
      }
      int my_e[kTok];
      float my_v[kTok];
#pragma unroll
      for (int u = 0; u < kTok; ++u) {
        my_e[u] = -1;
        my_v[u] = 0.f;
      }
      for (int r = 0; r < k; ++r) {
        uint32_t kmax[kTok], imin[kTok];
#pragma unroll
        for (int u = 0; u < kTok; ++u) kmax[u] = __reduce_max_sync(0xffffffffu, key[u]);
#pragma unroll
        for (int u = 0; u < kTok; ++u)
          imin[u] = __reduce_min_sync(0xffffffffu, key[u] == kmax[u] ? (uint32_t)e : 0xffffffffu);
#pragma unroll
        for (int u = 0; u < kTok; ++u) {
          if (lane == r) {
            my_e[u] = (int)imin[u];
            my_v[u] = key_value(kmax[u]);
          }
          if (key[u] == kmax[u] && (uint32_t)e == imin[u]) key[u] = 0u;
        }
      }
#pragma unroll
      for (int u = 0; u < kTok; ++u) {
        const int i = i0 + u * nw;
        if (i >= B) break;   // the same for the whole warp
        float g = 0.f;
        for (int r = 0; r < k; ++r) g += __shfl_sync(0xffffffffu, my_v[u], r);
        if (lane < k) out(i, lane, my_e[u], my_v[u] / g);
      }
    }
    return;
  }
  for (int i = warp; i < B; i += nw) {
    float cv[8];
    int ce[8];
    uint32_t valid = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int c = lane + 32 * j;
      ce[j] = 0;
      if (c < size) {
        valid |= 1u << j;
        ce[j] = order[c];
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) cv[j] = ((valid >> j) & 1u) ? prob(i, ce[j]) : 0.f;
    int my_e;
    float my_v;
    warp_topk(cv, ce, valid, k, my_e, my_v);
    float g = 0.f;
    for (int r = 0; r < k; ++r) g += __shfl_sync(0xffffffffu, my_v, r);
    if (lane < k) out(i, lane, my_e, my_v / g);
  }
}

template <class HatFn, class ProbFn, class OutFn>
__device__ inline void block_route_steps(int E, int kb, int k, int B, float top_p, HatFn hat,
                                         ProbFn prob, OutFn out, int32_t* __restrict__ coreset,
                                         int32_t* __restrict__ coreset_size,
                                         uint32_t* __restrict__ spec = nullptr,
                                         const float* hat_rows = nullptr) {
  __shared__ int order[kMaxExperts];
  // block top-k (p <= 0, the coreset is every token's routing): published for the expert
  // launch as soon as it is known
  const int size = block_coreset_steps(E, kb, B, top_p, hat, order, coreset, coreset_size,
                                       top_p <= 0.f && kb == k ? spec : nullptr, hat_rows, E);
  DMOE_STAMP(25);
  mask_topk_warps(k, B, size, order, prob, out);
  __syncthreads();
  DMOE_STAMP(26);
}

// Algorithm 1 for block b with the block's rows in global memory ([T, E] row-major). The
// hat rows hold TopKMask(s_i, kb); every token keeps its k <= kb best coreset members.
__device__ inline void block_route_cta(int b, const float* probs, const float* probs_hat, int E,
                                       int kb, int k, int B, float top_p,
                                       int32_t* __restrict__ topk_idx,
                                       float* __restrict__ topk_gate,
                                       int32_t* __restrict__ coreset,
                                       int32_t* __restrict__ coreset_size,
                                       uint32_t* __restrict__ spec = nullptr) {
  const size_t r0 = (size_t)b * B;
  block_route_steps(
      E, kb, k, B, top_p,
      [&](int i, int e) { return probs_hat[(r0 + i) * E + e]; },
      [&](int i, int e) { return probs[(r0 + i) * E + e]; },
      [&](int i, int r, int e, float g) {
        topk_idx[(r0 + i) * k + r] = e;
        topk_gate[(r0 + i) * k + r] = g;
      },
      coreset != nullptr ? coreset + (size_t)b * E : nullptr,
      coreset_size != nullptr ? coreset_size + b : nullptr,
      spec != nullptr ? spec + (size_t)b * spec_words(k) : nullptr, probs_hat + r0 * E);
}

}  // namespace dmoe
