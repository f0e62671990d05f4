// The dispatch of a decode-sized forward (at most 64 tokens), computed by one CTA of the
// routing launch: the unique experts and the expert -> (token, slot) lists, each expert's
// rows ordered by token (the canonical dispatch form). No order depends on atomics. Larger
// forwards take the two launches of dispatch.cu.
#pragma once

#ifndef DMOE_STAMP
#define DMOE_STAMP(st) ((void)0)
#endif

#include "block_reduce.cuh"
#include "dmoe_internal.cuh"

namespace dmoe {

// A two-word token mask per expert: one 32-bit atomic OR per (token, slot), one packed CTA
// scan for the offsets and the unique positions. Needs blockDim.x >= E (a multiple of 32,
// at most 256).
__device__ inline void dispatch_small_cta(const int32_t* topk_idx, int T, int E, int k,
                                          int32_t* __restrict__ n_unique,
                                          int32_t* __restrict__ unique_ids,
                                          int32_t* __restrict__ offsets,
                                          int32_t* __restrict__ rows, int32_t* __restrict__ pos,
                                          DevErrRecord* err) {
  __shared__ uint32_t msk[2][kMaxExperts];
  __shared__ int off_e[kMaxExperts];
  __shared__ int wtot[8];
  __shared__ int bad;
  const int tid = threadIdx.x, nthr = blockDim.x, lane = tid & 31, warp = tid >> 5;
  const int pairs = T * k;
  if (tid == 0) bad = 0;
  if (tid < E) {
    msk[0][tid] = 0u;
    msk[1][tid] = 0u;
  }
  __syncthreads();
  DMOE_STAMP(16);
  for (int i = tid; i < pairs; i += nthr) {
    const int t = i / k, e = topk_idx[i];
    if (e < 0 || e >= E) {
      record_error(err, kErrExpertId, kAtDispatch, i);
      bad = 1;
      continue;
    }
    const uint32_t bit = 1u << (t & 31);
    if (atomicOr(&msk[t >> 5][e], bit) & bit) {
      record_error(err, kErrDupExpert, kAtDispatch, i);
      bad = 1;
    }
  }
  __syncthreads();
  DMOE_STAMP(17);
  if (bad) return;  // uniform: the outputs are unspecified after a recorded fault
  // packed inclusive scan over the experts: low 16 bits count, high bits presence
  const int lo = tid < E ? __popc(msk[0][tid]) : 0;
  const int cnt = tid < E ? lo + __popc(msk[1][tid]) : 0;
  const int v = cnt | ((cnt > 0 ? 1 : 0) << 16);
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wtot[warp] = x;
  __syncthreads();
  int base = 0, all = 0;
  for (int w = 0; w < (nthr >> 5); ++w) {
    if (w < warp) base += wtot[w];
    all += wtot[w];
  }
  const int ex = base + x - v;
  const int off = ex & 0xffff, upos = ex >> 16, n_u = all >> 16;
  if (tid < E) {
    off_e[tid] = off;
    if (cnt > 0) {
      unique_ids[upos] = tid;
      offsets[upos] = off;
    }
  }
  for (int u = n_u + tid; u < E; u += nthr) unique_ids[u] = -1;
  for (int u = n_u + tid; u <= E; u += nthr) offsets[u] = pairs;
  if (tid == 0) {
    n_unique[0] = n_u;
    if ((all & 0xffff) != pairs) record_error(err, kErrBadDispatch, kAtDispatch, all & 0xffff);
  }
  __syncthreads();
  DMOE_STAMP(18);
  for (int i = tid; i < pairs; i += nthr) {
    const int t = i / k, e = topk_idx[i];
    const int w = t >> 5;
    const uint32_t below = msk[w][e] & ((1u << (t & 31)) - 1u);
    const int r = off_e[e] + __popc(below) + (w ? __popc(msk[0][e]) : 0);
    rows[r] = i;
    pos[i] = r;
  }
}

}  // namespace dmoe
