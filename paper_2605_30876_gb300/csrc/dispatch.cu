// Dispatch of a forward in two launches over 32-token chunks (one CTA per chunk):
//   dispatch_count_kernel  the chunk's token bitmap per expert (bits[c][e]: bit l for token
//                          32c + l); the last CTA to finish (atomic ticket) adds the bitmaps'
//                          counts over the chunks per expert (base[c][e] = pairs of e in
//                          chunks before c) and scans over the experts: the offsets, the
//                          unique list and U
//   dispatch_place_kernel  each (token, slot) goes to row off[e] + base[c][e] + the popcount
//                          of bits[c][e] below its token; in the fused layer call it also
//                          copies the x rows into dispatch order (16 CTAs per chunk)
// Every sum runs in a fixed order (no order depends on atomics), and each expert's rows are
// ordered by token, the canonical dispatch form. An id outside [0, E) or an expert twice in
// one token is recorded as a fault; the outputs are then unspecified (rows stay in range).
#include "block_reduce.cuh"
#include "dmoe_internal.cuh"
#include "trace_log.cuh"

// Debug builds (-DDMOE_TRACE): phase times of dispatch_count_kernel (%globaltimer, ns),
// g_dtr[cta * 16 + slot]: 0 entry, 1 ids loaded, 2 bitmap built, 3 bitmap stored, 4 ticket
// taken; the last CTA: 5 prefix over the chunks, 6 scans, 7 outputs written.
#ifdef DMOE_TRACE
__device__ uint64_t g_dtr[1024 * 16];
#define DTR_AT(slot)                                                                      \
  do {                                                                                    \
    if (threadIdx.x == 0) {                                                               \
      uint64_t t_;                                                                        \
      asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                             \
      g_dtr[(blockIdx.x % 1024) * 16 + (slot)] = t_;                                      \
    }                                                                                     \
  } while (0)
#else
#define DTR_AT(slot) ((void)0)
#endif

namespace dmoe {
namespace {

constexpr int kDispThreads = 256;
constexpr int kDispPerThread = (32 * kMaxTopK + kDispThreads - 1) / kDispThreads;

__global__ void __launch_bounds__(kDispThreads)
dispatch_count_kernel(const int32_t* __restrict__ topk_idx, int T, int E, int k,
                      uint32_t* __restrict__ gbits, int32_t* __restrict__ gbase,
                      int32_t* __restrict__ goff, int32_t* __restrict__ n_unique,
                      int32_t* __restrict__ unique_ids, int32_t* __restrict__ offsets,
                      DevErrRecord* err, int32_t* ticket) {
  __shared__ uint32_t bits[kMaxExperts];
  __shared__ int iscr[32];
  __shared__ int s_last;
  const int c = blockIdx.x, tid = threadIdx.x;
  const int t0 = c * 32, ntok = T - t0 < 32 ? T - t0 : 32, np = ntok * k;
  const int nchunks = gridDim.x, pairs = T * k;
  // the next launch reads the routing too: it may start once every CTA is past this wait
  pdl_wait();
  pdl_launch_dependents();
  KLOG(DMOE_KERNEL_DISPATCH, 0);
  DTR_AT(0);
  int ids[kDispPerThread];
#pragma unroll
  for (int j = 0; j < kDispPerThread; ++j) {
    const int p = tid + j * kDispThreads;
    ids[j] = p < np ? topk_idx[t0 * k + p] : 0;
  }
  for (int e = tid; e < E; e += kDispThreads) bits[e] = 0u;
  __syncthreads();
  DTR_AT(1);
#pragma unroll
  for (int j = 0; j < kDispPerThread; ++j) {
    const int p = tid + j * kDispThreads;
    if (p >= np) continue;
    const int i = t0 * k + p, e = ids[j];
    if (e < 0 || e >= E) {
      record_error(err, kErrExpertId, kAtDispatch, i);
      continue;
    }
    const uint32_t bit = 1u << ((i / k) & 31);
    if (atomicOr(&bits[e], bit) & bit) record_error(err, kErrDupExpert, kAtDispatch, i);
  }
  __syncthreads();
  DTR_AT(2);
  for (int e = tid; e < E; e += kDispThreads) gbits[(size_t)c * E + e] = bits[e];
  // the last CTA to get here sees every chunk's bitmap
  __syncthreads();
  DTR_AT(3);
  if (tid == 0) {
    __threadfence();
    s_last = atomicAdd(ticket, 1) == nchunks - 1 ? 1 : 0;
  }
  __syncthreads();
  DTR_AT(4);
  if (!s_last) return;
  __threadfence();
  int cnt = 0;
  if (tid < E) {
    for (int c0 = 0; c0 < nchunks; c0 += 32) {
      uint32_t w[32];   // one round of loads per 32 chunks
#pragma unroll
      for (int j = 0; j < 32; ++j)
        w[j] = c0 + j < nchunks ? __ldcg(gbits + (size_t)(c0 + j) * E + tid) : 0u;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (c0 + j < nchunks) {
          gbase[(size_t)(c0 + j) * E + tid] = cnt;
          cnt += __popc(w[j]);
        }
    }
  }
  DTR_AT(5);
  int total_pairs = 0, n_u = 0;
  const int off = block_exclusive_scan_i(tid < E ? cnt : 0, iscr, &total_pairs);
  const int present = (tid < E && cnt > 0) ? 1 : 0;
  const int upos = block_exclusive_scan_i(present, iscr, &n_u);
  DTR_AT(6);
  if (tid < E) {
    goff[tid] = off;
    if (present) {
      unique_ids[upos] = tid;
      offsets[upos] = off;
    }
  }
  for (int u = n_u + tid; u < E; u += kDispThreads) unique_ids[u] = -1;
  for (int u = n_u + tid; u <= E; u += kDispThreads) offsets[u] = pairs;
  if (tid == 0) {
    n_unique[0] = n_u;
    if (total_pairs != pairs) record_error(err, kErrBadDispatch, kAtDispatch, total_pairs);
    *ticket = 0;   // ready for the next call
  }
  DTR_AT(7);
  KLOG(DMOE_KERNEL_DISPATCH, 1);
}

// Placement of chunk blockIdx.x; with xperm, blockIdx.y takes its share of the chunk's
// (token, slot) pairs and also copies their x rows into dispatch order (kGatherRows rows
// in flight per thread).
constexpr int kPlaceSplit = 16;    // CTAs per chunk when the rows are copied too
constexpr int kGatherRows = 8;
__global__ void __launch_bounds__(kDispThreads)
dispatch_place_kernel(const int32_t* __restrict__ topk_idx, int T, int E, int k,
                      const uint32_t* __restrict__ gbits, const int32_t* __restrict__ gbase,
                      const int32_t* __restrict__ goff, int32_t* __restrict__ rows,
                      int32_t* __restrict__ pos, const __nv_bfloat16* __restrict__ x,
                      __nv_bfloat16* __restrict__ xperm, int d, int32_t* zero, int n_zero) {
  __shared__ uint32_t bits[kMaxExperts];
  __shared__ int base[kMaxExperts];
  __shared__ int s_r[32 * kMaxTopK], s_t[32 * kMaxTopK];
  const int c = blockIdx.x, tid = threadIdx.x;
  const int t0 = c * 32, ntok = T - t0 < 32 ? T - t0 : 32, np = ntok * k;
  const int pairs = T * k;
  // this CTA's pairs of the chunk
  const int per = (np + gridDim.y - 1) / gridDim.y;
  const int p0 = blockIdx.y * per, p1 = p0 + per < np ? p0 + per : np;
  // the routing was complete before the counting launch let this one start
  int ids[kDispPerThread];
#pragma unroll
  for (int j = 0; j < kDispPerThread; ++j) {
    const int p = p0 + tid + j * kDispThreads;
    ids[j] = p < p1 ? __ldcg(topk_idx + t0 * k + p) : 0;
  }
  pdl_wait();
  pdl_launch_dependents();   // after the wait: a waiting dependent would share the SMs
  KLOG(7, 0);
  if (zero != nullptr && blockIdx.x == 0 && blockIdx.y == 0)
    for (int i = tid; i < n_zero; i += kDispThreads) zero[i] = 0;
  for (int e = tid; e < E; e += kDispThreads) {
    bits[e] = gbits[(size_t)c * E + e];
    base[e] = gbase[(size_t)c * E + e] + goff[e];
  }
  __syncthreads();
#pragma unroll
  for (int j = 0; j < kDispPerThread; ++j) {
    const int p = p0 + tid + j * kDispThreads;
    const int e = ids[j];
    int r = -1;
    if (p < p1 && e >= 0 && e < E) {
      const int i = t0 * k + p, l = (i / k) & 31;
      r = base[e] + __popc(bits[e] & ((1u << l) - 1u));
      if (r >= 0 && r < pairs) {
        rows[r] = i;
        pos[i] = r;
      } else {
        r = -1;
      }
    }
    if (xperm != nullptr && p < p1) {
      s_r[p - p0] = r;
      s_t[p - p0] = t0 + p / k;
    }
  }
  if (xperm != nullptr) {
    __syncthreads();
    const int n = p1 - p0, vec = d / 8;   // rows, 16-byte pieces per row
    const uint4* src = reinterpret_cast<const uint4*>(x);
    uint4* dst = reinterpret_cast<uint4*>(xperm);
    for (int q0 = 0; q0 < n; q0 += kGatherRows)
      for (int i = tid; i < vec; i += kDispThreads) {
        uint4 v[kGatherRows];
#pragma unroll
        for (int q = 0; q < kGatherRows; ++q)
          if (q0 + q < n && s_r[q0 + q] >= 0) v[q] = src[(size_t)s_t[q0 + q] * vec + i];
#pragma unroll
        for (int q = 0; q < kGatherRows; ++q)
          if (q0 + q < n && s_r[q0 + q] >= 0) dst[(size_t)s_r[q0 + q] * vec + i] = v[q];
      }
  }
  KLOG(7, 1);
}

}  // namespace

cudaError_t launch_dispatch(const DispatchArgs& a, cudaStream_t s) {
  if (a.bits == nullptr || a.base == nullptr || a.off == nullptr || a.ticket == nullptr ||
      a.k > kMaxTopK || a.E > kMaxExperts || (a.xperm != nullptr && (a.x == nullptr || a.d % 8)))
    return cudaErrorInvalidValue;
  const int nchunks = (a.T + 31) / 32;
  prof_begin(DMOE_KERNEL_DISPATCH, s);
  cudaError_t e = launch_ex(dispatch_count_kernel, dim3(nchunks), dim3(kDispThreads), 0, s, true,
                            a.topk_idx, a.T, a.E, a.k, a.bits, a.base, a.off, a.n_unique,
                            a.unique_ids, a.offsets, a.err, a.ticket);
  if (e == cudaSuccess)
    e = launch_ex(dispatch_place_kernel, dim3(nchunks, a.xperm != nullptr ? kPlaceSplit : 1),
                  dim3(kDispThreads), 0, s, true, a.topk_idx, a.T, a.E, a.k,
                  static_cast<const uint32_t*>(a.bits), static_cast<const int32_t*>(a.base),
                  static_cast<const int32_t*>(a.off), a.rows, a.pos, a.x, a.xperm, a.d, a.zero,
                  a.n_zero);
  prof_end(DMOE_KERNEL_DISPATCH, s);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dmoe

#ifdef DMOE_TRACE
DMOE_KLOG_EXPORT(dmoe_debug_klog_dispatch)
extern "C" int dmoe_debug_dtr(void* host) {
  return (int)cudaMemcpyFromSymbol(host, g_dtr, sizeof(g_dtr));
}
#endif
