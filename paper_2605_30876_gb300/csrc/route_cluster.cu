// Routing of a decode-sized forward (T <= 64 tokens) in one launch of 8-CTA thread-block
// clusters (§4.2 router and Algorithm 1 of arXiv 2605.30876, plus the dispatch).
//
// Cluster c owns 32 experts; CTA r of the cluster owns the r-th eighth of d:
//   1. logits: TMA brings the W_r slice (d/8 rows x 32 experts, 128-B rows) and the x
//      slice (T rows x d/8); the W_r slice is split into three bf16 parts (hi + mid + lo
//      = w to 2^-27, x * part exact in fp32) and tensor cores (mma.sync, fp32 accumulate)
//      give the partial logits [T x 32], pushed over distributed shared memory to the CTA
//      that owns each token (t mod 8); CTA r then adds, in rank order, the eight partials of
//      its tokens and writes those logits.
//   2. one atomic ticket per CTA: the cluster of the last CTA to finish continues; the
//      others exit.
//   3. scores: one warp per token (8 CTAs x 8 warps = 64 tokens): softmax, top-k (token
//      mode: the routing; block mode: TopKMask, whose k nonzeros are stored straight into
//      the shared memory of the CTA that routes the token's block).
//   4. Algorithm 1 for block b by CTA b mod 8 (blocks in parallel); the scores MaskOutside
//      needs are read from the scoring CTAs' shared memory.
//   5. dispatch by CTA 0 (fused layer call) from the top-k ids gathered in its shared memory.
// Stages 3-5 are separated by cluster barriers (release/acquire at cluster scope) and pass
// their data through distributed shared memory; only the logits cross clusters, through
// global memory, read past the L1 (ld.global.cg) after the ticket's acquire.
#include <math.h>

// Debug builds (-DDMOE_TRACE): per-CTA timeline in g_ctrace[cta * 64 + stage] (stages 0
// 7 and 25: globaltimer, others: 1 = reached; + 32: clock64): 0 entry, 1 TMA landed, 8 x converted,
// 2 partial logits done, 3 logits reduced, 4 ticket, 9 score loads issued, 10 softmax,
// 11 top-k, 5 scores, 12 coreset, 13 MaskOutside, 6 Algorithm 1, 7 dispatch; 16-24: steps
// inside the dispatch, the coreset and MaskOutside (DMOE_STAMP in the shared headers);
// 25 coreset of the block known, 26 coreset received, 27 token's restricted top-k known.
#ifdef DMOE_TRACE
#include <stdint.h>
__device__ uint64_t g_ctrace[64 * 8 * 64];
#define CT_AT(st)                                                                       \
  do {                                                                                  \
    if (threadIdx.x == 0) {                                                             \
      const int c_ = ((blockIdx.y * gridDim.x + blockIdx.x) % 512) * 64 + (st);         \
      if ((st) == 0 || (st) == 7 || (st) == 25) {                                       \
        uint64_t t_;                                                                    \
        asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t_));                          \
        g_ctrace[c_] = t_;                                                              \
      } else {                                                                          \
        g_ctrace[c_] = 1;                                                               \
      }                                                                                 \
      g_ctrace[c_ + 32] = clock64();                                                    \
    }                                                                                   \
  } while (0)
#define DMOE_STAMP(st) CT_AT(st)
#else
#define CT_AT(st) ((void)0)
#endif

#include "dispatch_impl.cuh"
#include "dmoe_internal.cuh"
#include "routing_device.cuh"
#include "trace_log.cuh"

namespace dmoe {
namespace {

constexpr int kCl = kRouteClusterCtas;   // CTAs per cluster (split of d)
constexpr int kClExp = 32;             // experts per cluster
constexpr int kClMaxTok = 64;          // tokens of a decode-sized forward
constexpr int kClMaxDChunk = 256;      // d / kCl at most (one TMA box of rows)
constexpr int kClMaxCand = (kMaxExperts / kClExp) * kMaxTopK;   // candidates of one token



struct ClusterArgs {
  CUtensorMap wmap;   // W_r [d, E] fp32, box 32 experts x d/8 rows
  CUtensorMap xmap;   // x [T, d] bf16, box 64 columns x round16(T) rows, 128-B swizzle
  RouterArgs r;
  DispatchArgs dsp;   // dsp.n_unique == nullptr: no dispatch
  int32_t* ticket;    // zero between calls
  int box_rows;       // token rows of an x box (a multiple of 16, at most kClMaxTok)
  int logits_only;    // tile z of kClMaxTok tokens: stop once the logits are written
};

__device__ __forceinline__ uint32_t s_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;"
               ::: "memory");
}
// address of the same shared variable in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t peer_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(s_addr(p)), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_peer_u32(uint32_t addr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ void st_peer_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void st_peer_f32x2(uint32_t addr, float v0, float v1) {
  asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(addr), "f"(v0), "f"(v1)
               : "memory");
}

// Shared-memory layout after the logits (the W_r / x slices are dead by then), in bytes
// from the dynamic base: scores of this CTA's tokens, the top-k ids for the dispatch (rank
// 0), the coreset of each token's block, and the dense TopKMask rows of the blocks this CTA
// routes.
constexpr int kOffP = 0;                                      // f32 [8][kMaxExperts]
constexpr int kOffIdx = kOffP + 8 * kMaxExperts * 4;          // i32 [kClMaxTok * kMaxTopK]
constexpr int kOffCore = kOffIdx + kClMaxTok * kMaxTopK * 4;  // i32 [8][1 + kMaxExperts]
constexpr int kOffHat = kClMaxDChunk * kClExp * 4 + kClMaxTok * kClMaxDChunk * 2;  // f32 [kClMaxTok][kMaxExperts]
static_assert(kOffCore + 8 * (1 + kMaxExperts) * 4 <= kClMaxDChunk * kClExp * 4,
              "the routing scratch must fit where the W_r slice was");

// bf16 tensor-core product D[16 x 8] += A[16 x 16] B[16 x 8] (fp32 accumulators)
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__global__ void __launch_bounds__(256, 1)
route_cluster_kernel(const __grid_constant__ ClusterArgs f) {
  // 1024-B aligned: the swizzled x boxes take their swizzle phase from the address
  extern __shared__ __align__(1024) uint8_t dsm_raw[];
  uint8_t* dsm = dsm_raw + ((1024u - (s_addr(dsm_raw) & 1023u)) & 1023u);
  __shared__ __align__(8) uint64_t s_bar;
  __shared__ uint32_t s_last;
  // partial logits pushed by every CTA of the cluster to the owner of each token (token t:
  // CTA t mod 8): [source rank][t / 8][32 experts]
  __shared__ __align__(16) float s_part[kCl][kClMaxTok / kCl][kClExp];
  __shared__ float s_bias[kMaxExperts];
  __shared__ uint32_t s_loc[8][32];                  // one token's keys per warp
  __shared__ uint2 s_cand[8][kClMaxCand];            // merge: one token's candidates per warp
  const RouterArgs& a = f.r;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // logits-only launches take the tokens in tiles of kClMaxTok (blockIdx.z); otherwise
  // z = 0 and the tile is the whole forward
  const int tz = blockIdx.z * kClMaxTok;
  const int T = a.T - tz < kClMaxTok ? a.T - tz : kClMaxTok;
  // k: experts per token; kc: candidates per cluster and token = the TopKMask width
  // (block mode; kc >= k) or k (token mode)
  const int E = a.E, k = a.k, kc = a.kb, B = a.B;
  const int TB = f.box_rows;
  const uint32_t rank = cluster_rank();
  const int DC = a.d / kCl;                          // rows of d in this CTA's slice
  const int e0 = blockIdx.y * kClExp;
  const int n_clusters = gridDim.y;
  if (tid == 0) {
    // while the previous launch on the stream finishes: pull this CTA's W_r slice and the
    // shared expert's weights into L2. Only L2 is touched, and L2 is where a write by that
    // launch would land, so the loads below still see it.
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&f.wmap)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&f.xmap)) : "memory");
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                     reinterpret_cast<uint64_t>(&f.wmap)),
                 "r"(e0), "r"((int)rank * DC)
                 : "memory");
    issue_shared_prefetch(a.shared_pf, (blockIdx.z * gridDim.y + blockIdx.y) * kCl + (int)rank,
                          gridDim.x * gridDim.y * gridDim.z);
  }
  pdl_wait();
  // the expert launch may start now (not earlier: it reads the early coreset counter, which
  // the launch before this one clears)
  pdl_launch_dependents();
  KLOG(DMOE_KERNEL_ROUTER, 0);
  CT_AT(0);

  // ---- 1. partial logits over this CTA's slice of d
  float* Ws = reinterpret_cast<float*>(dsm);                                   // [DC][32]
  // x slice: boxes of 64 columns x TB rows with the 128-byte swizzle
  uint8_t* Xs = dsm + kClMaxDChunk * kClExp * 4;
  const int T16 = (T + 15) & ~15, nxb = (DC + 63) / 64;
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(s_addr(&s_bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    const uint32_t bytes = (uint32_t)DC * kClExp * 4 + (uint32_t)nxb * TB * 128;
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(s_addr(&s_bar)),
                 "r"(bytes)
                 : "memory");
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];" ::"r"(s_addr(Ws)),
        "l"(reinterpret_cast<uint64_t>(&f.wmap)), "r"(s_addr(&s_bar)), "r"(e0),
        "r"((int)rank * DC)
        : "memory");
    for (int bx = 0; bx < nxb; ++bx)
      asm volatile(
          "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
          " [%0], [%1, {%3, %4}], [%2];" ::"r"(s_addr(Xs) + (uint32_t)(bx * TB * 128)),
          "l"(reinterpret_cast<uint64_t>(&f.xmap)), "r"(s_addr(&s_bar)),
          "r"((int)rank * DC + 64 * bx), "r"(tz)
          : "memory");
  }
  for (int e = tid; e < E; e += 256) s_bias[e] = a.bias != nullptr ? a.bias[e] : 0.f;
  if (tid == 0) s_last = 0u;   // set by the last CTA's ticket (after the next cluster barrier)
  __syncthreads();
  {
    uint64_t t0;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
    for (;;) {
      uint32_t ok;
      asm volatile(
          "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n\t"
          "selp.u32 %0, 1, 0, p;\n\t}"
          : "=r"(ok)
          : "r"(s_addr(&s_bar))
          : "memory");
      if (ok) break;
      uint64_t t;
      asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
      if (t - t0 > 1000000000ull) {
        if (tid == 0) record_error(a.err, kErrTimeout, kAtRouter, (int)rank);
        break;
      }
    }
  }
  CT_AT(1);
  CT_AT(8);
  // tensor cores (mma.sync m16n8k16): warp tile = 16 tokens x 8 experts over the whole
  // slice. The B fragments come straight from the fp32 W_r slice (rows of 32 experts, 128
  // bytes, 128-byte swizzle: expert n of row k sits in 16-byte chunk (n / 4) xor (k mod 8),
  // so a warp's fragment loads hit 32 distinct banks) and are split there into three bf16
  // parts (hi + mid + lo = w to 2^-27; x * part is exact in fp32), one accumulator per part,
  // summed in that order at the end
  {
    const int g = lane >> 2, tq = lane & 3;
    const int ntile = (T16 / 16) * (kClExp / 8);
    const uint8_t* wsb = reinterpret_cast<const uint8_t*>(Ws);
    for (int tile = warp; tile < ntile; tile += 8) {
      const int mt = tile / (kClExp / 8), nt = tile % (kClExp / 8);
      const int r0 = mt * 16 + g;                   // A rows r0, r0 + 8 (same swizzle phase)
      const int n = nt * 8 + g;                     // B column (expert) of this thread
      float accp[3][4] = {};
#pragma unroll 8
      for (int k0 = 0; k0 < DC; k0 += 16) {
        const int bx = k0 >> 6, c = (k0 & 63) >> 3;   // box, 16-B chunk of k0
        const uint8_t* xb = Xs + bx * TB * 128;
        uint32_t af[4];
        af[0] = *reinterpret_cast<const uint32_t*>(xb + r0 * 128 + ((c ^ (r0 & 7)) << 4) + tq * 4);
        af[1] = *reinterpret_cast<const uint32_t*>(xb + (r0 + 8) * 128 + ((c ^ (r0 & 7)) << 4) + tq * 4);
        af[2] = *reinterpret_cast<const uint32_t*>(xb + r0 * 128 + (((c + 1) ^ (r0 & 7)) << 4) + tq * 4);
        af[3] = *reinterpret_cast<const uint32_t*>(xb + (r0 + 8) * 128 + (((c + 1) ^ (r0 & 7)) << 4) + tq * 4);
        // W_r[k][n] for k = k0 + 2tq, +1 (register 0) and +8, +9 (register 1)
        float w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int k = k0 + 2 * tq + (j & 1) + 8 * (j >> 1);
          w[j] = *reinterpret_cast<const float*>(
              wsb + k * 128 + ((((n >> 2) ^ (k & 7)) << 4) | ((n & 3) << 2)));
        }
        uint32_t bp[3][2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const __nv_bfloat162 hi = __floats2bfloat162_rn(w[2 * h], w[2 * h + 1]);
          const float2 hf = __bfloat1622float2(hi);
          const float q0 = w[2 * h] - hf.x, q1 = w[2 * h + 1] - hf.y;
          const __nv_bfloat162 mid = __floats2bfloat162_rn(q0, q1);
          const float2 mf = __bfloat1622float2(mid);
          const __nv_bfloat162 lo = __floats2bfloat162_rn(q0 - mf.x, q1 - mf.y);
          bp[0][h] = *reinterpret_cast<const uint32_t*>(&hi);
          bp[1][h] = *reinterpret_cast<const uint32_t*>(&mid);
          bp[2][h] = *reinterpret_cast<const uint32_t*>(&lo);
        }
#pragma unroll
        for (int part = 0; part < 3; ++part) mma_bf16_16816(accp[part], af, bp[part][0], bp[part][1]);
      }
      float acc[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) acc[i] = (accp[0][i] + accp[1][i]) + accp[2][i];
      // D rows r0, r0 + 8; columns 2tq, 2tq + 1 of the tile: to the owners of the tokens
      const int e = nt * 8 + 2 * tq;
      if (r0 < T)
        st_peer_f32x2(peer_addr(&s_part[rank][r0 >> 3][e], (uint32_t)(r0 & 7)), acc[0], acc[1]);
      if (r0 + 8 < T)
        st_peer_f32x2(peer_addr(&s_part[rank][(r0 + 8) >> 3][e], (uint32_t)((r0 + 8) & 7)),
                      acc[2], acc[3]);
    }
  }
  __syncthreads();
  {  // TopKMask rows start as zeros (scoring warps anywhere in the cluster add the winners)
    float4* hz = reinterpret_cast<float4*>(dsm + kOffHat);
    if (!f.logits_only)
      for (int i = tid; i < T * (kMaxExperts / 4); i += 256) hz[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  CT_AT(2);
  cluster_sync();   // every partial has reached its owner
  // CTA r adds the partials of tokens t = r (mod 8), in rank order, adds the bias, and keeps
  // the cluster's kc best experts of the token (candidates for the top-kc over all experts:
  // any expert of the top-kc is among the kc best of its own cluster)
  uint2* cand = a.cand;   // [T][clusters][kc]: (order key, id)
  {
    const int t = (int)rank + 8 * warp;
    if (t < T) {
      float v = 0.f;
#pragma unroll
      for (int q = 0; q < kCl; ++q) v += s_part[q][warp][lane];
      const bool ok = e0 + lane < E;
      v += ok ? s_bias[e0 + lane] : 0.f;
      if (ok) a.logits_part[(size_t)(tz + t) * E + e0 + lane] = v;
      if (!f.logits_only) {
        const uint32_t key = ok ? order_key(v) : 0u;
        s_loc[warp][lane] = key;
        __syncwarp();
        // rank among the cluster's 32 experts: larger key, ties to the lower lane (one
        // 64-bit comparison of key and inverted lane)
        const uint64_t mine = ((uint64_t)key << 32) | (uint32_t)(31 - lane);
        int r = 0;
#pragma unroll 8
        for (int j = 0; j < 32; ++j)
          r += ((((uint64_t)s_loc[warp][j]) << 32) | (uint32_t)(31 - j)) > mine ? 1 : 0;
        if (r < kc)
          cand[((size_t)t * n_clusters + blockIdx.y) * kc + r] =
              make_uint2(key, ok ? (uint32_t)(e0 + lane) : 0xffffffffu);
      }
    }
  }
  // this CTA's logits and candidates are written (no shared memory of a peer is touched
  // after this point unless the cluster goes on)
  __syncthreads();
  CT_AT(3);
  if (f.logits_only) {
    KLOG(DMOE_KERNEL_ROUTER, 1);
    return;
  }

  // ---- 2. the cluster of the last CTA to finish routes the forward: one ticket per CTA
  // (releases this CTA's logits and candidates, acquires everyone's at GPU scope); the last
  // CTA flags its cluster, whose barrier then passes the acquired writes on to its peers
  if (tid == 0) {
    uint32_t old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(f.ticket) : "memory");
    if (old == (uint32_t)(n_clusters * kCl) - 1)
      for (uint32_t q = 0; q < (uint32_t)kCl; ++q) st_peer_u32(peer_addr(&s_last, q), 1u);
  }
  cluster_sync();
  if (!s_last) {
    KLOG(DMOE_KERNEL_ROUTER, 1);
    return;
  }
  CT_AT(4);

  // ---- 3. scores: token t = 8 * rank + warp; its scores stay in this CTA's shared memory
  // (sP [8 warps][E]) and its TopKMask winners go to the CTA that routes its block
  float* sP = reinterpret_cast<float*>(dsm + kOffP);
  int32_t* sIdx = reinterpret_cast<int32_t*>(dsm + kOffIdx);  // [T * k], read in rank 0
  float* sHat = reinterpret_cast<float*>(dsm + kOffHat);
  constexpr int J = kMaxExperts / 32;
  {
    const int t = 8 * (int)rank + warp;
    if (t < T) {
      const int nc = n_clusters * kc;                      // candidates of the token
      const uint2* tc = cand + (size_t)t * nc;
      uint2 cd[kClMaxCand / 32];
#pragma unroll
      for (int q = 0; q < kClMaxCand / 32; ++q) {
        const int ci = lane + 32 * q;
        cd[q] = ci < nc ? __ldcg(tc + ci) : make_uint2(0u, 0xffffffffu);
      }
      float v[J];
      uint32_t valid = 0;
#pragma unroll
      for (int j = 0; j < J; ++j) {
        const int e = lane + 32 * j;
        v[j] = -INFINITY;
        if (e < E) {
          valid |= 1u << j;
          v[j] = __ldcg(a.logits_part + (size_t)t * E + e);   // logit + bias
        }
      }
      CT_AT(9);
      // scores: softmax over all experts (row kept in shared memory for MaskOutside)
      float mx = -INFINITY;
#pragma unroll
      for (int j = 0; j < J; ++j) mx = fmaxf(mx, v[j]);
      const float M = key_value(__reduce_max_sync(0xffffffffu, order_key(mx)));
      float sum = 0.f;
#pragma unroll
      for (int j = 0; j < J; ++j) {
        v[j] = ((valid >> j) & 1u) ? __expf(v[j] - M) : 0.f;
        sum += v[j];
      }
      const float inv = 1.f / warp_sum(sum);
      float* prow = sP + warp * kMaxExperts;
#pragma unroll
      for (int j = 0; j < J; ++j)
        if ((valid >> j) & 1u) {
          const float pv = v[j] * inv;
          prow[lane + 32 * j] = pv;
          if (a.probs_requested) a.probs[(size_t)t * E + lane + 32 * j] = pv;
        }
      CT_AT(10);
      // top-k over the clusters' candidates: each cluster's list is sorted (best first), so
      // k rounds of a tournament over the list heads (lane c holds cluster c's head; larger
      // score, ties to the lower id) give the winners in order; a winner's score is computed
      // exactly as in the row above
#pragma unroll
      for (int q = 0; q < kClMaxCand / 32; ++q) s_cand[warp][lane + 32 * q] = cd[q];
      __syncwarp();
      int head = 0;
      uint2 hc = lane < n_clusters ? s_cand[warp][lane * kc] : make_uint2(0u, 0xffffffffu);
      int my_idx = -1;
      float my_val = 0.f;
      for (int r = 0; r < kc; ++r) {
        const uint32_t kmax = __reduce_max_sync(0xffffffffu, hc.x);
        const uint32_t imin = __reduce_min_sync(0xffffffffu, hc.x == kmax ? hc.y : 0xffffffffu);
        if (lane == r) {
          my_idx = (int)imin;
          my_val = __expf(key_value(kmax) - M) * inv;
        }
        if (hc.x == kmax && hc.y == imin) {
          ++head;
          hc = head < kc ? s_cand[warp][lane * kc + head] : make_uint2(0u, 0xffffffffu);
        }
      }
      CT_AT(11);
      if (a.mode == DMOE_ROUTE_BLOCK) {
        // TopKMask: the kc winners into the zeroed row of token t in the CTA that routes
        // its block (block b: CTA b mod 8)
        if (lane < kc)
          st_peer_f32(peer_addr(sHat + t * kMaxExperts + my_idx, (uint32_t)((t / B) % kCl)),
                      my_val);
      } else {
        float tot = 0.f;
        for (int r = 0; r < k; ++r) tot += __shfl_sync(0xffffffffu, my_val, r);
        if (lane < k) {
          a.topk_idx[(size_t)t * k + lane] = my_idx;
          a.topk_gate[(size_t)t * k + lane] = my_val / tot;
          st_peer_u32(peer_addr(&sIdx[t * k + lane], 0), (uint32_t)my_idx);
        }
      }
    }
  }
  cluster_sync();
  CT_AT(5);

  // ---- 4. Algorithm 1: block b by CTA b mod 8 (Aggregate .. Top-P and the k floor), then
  // MaskOutside + TopK by the warp that scored each token, on its own score row
  if (a.mode == DMOE_ROUTE_BLOCK) {
    __shared__ int order[kMaxExperts];
    int* sCore = reinterpret_cast<int*>(dsm + kOffCore);    // [8 warps][1 + kMaxExperts]
    for (int b = (int)rank; b < a.n_blocks; b += kCl) {
      const int t0 = b * B;
      // block top-k: the coreset (k experts) is the routing of every token of the block; it
      // is published for the expert launch as soon as it is known
      const int size = block_coreset_steps(
          E, kc, B, a.top_p, [&](int i, int e) { return sHat[(t0 + i) * kMaxExperts + e]; }, order,
          a.coreset != nullptr ? a.coreset + (size_t)b * E : nullptr,
          a.coreset_size != nullptr ? a.coreset_size + b : nullptr,
          a.spec_words != nullptr && !a.spec_mask && a.top_p <= 0.f && kc == k
              ? a.spec_words + (size_t)b * spec_words(k)
              : nullptr,
          sHat + (size_t)t0 * kMaxExperts, kMaxExperts);
      if (a.spec_words != nullptr && a.spec_mask && warp == 0)
        publish_coreset_mask(a.spec_words + (size_t)b * kSpecMaskWords, order, size);
      CT_AT(25);
      // the coreset to the scoring warp of every token of the block (token t: CTA t / 8,
      // warp t mod 8): size, then the members in sorted order
      for (int i = tid; i < B * (size + 1); i += 256) {
        const int tt = t0 + i / (size + 1), c = i % (size + 1);
        st_peer_u32(peer_addr(sCore + (tt & 7) * (1 + kMaxExperts) + c, (uint32_t)(tt >> 3)),
                    (uint32_t)(c == 0 ? size : order[c - 1]));
      }
      __syncthreads();
    }
    CT_AT(12);
    cluster_sync();
    CT_AT(26);
    {
      const int t = 8 * (int)rank + warp;
      if (t < T) {
        const int* core = sCore + warp * (1 + kMaxExperts);
        const int size = core[0];
        const float* prow = sP + warp * kMaxExperts;
        int my_e = -1;
        float my_v = 0.f;
        if (size <= 32) {
          // one member per lane: k rounds of a tournament (larger score, ties to lower id)
          const int e = lane < size ? core[1 + lane] : -1;
          uint32_t key = e >= 0 ? order_key(prow[e]) : 0u;
          for (int r = 0; r < k; ++r) {
            const uint32_t kmax = __reduce_max_sync(0xffffffffu, key);
            const uint32_t imin =
                __reduce_min_sync(0xffffffffu, key == kmax ? (uint32_t)e : 0xffffffffu);
            if (lane == r) {
              my_e = (int)imin;
              my_v = key_value(kmax);
            }
            if (key == kmax && (uint32_t)e == imin) key = 0u;
          }
        } else {
          float cv[8];
          int ce[8];
          uint32_t valid = 0;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int c = lane + 32 * j;
            ce[j] = c < size ? core[1 + c] : 0;
            if (c < size) valid |= 1u << j;
            cv[j] = c < size ? prow[ce[j]] : 0.f;
          }
          warp_topk(cv, ce, valid, k, my_e, my_v);
        }
        CT_AT(27);
        float g = 0.f;
        for (int r = 0; r < k; ++r) g += __shfl_sync(0xffffffffu, my_v, r);
        if (lane < k) {
          a.topk_idx[(size_t)t * k + lane] = my_e;
          a.topk_gate[(size_t)t * k + lane] = my_v / g;
          st_peer_u32(peer_addr(&sIdx[t * k + lane], 0), (uint32_t)my_e);
        }
      }
    }
  } else if (rank == 0) {
    if (a.coreset != nullptr)
      for (int i = tid; i < a.n_blocks * E; i += 256) a.coreset[i] = -1;
    if (a.coreset_size != nullptr)
      for (int i = tid; i < a.n_blocks; i += 256) a.coreset_size[i] = 0;
  }
  CT_AT(13);
  cluster_sync();
  CT_AT(6);

  // ---- 5. dispatch
  if (rank == 0) {
    if (f.dsp.n_unique != nullptr)
      dispatch_small_cta(sIdx, T, E, k, f.dsp.n_unique, f.dsp.unique_ids, f.dsp.offsets,
                         f.dsp.rows, f.dsp.pos, f.dsp.err);
    if (tid == 0) *f.ticket = 0;  // ready for the next call
    CT_AT(7);
  }
  KLOG(DMOE_KERNEL_ROUTER, 1);
}

typedef CUresult (*EncodeTiledFnC)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFnC encoder() {
  static EncodeTiledFnC fn = nullptr;
  if (fn == nullptr) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFnC>(ptr);
  }
  return fn;
}

// Dynamic shared memory of a launch: the W_r and x slices, and for a routing launch the
// TopKMask rows after them (a logits-only launch stops before it needs them, and its
// smaller footprint lets two CTAs share an SM, so that the 64-token tiles of a large
// forward run in one wave)
size_t route_cluster_smem(bool logits_only) {
  const size_t stage1 = (size_t)kOffHat;
  const size_t stage4 = (size_t)kOffHat + (size_t)kClMaxTok * kMaxExperts * 4;
  return (logits_only || stage1 > stage4 ? stage1 : stage4) + 1024;
}

}  // namespace

#ifdef DMOE_TRACE
extern "C" int dmoe_debug_ctrace(void* host) {
  return (int)cudaMemcpyFromSymbol(host, g_ctrace, sizeof(g_ctrace));
}
DMOE_KLOG_EXPORT(dmoe_debug_klog_router)
extern "C" int dmoe_debug_ctrace_clear() {
  static uint64_t zeros[64 * 8 * 64];
  return (int)cudaMemcpyToSymbol(g_ctrace, zeros, sizeof(g_ctrace));
}
#endif

bool route_cluster_logits_ok(int d, int E) {
  // d % 256: each CTA's slice splits into eight runs of whole float4 groups
  return d % (kCl * 32) == 0 && d / kCl <= kClMaxDChunk && E % 8 == 0;
}

bool route_cluster_ok(int T, int d, int E) {
  return T <= kClMaxTok && route_cluster_logits_ok(d, E);
}

namespace {
cudaError_t launch_cluster_common(const RouterArgs& a, const DispatchArgs* dsp,
                                  int32_t* tickets, cudaStream_t s, bool logits_only);
}

cudaError_t launch_route_cluster(const RouterArgs& a, const DispatchArgs* dsp, int32_t* tickets,
                                 cudaStream_t s) {
  return launch_cluster_common(a, dsp, tickets, s, false);
}

cudaError_t launch_logits_cluster(const RouterArgs& a, cudaStream_t s) {
  return launch_cluster_common(a, nullptr, nullptr, s, true);
}

namespace {
cudaError_t launch_cluster_common(const RouterArgs& a, const DispatchArgs* dsp,
                                  int32_t* tickets, cudaStream_t s, bool logits_only) {
  EncodeTiledFnC enc = encoder();
  if (enc == nullptr) return cudaErrorInvalidValue;
  ClusterArgs f{};
  const int DC = a.d / kCl;
  {
    const cuuint64_t dims[2] = {(cuuint64_t)a.E, (cuuint64_t)a.d};
    const cuuint64_t strides[1] = {(cuuint64_t)a.E * 4};
    const cuuint32_t box[2] = {(cuuint32_t)kClExp, (cuuint32_t)DC};
    const cuuint32_t estr[2] = {1, 1};
    if (enc(&f.wmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(a.w_r), dims, strides,
            box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t dims[2] = {(cuuint64_t)a.d, (cuuint64_t)a.T};
    const cuuint64_t strides[1] = {(cuuint64_t)a.d * 2};
    f.box_rows = logits_only ? kClMaxTok : (a.T + 15) & ~15;
    const cuuint32_t box[2] = {64u, (cuuint32_t)f.box_rows};
    const cuuint32_t estr[2] = {1, 1};
    if (enc(&f.xmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<__nv_bfloat16*>(a.x), dims,
            strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  f.r = a;
  if (dsp != nullptr) f.dsp = *dsp;
  f.ticket = tickets;
  f.logits_only = logits_only ? 1 : 0;
  const size_t smem = route_cluster_smem(logits_only);
  const size_t smem_max = route_cluster_smem(false);
  static int mask = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 31 || !(mask & (1 << dev))) {
    cudaError_t e = cudaFuncSetAttribute(route_cluster_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem_max);
    if (e != cudaSuccess) return e;
    if (dev < 31) mask |= 1 << dev;
  }
  dim3 grid(kCl, (a.E + kClExp - 1) / kClExp,
            logits_only ? (a.T + kClMaxTok - 1) / kClMaxTok : 1);
  // programmatic dependent launch: the set-up overlaps the previous kernel on the stream;
  // the kernel waits for it (griddepcontrol.wait) before it reads anything
  return launch_cluster(route_cluster_kernel, grid, dim3(256), smem, s, kCl, true, f);
}
}  // namespace

}  // namespace dmoe
