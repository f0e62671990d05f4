// Expert execution of the MoE layer: grouped SwiGLU FFN over the unique experts of one
// forward (plus the shared expert), on tcgen05 tensor cores.
//
// Both GEMMs are "swap-AB": the expert weights are the MMA's M operand (128 weight rows per
// tile, streamed by TMA with the 128-byte swizzle), the few tokens routed to an expert are
// the N operand, K is the reduction dimension, and the fp32 accumulator lives in TMEM.
//
//   gather_kernel       x rows in dispatch order -> xperm [T*k, d]; clears the tile counters
//   moe_experts_kernel  one persistent launch with two kinds of unit:
//     gate/up unit      (group, 64 rows of I, token tile): the A tile stacks 64 rows of
//                       W_gate over the same 64 rows of W_up, so one M=128 MMA chain gives
//                       gate (TMEM lanes 0-63) and up (lanes 64-127) of those rows; the
//                       epilogue warps holding "up" pass it through shared memory to the
//                       warps holding "gate", which write h = silu(gate) * up as bf16 H and
//                       then publish the tile (h_ready counter)
//     down unit         (group, 128 rows of d, token tile): D = W_down * H^T; the epilogue
//                       stores the rows per (token, slot) as bf16 (half the bytes of fp32
//                       through HBM twice; the combine adds them in fp32)
//   combine_kernel      y_t = sum over slots (slot order) of g_tj * row + shared -> bf16
//
// A group is one unique expert (dispatch order) or the shared expert (all T tokens). The
// expert kernel is warp-specialised: warp 0 issues TMA, warp 1 issues MMAs, warps 2-9 run
// the epilogue; each pipeline stage carries K = 128 (two 128-B-wide boxes per operand; 64
// for 256-row token tiles). The unit list is derived on
// the device from the dispatch output, so no host round-trip is needed. Consecutive
// kernels are chained with programmatic dependent launch: each kernel's set-up (barriers,
// TMEM, tensor-map prefetch) overlaps the previous kernel, and griddepcontrol.wait orders
// the reads of its outputs.
#include <math.h>

#include <mutex>

#include "dmoe_internal.cuh"
#include "sm100_ptx.cuh"
#include "trace_log.cuh"

namespace dmoe {
namespace {

constexpr int kThreads = 320;                      // 10 warps
constexpr int kEpiThreads = 256;                   // warps 2-9: the epilogue
constexpr int kBoxBytes = 64 * 128;                // one TMA box: 64 rows x 128 B
constexpr int kMaxKBoxes = 2;                      // K boxes per stage: 1 or 2 (K = 64, 128)
constexpr int kATileBytes = kTileM * 128;          // 16 KB: 128 rows x 64 K (one K box)
constexpr int kMaxGroups = kMaxExperts + 1;
constexpr uint64_t kWaitTimeoutNs = 1000000000ull;  // 1 s
constexpr int kMaxStages = 8;
constexpr int64_t kDownPrefetchMax = (int64_t)64 << 20;   // half of the 129 MB L2
constexpr int kXchgStride = 17;                    // floats per row of the exchange buffers
constexpr int kSpecBlocks = 64;                    // blocks of a block top-k forward, at most
constexpr int kSpecPairs = kSpecBlocks * kMaxTopK;   // (block, coreset member) pairs, at most

struct GemmParams {
  const int32_t* n_unique;
  const int32_t* unique_ids;
  const int32_t* offsets;
  const int32_t* rows;    // dispatch rows: t * k + slot (the x row of a routed token row)
  __nv_bfloat16* h;       // [T*k, I]
  __nv_bfloat16* hs;      // [T, Is]
  __nv_bfloat16* yslot;   // [T*k, d] bf16 (the combine sums them in fp32)
  __nv_bfloat16* yshared; // [T, d] bf16
  int32_t* h_ready;       // [(E+1) * ntiles]: gate/up tiles done per (group, token tile)
  DevErrRecord* err;
  const void* w_down;     // routed W_down, prefetched into L2 for the unique experts
  const void* ws_gate; const void* ws_up; const void* ws_down;  // shared, prefetched if set
  int T, d, E, k, I, Is;
  int n_max;              // token tile = rows of the B box
  int n_half;             // rows of the half box (token tiles of at most this many rows)
  int kbs;                // K boxes per stage (1 for 256-row token tiles, else 2)
  int dpair;              // 128-row tiles of W_down per down unit (2: a pair sharing the H
                          // stages, K = 64 per stage; 1)
  int ntiles;             // token tiles per group at most
  int stages;
  int n_acc;              // accumulator buffers in TMEM
  uint32_t tmem_cols;
  int has_shared;
  // Block top-k (spec_words != nullptr): the groups come from the coresets that the block
  // routing launch publishes (n_blocks blocks of blk rows). The unique experts are their
  // union, ascending; an expert's token rows are its blocks' rows in block order, which is
  // the dispatch's order. This launch then does the dispatch itself: its CTAs copy every
  // (block, coreset member) pair's rows of x to their place in xperm (x_ready[g ntiles + n]
  // counts the copied rows of token tile n of group g; a gate/up unit loads its tile's rows
  // once they are all there) and write
  // n_unique, unique_ids and pos (the row of every (token, slot), from topk_idx).
  const uint32_t* spec_words;
  int n_blocks, blk;
  const int32_t* topk_idx;
  int32_t* pos_out;
  int32_t* n_unique_out;
  int32_t* unique_ids_out;
  int32_t* x_ready;          // [groups x ntiles], zero at the start (the routing launch
                             // clears it)
  const __nv_bfloat16* x;
  __nv_bfloat16* xperm;
};

struct Maps {
  CUtensorMap wg, wu, sg, su;   // gate/up weights, 64-row boxes (routed [E*I,d], shared [Is,d])
  CUtensorMap wd, sd;           // down weights, 128-row boxes (routed [E*d,I], shared [d,Is])
  CUtensorMap xp, x;            // gate/up token rows: xperm [T*k,d], x [T,d]
  CUtensorMap h, hs;            // down token rows: H [T*k,I], Hs [T,Is]
  CUtensorMap xph, hh;          // xperm and H with half-height boxes (small token tiles)
};

using ptx::fence_proxy_async_global;
using ptx::ld_acquire;
using ptx::named_bar_sync;
using ptx::red_release_add;

__device__ __forceinline__ float silu_f(float z) { return z / (1.f + __expf(-z)); }

// A bf16 store that asks L2 to keep the line (the slot rows are read back by the combine
// right after this launch, while the weights stream through L2 with evict-first)
__device__ __forceinline__ void st_bf16_keep(__nv_bfloat16* p, __nv_bfloat16 v, uint64_t pol) {
  asm volatile("st.global.L2::cache_hint.b16 [%0], %1, %2;" ::"l"(p),
               "h"(*reinterpret_cast<const unsigned short*>(&v)), "l"(pol)
               : "memory");
}

// AND of `v` over the kEpiThreads epilogue threads (named barrier 1), so that they take the
// warp-collective TMEM loads, or leave the unit loop, together
__device__ __forceinline__ bool epi_all_threads(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, 1, %2, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v), "n"(kEpiThreads)
      : "memory");
  return r != 0;
}

// Debug builds (-DDMOE_TRACE) record a per-CTA timeline of the expert kernel: slot 0 entry,
// 1 after the unit list, 62 exit; for the i-th unit of the CTA (i < 8), at 2 + 6i: unit id,
// producer start, last TMA issued, H ready (down units; for block top-k gate/up units: the
// group's token rows copied), last MMA commit, epilogue done;
// at 50 + i: the epilogue's first TMEM read of that unit; 63: this CTA's copies of the
// token rows done (block top-k).
#ifdef DMOE_TRACE
__device__ uint64_t g_trace[kMaxPersistentCtas * 64];
#define DMOE_TRACE_AT(slot) (g_trace[blockIdx.x * 64 + (slot)] = ptx::globaltimer_ns())
#define DMOE_TRACE_SET(slot, v) (g_trace[blockIdx.x * 64 + (slot)] = (uint64_t)(v))
#else
#define DMOE_TRACE_AT(slot) ((void)0)
#define DMOE_TRACE_SET(slot, v) ((void)0)
#endif

// The expert FFN of one forward in one persistent launch. Units: first every gate/up tile
// (group, 64 rows of I, token tile), then every down tile (group, 128 rows of d, token
// tile); the shared expert's group comes first in both lists. A CTA takes units
// blockIdx.x, blockIdx.x + gridDim.x, ... so its gate/up units always precede its down
// units and a gate/up unit never waits on another unit. A down unit loads its W_down
// tiles at once and only then waits (bounded) for the gate/up tiles of its token rows to
// be published (h_ready), so weight streaming of both phases overlaps. kSpec: the block
// top-k form (GemmParams::spec_words), compiled separately so that the other form carries
// none of its code.
template <bool kSpec>
__global__ void __launch_bounds__(kThreads, 1)
moe_experts_kernel(const __grid_constant__ Maps tm, const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = ptx::smem_addr(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);  // 1024-B aligned

  const int stages = p.stages;
  const int kbs = p.kbs;                                      // K boxes per stage
  const int stage_k = kbs * kTileK;
  const uint32_t a_stage = (uint32_t)kbs * kATileBytes;
  const uint32_t b_box = (uint32_t)p.n_max * 128u;            // one B box (slot size)
  const uint32_t b_stage = (uint32_t)kbs * b_box;
  const uint32_t off_a = 0;
  const uint32_t off_b = off_a + (uint32_t)stages * a_stage;
  const uint32_t off_x = off_b + (uint32_t)stages * b_stage;
  const uint32_t x_bytes = 2u * 128u * kXchgStride * 4u;       // 2 x [128][17] fp32
  const uint32_t off_bar = (off_x + x_bytes + 7u) & ~7u;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + off_bar);
  uint64_t* empty = full + stages;
  uint64_t* acc_full = empty + stages;
  uint64_t* acc_empty = acc_full + 4;
  uint64_t* drain = acc_empty + 4;
  int* misc = reinterpret_cast<int*>(drain + 1);
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(misc + 0);
  volatile int* s_abort = misc + 1;
  int* s_sched = misc + 4;                         // G, U, gu_units, dn_units, dpair
  int* gu_prefix = misc + 12;                      // [kMaxGroups + 1], by slot
  int* dn_prefix = gu_prefix + (kMaxGroups + 1);   // [kMaxGroups + 1], by slot
  int* g_row0 = dn_prefix + (kMaxGroups + 1);      // by group
  int* g_cnt = g_row0 + kMaxGroups;
  int* g_e = g_cnt + kMaxGroups;
  // block top-k planning: blocks per expert (bit b of s_bmask[2e + b / 32]), each block's
  // coreset, per expert its group and the blocks of the groups before it
  uint32_t* s_bmask = reinterpret_cast<uint32_t*>(g_e + kMaxGroups);   // [2 * kMaxExperts]
  int16_t* s_upos = reinterpret_cast<int16_t*>(s_bmask + 2 * kMaxExperts);   // [kMaxExperts]
  int16_t* s_bpos = s_upos + kMaxExperts;                                      // [kMaxExperts]
  uint8_t* s_bcore = reinterpret_cast<uint8_t*>(s_bpos + kMaxExperts);   // [kSpecPairs]
  float* xchg = reinterpret_cast<float*>(smem + off_x);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) DMOE_TRACE_AT(0);
  KLOG(DMOE_KERNEL_EXPERTS, 0);

  if (tid == 0) {
    for (int s = 0; s < stages; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 4; ++a) {
      ptx::mbar_init(&acc_full[a], 1);
      ptx::mbar_init(&acc_empty[a], kEpiThreads);
    }
    ptx::mbar_init(drain, 1);
    ptx::fence_mbarrier_init();
    *s_abort = 0;
    ptx::prefetch_tensormap(&tm.wg);
    ptx::prefetch_tensormap(&tm.wu);
    ptx::prefetch_tensormap(&tm.wd);
    ptx::prefetch_tensormap(&tm.xp);
    ptx::prefetch_tensormap(&tm.h);
  }
  if (warp == 1) {
    ptx::tmem_alloc(s_tmem, p.tmem_cols);
    ptx::tmem_relinquish();
  }
  constexpr bool spec = kSpec;
  if (!spec) pdl_wait();  // dispatch output and the gathered rows are complete from here on

  // ---------------- groups and unit lists (slot 0 = the shared expert when present)
  if (warp == 0) {
    int U;
    if (spec) {
      // Block top-k: poll every block's published coreset words until all are nonzero (a
      // nonzero word is complete), recording each block's members and, per expert, the
      // blocks that use it
      const int nw = spec_words(p.k), total = p.n_blocks * nw;
      for (int i = lane; i < 2 * kMaxExperts; i += 32) s_bmask[i] = 0u;
      __syncwarp();
      bool bad = false;
      const uint64_t t0 = ptx::globaltimer_ns();
      for (;;) {
        bool all = true;
        for (int i = lane; i < total; i += 32) {
          const uint32_t w = ptx::ld_relaxed_u32(p.spec_words + i);
          if (w == 0u) {
            all = false;
            continue;
          }
          const int b = i / nw, r0 = 3 * (i % nw);
#pragma unroll
          for (int j = 0; j < 3; ++j) {
            if (r0 + j >= p.k) break;
            const int e = (int)((w >> (8 * j)) & 0xffu);
            if (e >= p.E) {
              bad = true;
            } else {
              s_bcore[b * p.k + r0 + j] = (uint8_t)e;
              atomicOr(&s_bmask[2 * e + (b >> 5)], 1u << (b & 31));
            }
          }
        }
        if (__all_sync(0xffffffffu, all)) break;
        if (ptx::globaltimer_ns() - t0 > kWaitTimeoutNs) {   // the coresets did not come
          if (lane == 0) record_error(p.err, kErrTimeout, kAtGateUp, -1);
          bad = true;
          break;
        }
      }
      bad = __any_sync(0xffffffffu, bad);
      __syncwarp();
      // the unique experts ascending (lane l: experts 8l .. 8l + 7): group u's rows are its
      // blocks' rows, so it starts at blk * (blocks of the groups before it)
      int nbq[8], cu = 0, cb = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int e = 8 * lane + q;
        nbq[q] = e < p.E ? __popc(s_bmask[2 * e]) + __popc(s_bmask[2 * e + 1]) : 0;
        cu += nbq[q] > 0 ? 1 : 0;
        cb += nbq[q];
      }
      int iu = cu, ib = cb;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int a = __shfl_up_sync(0xffffffffu, iu, o);
        const int c = __shfl_up_sync(0xffffffffu, ib, o);
        if (lane >= o) { iu += a; ib += c; }
      }
      int u = iu - cu, bp = ib - cb;
#pragma unroll
      for (int q = 0; q < 8; ++q)
        if (nbq[q] > 0) {
          const int e = 8 * lane + q;
          s_upos[e] = (int16_t)u;
          s_bpos[e] = (int16_t)bp;
          g_e[u] = e;
          g_row0[u] = p.blk * bp;
          g_cnt[u] = p.blk * nbq[q];
          ++u;
          bp += nbq[q];
        }
      U = bad ? 0 : __shfl_sync(0xffffffffu, iu, 31);
      if (bad && lane == 0) record_error(p.err, kErrBadDispatch, kAtGateUp, -1);
      if (lane == 0 && p.has_shared) {
        g_row0[U] = 0;
        g_cnt[U] = p.T;
        g_e[U] = -1;
      }
      __syncwarp();
    } else {
      U = *p.n_unique;
      if (U < 0 || U > p.E) {
        if (lane == 0) record_error(p.err, kErrBadDispatch, kAtGateUp, U);
        U = 0;
      }
    }
    const int G = U + (p.has_shared ? 1 : 0);
    int carry_gu = 0, carry_dn = 0;
    for (int base = 0; base < G; base += 32) {
      const int slot = base + lane;
      int gu = 0, dn = 0;
      if (slot < G) {
        const int g = p.has_shared ? (slot == 0 ? U : slot - 1) : slot;
        int cnt, row0, e, Ig;
        if (spec) {
          cnt = g_cnt[g];
          row0 = g_row0[g];
          e = g_e[g];
          Ig = g < U ? p.I : p.Is;
        } else if (g < U) {
          row0 = p.offsets[g];
          cnt = p.offsets[g + 1] - row0;
          e = p.unique_ids[g];
          Ig = p.I;
          if (e < 0 || e >= p.E || cnt < 0 || cnt > p.T || row0 < 0 ||
              row0 + cnt > p.T * p.k) {
            record_error(p.err, kErrBadDispatch, kAtGateUp, g);
            cnt = 0;
            e = 0;
            row0 = 0;
          }
        } else {
          row0 = 0;
          cnt = p.T;
          e = -1;
          Ig = p.Is;
        }
        g_row0[g] = row0;
        g_cnt[g] = cnt;
        g_e[g] = e;
        const int nt = (cnt + p.n_max - 1) / p.n_max;
        gu = nt * (Ig / 64);
        dn = nt * (p.d / kTileM);
      }
      int igu = gu, idn = dn;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int a = __shfl_up_sync(0xffffffffu, igu, o);
        const int b = __shfl_up_sync(0xffffffffu, idn, o);
        if (lane >= o) { igu += a; idn += b; }
      }
      if (slot < G) {
        gu_prefix[slot + 1] = carry_gu + igu;
        dn_prefix[slot + 1] = carry_dn + idn;
      }
      carry_gu += __shfl_sync(0xffffffffu, igu, 31);
      carry_dn += __shfl_sync(0xffffffffu, idn, 31);
    }
    // pairs of down tiles only when the down units are many per CTA (a pair unit pulls 25 %
    // less per tile but holds less of its weights before H is ready: with about one or two
    // single units per CTA it lengthens the tail); a pair count is the single count / 2
    const int dpair = (p.dpair == 2 && carry_dn >= 4 * (int)gridDim.x) ? 2 : 1;
    if (dpair == 2) {
      __syncwarp();
      for (int i = lane; i <= G; i += 32) dn_prefix[i] /= 2;
      carry_dn /= 2;
    }
    if (lane == 0) {
      gu_prefix[0] = 0;
      dn_prefix[0] = 0;
      s_sched[0] = G;
      s_sched[1] = U;
      s_sched[2] = carry_gu;
      s_sched[3] = carry_dn;
      s_sched[4] = dpair;
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  const int G = s_sched[0], U = s_sched[1], n_gu = s_sched[2], n_dn = s_sched[3];
  const int dpair = s_sched[4];   // 128-row tiles of W_down per down unit
  const int units = n_gu + n_dn;
  if (tid == 0) DMOE_TRACE_AT(1);
  if (tid == 64) {
    // Pull the down-projection weights of every unique expert into L2 now, spread over all
    // CTAs: the down units of the second wave then read them from L2, and HBM keeps
    // streaming while the gate/up results are produced and published. Only while they
    // fit in half of L2: beyond that the prefetched lines are evicted before their use
    // and only add HBM traffic (token routing at 2048 tokens: 256 experts, 537 MB).
    L2Prefetch pf;
    pf.ptr[2] = p.w_down;
    pf.bytes = (int64_t)p.d * p.I * 2;
    const int64_t per = (pf.bytes + kPrefetchChunk - 1) / kPrefetchChunk;
    const int total = (int)(3 * per * U);
    if (pf.bytes * U <= kDownPrefetchMax)
      for (int c = (int)(2 * per * U) + blockIdx.x; c < total; c += gridDim.x)
        l2_prefetch_chunk(pf, spec ? g_e : p.unique_ids, U, c);
    if (p.ws_gate != nullptr) {
      L2Prefetch sp;
      sp.ptr[0] = p.ws_gate;
      sp.ptr[1] = p.ws_up;
      sp.ptr[2] = p.ws_down;
      sp.bytes = (int64_t)p.d * p.Is * 2;
      const int sper = (int)((sp.bytes + kPrefetchChunk - 1) / kPrefetchChunk);
      for (int c = blockIdx.x; c < 3 * sper; c += gridDim.x) l2_prefetch_chunk(sp, nullptr, 1, c);
    }
  }

  // unit -> phase, group, m tile, n tile
  struct Unit { bool gu; int g, m, n; };
  auto decode = [&](int u) -> Unit {
    Unit r;
    r.gu = u < n_gu;
    const int* pre = r.gu ? gu_prefix : dn_prefix;
    const int v = r.gu ? u : u - n_gu;
    int lo = 0, hi = G - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (pre[mid] <= v) lo = mid; else hi = mid - 1;
    }
    r.g = p.has_shared ? (lo == 0 ? U : lo - 1) : lo;
    // token tile innermost: the CTAs that take a weight tile's token tiles take them at
    // the same time, so that the tile comes from HBM once and from L2 for the others
    const int nt = (g_cnt[r.g] + p.n_max - 1) / p.n_max;
    const int local = v - pre[lo];
    r.m = local / nt;
    r.n = local - r.m * nt;
    return r;
  };
  auto wait = [&](uint64_t* bar, uint32_t parity, int value) -> bool {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::globaltimer_ns();
    for (uint32_t i = 1;; ++i) {
      if (ptx::mbar_try_wait(bar, parity)) return true;
      if ((i & 63u) == 0u) {
        if (*s_abort) return false;
        if (ptx::globaltimer_ns() - t0 > kWaitTimeoutNs) {
          record_error(p.err, kErrTimeout, kAtGateUp, value);
          *s_abort = 1;
          return false;
        }
      }
    }
  };

  if (warp == 0) {
    // ================= TMA producer
    if (lane == 0) {
      const uint64_t pol_first = ptx::policy_evict_first();   // weights read by one tile
      const uint64_t pol_norm = ptx::policy_evict_normal();   // ... or by several
      const uint64_t pol_x = ptx::policy_evict_last();    // activations: re-read by tiles
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      bool ok = true;
      int li = 0;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++li) {
        const Unit un = decode(u);
        const bool shared = un.g >= U;
        const uint64_t pol_w = g_cnt[un.g] > p.n_max ? pol_norm : pol_first;
        // a routed token tile of at most n_half rows loads the half-height box
        const int nvalid = min(p.n_max, g_cnt[un.g] - un.n * p.n_max);
        const bool half = !shared && nvalid <= p.n_half;
        const uint32_t b_bytes = (uint32_t)kbs * (half ? (uint32_t)p.n_half * 128u : b_box);
        const uint32_t tx_bytes = a_stage + b_bytes;
        if (li < 8) { DMOE_TRACE_SET(2 + 6 * li, u); DMOE_TRACE_AT(3 + 6 * li); }
        if (un.gu) {
          const int arow = shared ? un.m * 64 : g_e[un.g] * p.I + un.m * 64;
          const int brow = (shared ? 0 : g_row0[un.g]) + un.n * p.n_max;
          const CUtensorMap* mg = shared ? &tm.sg : &tm.wg;
          const CUtensorMap* mu = shared ? &tm.su : &tm.wu;
          const CUtensorMap* mb = shared ? &tm.x : (half ? &tm.xph : &tm.xp);
          const int kc = p.d / stage_k;
          auto load_gu = [&](int st, int c, bool with_a, bool with_b) {
            uint8_t* a_dst = smem + off_a + st * a_stage;
            uint8_t* b_dst = smem + off_b + st * b_stage;
            for (int kb = 0; kb < kbs; ++kb) {
              const int kx = c * stage_k + kb * kTileK;
              if (with_a) {
                ptx::tma_load_2d(a_dst + kb * kATileBytes, mg, &full[st], kx, arow, pol_w);
                ptx::tma_load_2d(a_dst + kb * kATileBytes + kBoxBytes, mu, &full[st], kx, arow,
                                 pol_w);
              }
              if (with_b) ptx::tma_load_2d(b_dst + kb * b_box, mb, &full[st], kx, brow, pol_x);
            }
          };
          int c0 = 0;
          if (spec && !shared) {
            // block top-k: the weight stages first, the token rows once this launch's copies
            // of the tile's rows are all in xperm
            const int pre = kc < stages ? kc : stages;
            const int stage0 = stage;
            for (int c = 0; c < pre; ++c) {
              if (!wait(&empty[stage], phase ^ 1u, u)) { ok = false; break; }
              ptx::mbar_arrive_expect_tx(&full[stage], tx_bytes);
              load_gu(stage, c, true, false);
              ++issued;
              if (++stage == stages) { stage = 0; phase ^= 1u; }
            }
            if (!ok) break;
            // the rows of this token tile (a pair's rows lie in one tile: n_max % blk == 0)
            const int32_t* flag = p.x_ready + un.g * p.ntiles + un.n;
            const int need = min(p.n_max, g_cnt[un.g] - un.n * p.n_max);
            if (ld_acquire(flag) < need) {
              const uint64_t t0 = ptx::globaltimer_ns();
              while (ld_acquire(flag) < need) {
                if (*s_abort) { ok = false; break; }
                if (ptx::globaltimer_ns() - t0 > kWaitTimeoutNs) {
                  record_error(p.err, kErrTimeout, kAtGather, u);
                  *s_abort = 1;
                  ok = false;
                  break;
                }
              }
            }
            fence_proxy_async_global();   // the copies (generic stores) before these loads
            if (li < 8) DMOE_TRACE_AT(5 + 6 * li);
            int st = stage0;
            for (int c = 0; c < pre; ++c) {
              if (ok)
                load_gu(st, c, false, true);
              else
                ptx::mbar_complete_tx_local(&full[st], b_bytes);   // keep the accounting whole
              if (++st == stages) st = 0;
            }
            if (!ok) break;
            c0 = pre;
          }
          for (int c = c0; c < kc; ++c) {
            if (!wait(&empty[stage], phase ^ 1u, u)) { ok = false; break; }
            ptx::mbar_arrive_expect_tx(&full[stage], tx_bytes);
            load_gu(stage, c, true, true);
            ++issued;
            if (++stage == stages) { stage = 0; phase ^= 1u; }
          }
        } else {
          // a pair unit takes 128-row tiles 2m and 2m+1 of W_down over K = 64 per stage (its
          // two A boxes side by side at the same K), both against the stage's one H box
          const bool pr = dpair == 2;
          const int ksz = pr ? kTileK : stage_k;               // K per stage
          const int nbb = pr ? 1 : kbs;                        // B boxes per stage
          const uint32_t b_bytes_d =
              (uint32_t)nbb * (half ? (uint32_t)p.n_half * 128u : b_box);
          const uint32_t tx_d = a_stage + b_bytes_d;
          const int Kg = shared ? p.Is : p.I;
          const int arow = (shared ? 0 : g_e[un.g] * p.d) + un.m * dpair * kTileM;
          const int brow = (shared ? 0 : g_row0[un.g]) + un.n * p.n_max;
          const CUtensorMap* ma = shared ? &tm.sd : &tm.wd;
          const CUtensorMap* mb = shared ? &tm.hs : (half ? &tm.hh : &tm.h);
          const int kc = Kg / ksz;
          const int pre = kc < stages ? kc : stages;
          const int stage0 = stage;
          auto load_a = [&](int st, int c) {
            uint8_t* a_dst = smem + off_a + st * a_stage;
            if (pr) {
              ptx::tma_load_2d(a_dst, ma, &full[st], c * ksz, arow, pol_w);
              ptx::tma_load_2d(a_dst + kATileBytes, ma, &full[st], c * ksz, arow + kTileM, pol_w);
            } else {
              for (int kb = 0; kb < kbs; ++kb)
                ptx::tma_load_2d(a_dst + kb * kATileBytes, ma, &full[st], c * ksz + kb * kTileK,
                                 arow, pol_w);
            }
          };
          // weights first: they do not depend on the gate/up phase
          for (int c = 0; c < pre; ++c) {
            if (!wait(&empty[stage], phase ^ 1u, u)) { ok = false; break; }
            ptx::mbar_arrive_expect_tx(&full[stage], tx_d);
            load_a(stage, c);
            ++issued;
            if (++stage == stages) { stage = 0; phase ^= 1u; }
          }
          if (!ok) break;
          // then the H rows, once every gate/up tile of this token tile is published
          const int target = Kg / 64;
          const int32_t* flag = p.h_ready + un.g * p.ntiles + un.n;
          if (ld_acquire(flag) < target) {
            const uint64_t t0 = ptx::globaltimer_ns();
            while (ld_acquire(flag) < target) {
              __nanosleep(64);
              if (*s_abort) { ok = false; break; }
              if (ptx::globaltimer_ns() - t0 > kWaitTimeoutNs) {
                record_error(p.err, kErrTimeout, kAtDown, u);
                *s_abort = 1;
                ok = false;
                break;
              }
            }
          }
          fence_proxy_async_global();
          if (li < 8) DMOE_TRACE_AT(5 + 6 * li);
          int st = stage0;
          for (int c = 0; c < pre; ++c) {
            if (ok) {
              uint8_t* b_dst = smem + off_b + st * b_stage;
              for (int kb = 0; kb < nbb; ++kb)
                ptx::tma_load_2d(b_dst + kb * b_box, mb, &full[st], c * ksz + kb * kTileK, brow,
                                 pol_x);
            } else {
              // keep the barrier accounting whole: complete the stage without B data
              ptx::mbar_complete_tx_local(&full[st], b_bytes_d);
            }
            if (++st == stages) st = 0;
          }
          if (!ok) break;
          for (int c = pre; c < kc; ++c) {
            if (!wait(&empty[stage], phase ^ 1u, u)) { ok = false; break; }
            ptx::mbar_arrive_expect_tx(&full[stage], tx_d);
            load_a(stage, c);
            uint8_t* b_dst = smem + off_b + stage * b_stage;
            for (int kb = 0; kb < nbb; ++kb)
              ptx::tma_load_2d(b_dst + kb * b_box, mb, &full[stage], c * ksz + kb * kTileK, brow,
                               pol_x);
            ++issued;
            if (++stage == stages) { stage = 0; phase ^= 1u; }
          }
        }
        if (li < 8) DMOE_TRACE_AT(4 + 6 * li);
      }
      if (!ok) {
        // let the copies already in flight land before the CTA exits
        int st = stage;
        uint32_t ph = phase;
        const int n = issued < stages ? issued : stages;
        for (int i = 0; i < n; ++i) {
          if (--st < 0) { st = stages - 1; ph ^= 1u; }
          const uint64_t t0 = ptx::globaltimer_ns();
          while (!ptx::mbar_try_wait(&full[st], ph) &&
                 ptx::globaltimer_ns() - t0 < kWaitTimeoutNs / 10) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ================= MMA issuer
    if (lane == 0) {
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool ok = true;
      int li = 0;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++li) {
        const Unit un = decode(u);
        const bool shared = un.g >= U;
        const bool pr = !un.gu && dpair == 2;     // a pair of down tiles, two accumulators
        const int Kg = un.gu ? p.d : (shared ? p.Is : p.I);
        const int kc = Kg / (pr ? kTileK : stage_k);
        const int nvalid = min(p.n_max, g_cnt[un.g] - un.n * p.n_max);
        const uint32_t n_mma = (uint32_t)((nvalid + 15) & ~15);
        const uint32_t idesc = ptx::idesc_bf16(kTileM, n_mma);
        // the second accumulator of a pair: the next slot
        int acc2 = acc + 1;
        uint32_t acc2_phase = acc_phase;
        if (acc2 == p.n_acc) { acc2 = 0; acc2_phase ^= 1u; }
        if (!wait(&acc_empty[acc], acc_phase ^ 1u, u)) { ok = false; break; }
        if (pr && !wait(&acc_empty[acc2], acc2_phase ^ 1u, u)) { ok = false; break; }
        ptx::tc_fence_after();
        const uint32_t d0 = tmem_base + (uint32_t)acc * (uint32_t)p.n_max;
        const uint32_t d1 = tmem_base + (uint32_t)acc2 * (uint32_t)p.n_max;
        for (int c = 0; c < kc; ++c) {
          if (!wait(&full[stage], phase, u)) { ok = false; break; }
          ptx::tc_fence_after();
          if (!*s_abort) {
            const uint32_t a0 = ptx::smem_addr(smem + off_a + stage * a_stage);
            const uint32_t b0 = ptx::smem_addr(smem + off_b + stage * b_stage);
            if (pr) {
#pragma unroll
              for (int kk = 0; kk < kTileK / 16; ++kk) {
                const uint64_t bd = ptx::sdesc_k_sw128(b0 + kk * 32);
                const uint32_t accum = (c > 0 || kk > 0) ? 1u : 0u;
                ptx::mma_bf16(d0, ptx::sdesc_k_sw128(a0 + kk * 32), bd, idesc, accum);
                ptx::mma_bf16(d1, ptx::sdesc_k_sw128(a0 + kATileBytes + kk * 32), bd, idesc,
                              accum);
              }
            } else {
              for (int kb = 0; kb < kbs; ++kb)
#pragma unroll
                for (int kk = 0; kk < kTileK / 16; ++kk)
                  ptx::mma_bf16(d0, ptx::sdesc_k_sw128(a0 + kb * kATileBytes + kk * 32),
                                ptx::sdesc_k_sw128(b0 + kb * b_box + kk * 32), idesc,
                                (c > 0 || kb > 0 || kk > 0) ? 1u : 0u);
            }
          }
          ptx::mma_commit(&empty[stage]);
          if (++stage == stages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        ptx::mma_commit(&acc_full[acc]);
        if (pr) ptx::mma_commit(&acc_full[acc2]);
        if (li < 8) DMOE_TRACE_AT(6 + 6 * li);
        if (pr) {
          acc = acc2;
          acc_phase = acc2_phase;
        }
        if (++acc == p.n_acc) { acc = 0; acc_phase ^= 1u; }
      }
      // make sure no MMA is still running when TMEM is released
      ptx::mma_commit(drain);
      const uint64_t t0 = ptx::globaltimer_ns();
      while (!ptx::mbar_try_wait(drain, 0) && ptx::globaltimer_ns() - t0 < kWaitTimeoutNs) {
      }
    }
  } else {
    // ================= epilogue: warps 2..9, TMEM lanes 32*(warp%4) ..; two column groups
    // (warps 2-5 and 6-9) take alternate 16-column slices of the accumulator, each with its
    // own exchange tile and named barrier (the epilogue math is latency-bound: two groups
    // finish a tile in about half the time)
    if (spec && U > 0) {
      // this CTA's share of the dispatch's copies: the rows of pair (block b, coreset member
      // e) go to xperm rows blk * (s_bpos[e] + rank of b among e's blocks), a pair split into
      // up to four parts when the pairs are fewer than the CTAs; the group counts its copied
      // rows (one release add per part, after every epilogue thread's stores)
      const int et = tid - 64;
      const int npairs = p.n_blocks * p.k;
      int parts = (int)gridDim.x / npairs;
      parts = parts < 1 ? 1 : (parts > 4 ? 4 : parts);
      while (p.blk % parts != 0) --parts;
      const int prow = p.blk / parts;                 // rows per part
      const int n16 = prow * p.d / 8;                 // 16-byte pieces per part
      for (int w = blockIdx.x; w < npairs * parts; w += gridDim.x) {
        const int i = w / parts, part = w - i * parts;
        const int b = i / p.k, e = s_bcore[i];
        const uint32_t lo = s_bmask[2 * e], hi = s_bmask[2 * e + 1];
        const int rank = b < 32 ? __popc(lo & ((1u << b) - 1u))
                                : __popc(lo) + __popc(hi & ((1u << (b - 32)) - 1u));
        const uint4* src = reinterpret_cast<const uint4*>(
            p.x + ((size_t)b * p.blk + (size_t)part * prow) * p.d);
        uint4* dst = reinterpret_cast<uint4*>(
            p.xperm + ((size_t)p.blk * (s_bpos[e] + rank) + (size_t)part * prow) * p.d);
        for (int v0 = et; v0 < n16; v0 += kEpiThreads * 8) {
          uint4 r[8];
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (v0 + q * kEpiThreads < n16) r[q] = __ldg(src + v0 + q * kEpiThreads);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            if (v0 + q * kEpiThreads < n16) dst[v0 + q * kEpiThreads] = r[q];
        }
        __threadfence();
        named_bar_sync(4, kEpiThreads);
        if (et == 0)
          red_release_add(p.x_ready + s_upos[e] * p.ntiles + (p.blk * rank) / p.n_max, prow);
      }
      if (et == 0) DMOE_TRACE_AT(63);
    }
    if (spec && warp == 2) {
      // the dispatch's outputs: the row of every (token, slot) of this CTA's share of the
      // tokens (expert e = topk_idx[t, j] of block b: the group's rows start at
      // blk * s_bpos[e], block b is its rank-th block), once the routing launch has ended
      pdl_wait();
      const int per = (p.T + (int)gridDim.x - 1) / (int)gridDim.x;
      const int t_begin = (int)blockIdx.x * per;
      const int t_end = min(p.T, t_begin + per);
      for (int i = t_begin * p.k + lane; i < t_end * p.k; i += 32) {
        const int t = i / p.k, b = t / p.blk;
        const int e = __ldcg(p.topk_idx + i);
        int r = -1;
        if (U > 0 && e >= 0 && e < p.E && b < p.n_blocks) {
          const uint32_t lo = s_bmask[2 * e], hi = s_bmask[2 * e + 1];
          const bool in = b < 32 ? ((lo >> b) & 1u) != 0u : ((hi >> (b - 32)) & 1u) != 0u;
          const int rank = b < 32 ? __popc(lo & ((1u << b) - 1u))
                                  : __popc(lo) + __popc(hi & ((1u << (b - 32)) - 1u));
          if (in) r = p.blk * (s_bpos[e] + rank) + (t - b * p.blk);
        }
        if (r < 0) {
          record_error(p.err, kErrBadDispatch, kAtDown, i);
          r = 0;
        }
        p.pos_out[i] = r;
      }
      if (blockIdx.x == 0) {
        if (lane == 0) *p.n_unique_out = U;
        for (int u = lane; u < p.E; u += 32) p.unique_ids_out[u] = u < U ? g_e[u] : -1;
      }
      // visible before this launch releases the combine (at its end): the combine reads
      // pos before its dependency wait
      __threadfence();
    }
    const int q = warp & 3;
    const int cg = (warp - 2) >> 2;                 // column group
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    float* xg = xchg + cg * (128 * kXchgStride);    // this group's exchange tile
    const int gbar = 2 + cg;                        // this group's named barrier
    const uint64_t pol_keep = ptx::policy_evict_last();   // the slot rows, for the combine
    int acc = 0, li = 0;
    uint32_t acc_phase = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++li) {
      const Unit un = decode(u);
      const bool shared = un.g >= U;
      const int nvalid = min(p.n_max, g_cnt[un.g] - un.n * p.n_max);
      const int n_mma = (nvalid + 15) & ~15;
      const bool pr = !un.gu && dpair == 2;     // a pair of down tiles: two accumulators
      int acc2 = acc + 1;
      uint32_t acc2_phase = acc_phase;
      if (acc2 == p.n_acc) { acc2 = 0; acc2_phase ^= 1u; }
      if (!epi_all_threads(wait(&acc_full[acc], acc_phase, u) &&
                           (!pr || wait(&acc_full[acc2], acc2_phase, u))))
        break;
      ptx::tc_fence_after();
      if (tid == 64 && li < 8) DMOE_TRACE_AT(50 + li);
      const uint32_t tbase = tmem_base + lane_off + (uint32_t)acc * (uint32_t)p.n_max;
      const int col0 = un.n * p.n_max;              // first token column of the tile
      if (un.gu) {
        // lanes 0-63: gate rows, lanes 64-127: up rows of the same 64 intermediate units
        const bool is_gate = q < 2;
        const int r64 = (q & 1) * 32 + lane;         // row within the 64-row slice
        const int Ig = shared ? p.Is : p.I;
        __nv_bfloat16* hout = shared ? p.hs : p.h;
        const int hrow0 = (shared ? 0 : g_row0[un.g]) + col0;
        // per 16-token slice: every accumulator row's 16 values go to the exchange tile
        // (gate rows 0-63, up rows 64-127), then each of the group's 128 threads takes 8
        // adjacent H columns of one token (loads, SwiGLU, one 16-byte store). Interleaving
        // the exchange loads with the H stores instead serialises them: the compiler
        // cannot tell the two memories apart.
        const int et = tid - 64 - 128 * cg, xc = et >> 3, hc = (et & 7) * 8;
        for (int c0 = 16 * cg; c0 < n_mma; c0 += 32) {
          float v[16];
          ptx::tmem_ld16(tbase + c0, v);
          ptx::tmem_ld_wait();
          {
            float* xr = xg + ((is_gate ? 0 : 64) + r64) * kXchgStride;
#pragma unroll
            for (int c = 0; c < 16; ++c) xr[c] = v[c];
          }
          named_bar_sync(gbar, 128);
          float gv[8], uv[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            gv[j] = xg[(hc + j) * kXchgStride + xc];
            uv[j] = xg[(64 + hc + j) * kXchgStride + xc];
          }
          uint32_t hp[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const __nv_bfloat162 h2 = __floats2bfloat162_rn(silu_f(gv[2 * j]) * uv[2 * j],
                                                            silu_f(gv[2 * j + 1]) * uv[2 * j + 1]);
            hp[j] = *reinterpret_cast<const uint32_t*>(&h2);
          }
          if (c0 + xc < nvalid)
            *reinterpret_cast<uint4*>(hout + (size_t)(hrow0 + c0 + xc) * Ig + un.m * 64 + hc) =
                make_uint4(hp[0], hp[1], hp[2], hp[3]);
          named_bar_sync(gbar, 128);   // the exchange tile is rewritten by the next slice
        }
        if (tid == 64 && li < 4) DMOE_TRACE_AT(54 + li);
        ptx::tc_fence_before();
        ptx::mbar_arrive(&acc_empty[acc]);
        // publish the tile: the barrier orders every epilogue thread's H stores before one
        // release add; a reader acquires the counter, then fences the async proxy
        named_bar_sync(4, kEpiThreads);
        if (tid == 64 && li < 8) DMOE_TRACE_AT(58 + (li < 4 ? li : 3));
        if (tid == 64) red_release_add(p.h_ready + un.g * p.ntiles + un.n, 1);
      } else {
        __nv_bfloat16* out = shared ? p.yshared + (size_t)col0 * p.d
                                    : p.yslot + (size_t)(g_row0[un.g] + col0) * p.d;
        for (int h = 0; h < (pr ? 2 : 1); ++h) {
          const int slot = h == 0 ? acc : acc2;
          const uint32_t tb = tmem_base + lane_off + (uint32_t)slot * (uint32_t)p.n_max;
          const int drow = (un.m * dpair + h) * kTileM + q * 32 + lane;
          for (int c0 = 16 * cg; c0 < n_mma; c0 += 32) {
            float v[16];
            ptx::tmem_ld16(tb + c0, v);
            ptx::tmem_ld_wait();
#pragma unroll
            for (int c = 0; c < 16; ++c)
              if (c0 + c < nvalid)
                st_bf16_keep(out + (size_t)(c0 + c) * p.d + drow, __float2bfloat16_rn(v[c]),
                             pol_keep);
          }
          ptx::tc_fence_before();
          ptx::mbar_arrive(&acc_empty[slot]);
        }
      }
      if (tid == 64 && li < 8) DMOE_TRACE_AT(7 + 6 * li);
      if (pr) {
        acc = acc2;
        acc_phase = acc2_phase;
      }
      if (++acc == p.n_acc) { acc = 0; acc_phase ^= 1u; }
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  // the combine may start now: launched earlier, its waiting CTAs would share the SMs with
  // this launch and slow it down
  pdl_launch_dependents();
  if (tid == 0) DMOE_TRACE_AT(62);
  KLOG(DMOE_KERNEL_EXPERTS, 1);
  if (warp == 1) {
    __syncwarp();
    ptx::tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

// xperm[r, :] = x[rows[r] / k, :]; block 0 also clears the gate/up tile counters.
__global__ void __launch_bounds__(256)
gather_kernel(const __nv_bfloat16* __restrict__ x, const int32_t* __restrict__ rows,
              __nv_bfloat16* __restrict__ xperm, int32_t* __restrict__ h_ready, int n_ready,
              int pairs, int k, int d) {
  pdl_wait();
  pdl_launch_dependents();   // after the wait: a waiting dependent would share the SMs
  KLOG(DMOE_KERNEL_GATHER, 0);
  if (blockIdx.x == 0)
    for (int i = threadIdx.x; i < n_ready; i += blockDim.x) h_ready[i] = 0;
  const int vec = d / 8;  // uint4 per row
  for (int r = blockIdx.x; r < pairs; r += gridDim.x) {
    const int t = rows[r] / k;
    const uint4* src = reinterpret_cast<const uint4*>(x + (size_t)t * d);
    uint4* dst = reinterpret_cast<uint4*>(xperm + (size_t)r * d);
    for (int i = threadIdx.x; i < vec; i += blockDim.x) dst[i] = src[i];
  }
  KLOG(DMOE_KERNEL_GATHER, 1);
}

// kCombineCols consecutive row values: the raw 16-byte pieces (one for 8 bf16, two for 8
// fp32), loaded first and converted to fp32 as they are used (registers bound the CTAs per
// SM, and with them the loads in flight).
constexpr int kCombineCols = 8;
template <typename Row> struct Raw8;
template <> struct Raw8<__nv_bfloat16> {
  uint4 a;
  __device__ __forceinline__ void load(const __nv_bfloat16* src) {
    a = *reinterpret_cast<const uint4*>(src);
  }
  __device__ __forceinline__ void unpack(float (&v)[8]) const {
    const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[i]));
      v[2 * i] = f.x;
      v[2 * i + 1] = f.y;
    }
  }
};
template <> struct Raw8<float> {
  float4 a, b;
  __device__ __forceinline__ void load(const float* src) {
    a = *reinterpret_cast<const float4*>(src);
    b = *reinterpret_cast<const float4*>(src + 4);
  }
  __device__ __forceinline__ void unpack(float (&v)[8]) const {
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
};

// y[t, :] = bf16( sum_j g[t,j] * yslot[pos[t*k + j], :] (slot order) + yshared[t, :] );
// block (0, 0) also clears `zero[0 .. n_zero)` and `zero2[0 .. n_zero2)` (counters and
// flags of the launches before, now done). With meta_early the slot indices and gates are
// read before the dependency wait: the caller guarantees that they were complete before the
// launch before this one could let this one start (the decode-size expert launch releases
// it only at its end, after its own wait for the routing launch that wrote them).
template <typename Row>
__global__ void __launch_bounds__(256, sizeof(Row) == 2 ? 3 : 1)   // bf16 rows: three CTAs per SM
combine_kernel(const Row* __restrict__ yslot, const Row* __restrict__ yshared,
               const int32_t* __restrict__ pos, const float* __restrict__ gate,
               __nv_bfloat16* __restrict__ y, int k, int d, int has_shared, int32_t* zero,
               int n_zero, uint32_t* zero2, int n_zero2, int meta_early) {
  pdl_launch_dependents();
  const int t = blockIdx.y;
  const int c = (blockIdx.x * blockDim.x + threadIdx.x) * kCombineCols;
  // the slot indices and gates, eight slots at a time
  int r[8];
  float gj[8];
  auto load_meta = [&](int j0) {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j0 + j < k) {
        r[j] = __ldcg(pos + t * k + j0 + j);
        gj[j] = __ldcg(gate + t * k + j0 + j);
      }
  };
  if (meta_early) load_meta(0);
  pdl_wait();
  KLOG(DMOE_KERNEL_COMBINE, 0);
  if (blockIdx.x == 0 && blockIdx.y == 0) {
    for (int i = threadIdx.x; i < n_zero; i += blockDim.x) zero[i] = 0;
    for (int i = threadIdx.x; i < n_zero2; i += blockDim.x) zero2[i] = 0u;
  }
  if (c >= d) return;
  // eight slots at a time: their row loads (and the shared row's) are issued before the
  // first product; the sum keeps the slot order
  float acc[kCombineCols];
#pragma unroll
  for (int i = 0; i < kCombineCols; ++i) acc[i] = 0.f;
  Raw8<Row> raw_s;
  if (has_shared) raw_s.load(yshared + (size_t)t * d + c);
  for (int j0 = 0; j0 < k; j0 += 8) {
    if (!meta_early || j0 > 0) load_meta(j0);
    Raw8<Row> raw[8];
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j0 + j < k) raw[j].load(yslot + (size_t)r[j] * d + c);
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (j0 + j < k) {
        float v[kCombineCols];
        raw[j].unpack(v);
#pragma unroll
        for (int i = 0; i < kCombineCols; ++i) acc[i] = fmaf(gj[j], v[i], acc[i]);
      }
  }
  if (has_shared) {
    float vs[kCombineCols];
    raw_s.unpack(vs);
#pragma unroll
    for (int i = 0; i < kCombineCols; ++i) acc[i] += vs[i];
  }
  uint32_t out[kCombineCols / 2];
#pragma unroll
  for (int i = 0; i < kCombineCols / 2; ++i) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(acc[2 * i], acc[2 * i + 1]);
    out[i] = *reinterpret_cast<const uint32_t*>(&h);
  }
  *reinterpret_cast<uint4*>(y + (size_t)t * d + c) = make_uint4(out[0], out[1], out[2], out[3]);
  KLOG(DMOE_KERNEL_COMBINE, 1);
}

// ------------------------------------------------------------------ host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// bf16 matrix [rows, cols] row-major, box = 64 columns (128 B) x box_rows rows, 128-B swizzle.
bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kTileK, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

uint32_t pow2_cols(uint32_t c) {
  uint32_t r = 32;
  while (r < c) r <<= 1;
  return r;
}

size_t experts_fixed_smem() {
  // alignment slack + exchange buffers + barriers + misc/group arrays + block top-k planning
  return 1024 + 2 * 128 * kXchgStride * 4 + 8 + 8 * (2 * kMaxStages + 9) +
         sizeof(int) * (12 + 5 * (kMaxGroups + 1)) + 64 + 4 * 2 * kMaxExperts +
         2 * 2 * kMaxExperts + kSpecPairs;
}

int max_smem_optin() {
  int dev = 0, v = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  return v;
}

}  // namespace

#ifdef DMOE_TRACE
extern "C" int dmoe_debug_trace(void* host, size_t bytes) {
  if (bytes > sizeof(g_trace)) bytes = sizeof(g_trace);
  return (int)cudaMemcpyFromSymbol(host, g_trace, bytes);
}
extern "C" int dmoe_debug_trace_clear() {
  static uint64_t zeros[kMaxPersistentCtas * 64] = {};
  return (int)cudaMemcpyToSymbol(g_trace, zeros, sizeof(zeros));
}
DMOE_KLOG_EXPORT(dmoe_debug_klog_experts)
#endif

int experts_ready_counters(int T, int E, int n_max) {
  return (E + 1) * ((T + n_max - 1) / n_max);
}

bool experts_spec_ok(const dmoe_layer_desc& d, int n_max) {
  // blocks of whole 8-row groups (a block's box starts on a 1 KB swizzle boundary), whole
  // blocks per token tile, at most kSpecBlocks blocks (a 64-bit block mask per expert)
  return d.mode == DMOE_ROUTE_BLOCK && d.top_p <= 0.f && mask_top_k(d) == d.top_k &&
         d.n_blocks >= 1 && d.n_blocks <= kSpecBlocks && d.block_size % 8 == 0 &&
         n_max % d.block_size == 0 && d.n_experts <= kMaxExperts;
}

cudaError_t launch_experts(const ExpertArgs& a, cudaStream_t s) {
  const int pairs = a.T * a.k;
  const bool has_shared = a.Is > 0;
  const int n_ready = experts_ready_counters(a.T, a.E, a.n_max);
  const bool spec = a.spec_words != nullptr;
  // 1. gather x in dispatch order; clear the gate/up tile counters (unless the dispatch
  //    placement of the fused layer call has done both, or, for block top-k, the block
  //    routing launch has cleared them and the token rows are read from x by block)
  if (!a.gathered && !spec) {
    const int grid = pairs < 1024 ? pairs : 1024;
    prof_begin(DMOE_KERNEL_GATHER, s);
    cudaError_t e = launch_ex(gather_kernel, dim3(grid), dim3(256), 0, s, true, a.x, a.rows,
                              a.xperm, a.h_ready, n_ready, pairs, a.k, a.d);
    prof_end(DMOE_KERNEL_GATHER, s);
    if (e != cudaSuccess) return e;
  }
  GemmParams gp{};
  gp.n_unique = a.n_unique;
  gp.unique_ids = a.unique_ids;
  gp.offsets = a.offsets;
  gp.h = a.h;
  gp.hs = a.hs;
  gp.yslot = static_cast<__nv_bfloat16*>(a.yslot);
  gp.yshared = static_cast<__nv_bfloat16*>(a.yshared);
  gp.h_ready = a.h_ready;
  gp.err = a.err;
  gp.w_down = a.w_down;
  if (has_shared && a.prefetch_shared) {
    gp.ws_gate = a.ws_gate;
    gp.ws_up = a.ws_up;
    gp.ws_down = a.ws_down;
  }
  gp.T = a.T; gp.d = a.d; gp.E = a.E; gp.k = a.k; gp.I = a.I; gp.Is = a.Is;
  gp.n_max = a.n_max;
  gp.n_half = ((a.n_max / 2) + 15) & ~15;
  gp.kbs = a.n_max >= 256 ? 1 : kMaxKBoxes;
  // pairs of down tiles share their H stages: 25 % less to pull per SM and half the down
  // units, so that each CTA takes about one (needs two K boxes per stage for the pair's A
  // and an even number of 128-row tiles of d)
  gp.dpair = (gp.kbs == 2 && (a.d / kTileM) % 2 == 0) ? 2 : 1;
  gp.ntiles = (a.T + a.n_max - 1) / a.n_max;
  gp.has_shared = has_shared ? 1 : 0;
  if (spec) {
    gp.spec_words = a.spec_words;
    gp.n_blocks = a.spec_blocks;
    gp.blk = a.T / a.spec_blocks;
    gp.topk_idx = a.topk_idx;
    gp.pos_out = a.pos_out;
    gp.n_unique_out = a.n_unique_out;
    gp.unique_ids_out = a.unique_ids_out;
    gp.x_ready = a.h_ready + experts_ready_counters(a.T, a.E, a.n_max);
    gp.x = a.x;
    gp.xperm = a.xperm;
  }

  // 2. gate/up + SwiGLU and down projection in one persistent launch
  Maps m;
  bool ok = make_map(&m.wg, a.w_gate, (uint64_t)a.E * a.I, a.d, 64) &&
            make_map(&m.wu, a.w_up, (uint64_t)a.E * a.I, a.d, 64) &&
            make_map(&m.wd, a.w_down, (uint64_t)a.E * a.d, a.I, kTileM) &&
            make_map(&m.xp, a.xperm, (uint64_t)pairs, a.d, (uint32_t)a.n_max) &&
            make_map(&m.x, a.x, (uint64_t)a.T, a.d, (uint32_t)a.n_max) &&
            make_map(&m.h, a.h, (uint64_t)pairs, a.I, (uint32_t)a.n_max) &&
            make_map(&m.xph, a.xperm, (uint64_t)pairs, a.d, (uint32_t)gp.n_half) &&
            make_map(&m.hh, a.h, (uint64_t)pairs, a.I, (uint32_t)gp.n_half);
  if (ok && has_shared)
    ok = make_map(&m.sg, a.ws_gate, (uint64_t)a.Is, a.d, 64) &&
         make_map(&m.su, a.ws_up, (uint64_t)a.Is, a.d, 64) &&
         make_map(&m.sd, a.ws_down, (uint64_t)a.d, a.Is, kTileM) &&
         make_map(&m.hs, a.hs, (uint64_t)a.T, a.Is, (uint32_t)a.n_max);
  if (!has_shared) { m.sg = m.wg; m.su = m.wu; m.sd = m.wd; m.hs = m.h; }
  if (!ok) return cudaErrorInvalidValue;

  const size_t stage_bytes = (size_t)gp.kbs * ((size_t)kATileBytes + (size_t)a.n_max * 128);
  const size_t fixed = experts_fixed_smem();
  const int limit = max_smem_optin();
  int stages = (int)((limit - (int)fixed) / (int)stage_bytes);
  if (stages > kMaxStages) stages = kMaxStages;
  if (stages < 2) return cudaErrorInvalidConfiguration;
  gp.stages = stages;
  gp.n_acc = 512 / a.n_max;
  if (gp.n_acc > 4) gp.n_acc = 4;
  gp.tmem_cols = pow2_cols((uint32_t)(gp.n_acc * a.n_max));
  const size_t smem = fixed + (size_t)stages * stage_bytes;
  static int attr_dev_mask = 0;  // the dynamic smem limit is a per-device function attribute
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 31 || !(attr_dev_mask & (1 << dev))) {
    cudaError_t e = cudaFuncSetAttribute(moe_experts_kernel<false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, limit);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(moe_experts_kernel<true>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, limit);
    if (e != cudaSuccess) return e;
    if (dev < 31) attr_dev_mask |= 1 << dev;
  }
  int grid = device_sm_count();
  // block top-k with few blocks: the CTAs start while the block routing launch (one CTA
  // per block) still runs; leave its SMs free, so that no CTA starts only when it ends
  if (spec && a.spec_blocks <= 16 && grid > 4 * a.spec_blocks) grid -= a.spec_blocks;
  if (grid > kMaxPersistentCtas) grid = kMaxPersistentCtas;
  prof_begin(DMOE_KERNEL_EXPERTS, s);
  cudaError_t e = spec ? launch_ex(moe_experts_kernel<true>, dim3(grid), dim3(kThreads), smem, s,
                                   !prof_serial(DMOE_KERNEL_EXPERTS), m, gp)
                        : launch_ex(moe_experts_kernel<false>, dim3(grid), dim3(kThreads), smem,
                                    s, !prof_serial(DMOE_KERNEL_EXPERTS), m, gp);
  prof_end(DMOE_KERNEL_EXPERTS, s);
  if (e != cudaSuccess) return e;

  // 3. gate-weighted combine of the bf16 rows (the slot rows and gates were complete before
  //    this launch released it: the combine may read them before its dependency wait)
  return launch_combine(a, s, nullptr, 0, nullptr, 0, true, true);
}

cudaError_t launch_combine(const ExpertArgs& a, cudaStream_t s, int32_t* zero, int n_zero,
                           uint32_t* zero2, int n_zero2, bool meta_early, bool rows_bf16) {
  // CTAs of 256 threads; fewer (down to 32) while that leaves fewer than 128 CTAs, so
  // that a decode-sized forward spreads its rows over most SMs
  int thr = 256;
  while (thr > 32 && (a.d / kCombineCols + thr - 1) / thr * a.T < 128) thr >>= 1;
  dim3 cgrid((a.d / kCombineCols + thr - 1) / thr, a.T);
  prof_begin(DMOE_KERNEL_COMBINE, s);
  cudaError_t e =
      rows_bf16
          ? launch_ex(combine_kernel<__nv_bfloat16>, cgrid, dim3(thr), 0, s, true,
                      static_cast<const __nv_bfloat16*>(a.yslot),
                      static_cast<const __nv_bfloat16*>(a.yshared), a.pos, a.topk_gate,
                      a.y, a.k, a.d, a.Is > 0 ? 1 : 0, zero, n_zero, zero2, n_zero2,
                      meta_early ? 1 : 0)
          : launch_ex(combine_kernel<float>, cgrid, dim3(thr), 0, s, true,
                      static_cast<const float*>(a.yslot), static_cast<const float*>(a.yshared),
                      a.pos, a.topk_gate, a.y, a.k, a.d, a.Is > 0 ? 1 : 0, zero, n_zero,
                      zero2, n_zero2, meta_early ? 1 : 0);
  prof_end(DMOE_KERNEL_COMBINE, s);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dmoe
