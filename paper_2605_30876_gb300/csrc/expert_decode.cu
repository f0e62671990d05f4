// Expert FFN of a decode-sized forward (at most 64 tokens) in one persistent launch on
// tcgen05 tensor cores (§4.2 of arXiv 2605.30876: every unique expert of the forward runs
// once on the tokens routed to it; plus the shared expert on all tokens).
//
// A group is the shared expert (group 0, when present) or the u-th unique expert of the
// dispatch. With at most 64 tokens every group is computed over all T tokens at once: the
// B operand of gate/up is x itself (no gather), the extra MMA columns cost nothing next to
// the weight stream, and the down epilogue keeps only the columns of the tokens routed to
// the group. The work is a list of units spread round-robin over one CTA per SM:
//   gate/up unit (group, hg rows of I, hg = 64 or 32): hg rows of W_gate stacked over the
//     same hg rows of W_up, one M = 2 hg MMA chain over K = d (gate in the first hg rows of
//     the accumulator, up in the rest); the epilogue writes h = silu(gate) * up as bf16 into
//     the group's H (global, L2-resident) and publishes the tile on the group's counter;
//   down unit (group, 128 rows of d): D = W_down tile x H^T over K = I; the producer loads
//     the weight stages first and the H stages once every gate/up tile of the group is
//     published; the epilogue stores the fp32 rows per (token, slot).
// Down units continue the round-robin where the gate/up units stopped. hg is chosen on the
// device once the unique-expert count is known: 32 when the 32-row gate/up units still fit
// in one round over the CTAs, else 64. With few unique experts the 64-row units would
// leave half of the SMs on down tiles only, and one SM's TMA rate, not HBM, would set the
// pace of the gate/up stream; the 32-row units put a gate/up tile on every SM and keep the
// weight bytes per SM near the mean. Every stage carries 32 KB of weights: K = 128 for
// hg = 64 and for the down tiles, K = 256 for hg = 32 (four 128-B boxes per weight row).
// The combine launch that follows clears the group counters for the next call.
//
// Warp roles (224 threads): warp 0 lane 0 issues TMA, lane 0 of warps 1 and 6 issue the MMAs
// (each the first or second half of every stage's K boxes, into its own part of the
// accumulator: one thread issues a tcgen05.mma only every ~58 cycles, whatever its shape,
// and these chains are short), warps 2-5 run the epilogues (TMEM lane quadrant = warp % 4),
// which add the two parts. Every wait is bounded (1 s): a timeout is recorded and the CTA
// unwinds.
#include <math.h>

#include <mutex>

#include "dmoe_internal.cuh"
#include "sm100_ptx.cuh"
#include "trace_log.cuh"

namespace dmoe {
namespace {

constexpr int kThr = 224;
constexpr int kKB = 2;                          // K boxes per down stage: K = 128
constexpr int kStageK = kKB * kTileK;
constexpr int kABox = kTileM * 128;             // 128 rows x 128 B (W_down)
constexpr int kAStage = kKB * kABox;            // 32 KB of weights in every stage
constexpr int kMaxKBG = 4;                      // K boxes per gate/up stage (hg = 32)
constexpr int kMaxStagesD = 6;
constexpr int kXStride = 17;                    // floats per row of the SwiGLU exchange
constexpr int kXchgBytes = 2 * 64 * kXStride * 4;
constexpr uint64_t kTimeoutNs = 1000000000ull;  // 1 s
constexpr int kMaxTok = 64;                     // tokens of a decode-sized forward

// Debug builds (-DDMOE_TRACE): per-CTA timeline of the first unit of each kind,
// g_dtrace[cta * 32 + slot] (globaltimer ns): 0 entry, 1 unit list known, 2 gate/up first
// stage landed, 3 gate/up MMAs committed, 4 gate/up tile published, 5 down weights issued,
// 6 H ready seen, 7 down MMAs committed, 8 down rows stored, 9 exit, 10 gate/up unit id,
// 11 down unit id, 12/13 first/last down stage landed, 14 down accumulator ready, 15 down
// accumulator staged, 16 staging complete, 17 row copies issued, 18 coresets seen by the
// polling warp, 19 its CTA past the barrier after the poll, 26/27 fourth / last gate/up
// stage landed, 28/29 first / last gate/up stage issued, 30 past the TMEM barrier, 31 the
// producer's cache policies made.
#ifdef DMOE_TRACE
__device__ uint64_t g_dtrace[kMaxPersistentCtas * 32];
#define ED_AT(slot) (g_dtrace[blockIdx.x * 32 + (slot)] = ptx::globaltimer_ns())
#define ED_SET(slot, v) (g_dtrace[blockIdx.x * 32 + (slot)] = (uint64_t)(v))
#else
#define ED_AT(slot) ((void)0)
#define ED_SET(slot, v) ((void)0)
#endif

struct DParams {
  const int32_t* n_unique;
  const int32_t* unique_ids;
  const int32_t* offsets;
  const int32_t* rows;
  __nv_bfloat16* hdense;     // [(E+1) * n_pad, imax]: H of group g in rows g*n_pad ..
  float* yslot;              // [T*k, d]
  float* yshared;            // [T, d]
  int32_t* h_ready;          // [E+1]: published gate/up tiles per group (zero between calls;
                             // the combine launch clears them)
  const uint32_t* spec_words;   // block top-k: published coresets (spec_words(k) words per
                                // block, three ids and a marker byte each), or nullptr
  int spec_blocks;
  int spec_mask;             // the words are coreset masks (kSpecMaskWords per block): their
                             // union contains the unique experts, whose rows the dispatch gives
  DevErrRecord* err;
  int T, d, E, k, I, Is;
  int imax;                  // max(I, Is): row length of hdense
  int n_pad;                 // token rows of every B box (multiple of 16)
  int ring_bytes;            // pipeline ring (multiple of 1 KB)
  int h32_ok;                // 32-row gate/up units allowed (d % 256 == 0, >= 3 slots fit)
  int has_shared;
  int n_acc;                 // TMEM accumulators of n_pad columns
  uint32_t tmem_cols;
};

struct DMaps {
  CUtensorMap wg, wu, wd;    // routed: [E*I, d] (64-row boxes) x2, [E*d, I] (128-row boxes)
  CUtensorMap sg, su, sd;    // shared: [Is, d] x2, [d, Is]
  CUtensorMap wg32, wu32;    // routed gate/up, 32-row boxes
  CUtensorMap sg32, su32;    // shared gate/up, 32-row boxes
  CUtensorMap x;             // x [T, d], n_pad-row boxes (rows >= T read as zeros)
  CUtensorMap h;             // hdense, n_pad-row boxes, 128-B swizzle (down B operand)
  CUtensorMap hst;           // hdense, 32 columns x n_pad rows, no swizzle (tile stores)
  CUtensorMap ys, ysh;       // yslot [T*k, d], yshared [T, d] fp32: 128 columns x 8 rows
};

// One group of the forward.
struct Grp {
  bool shared;
  int e;      // expert id (routed)
  int row0;   // first dispatch row (routed)
  int n;      // tokens routed to the group (T for the shared expert)
  int Ig;     // intermediate size
};

using ptx::bulk_commit_wait_all;
using ptx::bulk_commit_wait_read;
using ptx::bulk_store;
using ptx::epi_all;
using ptx::fence_proxy_async_global;
using ptx::ld_acquire;
using ptx::ld_relaxed_u32;
using ptx::named_bar_sync;
using ptx::red_release_add;
using ptx::tma_store_2d;
// silu with the fast divide: H is rounded to bf16 right after
__device__ __forceinline__ float silu_f(float z) { return __fdividef(z, 1.f + __expf(-z)); }

// kMask: the coresets are published as masks (DParams::spec_mask), compiled separately so
// that the launch on ids carries none of that code
template <bool kMask>
__global__ void __launch_bounds__(kThr, 1)
moe_decode_kernel(const __grid_constant__ DMaps tm, const __grid_constant__ DParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (ptx::smem_addr(smem_raw) & 1023u)) & 1023u);
  const int bbox = p.n_pad * 128;                 // one K box of token rows
  const int bstage = kKB * bbox;                  // B bytes of a down stage
  const int SP = p.n_pad + 1;                     // floats per row of the down staging tile
  // ring of S slots [32 KB of weights | token boxes]; S and the slot size follow hg below
  uint8_t* ring = smem;
  // staging: a gate/up tile's H box, or a down tile as [token][128 rows] fp32 (128 x SP floats)
  float* stage_t = reinterpret_cast<float*>(ring + p.ring_bytes);
  float* xchg = stage_t + kTileM * SP;
  int* tok = reinterpret_cast<int*>(xchg + 2 * 64 * kXStride);      // [kMaxTok]
  uint64_t* full = reinterpret_cast<uint64_t*>(tok + kMaxTok);
  uint64_t* empty = full + kMaxStagesD;
  uint64_t* acc_full = empty + kMaxStagesD;
  uint64_t* acc_empty = acc_full + 4;
  uint64_t* drain = acc_empty + 4;
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);
  int* s_u = const_cast<int*>(s_abort) + 1;
  uint8_t* s_spec = reinterpret_cast<uint8_t*>(s_u + 1);   // [kMaxExperts]: unique ids
  uint32_t* s_mask = reinterpret_cast<uint32_t*>(s_spec + kMaxExperts);   // [kMaxExperts / 32]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nb = gridDim.x, b = blockIdx.x;
  KLOG(DMOE_KERNEL_EXPERTS, 0);
  if (tid == 0) ED_AT(0);

  if (tid == 0) {
    for (int s = 0; s < kMaxStagesD; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 2);       // both MMA issuers commit
    }
    for (int a = 0; a < 4; ++a) {
      ptx::mbar_init(&acc_full[a], 2);
      ptx::mbar_init(&acc_empty[a], 128);
    }
    ptx::mbar_init(drain, 2);
    ptx::fence_mbarrier_init();
    *s_abort = 0;
  } else if (tid == 32) {
    // the descriptors of the first copies
    const CUtensorMap* maps[7] = {&tm.wg32, &tm.wu32, &tm.wg, &tm.wu, &tm.x, &tm.sg32, &tm.su32};
#pragma unroll
    for (int i = 0; i < 7; ++i) ptx::prefetch_tensormap(maps[i]);
  }
  if (warp == 1) {
    ptx::tmem_alloc(s_tmem, p.tmem_cols);
    ptx::tmem_relinquish();
  }
  // What does not depend on the unit list is read and derived before any wait, so that
  // nothing but the list is left once the coresets or the dispatch are in: the producer's
  // diagnostic hold (normally 0: every down unit waits for this many more gate/up tiles
  // than its group has, so that its bounded wait runs out) and the shapes of both unit
  // heights.
  int hold = 0;
  if (tid == 0) hold = *reinterpret_cast<volatile int32_t*>(&p.err->hold);
  const int has_shared = p.has_shared, pI = p.I, pIs = p.Is;
  const int ngu64_s = has_shared ? pIs / 64 : 0, ngu64_r = pI / 64;
  const int slot32 = kAStage + (kTileM / 32) * bbox, slot64 = kAStage + (kTileM / 64) * bbox;
  const int S32 = min(p.ring_bytes / slot32, kMaxStagesD);
  const int S64 = min(p.ring_bytes / slot64, kMaxStagesD);
  const int ngu_s32 = has_shared ? pIs / 32 : 0, ngu_r32 = pI / 32;
  const int kc32 = p.d / (kMaxKBG * kTileK), kc64 = p.d / (2 * kTileK);
  const int ndn = p.d / kTileM;
  const bool h32_ok = p.h32_ok != 0;

  // Block top-k: the unique experts are the union of the blocks' coresets (every token of a
  // block is routed to all k experts of its coreset), published by the routing launch
  // before it ends; the weight stream starts on them, and only the down epilogue waits for
  // the dispatch. Otherwise (or if the coresets do not come) everything waits for it.
  bool spec = p.spec_words != nullptr;
  int early = 0;   // stages of the first gate/up unit the producer sent right after the poll
  if (spec) {
    if (warp == 0) {
      // poll every block's words until all are nonzero; a nonzero word is complete (one
      // 32-bit store), so its ids go into the shared mask as it is seen (or-ing twice is
      // harmless)
      const int nw = spec_words(p.k), total = p.spec_blocks * nw;
      if (lane < kMaxExperts / 32) s_mask[lane] = 0u;
      __syncwarp();
      bool bad = false;
      const uint64_t t0 = ptx::globaltimer_ns();
      for (;;) {
        bool all = true;
        if (kMask) {
          // masks: a block's words are read once its marker (stored last, with release
          // semantics) is seen by an acquire load; or-ing a mask twice is harmless
          for (int b = lane; b < p.spec_blocks; b += 32) {
            const uint32_t* wb = p.spec_words + (size_t)b * kSpecMaskWords;
            if (ld_acquire(reinterpret_cast<const int32_t*>(wb + kMaxExperts / 32)) == 0) {
              all = false;
              continue;
            }
#pragma unroll
            for (int w = 0; w < kMaxExperts / 32; ++w) {
              const uint32_t m = ld_relaxed_u32(wb + w);
              if (m != 0u) {
                if (32 * w >= p.E || (32 * w + 31 >= p.E && (m >> (p.E - 32 * w)) != 0u))
                  bad = true;
                atomicOr(&s_mask[w], m);
              }
            }
          }
        } else
        for (int i = lane; i < total; i += 32) {
          const uint32_t w = ld_relaxed_u32(p.spec_words + i);
          if (w == 0u) {
            all = false;
            continue;
          }
          const int r0 = 3 * (i % nw);
#pragma unroll
          for (int j = 0; j < 3; ++j) {
            if (r0 + j >= p.k) break;
            const int e = (int)((w >> (8 * j)) & 0xffu);
            if (e >= p.E) bad = true;
            else atomicOr(&s_mask[e >> 5], 1u << (e & 31));
          }
        }
        if (__all_sync(0xffffffffu, all)) {
          if (lane == 0) ED_AT(18);
          break;
        }
        if (ptx::globaltimer_ns() - t0 > kTimeoutNs) {   // the coresets did not come
          bad = true;
          break;
        }
      }
      bad = __any_sync(0xffffffffu, bad);
      __syncwarp();
      // the ascending id list: lane w expands mask word w at its prefix position
      const uint32_t mw = lane < kMaxExperts / 32 ? s_mask[lane] : 0u;
      const int c = __popc(mw);
      int incl = c;
#pragma unroll
      for (int o = 1; o < kMaxExperts / 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const int u_all = __shfl_sync(0xffffffffu, incl, kMaxExperts / 32 - 1);
      if (!bad) {
        int u = incl - c;
        for (uint32_t bits = mw; bits != 0u; bits &= bits - 1u)
          s_spec[u++] = (uint8_t)(lane * 32 + __ffs((int)bits) - 1);
      }
      if (lane == 0) *s_u = bad ? -1 : u_all;
      __syncwarp();
      if (lane == 0 && !bad) {
        // This lane is the producer: the first ring slots of its first gate/up unit are
        // filled now, before the CTA barrier and the unit bookkeeping below (the same copies
        // the producer loop would make; fresh ring slots need no wait).
        const bool h32e = h32_ok && 2 * (ngu64_s + u_all * ngu64_r) <= nb;
        const int hge = h32e ? 32 : 64, kbge = kTileM / hge;
        const int slote = h32e ? slot32 : slot64, Se = h32e ? S32 : S64;
        const int ngse = h32e ? ngu_s32 : ngu64_s, ngre = h32e ? ngu_r32 : ngu64_r;
        const int kce = h32e ? kc32 : kc64;
        if (b < ngse + u_all * ngre) {
          const bool sh = b < ngse;
          const int m = sh ? b : (b - ngse) % ngre;
          const int e = sh ? 0 : (int)s_spec[(b - ngse) / ngre];
          const CUtensorMap* mg = h32e ? (sh ? &tm.sg32 : &tm.wg32) : (sh ? &tm.sg : &tm.wg);
          const CUtensorMap* mu = h32e ? (sh ? &tm.su32 : &tm.wu32) : (sh ? &tm.su : &tm.wu);
          const int arow = (sh ? 0 : e * pI) + m * hge;
          const uint64_t pw = ptx::policy_evict_first(), px = ptx::policy_evict_last();
          early = Se < kce ? Se : kce;
          ED_AT(28);
          for (int c = 0; c < early; ++c) {
            ptx::mbar_arrive_expect_tx(&full[c], kAStage + kbge * bbox);
            uint8_t* a_dst = smem + c * slote;
            uint8_t* b_dst = a_dst + kAStage;
            for (int kb = 0; kb < kbge; ++kb) {
              const int kx = (c * kbge + kb) * kTileK;
              ptx::tma_load_2d(a_dst + kb * 2 * hge * 128, mg, &full[c], kx, arow, pw);
              ptx::tma_load_2d(a_dst + kb * 2 * hge * 128 + hge * 128, mu, &full[c], kx, arow,
                               pw);
              ptx::tma_load_2d(b_dst + kb * bbox, &tm.x, &full[c], kx, 0, px);
            }
          }
        }
      }
    }
    __syncthreads();
    if (tid == 0) ED_AT(19);
    spec = *s_u >= 0;
  }
  if (!spec) {
    pdl_wait();   // the dispatch is complete from here on
    if (tid == 0) {
      int u = __ldcg(p.n_unique);
      if (u < 0 || u > p.E) {
        record_error(p.err, kErrBadDispatch, kAtGateUp, u);
        u = 0;
      }
      *s_u = u;
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  if (tid == 0) ED_AT(30);
  const uint32_t tmem_base = *s_tmem;
  const int U = *s_u;
  const int G = U + has_shared;
  // gate/up unit height: 32 rows of I when even the 32-row units fit in one round over the
  // CTAs (a forward with few unique experts), else 64
  const bool h32 = h32_ok && 2 * (ngu64_s + U * ngu64_r) <= nb;
  const int hg = h32 ? 32 : 64;
  const int kbg = h32 ? kTileM / 32 : kTileM / 64;   // K boxes per gate/up stage (32 KB)
  const int slot = h32 ? slot32 : slot64;
  const int S = h32 ? S32 : S64;
  auto slot_a = [&](int st) { return ring + st * slot; };
  auto slot_b = [&](int st) { return ring + st * slot + kAStage; };
  const int abox_g = 2 * hg * 128;                // one K box of the stacked gate|up rows
  const int ngu_s = h32 ? ngu_s32 : ngu64_s, ngu_r = h32 ? ngu_r32 : ngu64_r;
  const int NGU = ngu_s + U * ngu_r;
  const int ND = G * ndn;
  // first down unit of this CTA: the round-robin continues after the NGU gate/up units
  const int nrem = NGU % nb;
  const int v0 = b >= nrem ? b - nrem : b - nrem + nb;
  if (tid == 0) ED_AT(1);

  // the group's expert and size (all the weight stream needs)
  auto group_w = [&](int gi) -> Grp {
    Grp g;
    g.row0 = 0;
    g.n = 0;
    if (gi < p.has_shared) {
      g.shared = true;
      g.e = 0;
      g.Ig = p.Is;
      return g;
    }
    const int u = gi - p.has_shared;
    int e = spec ? (int)s_spec[u] : __ldcg(p.unique_ids + u);
    if (e < 0 || e >= p.E) {
      record_error(p.err, kErrBadDispatch, kAtGateUp, u);
      e = 0;
    }
    g.shared = false;
    g.e = e;
    g.Ig = p.I;
    return g;
  };
  // ... and its rows of the dispatch (once the dispatch is complete)
  auto group = [&](int gi) -> Grp {
    Grp g = group_w(gi);
    if (g.shared) {
      g.n = p.T;
      return g;
    }
    int u = gi - p.has_shared;
    if (kMask && spec) {
      // the group is a member of the coresets' union; its rows are those of its place in
      // the dispatch's unique list (ascending), none if no token kept it
      const int nd = __ldcg(p.n_unique), e = g.e;
      int lo = 0, hi = nd;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (__ldcg(p.unique_ids + mid) < e) lo = mid + 1;
        else hi = mid;
      }
      if (lo >= nd || __ldcg(p.unique_ids + lo) != e) {
        g.row0 = 0;
        g.n = 0;
        return g;
      }
      u = lo;
    }
    int row0 = __ldcg(p.offsets + u);
    int n = __ldcg(p.offsets + u + 1) - row0;
    if (n < 0 || n > p.T || row0 < 0 || row0 + n > p.T * p.k) {
      record_error(p.err, kErrBadDispatch, kAtDown, u);
      n = 0;
      row0 = 0;
    }
    g.row0 = row0;
    g.n = n;
    return g;
  };
  // gate/up unit -> (group, 64-row tile)
  auto gu_unit = [&](int u, int& gi, int& m) {
    if (u < ngu_s) {
      gi = 0;
      m = u;
    } else {
      gi = p.has_shared + (u - ngu_s) / ngu_r;
      m = (u - ngu_s) % ngu_r;
    }
  };
  auto wait = [&](uint64_t* bar, uint32_t parity, int value) -> bool {
    if (*s_abort) return false;
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::globaltimer_ns();
    for (uint32_t i = 1;; ++i) {
      if (ptx::mbar_try_wait(bar, parity)) return true;
      if ((i & 63u) == 0u) {
        if (*s_abort) return false;
        if (ptx::globaltimer_ns() - t0 > kTimeoutNs) {
          record_error(p.err, kErrTimeout, kAtGateUp, value);
          *s_abort = 1;
          return false;
        }
      }
    }
  };
  const int kc = h32 ? kc32 : kc64;   // stages of one gate/up tile

  if (warp == 0 && lane == 0) {
    // ================= TMA producer
    const uint64_t pol_w = ptx::policy_evict_first();   // weights: streamed once
    const uint64_t pol_x = ptx::policy_evict_last();    // x and H: re-read by many tiles
    ED_AT(31);
    // the stages sent right after the poll
    int stage = early == S ? 0 : early, issued = early;
    uint32_t phase = early == S ? 1u : 0u;
    bool ok = true;
    bool first = true;
    for (int u = b; u < NGU && ok; u += nb) {
      int gi, m;
      gu_unit(u, gi, m);
      const Grp g = group_w(gi);
      const CUtensorMap* mg =
          hg == 32 ? (g.shared ? &tm.sg32 : &tm.wg32) : (g.shared ? &tm.sg : &tm.wg);
      const CUtensorMap* mu =
          hg == 32 ? (g.shared ? &tm.su32 : &tm.wu32) : (g.shared ? &tm.su : &tm.wu);
      const int arow = (g.shared ? 0 : g.e * p.I) + m * hg;
      if (first) ED_SET(10, u);
      for (int c = first ? early : 0; c < kc; ++c) {
        if (!wait(&empty[stage], phase ^ 1u, u)) { ok = false; break; }
        if (first && c == 0) ED_AT(28);
        if (first && c == kc - 1) ED_AT(29);
        ptx::mbar_arrive_expect_tx(&full[stage], kAStage + kbg * bbox);
        uint8_t* a_dst = slot_a(stage);
        uint8_t* b_dst = slot_b(stage);
        for (int kb = 0; kb < kbg; ++kb) {
          const int kx = (c * kbg + kb) * kTileK;
          ptx::tma_load_2d(a_dst + kb * abox_g, mg, &full[stage], kx, arow, pol_w);
          ptx::tma_load_2d(a_dst + kb * abox_g + hg * 128, mu, &full[stage], kx, arow, pol_w);
          ptx::tma_load_2d(b_dst + kb * bbox, &tm.x, &full[stage], kx, 0, pol_x);
        }
        ++issued;
        if (++stage == S) { stage = 0; phase ^= 1u; }
      }
      first = false;
    }
    first = true;
    for (int v = v0; v < ND && ok; v += nb) {
      const int gi = v / ndn, i = v % ndn;
      const Grp g = group_w(gi);
      const CUtensorMap* md = g.shared ? &tm.sd : &tm.wd;
      const int arow = (g.shared ? 0 : g.e * p.d) + i * kTileM;
      const int ndk = g.Ig / kStageK;
      const int pre = ndk < S ? ndk : S;
      const int st0 = stage;
      if (first) ED_SET(11, v);
      // weights first: they do not depend on the gate/up phase
      int done = 0;
      for (int c = 0; c < pre; ++c, ++done) {
        if (!wait(&empty[stage], phase ^ 1u, v)) { ok = false; break; }
        ptx::mbar_arrive_expect_tx(&full[stage], kAStage + bstage);
        uint8_t* a_dst = slot_a(stage);
#pragma unroll
        for (int kb = 0; kb < kKB; ++kb)
          ptx::tma_load_2d(a_dst + kb * kABox, md, &full[stage], c * kStageK + kb * kTileK, arow,
                           pol_w);
        ++issued;
        if (++stage == S) { stage = 0; phase ^= 1u; }
      }
      if (first) ED_AT(5);
      // then the H rows, once every gate/up tile of the group is published
      const int target = g.Ig / hg + hold;
      if (ok && ld_acquire(p.h_ready + gi) < target) {
        const uint64_t t0 = ptx::globaltimer_ns();
        while (ld_acquire(p.h_ready + gi) < target) {
          if (*s_abort) { ok = false; break; }
          if (ptx::globaltimer_ns() - t0 > kTimeoutNs) {
            record_error(p.err, kErrTimeout, kAtDown, v);
            *s_abort = 1;
            ok = false;
            break;
          }
        }
      }
      fence_proxy_async_global();
      if (first) ED_AT(6);
      {
        int st = st0;
        for (int c = 0; c < done; ++c) {
          if (ok) {
            uint8_t* b_dst = slot_b(st);
#pragma unroll
            for (int kb = 0; kb < kKB; ++kb)
              ptx::tma_load_2d(b_dst + kb * bbox, &tm.h, &full[st], c * kStageK + kb * kTileK,
                               gi * p.n_pad, pol_x);
          } else {
            // keep the barrier accounting whole: complete the stage without B data
            ptx::mbar_complete_tx_local(&full[st], bstage);
          }
          if (++st == S) st = 0;
        }
      }
      for (int c = pre; c < ndk && ok; ++c) {
        if (!wait(&empty[stage], phase ^ 1u, v)) { ok = false; break; }
        ptx::mbar_arrive_expect_tx(&full[stage], kAStage + bstage);
        uint8_t* a_dst = slot_a(stage);
        uint8_t* b_dst = slot_b(stage);
#pragma unroll
        for (int kb = 0; kb < kKB; ++kb) {
          const int kx = c * kStageK + kb * kTileK;
          ptx::tma_load_2d(a_dst + kb * kABox, md, &full[stage], kx, arow, pol_w);
          ptx::tma_load_2d(b_dst + kb * bbox, &tm.h, &full[stage], kx, gi * p.n_pad, pol_x);
        }
        ++issued;
        if (++stage == S) { stage = 0; phase ^= 1u; }
      }
      first = false;
    }
    if (!ok) {
      // let the copies already in flight land before the CTA exits
      int st = stage;
      uint32_t ph = phase;
      const int n = issued < S ? issued : S;
      for (int i = 0; i < n; ++i) {
        if (--st < 0) { st = S - 1; ph ^= 1u; }
        const uint64_t t0 = ptx::globaltimer_ns();
        while (!ptx::mbar_try_wait(&full[st], ph) &&
               ptx::globaltimer_ns() - t0 < kTimeoutNs / 10) {
        }
      }
    }
  } else if ((warp == 1 || warp == 6) && lane == 0) {
    // ================= MMA issuers: `half` 0 takes the first half of every stage's K boxes
    // into part 0 of the accumulator, `half` 1 the second half into part 1
    const int half = warp == 6 ? 1 : 0;
    int stage = 0, acc = 0;
    uint32_t phase = 0, acc_phase = 0;
    bool ok = true, first = half == 0;
    // nstages stages of kboxes K boxes each; A boxes abox bytes apart, M = mrows
    auto run = [&](int nstages, int kboxes, int abox, uint32_t mrows, int value, bool gu) {
      const uint32_t n_mma = (uint32_t)((p.T + 15) & ~15);
      const uint32_t idesc = ptx::idesc_bf16(mrows, n_mma);
      if (!wait(&acc_empty[acc], acc_phase ^ 1u, value)) { ok = false; return; }
      ptx::tc_fence_after();
      const uint32_t d0 = tmem_base + (uint32_t)((half * p.n_acc + acc) * p.n_pad);
      const int kb0 = half * (kboxes / 2), kb1 = kb0 + kboxes / 2;
      for (int c = 0; c < nstages; ++c) {
        if (!wait(&full[stage], phase, value)) { ok = false; return; }
        if (gu && first && c == 0) ED_AT(2);
        if (gu && first && c == 3) ED_AT(26);
        if (gu && first && c == nstages - 1) ED_AT(27);
        if (!gu && first && c == 0) ED_AT(12);
        if (!gu && first && c == nstages - 1) ED_AT(13);
        ptx::tc_fence_after();
        const uint32_t a0 = ptx::smem_addr(slot_a(stage));
        const uint32_t b0 = ptx::smem_addr(slot_b(stage));
        for (int kb = kb0; kb < kb1; ++kb)
#pragma unroll
          for (int kk = 0; kk < kTileK / 16; ++kk)
            ptx::mma_bf16(d0, ptx::sdesc_k_sw128(a0 + kb * abox + kk * 32),
                          ptx::sdesc_k_sw128(b0 + kb * bbox + kk * 32), idesc,
                          (c > 0 || kb > kb0 || kk > 0) ? 1u : 0u);
        ptx::mma_commit(&empty[stage]);
        if (++stage == S) { stage = 0; phase ^= 1u; }
      }
      ptx::mma_commit(&acc_full[acc]);
      if (++acc == p.n_acc) { acc = 0; acc_phase ^= 1u; }
    };
    for (int u = b; u < NGU && ok; u += nb) {
      int gi, m;
      gu_unit(u, gi, m);
      // all T token columns: the B box is x (rows >= T are zeros)
      run(kc, kbg, abox_g, (uint32_t)(2 * hg), u, true);
      if (first) ED_AT(3);
      first = false;
    }
    first = half == 0;
    for (int v = v0; v < ND && ok; v += nb) {
      const Grp g = group_w(v / ndn);
      run(g.Ig / kStageK, kKB, kABox, (uint32_t)kTileM, v, false);
      if (first) ED_AT(7);
      first = false;
    }
    // no MMA may still run when TMEM is released
    ptx::mma_commit(drain);
    const uint64_t t0 = ptx::globaltimer_ns();
    while (!ptx::mbar_try_wait(drain, 0) && ptx::globaltimer_ns() - t0 < kTimeoutNs) {
    }
  } else if (warp >= 2 && warp <= 5) {
    // ================= epilogue: warps 2..5, TMEM lanes 32*(warp%4) ..
    const int q = warp & 3;
    const int et = tid - 64;                      // 0..127
    const int row = q * 32 + lane;                // accumulator row of this thread
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const bool is_gate = q < 2;
    // gate/up accumulator (M = 2 hg): row r sits in TMEM lane r for M = 128 and in lane
    // 32 (r / 16) + r % 16 for M = 64, so each quadrant holds rq = hg / 2 rows in its first
    // rq lanes: gate rows in quadrants 0-1, the matching up rows in quadrants 2-3
    const int rq = hg / 2;
    const bool g_act = lane < rq;
    const int rr = (q & 1) * rq + lane;           // row within the hg-row slice
    const int n_mma = (p.T + 15) & ~15;
    const uint32_t part1 = (uint32_t)(p.n_acc * p.n_pad);   // column offset of part 1
    // 16 columns of an accumulator: the sum of its two parts
    auto acc_ld16 = [&](uint32_t taddr, float (&v)[16]) {
      float w[16];
      ptx::tmem_ld16(taddr, v);
      ptx::tmem_ld16(taddr + part1, w);
      ptx::tmem_ld_wait();
#pragma unroll
      for (int c = 0; c < 16; ++c) {
        asm volatile("" : "+f"(v[c]), "+f"(w[c]));   // the values exist only after the wait
        v[c] += w[c];
      }
    };
    int acc = 0;
    uint32_t acc_phase = 0;
    bool first = true;
    for (int u = b; u < NGU; u += nb) {
      int gi, m;
      gu_unit(u, gi, m);
      const bool ok = epi_all(wait(&acc_full[acc], acc_phase, u));
      if (!ok) break;
      if (first && et == 0) ED_AT(20);
      ptx::tc_fence_after();
      const uint32_t tbase = tmem_base + lane_off + (uint32_t)(acc * p.n_pad);
      // the H tile (n_pad token rows x hg columns, bf16) is laid out in the staging tile as
      // hg / 32 row-major boxes of 32 columns, then stored by TMA
      uint8_t* hbox = reinterpret_cast<uint8_t*>(stage_t);
      // per 16-token slice: every row's 16 values go to the exchange tile (gate rows
      // 0..hg-1, up rows hg..2hg-1), then all 128 threads take hg / 8 adjacent columns of one
      // token each (loads first, then the SwiGLU, then one 8- or 16-byte store)
      const int cpt = hg >> 3, xc = et >> 3, col0 = (et & 7) * cpt;
      uint8_t* hdst = hbox + (col0 >> 5) * p.n_pad * 64 + (col0 & 31) * 2;
      for (int c0 = 0; c0 < n_mma; c0 += 16) {
        float v[16];
        acc_ld16(tbase + c0, v);
        if (first && et == 0 && c0 == 0) ED_AT(23);
        if (g_act) {
          float* xr = xchg + ((is_gate ? 0 : hg) + rr) * kXStride;
#pragma unroll
          for (int c = 0; c < 16; ++c) xr[c] = v[c];
        }
        named_bar_sync(2, 128);
        if (first && et == 0 && c0 == 0) ED_AT(24);
        float gv[8], uv[8];
#pragma unroll
        for (int j = 0; j < 8; ++j)
          if (j < cpt) {
            gv[j] = xchg[(col0 + j) * kXStride + xc];
            uv[j] = xchg[(hg + col0 + j) * kXStride + xc];
          }
        uint32_t hp[4];
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (2 * j < cpt) {
            const __nv_bfloat162 h2 = __floats2bfloat162_rn(silu_f(gv[2 * j]) * uv[2 * j],
                                                            silu_f(gv[2 * j + 1]) * uv[2 * j + 1]);
            hp[j] = *reinterpret_cast<const uint32_t*>(&h2);
          }
        uint8_t* hrow = hdst + (c0 + xc) * 64;
        if (cpt == 4)
          *reinterpret_cast<uint2*>(hrow) = make_uint2(hp[0], hp[1]);
        else
          *reinterpret_cast<uint4*>(hrow) = make_uint4(hp[0], hp[1], hp[2], hp[3]);
        named_bar_sync(2, 128);   // the exchange tile is rewritten by the next slice
      }
      if (first && et == 0) ED_AT(25);
      ptx::tc_fence_before();
      ptx::mbar_arrive(&acc_empty[acc]);
      if (++acc == p.n_acc) { acc = 0; acc_phase ^= 1u; }
      // publish the tile: one bulk store of the box, waited to completion, then one release
      // add; a reader acquires the counter, then fences the async proxy
      ptx::fence_proxy_async_smem();
      named_bar_sync(2, 128);
      if (et == 0) {
        if (first) ED_AT(21);
        for (int j = 0; j < hg / 32; ++j)
          tma_store_2d(&tm.hst, hbox + j * p.n_pad * 64, m * hg + 32 * j, gi * p.n_pad);
        bulk_commit_wait_all();
        if (first) ED_AT(22);
        fence_proxy_async_global();
        red_release_add(p.h_ready + gi, 1);
        if (first) ED_AT(4);
      }
      named_bar_sync(2, 128);   // the box is rewritten by the next tile
      first = false;
    }
    first = true;
    if (spec && v0 < ND) {
      // the rows of the dispatch from here on; the coresets must have given its unique list
      pdl_wait();
      if (warp == 2) {
        // ids: the lists are equal; masks: the dispatch's list is inside the union
        const int nd = __ldcg(p.n_unique);
        bool bad = kMask ? (nd < 0 || nd > U) : nd != U;
        if (!bad && kMask) {
          for (int u = lane; u < nd; u += 32) {
            const int e = __ldcg(p.unique_ids + u);
            if (e < 0 || e >= p.E || ((s_mask[e >> 5] >> (e & 31)) & 1u) == 0u) bad = true;
          }
        } else if (!bad) {
          for (int u = lane; u < U; u += 32)
            if (__ldcg(p.unique_ids + u) != (int)s_spec[u]) bad = true;
        }
        if (__any_sync(0xffffffffu, bad) && lane == 0)
          record_error(p.err, kErrBadDispatch, kAtDown, -1);
      }
    }
    for (int v = v0; v < ND; v += nb) {
      const int gi = v / ndn, i = v % ndn;
      const Grp g = group(gi);
      if (!g.shared && et < g.n) tok[et] = __ldcg(p.rows + g.row0 + et) / p.k;
      const bool ok = epi_all(wait(&acc_full[acc], acc_phase, v));   // also orders tok[]
      if (!ok) break;
      if (first && et == 0) ED_AT(14);
      ptx::tc_fence_after();
      const uint32_t tbase = tmem_base + lane_off + (uint32_t)(acc * p.n_pad);
      // the accumulator column of token t is the group's output for t: the tile goes through
      // shared memory as [token][128 rows] fp32, then one 512-B bulk copy per kept row (every
      // token for the shared expert, the routed ones in dispatch order otherwise)
      float* stg = stage_t;
      for (int c0 = 0; c0 < n_mma; c0 += 16) {
        float vv[16];
        acc_ld16(tbase + c0, vv);
#pragma unroll
        for (int c = 0; c < 16; ++c)
          if (c0 + c < p.T) stg[(c0 + c) * kTileM + row] = vv[c];
      }
      ptx::tc_fence_before();
      ptx::mbar_arrive(&acc_empty[acc]);
      if (++acc == p.n_acc) { acc = 0; acc_phase ^= 1u; }
      if (first && et == 0) ED_AT(15);
      ptx::fence_proxy_async_smem();
      named_bar_sync(2, 128);
      if (et < 32) {
        if (first && et == 0) ED_AT(16);
        const int nrows = g.shared ? p.T : g.n;
        // every token kept (the shared expert; a routed group that all T tokens use, whose
        // dispatch rows are then tokens 0..T-1 in order): the staging tile is the rows' image,
        // stored 8 rows per tensor copy; otherwise one 512-B row copy per lane
        bool dense = nrows == p.T && (p.T & 7) == 0;
        if (dense && !g.shared)
          for (int r = et; r < nrows; r += 32) dense = dense && tok[r] == r;
        dense = __all_sync(0xffffffffu, dense);
        if (dense) {
          if (et == 0)
            for (int r8 = 0; r8 < nrows; r8 += 8)
              tma_store_2d(g.shared ? &tm.ysh : &tm.ys, stg + r8 * kTileM, i * kTileM,
                           (g.shared ? 0 : g.row0) + r8);
        } else {
          const size_t col = (size_t)i * kTileM;
          for (int r = et; r < nrows; r += 32) {
            const int t = g.shared ? r : tok[r];
            float* dst = g.shared ? p.yshared + (size_t)r * p.d + col
                                  : p.yslot + (size_t)(g.row0 + r) * p.d + col;
            if (t >= 0 && t < p.T) bulk_store(dst, stg + t * kTileM, kTileM * 4);
          }
        }
        if (first && et == 0) ED_AT(17);
        bulk_commit_wait_read();   // the staging tile is rewritten by the next unit
      }
      named_bar_sync(2, 128);   // tok[] and the staging tile are rewritten by the next unit
      if (first && et == 0) ED_AT(8);
      first = false;
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  // the combine may start now: launched earlier, its waiting CTAs would share SMs with the
  // routing launch of this forward and slow it down
  pdl_launch_dependents();
  if (warp == 1) {
    __syncwarp();
    ptx::tmem_dealloc(tmem_base, p.tmem_cols);
  }
  if (tid == 0) ED_AT(9);
  KLOG(DMOE_KERNEL_EXPERTS, 1);
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

// bf16 matrix [rows, cols] row-major, box = 64 columns (128 B) x box_rows rows with the
// 128-B swizzle, or (plain) box_cols columns x box_rows rows without swizzle.
bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows,
              bool plain = false, uint32_t box_cols = 64) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {plain ? box_cols : 64u, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             plain ? CU_TENSOR_MAP_SWIZZLE_NONE : CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// fp32 matrix [rows, cols] row-major, box = 128 columns x 8 rows, no swizzle.
bool make_map_f32(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 4};
  const cuuint32_t box[2] = {(cuuint32_t)kTileM, 8};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
             CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Opt-in shared memory per CTA; without a device (host-side planning) the sm_100-family
// figure, 227 KB.
int max_smem_optin() {
  int dev = 0, v = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
      v <= 0) {
    cudaGetLastError();
    v = 227 * 1024;
  }
  return v;
}

uint32_t pow2_cols(uint32_t n) {
  uint32_t c = 32;
  while (c < n) c <<= 1;
  return c;
}

// Shared memory besides the ring: staging tile, SwiGLU exchange, token list, barriers.
size_t fixed_smem(int n_pad) {
  return 1024 /* alignment */ + (size_t)kTileM * (n_pad + 1) * 4 + kXchgBytes + kMaxTok * 4 +
         (size_t)(2 * kMaxStagesD + 9) * 8 + 16 + kMaxExperts + kMaxExperts / 8 + 48;
}

// Pipeline ring: the shared memory left by the fixed part. A slot holds 32 KB of weights
// and two K boxes of token rows (64-row gate/up units, down tiles) or four (32-row gate/up
// units, K = 256 per stage; allowed when d is a multiple of 256 and three slots fit).
struct Ring {
  int bytes, stages2, h32_ok;
};
Ring plan_ring(int T, int d) {
  const int n_pad = ((T + 15) / 16) * 16;
  long avail = (long)max_smem_optin() - (long)fixed_smem(n_pad);
  avail = avail > 0 ? (avail & ~1023L) : 0;
  Ring r;
  r.bytes = (int)avail;
  r.stages2 = (int)(avail / (kAStage + kKB * n_pad * 128));
  r.h32_ok = d % (kMaxKBG * kTileK) == 0 && avail / (kAStage + kMaxKBG * n_pad * 128) >= 3;
  return r;
}

}  // namespace

#ifdef DMOE_TRACE
DMOE_KLOG_EXPORT(dmoe_debug_klog_decode)
extern "C" int dmoe_debug_dtrace(void* host) {
  return (int)cudaMemcpyFromSymbol(host, g_dtrace, sizeof(g_dtrace));
}
extern "C" int dmoe_debug_dtrace_clear() {
  static uint64_t zeros[kMaxPersistentCtas * 32];
  return (int)cudaMemcpyToSymbol(g_dtrace, zeros, sizeof(zeros));
}
#endif

bool experts_decode_ok(int T, int d, int I, int Is) {
  if (T < 1 || T > kMaxTok || d % kTileM != 0 || I % kStageK != 0 || (Is > 0 && Is % kStageK != 0))
    return false;
  return plan_ring(T, d).stages2 >= 2;
}

cudaError_t launch_experts_decode(const ExpertArgs& a, cudaStream_t s) {
  const bool has_shared = a.Is > 0;
  const Ring ring = plan_ring(a.T, a.d);
  if (ring.stages2 < 2) return cudaErrorInvalidConfiguration;
  const int n_pad = ((a.T + 15) / 16) * 16;
  const int imax = a.I > a.Is ? a.I : a.Is;

  DMaps m;
  bool ok = make_map(&m.wg, a.w_gate, (uint64_t)a.E * a.I, a.d, 64) &&
            make_map(&m.wu, a.w_up, (uint64_t)a.E * a.I, a.d, 64) &&
            make_map(&m.wg32, a.w_gate, (uint64_t)a.E * a.I, a.d, 32) &&
            make_map(&m.wu32, a.w_up, (uint64_t)a.E * a.I, a.d, 32) &&
            make_map(&m.wd, a.w_down, (uint64_t)a.E * a.d, a.I, kTileM) &&
            make_map(&m.x, a.x, (uint64_t)a.T, a.d, (uint32_t)n_pad) &&
            make_map(&m.h, a.hdense, (uint64_t)(a.E + 1) * n_pad, (uint64_t)imax,
                     (uint32_t)n_pad) &&
            make_map(&m.hst, a.hdense, (uint64_t)(a.E + 1) * n_pad, (uint64_t)imax,
                     (uint32_t)n_pad, true, 32) &&
            make_map_f32(&m.ys, a.yslot, (uint64_t)a.T * a.k, a.d) &&
            make_map_f32(&m.ysh, a.yshared, (uint64_t)a.T, a.d);
  if (ok && has_shared)
    ok = make_map(&m.sg, a.ws_gate, (uint64_t)a.Is, a.d, 64) &&
         make_map(&m.su, a.ws_up, (uint64_t)a.Is, a.d, 64) &&
         make_map(&m.sg32, a.ws_gate, (uint64_t)a.Is, a.d, 32) &&
         make_map(&m.su32, a.ws_up, (uint64_t)a.Is, a.d, 32) &&
         make_map(&m.sd, a.ws_down, (uint64_t)a.d, a.Is, kTileM);
  if (!has_shared) { m.sg = m.wg; m.su = m.wu; m.sd = m.wd; m.sg32 = m.wg32; m.su32 = m.wu32; }
  if (!ok) return cudaErrorInvalidValue;

  DParams p{};
  p.n_unique = a.n_unique;
  p.unique_ids = a.unique_ids;
  p.offsets = a.offsets;
  p.rows = a.rows;
  p.hdense = a.hdense;
  p.yslot = static_cast<float*>(a.yslot);
  p.yshared = static_cast<float*>(a.yshared);
  p.h_ready = a.h_ready;
  p.spec_words = a.spec_words;
  p.spec_blocks = a.spec_blocks;
  p.spec_mask = a.spec_mask ? 1 : 0;
  p.err = a.err;
  p.T = a.T; p.d = a.d; p.E = a.E; p.k = a.k; p.I = a.I; p.Is = a.Is;
  p.imax = imax;
  p.n_pad = n_pad;
  p.ring_bytes = ring.bytes;
  p.h32_ok = ring.h32_ok;
  p.has_shared = has_shared ? 1 : 0;
  p.n_acc = 256 / n_pad > 4 ? 4 : 256 / n_pad;   // accumulators of two parts each
  p.tmem_cols = pow2_cols((uint32_t)(2 * p.n_acc * n_pad));
  const size_t smem = (size_t)ring.bytes + fixed_smem(n_pad);

  static std::mutex mu;
  static int attr_dev_mask = 0;  // the dynamic smem limit is a per-device function attribute
  int dev = 0;
  cudaGetDevice(&dev);
  {
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= 31 || !(attr_dev_mask & (1 << dev))) {
      cudaError_t e = cudaFuncSetAttribute(moe_decode_kernel<false>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           max_smem_optin());
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(moe_decode_kernel<true>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem_optin());
      if (e != cudaSuccess) return e;
      if (dev < 31) attr_dev_mask |= 1 << dev;
    }
  }
  // one CTA per SM; when the stream starts on the published coresets, the last routing
  // cluster still holds its SMs, and a CTA placed there would start only when it ends
  int grid = device_sm_count();
  if (a.spec_words != nullptr && grid > 2 * kRouteClusterCtas) grid -= kRouteClusterCtas;
  if (grid > kMaxPersistentCtas) grid = kMaxPersistentCtas;
  prof_begin(DMOE_KERNEL_EXPERTS, s);
  cudaError_t e =
      p.spec_mask ? launch_ex(moe_decode_kernel<true>, dim3(grid), dim3(kThr), smem, s,
                              !prof_serial(DMOE_KERNEL_EXPERTS), m, p)
                  : launch_ex(moe_decode_kernel<false>, dim3(grid), dim3(kThr), smem, s,
                              !prof_serial(DMOE_KERNEL_EXPERTS), m, p);
  prof_end(DMOE_KERNEL_EXPERTS, s);
  if (e != cudaSuccess) return e;
  // the expert launch releases the combine at its end, after its wait for the routing
  // launch (which wrote the slot indices and gates): the combine may read them at once
  return launch_combine(a, s, a.h_ready, a.E + 1, a.spec_words,
                        a.spec_words != nullptr
                            ? a.spec_blocks * (a.spec_mask ? kSpecMaskWords : spec_words(a.k))
                            : 0,
                        /*meta_early=*/true);
}

}  // namespace dmoe
