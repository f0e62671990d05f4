// Expert execution of the MoE layer: grouped SwiGLU FFN over the unique experts of one
// forward (plus the shared expert), on tcgen05 tensor cores.
//
// Both GEMMs are "swap-AB": the expert weights are the MMA's M operand (128 weight rows per
// tile, streamed by TMA with the 128-byte swizzle), the few tokens routed to an expert are
// the N operand, K is the reduction dimension, and the fp32 accumulator lives in TMEM.
//
//   gather_kernel     x rows in dispatch order -> xperm [T*k, d]
//   gate/up kernel    per (group, 64 rows of I, token tile): the A tile stacks 64 rows of
//                     W_gate over the same 64 rows of W_up, so one M=128 MMA chain gives
//                     gate (TMEM lanes 0-63) and up (lanes 64-127) of those rows; the
//                     epilogue warps holding "up" pass it through shared memory to the
//                     warps holding "gate", which write h = silu(gate) * up as bf16 H.
//   down kernel       per (group, 128 rows of d, token tile): D = W_down * H^T; the
//                     epilogue stores the fp32 rows per (token, slot)
//   combine_kernel    y_t = sum over slots (slot order) of g_tj * row + shared -> bf16
//
// A group is one unique expert (dispatch order) or the shared expert (all T tokens). Both
// GEMM kernels are persistent (one CTA per SM) and warp-specialised: warp 0 issues TMA,
// warp 1 issues MMAs, warps 2-5 run the epilogue. The unit list is derived on the device
// from the dispatch output, so no host round-trip is needed. Consecutive kernels are
// chained with programmatic dependent launch: each kernel's set-up (barriers, TMEM,
// tensor-map prefetch) overlaps the previous kernel, and griddepcontrol.wait orders the
// reads of its outputs.
#include <math.h>

#include <mutex>

#include "dmoe_internal.cuh"
#include "sm100_ptx.cuh"

namespace dmoe {
namespace {

constexpr int kThreads = 192;                      // 6 warps
constexpr int kATileBytes = kTileM * kTileK * 2;   // 16 KB: 128 rows x 64 K
constexpr int kHalfTileBytes = kATileBytes / 2;    // 8 KB: 64 rows x 64 K
constexpr int kMaxGroups = kMaxExperts + 1;
constexpr uint64_t kWaitTimeoutNs = 1000000000ull;  // 1 s
constexpr int kMaxStages = 12;
constexpr int kXchgStride = 17;                    // floats per row of the exchange buffer

struct GemmParams {
  const int32_t* n_unique;
  const int32_t* unique_ids;
  const int32_t* offsets;
  __nv_bfloat16* h;       // [T*k, I]
  __nv_bfloat16* hs;      // [T, Is]
  float* yslot;           // [T*k, d]
  float* yshared;         // [T, d]
  DevErrRecord* err;
  int T, d, E, k, I, Is;
  int n_max;              // token tile = rows of the B box
  int stages;
  int n_acc;              // accumulator buffers in TMEM
  uint32_t tmem_cols;
  int has_shared;
};

__device__ __forceinline__ void named_bar_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

// AND of `v` over the 128 epilogue threads (named barrier 1), so that they leave the unit
// loop together when a wait gives up.
__device__ __forceinline__ bool epi_all(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, 1, 128, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ float silu_f(float z) { return z / (1.f + __expf(-z)); }

template <bool kGateUp>
__global__ void __launch_bounds__(kThreads, 1)
expert_gemm_kernel(const __grid_constant__ CUtensorMap tm_a0,   // W_gate [E*I, d] (64-row box) | W_down [E*d, I]
                   const __grid_constant__ CUtensorMap tm_a1,   // W_up   [E*I, d] (64-row box) | unused
                   const __grid_constant__ CUtensorMap tm_b,    // xperm [T*k, d] | H [T*k, I]
                   const __grid_constant__ CUtensorMap tm_sa0,  // W_sgate [Is, d] | W_sdown [d, Is]
                   const __grid_constant__ CUtensorMap tm_sa1,  // W_sup   [Is, d] | unused
                   const __grid_constant__ CUtensorMap tm_sb,   // x [T, d] | Hs [T, Is]
                   const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-B aligned base (the swizzled tiles need it)
  const uint32_t raw_addr = ptx::smem_addr(smem_raw);
  uint8_t* smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);

  constexpr int kRowsPerTile = kGateUp ? kTileM / 2 : kTileM;  // weight rows of I or d per tile
  const int stages = p.stages;
  const uint32_t b_bytes = (uint32_t)p.n_max * 128u;
  const uint32_t off_a = 0;
  const uint32_t off_b = off_a + (uint32_t)stages * kATileBytes;
  const uint32_t off_x = off_b + (uint32_t)stages * b_bytes;           // epilogue exchange
  const uint32_t x_bytes = kGateUp ? 2u * 64u * kXchgStride * 4u : 0u;  // 2 buffers [64][17] fp32
  const uint32_t off_bar = (off_x + x_bytes + 7u) & ~7u;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + off_bar);
  uint64_t* empty = full + stages;
  uint64_t* acc_full = empty + stages;
  uint64_t* acc_empty = acc_full + 4;
  uint64_t* drain = acc_empty + 4;
  int* misc = reinterpret_cast<int*>(drain + 1);
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(misc + 0);
  volatile int* s_abort = misc + 1;
  int* s_sched = misc + 4;                     // G, U, units
  int* g_prefix = misc + 8;                    // [kMaxGroups + 1] tile prefix
  int* g_row0 = g_prefix + (kMaxGroups + 1);   // [kMaxGroups]
  int* g_cnt = g_row0 + kMaxGroups;            // [kMaxGroups]
  int* g_e = g_cnt + kMaxGroups;               // [kMaxGroups]
  float* xchg = reinterpret_cast<float*>(smem + off_x);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int mtiles_routed = (kGateUp ? p.I : p.d) / kRowsPerTile;
  const int mtiles_shared = (kGateUp ? p.Is : p.d) / kRowsPerTile;

  // ---------------- set-up that does not read the previous kernel's output
  if (tid == 0) {
    for (int s = 0; s < stages; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 4; ++a) {
      ptx::mbar_init(&acc_full[a], 1);
      ptx::mbar_init(&acc_empty[a], 128);
    }
    ptx::mbar_init(drain, 1);
    ptx::fence_mbarrier_init();
    *s_abort = 0;
    ptx::prefetch_tensormap(&tm_a0);
    if (kGateUp) ptx::prefetch_tensormap(&tm_a1);
    ptx::prefetch_tensormap(&tm_b);
    if (p.has_shared) {
      ptx::prefetch_tensormap(&tm_sa0);
      ptx::prefetch_tensormap(&tm_sb);
    }
  }
  if (warp == 1) {
    ptx::tmem_alloc(s_tmem, p.tmem_cols);
    ptx::tmem_relinquish();
  }
  pdl_launch_dependents();
  pdl_wait();  // the dispatch output (and H for the down kernel) is complete from here on

  // ---------------- the unit list, from the dispatch output
  if (warp == 0) {
    int U = *p.n_unique;
    if (U < 0 || U > p.E) {
      if (lane == 0) record_error(p.err, kErrBadDispatch, kGateUp ? kAtGateUp : kAtDown, U);
      U = 0;
    }
    const int G = U + (p.has_shared ? 1 : 0);
    int carry = 0;
    for (int base = 0; base < G; base += 32) {
      const int g = base + lane;
      int tiles = 0;
      if (g < G) {
        int cnt, row0, e, mt;
        if (g < U) {
          row0 = p.offsets[g];
          cnt = p.offsets[g + 1] - row0;
          e = p.unique_ids[g];
          mt = mtiles_routed;
          if (e < 0 || e >= p.E || cnt < 0 || cnt > p.T || row0 < 0 ||
              row0 + cnt > p.T * p.k) {
            record_error(p.err, kErrBadDispatch, kGateUp ? kAtGateUp : kAtDown, g);
            cnt = 0;
            e = 0;
            row0 = 0;
          }
        } else {
          row0 = 0;
          cnt = p.T;
          e = -1;
          mt = mtiles_shared;
        }
        g_row0[g] = row0;
        g_cnt[g] = cnt;
        g_e[g] = e;
        tiles = ((cnt + p.n_max - 1) / p.n_max) * mt;
      }
      int incl = tiles;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += u;
      }
      if (g < G) g_prefix[g + 1] = carry + incl;
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) {
      g_prefix[0] = 0;
      s_sched[0] = G;
      s_sched[1] = U;
      s_sched[2] = carry;
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem_base = *s_tmem;
  const int G = s_sched[0], U = s_sched[1], units = s_sched[2];

  // unit -> (group, m tile, n tile); m varies fastest so that neighbouring CTAs share the
  // token tile of one expert
  auto decode = [&](int u, int& g, int& m_idx, int& n_idx) {
    int lo = 0, hi = G - 1;  // largest g with g_prefix[g] <= u
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (g_prefix[mid] <= u) lo = mid; else hi = mid - 1;
    }
    g = lo;
    const int local = u - g_prefix[g];
    const int mt = (g < U) ? mtiles_routed : mtiles_shared;
    n_idx = local / mt;
    m_idx = local - n_idx * mt;
  };
  const int where = kGateUp ? kAtGateUp : kAtDown;
  auto wait = [&](uint64_t* bar, uint32_t parity, int value) -> bool {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::globaltimer_ns();
    for (uint32_t i = 1;; ++i) {
      if (ptx::mbar_try_wait(bar, parity)) return true;
      if ((i & 63u) == 0u) {
        if (*s_abort) return false;
        if (ptx::globaltimer_ns() - t0 > kWaitTimeoutNs) {
          record_error(p.err, kErrTimeout, where, value);
          *s_abort = 1;
          return false;
        }
      }
    }
  };

  if (warp == 0) {
    // ================= TMA producer
    if (lane == 0) {
      const uint64_t pol_w = ptx::policy_evict_first();   // weights: streamed once
      const uint64_t pol_x = ptx::policy_evict_last();    // activations: re-read by tiles
      const uint32_t tx_bytes = kATileBytes + b_bytes;
      int stage = 0;
      uint32_t phase = 0;
      int issued = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        int g, m_idx, n_idx;
        decode(u, g, m_idx, n_idx);
        const bool shared = g >= U;
        const int Kg = kGateUp ? p.d : (shared ? p.Is : p.I);
        const int kc = Kg / kTileK;
        const int arow = shared ? m_idx * kRowsPerTile
                                : g_e[g] * (kGateUp ? p.I : p.d) + m_idx * kRowsPerTile;
        const int brow = (shared ? 0 : g_row0[g]) + n_idx * p.n_max;
        const CUtensorMap* ma0 = shared ? &tm_sa0 : &tm_a0;
        const CUtensorMap* ma1 = shared ? &tm_sa1 : &tm_a1;
        const CUtensorMap* mb = shared ? &tm_sb : &tm_b;
        for (int c = 0; c < kc; ++c) {
          if (!wait(&empty[stage], phase ^ 1u, u)) { ok = false; break; }
          ptx::mbar_arrive_expect_tx(&full[stage], tx_bytes);
          const int kx = c * kTileK;
          uint8_t* a_dst = smem + off_a + stage * kATileBytes;
          ptx::tma_load_2d(a_dst, ma0, &full[stage], kx, arow, pol_w);
          if (kGateUp)
            ptx::tma_load_2d(a_dst + kHalfTileBytes, ma1, &full[stage], kx, arow, pol_w);
          ptx::tma_load_2d(smem + off_b + stage * b_bytes, mb, &full[stage], kx, brow, pol_x);
          ++issued;
          if (++stage == stages) { stage = 0; phase ^= 1u; }
        }
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
      const uint32_t acc_cols = (uint32_t)p.n_max;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        int g, m_idx, n_idx;
        decode(u, g, m_idx, n_idx);
        const bool shared = g >= U;
        const int Kg = kGateUp ? p.d : (shared ? p.Is : p.I);
        const int kc = Kg / kTileK;
        const int nvalid = min(p.n_max, g_cnt[g] - n_idx * p.n_max);
        const uint32_t n_mma = (uint32_t)((nvalid + 15) & ~15);
        const uint32_t idesc = ptx::idesc_bf16(kTileM, n_mma);
        if (!wait(&acc_empty[acc], acc_phase ^ 1u, u)) { ok = false; break; }
        ptx::tc_fence_after();
        const uint32_t d0 = tmem_base + (uint32_t)acc * acc_cols;
        for (int c = 0; c < kc; ++c) {
          if (!wait(&full[stage], phase, u)) { ok = false; break; }
          ptx::tc_fence_after();
          const uint32_t a0 = ptx::smem_addr(smem + off_a + stage * kATileBytes);
          const uint32_t bb = ptx::smem_addr(smem + off_b + stage * b_bytes);
#pragma unroll
          for (int kk = 0; kk < kTileK / 16; ++kk)
            ptx::mma_bf16(d0, ptx::sdesc_k_sw128(a0 + kk * 32), ptx::sdesc_k_sw128(bb + kk * 32),
                          idesc, (c > 0 || kk > 0) ? 1u : 0u);
          ptx::mma_commit(&empty[stage]);
          if (++stage == stages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        ptx::mma_commit(&acc_full[acc]);
        if (++acc == p.n_acc) { acc = 0; acc_phase ^= 1u; }
      }
      // make sure no MMA is still running when TMEM is released
      ptx::mma_commit(drain);
      const uint64_t t0 = ptx::globaltimer_ns();
      while (!ptx::mbar_try_wait(drain, 0) && ptx::globaltimer_ns() - t0 < kWaitTimeoutNs) {
      }
    }
  } else {
    // ================= epilogue: warps 2..5, TMEM lanes 32*(warp%4) ..
    const int q = warp & 3;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    int acc = 0, xb = 0;
    uint32_t acc_phase = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x) {
      int g, m_idx, n_idx;
      decode(u, g, m_idx, n_idx);
      const bool shared = g >= U;
      const int nvalid = min(p.n_max, g_cnt[g] - n_idx * p.n_max);
      const int n_mma = (nvalid + 15) & ~15;
      if (!epi_all(wait(&acc_full[acc], acc_phase, u))) break;
      ptx::tc_fence_after();
      const uint32_t tbase = tmem_base + lane_off + (uint32_t)acc * (uint32_t)p.n_max;
      const int col0 = n_idx * p.n_max;              // first token column of the tile
      if (kGateUp) {
        // lanes 0-63: gate rows, lanes 64-127: up rows of the same 64 intermediate units
        const bool is_gate = q < 2;
        const int r64 = (q & 1) * 32 + lane;         // row within the 64-row slice
        const int Ig = shared ? p.Is : p.I;
        __nv_bfloat16* hout = shared ? p.hs : p.h;
        const int hrow0 = (shared ? 0 : g_row0[g]) + col0;
        const int icol = m_idx * 64 + r64;
        for (int c0 = 0; c0 < n_mma; c0 += 16) {
          float v[16];
          ptx::tmem_ld16(tbase + c0, v);
          ptx::tmem_ld_wait();
          float* buf = xchg + xb * (64 * kXchgStride);
          if (!is_gate) {
#pragma unroll
            for (int c = 0; c < 16; ++c) buf[r64 * kXchgStride + c] = v[c];
          }
          named_bar_sync(2, 128);
          if (is_gate) {
#pragma unroll
            for (int c = 0; c < 16; ++c)
              if (c0 + c < nvalid)
                hout[(size_t)(hrow0 + c0 + c) * Ig + icol] =
                    __float2bfloat16(silu_f(v[c]) * buf[r64 * kXchgStride + c]);
          }
          xb ^= 1;
        }
      } else {
        const int drow = m_idx * kTileM + q * 32 + lane;
        float* out = shared ? p.yshared + (size_t)col0 * p.d
                            : p.yslot + (size_t)(g_row0[g] + col0) * p.d;
        for (int c0 = 0; c0 < n_mma; c0 += 16) {
          float v[16];
          ptx::tmem_ld16(tbase + c0, v);
          ptx::tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < 16; ++c)
            if (c0 + c < nvalid) out[(size_t)(c0 + c) * p.d + drow] = v[c];
        }
      }
      ptx::tc_fence_before();
      ptx::mbar_arrive(&acc_empty[acc]);
      if (++acc == p.n_acc) { acc = 0; acc_phase ^= 1u; }
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    ptx::tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

// xperm[r, :] = x[rows[r] / k, :]
__global__ void __launch_bounds__(256)
gather_kernel(const __nv_bfloat16* __restrict__ x, const int32_t* __restrict__ rows,
              __nv_bfloat16* __restrict__ xperm, int pairs, int k, int d) {
  pdl_launch_dependents();
  pdl_wait();
  const int vec = d / 8;  // uint4 per row
  for (int r = blockIdx.x; r < pairs; r += gridDim.x) {
    const int t = rows[r] / k;
    const uint4* src = reinterpret_cast<const uint4*>(x + (size_t)t * d);
    uint4* dst = reinterpret_cast<uint4*>(xperm + (size_t)r * d);
    for (int i = threadIdx.x; i < vec; i += blockDim.x) dst[i] = src[i];
  }
}

// y[t, :] = bf16( sum_j g[t,j] * yslot[pos[t*k + j], :] (slot order) + yshared[t, :] )
__global__ void __launch_bounds__(256)
combine_kernel(const float* __restrict__ yslot, const float* __restrict__ yshared,
               const int32_t* __restrict__ pos, const float* __restrict__ gate,
               __nv_bfloat16* __restrict__ y, int k, int d, int has_shared) {
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.y;
  const int c = (blockIdx.x * blockDim.x + threadIdx.x) * 4;
  if (c >= d) return;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int j = 0; j < k; ++j) {
    const int r = pos[t * k + j];
    const float gj = gate[t * k + j];
    const float4 v = *reinterpret_cast<const float4*>(yslot + (size_t)r * d + c);
    acc.x = fmaf(gj, v.x, acc.x);
    acc.y = fmaf(gj, v.y, acc.y);
    acc.z = fmaf(gj, v.z, acc.z);
    acc.w = fmaf(gj, v.w, acc.w);
  }
  if (has_shared) {
    const float4 v = *reinterpret_cast<const float4*>(yshared + (size_t)t * d + c);
    acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
  }
  __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x, acc.y);
  __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z, acc.w);
  uint2 out;
  out.x = *reinterpret_cast<uint32_t*>(&lo);
  out.y = *reinterpret_cast<uint32_t*>(&hi);
  *reinterpret_cast<uint2*>(y + (size_t)t * d + c) = out;
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

size_t gemm_fixed_smem(bool gate_up) {
  // alignment slack + exchange buffers + barriers + misc/group arrays
  return 1024 + (gate_up ? 2 * 64 * kXchgStride * 4 : 0) + 8 +
         8 * (2 * kMaxStages + 9) + sizeof(int) * (8 + 4 * (kMaxGroups + 1)) + 64;
}

int max_smem_optin() {
  int dev = 0, v = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  return v;
}

template <bool kGateUp>
cudaError_t launch_gemm(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& b,
                        const CUtensorMap& sa0, const CUtensorMap& sa1, const CUtensorMap& sb,
                        GemmParams gp, cudaStream_t s) {
  const size_t stage_bytes = (size_t)kATileBytes + (size_t)gp.n_max * 128;
  const size_t fixed = gemm_fixed_smem(kGateUp);
  const int limit = max_smem_optin();
  int stages = (int)((limit - (int)fixed) / (int)stage_bytes);
  if (stages > kMaxStages) stages = kMaxStages;
  if (stages < 2) return cudaErrorInvalidConfiguration;
  gp.stages = stages;
  const uint32_t acc_cols = (uint32_t)gp.n_max;
  gp.n_acc = (int)(512 / acc_cols);
  if (gp.n_acc > 4) gp.n_acc = 4;
  gp.tmem_cols = pow2_cols(gp.n_acc * acc_cols);
  const size_t smem = fixed + (size_t)stages * stage_bytes;
  static int attr_dev_mask = 0;  // per-device: the dynamic smem limit is a function attribute
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 31 || !(attr_dev_mask & (1 << dev))) {
    cudaError_t e = cudaFuncSetAttribute(expert_gemm_kernel<kGateUp>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, limit);
    if (e != cudaSuccess) return e;
    if (dev < 31) attr_dev_mask |= 1 << dev;
  }
  int grid = device_sm_count();
  if (grid > kMaxPersistentCtas) grid = kMaxPersistentCtas;
  const int kid = kGateUp ? DMOE_KERNEL_GATE_UP : DMOE_KERNEL_DOWN;
  prof_begin(kid, s);
  cudaError_t e = launch_ex(expert_gemm_kernel<kGateUp>, dim3(grid), dim3(kThreads), smem, s,
                            true, a0, a1, b, sa0, sa1, sb, gp);
  prof_end(kid, s);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_experts(const ExpertArgs& a, cudaStream_t s) {
  const int pairs = a.T * a.k;
  const bool has_shared = a.Is > 0;
  // 1. gather x in dispatch order
  {
    int grid = pairs < 1024 ? pairs : 1024;
    prof_begin(DMOE_KERNEL_GATHER, s);
    cudaError_t e = launch_ex(gather_kernel, dim3(grid), dim3(256), 0, s, true, a.x, a.rows,
                              a.xperm, pairs, a.k, a.d);
    prof_end(DMOE_KERNEL_GATHER, s);
    if (e != cudaSuccess) return e;
  }
  GemmParams gp{};
  gp.n_unique = a.n_unique;
  gp.unique_ids = a.unique_ids;
  gp.offsets = a.offsets;
  gp.h = a.h;
  gp.hs = a.hs;
  gp.yslot = a.yslot;
  gp.yshared = a.yshared;
  gp.err = a.err;
  gp.T = a.T; gp.d = a.d; gp.E = a.E; gp.k = a.k; gp.I = a.I; gp.Is = a.Is;
  gp.n_max = a.n_max;
  gp.has_shared = has_shared ? 1 : 0;

  // 2. gate/up + SwiGLU: 64-row boxes of W_gate and W_up stacked in one A tile
  CUtensorMap m_wg, m_wu, m_xp, m_sg, m_su, m_x;
  bool ok = make_map(&m_wg, a.w_gate, (uint64_t)a.E * a.I, a.d, 64) &&
            make_map(&m_wu, a.w_up, (uint64_t)a.E * a.I, a.d, 64) &&
            make_map(&m_xp, a.xperm, (uint64_t)pairs, a.d, (uint32_t)a.n_max) &&
            make_map(&m_x, a.x, (uint64_t)a.T, a.d, (uint32_t)a.n_max);
  if (ok && has_shared)
    ok = make_map(&m_sg, a.ws_gate, (uint64_t)a.Is, a.d, 64) &&
         make_map(&m_su, a.ws_up, (uint64_t)a.Is, a.d, 64);
  if (!has_shared) { m_sg = m_wg; m_su = m_wu; }
  if (!ok) return cudaErrorInvalidValue;
  cudaError_t e = launch_gemm<true>(m_wg, m_wu, m_xp, m_sg, m_su, m_x, gp, s);
  if (e != cudaSuccess) return e;

  // 3. down projection
  CUtensorMap m_wd, m_h, m_sd, m_hs;
  ok = make_map(&m_wd, a.w_down, (uint64_t)a.E * a.d, a.I, kTileM) &&
       make_map(&m_h, a.h, (uint64_t)pairs, a.I, (uint32_t)a.n_max);
  if (ok && has_shared)
    ok = make_map(&m_sd, a.ws_down, (uint64_t)a.d, a.Is, kTileM) &&
         make_map(&m_hs, a.hs, (uint64_t)a.T, a.Is, (uint32_t)a.n_max);
  if (!has_shared) { m_sd = m_wd; m_hs = m_h; }
  if (!ok) return cudaErrorInvalidValue;
  e = launch_gemm<false>(m_wd, m_wd, m_h, m_sd, m_sd, m_hs, gp, s);
  if (e != cudaSuccess) return e;

  // 4. gate-weighted combine
  dim3 grid((a.d / 4 + 255) / 256, a.T);
  prof_begin(DMOE_KERNEL_COMBINE, s);
  e = launch_ex(combine_kernel, grid, dim3(256), 0, s, true, a.yslot, a.yshared, a.pos,
                a.topk_gate, a.y, a.k, a.d, has_shared ? 1 : 0);
  prof_end(DMOE_KERNEL_COMBINE, s);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dmoe
