// Router logits of a large forward on tcgen05 tensor cores (§4.2 of arXiv 2605.30876: the
// router scores every expert from the token's hidden state, s = softmax(x W_r + b); here
// the fp32 products x W_r as partial sums over S slices of d, which router_softmax_kernel
// adds in slice order, with b, before the softmax and top-k).
//
// fp32 products on bf16 tensor cores: W_r is split into three bf16 parts, hi + mid + lo = w
// to 2^-27 (hi = bf16(w), mid = bf16(w - hi), lo = bf16(w - hi - mid)); x is bf16, so every
// product x * part is exact in fp32. The MMAs accumulate in fp32 with a rounding error of
// up to about one unit in the last place of the accumulator per MMA (measured: with one
// accumulator over all of d = 2048, 384 MMAs, the scores came out up to 2.4e-5 relative
// off); so a CTA takes at most 256 of d (16 MMAs into its hi accumulator), the mid and lo
// products (2^-8 and 2^-16 of the total) go to a second accumulator, and the slices are
// added on the CUDA cores.
//
//   router_wsplit_kernel      the three parts of W_r, each stored K-major ([E, d] bf16: row
//                             e holds expert e's weights over d), the MMA's B operand
//   router_logits_tc_kernel   one CTA per (128 tokens, slice of d, group of N experts; N =
//                             E / nsplit, a multiple of 32, at most 256), no cross-CTA step:
//     warp 0     TMA, two stages: x chunk (128 tokens x 64 of d, 128-B swizzle, rows past
//                T read as zero) and the three parts' chunks (N rows x 64)
//     warp 1     TMEM allocation; lane 0 issues D[128 x N] += x * part^T, 4 K-steps of 16
//                per chunk and part (hi into one accumulator, mid and lo into the other)
//     warps 0-3  (after the MMAs; one TMEM lane quadrant each) put hi + (mid + lo) into
//                shared memory (the stages are free by then) as E / 32 boxes of 32
//                experts x 128 tokens with the 128-B swizzle, which thread 0 then stores by
//                TMA (rows past T are not written)
// Every mbarrier wait is bounded (1 s): a timeout is recorded and the CTA unwinds.
#include "dmoe_internal.cuh"
#include "sm100_ptx.cuh"
#include "trace_log.cuh"

// Debug builds (-DDMOE_TRACE): per-CTA phase times of router_logits_tc_kernel (%globaltimer,
// ns), g_rtc[cta * 16 + slot]: 0 entry, 1 set-up done, 2 last TMA issued, 3 first stage
// landed, 4 last MMA issued, 5 accumulator ready, 7 rows staged in shared memory, 6 rows
// stored.
#ifdef DMOE_TRACE
__device__ uint64_t g_rtc[1024 * 16];
#define RTC_AT(slot) \
  (g_rtc[((blockIdx.y * gridDim.x + blockIdx.x) % 1024) * 16 + (slot)] = ptx::globaltimer_ns())
#else
#define RTC_AT(slot) ((void)0)
#endif

namespace dmoe {
namespace {

constexpr int kLtM = 128;                     // tokens per tile (MMA M)
constexpr int kLtKC = 64;                     // d per chunk: one 128-B row of bf16
constexpr int kLtMaxDS = 256;                 // d per CTA at most (16 hi MMAs)
constexpr int kLtThreads = 128;
constexpr int kLtXBytes = kLtM * 128;         // 16 KB
constexpr uint64_t kLtTimeoutNs = 1000000000ull;

struct LtArgs {
  CUtensorMap xmap;   // x [T, d] bf16, box 64 columns x 128 rows, 128-B swizzle
  CUtensorMap pmap;   // parts [3E, d] bf16, box 64 columns x N rows, 128-B swizzle
  CUtensorMap omap;   // partials [S, T, E] fp32, box 32 x 128 x 1, 128-B swizzle
  DevErrRecord* err;
  L2Prefetch shared_pf;
  int T, d, E, ds;    // ds: d per slice (blockIdx.y)
  int N;              // experts per CTA (blockIdx.z: experts N z .. N z + N - 1)
};

// parts[p][e][i] for the tile of 32 experts x 64 of d: thread (e, 8-wide run of d) reads
// its eight weights (a warp reads eight 128-B rows) and writes 16 bytes to each part.
__global__ void __launch_bounds__(256)
router_wsplit_kernel(const float* __restrict__ w_r, __nv_bfloat16* __restrict__ parts, int d,
                     int E) {
  const int e = blockIdx.x * 32 + (threadIdx.x & 31);
  const int k0 = blockIdx.y * 64 + (threadIdx.x >> 5) * 8;
  // The split needs no dependency wait: this launch reads only W_r (an input) and writes
  // only the parts, which only the logits launch of an earlier call reads. That launch is
  // always followed by router_softmax_kernel, which releases its dependents only after its
  // own dependency wait (the logits launch has ended by then); so by the time any later
  // launch, this one included, can start, the earlier logits launch has ended. The wait at
  // the end makes this launch end only after the launch before it, so that the logits
  // launch after this one, which waits for this one, also reads x only after the launch
  // that may have written it.
  pdl_launch_dependents();
  KLOG(8, 0);
  if (e >= E) {
    pdl_wait();
    return;
  }
  float w[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) w[j] = w_r[(size_t)(k0 + j) * E + e];
  uint32_t hp[4], mp[4], lp[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const __nv_bfloat162 hi = __floats2bfloat162_rn(w[2 * j], w[2 * j + 1]);
    const float2 hf = __bfloat1622float2(hi);
    const float q0 = w[2 * j] - hf.x, q1 = w[2 * j + 1] - hf.y;
    const __nv_bfloat162 mid = __floats2bfloat162_rn(q0, q1);
    const float2 mf = __bfloat1622float2(mid);
    const __nv_bfloat162 lo = __floats2bfloat162_rn(q0 - mf.x, q1 - mf.y);
    hp[j] = *reinterpret_cast<const uint32_t*>(&hi);
    mp[j] = *reinterpret_cast<const uint32_t*>(&mid);
    lp[j] = *reinterpret_cast<const uint32_t*>(&lo);
  }
  const size_t pe = (size_t)E * d;
  const size_t o = (size_t)e * d + k0;
  *reinterpret_cast<uint4*>(parts + o) = make_uint4(hp[0], hp[1], hp[2], hp[3]);
  *reinterpret_cast<uint4*>(parts + pe + o) = make_uint4(mp[0], mp[1], mp[2], mp[3]);
  *reinterpret_cast<uint4*>(parts + 2 * pe + o) = make_uint4(lp[0], lp[1], lp[2], lp[3]);
  KLOG(8, 1);
  pdl_wait();
}

__global__ void __launch_bounds__(kLtThreads, 1)
router_logits_tc_kernel(const __grid_constant__ LtArgs f) {
  extern __shared__ uint8_t lt_raw[];
  uint8_t* smem = lt_raw + ((1024u - (ptx::smem_addr(lt_raw) & 1023u)) & 1023u);
  __shared__ __align__(8) uint64_t full[2], empty[2], acc_full;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) RTC_AT(0);
  const int E = f.E, N = f.N;
  const int e_base = blockIdx.z * N;
  const int m0 = blockIdx.x * kLtM;
  const int k_base = blockIdx.y * f.ds;
  const int nch = f.ds / kLtKC;
  const int pbytes = N * 128;                 // one part's chunk
  const int slot = kLtXBytes + 3 * pbytes;
  // TMEM: the hi accumulator in columns 0 .. N-1, the mid/lo one from column t_ml
  uint32_t t_ml = 32;
  while (t_ml < (uint32_t)N) t_ml <<= 1;
  const uint32_t t_cols = 2 * t_ml;
  auto x_buf = [&](int s) { return smem + s * slot; };
  auto p_buf = [&](int s, int part) { return smem + s * slot + kLtXBytes + part * pbytes; };

  if (tid == 0) {
    ptx::prefetch_tensormap(&f.xmap);
    ptx::prefetch_tensormap(&f.pmap);
    for (int s = 0; s < 2; ++s) {
      ptx::mbar_init(&full[s], 1);
      ptx::mbar_init(&empty[s], 1);
    }
    ptx::mbar_init(&acc_full, 1);
    ptx::fence_mbarrier_init();
    s_abort = 0;
    // the shared expert's weights are pulled into L2 for the expert launch
    issue_shared_prefetch(f.shared_pf,
                          (int)((blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x),
                          (int)(gridDim.x * gridDim.y * gridDim.z));
  }
  if (warp == 1) {
    ptx::tmem_alloc(&s_tmem, t_cols);
    ptx::tmem_relinquish();
  }
  pdl_wait();   // the parts of this call are written
  pdl_launch_dependents();
  KLOG(DMOE_KERNEL_ROUTER, 0);
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem = s_tmem;
  if (tid == 0) RTC_AT(1);

  auto wait = [&](uint64_t* bar, uint32_t parity, int where) -> bool {
    if (*(volatile int*)&s_abort) return false;
    if (ptx::mbar_wait(bar, parity, kLtTimeoutNs)) return true;
    record_error(f.err, kErrTimeout, kAtRouter, where);
    *(volatile int*)&s_abort = 1;
    return false;
  };

  if (warp == 0) {
    if (lane == 0) {
      // ================= TMA producer
      const uint64_t pol = ptx::policy_evict_last();   // x and the parts are re-read by tiles
      for (int c = 0; c < nch; ++c) {
        const int s = c & 1;
        const uint32_t ph = (uint32_t)((c >> 1) & 1);
        if (c >= 2 && !wait(&empty[s], ph ^ 1u, 100 + c)) break;
        ptx::mbar_arrive_expect_tx(&full[s], (uint32_t)slot);
        const int k0 = k_base + c * kLtKC;
        ptx::tma_load_2d(x_buf(s), &f.xmap, &full[s], k0, m0, pol);
#pragma unroll
        for (int part = 0; part < 3; ++part)
          ptx::tma_load_2d(p_buf(s, part), &f.pmap, &full[s], k0, part * E + e_base, pol);
      }
      RTC_AT(2);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ================= MMA issuer
      const uint32_t idesc = ptx::idesc_bf16(kLtM, (uint32_t)N);
      for (int c = 0; c < nch; ++c) {
        const int s = c & 1;
        const uint32_t ph = (uint32_t)((c >> 1) & 1);
        if (!wait(&full[s], ph, 300 + c)) break;
        if (c == 0) RTC_AT(3);
        ptx::tc_fence_after();
        const uint32_t xa = ptx::smem_addr(x_buf(s));
#pragma unroll
        for (int ks = 0; ks < kLtKC / 16; ++ks) {
          const uint64_t ad = ptx::sdesc_k_sw128(xa + ks * 32);
          const uint32_t first = (c == 0 && ks == 0) ? 0u : 1u;
          ptx::mma_bf16(tmem, ad, ptx::sdesc_k_sw128(ptx::smem_addr(p_buf(s, 0)) + ks * 32),
                        idesc, first);
          ptx::mma_bf16(tmem + t_ml, ad,
                        ptx::sdesc_k_sw128(ptx::smem_addr(p_buf(s, 1)) + ks * 32), idesc, first);
          ptx::mma_bf16(tmem + t_ml, ad,
                        ptx::sdesc_k_sw128(ptx::smem_addr(p_buf(s, 2)) + ks * 32), idesc, 1u);
        }
        ptx::mma_commit(&empty[s]);
      }
      ptx::mma_commit(&acc_full);   // also after a failed wait: the issued MMAs drain
      RTC_AT(4);
    }
  }
  __syncwarp();

  // epilogue: thread = token row (TMEM lane); the slice's partial row hi + (mid + lo)
  const bool have_acc = ptx::mbar_wait(&acc_full, 0, kLtTimeoutNs);
  if (!have_acc && lane == 0) record_error(f.err, kErrTimeout, kAtRouter, 700);
  ptx::tc_fence_after();
  if (tid == 0) RTC_AT(5);
  {
    // box b (experts 32b .. 32b + 31) at b * 16 KB: row r = token, 16-byte chunk j of the row
    // at j xor (r mod 8); the eight rows of a lane group hit eight different chunks
    uint8_t* boxes = smem;
    const int r = warp * 32 + lane;
    const uint32_t lanes = (uint32_t)(warp * 32) << 16;
    for (int c0 = 0; c0 < N; c0 += 32) {
      float h[32], ml[32];
      ptx::tmem_ld32(tmem + lanes + (uint32_t)c0, h);
      ptx::tmem_ld32(tmem + lanes + t_ml + (uint32_t)c0, ml);
      ptx::tmem_ld_wait();
      uint8_t* row = boxes + (c0 / 32) * (kLtM * 128) + r * 128;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        *reinterpret_cast<float4*>(row + ((j ^ (r & 7)) << 4)) =
            make_float4(h[4 * j] + ml[4 * j], h[4 * j + 1] + ml[4 * j + 1],
                        h[4 * j + 2] + ml[4 * j + 2], h[4 * j + 3] + ml[4 * j + 3]);
    }
    ptx::fence_proxy_async_smem();   // the boxes are read by the TMA store
    if (tid == 0) RTC_AT(7);
    __syncthreads();
    if (tid == 0) {
      if (have_acc)
        for (int b = 0; b < N / 32; ++b)
          ptx::tma_store_3d(&f.omap, boxes + b * (kLtM * 128), e_base + 32 * b, m0,
                            (int)blockIdx.y);
      ptx::bulk_commit_wait_read();   // the shared memory stays until the stores read it
    }
  }
  ptx::tc_fence_before();
  __syncthreads();
  if (tid == 0) RTC_AT(6);
  if (warp == 1) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem, t_cols);
  }
  KLOG(DMOE_KERNEL_ROUTER, 1);
}

typedef CUresult (*EncodeFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                             const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                             const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                             CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn_lt() {
  static EncodeFn fn = nullptr;
  if (fn == nullptr) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(ptr);
  }
  return fn;
}

bool encode_bf16_2d(EncodeFn enc, CUtensorMap* m, const void* base, uint64_t rows,
                    uint64_t cols, uint32_t box_rows) {
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  const cuuint32_t box[2] = {64u, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

size_t lt_smem_bytes(int E) { return 2 * ((size_t)kLtXBytes + 3 * (size_t)E * 128) + 1024; }

bool encode_part_3d(EncodeFn enc, CUtensorMap* m, float* base, int S, int T, int E) {
  const cuuint64_t dims[3] = {(cuuint64_t)E, (cuuint64_t)T, (cuuint64_t)S};
  const cuuint64_t strides[2] = {(cuuint64_t)E * 4, (cuuint64_t)T * E * 4};
  const cuuint32_t box[3] = {32u, (cuuint32_t)kLtM, 1u};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, base, dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

}  // namespace

bool router_tc_ok(int T, int d, int E) {
  return T >= kLtM && d % kLtKC == 0 && E % 32 == 0 && E <= kMaxExperts;
}

// Slices of d: each CTA takes at most 256 of d; of the splits that divide d into whole
// 64-wide chunks (at most 16, two rounds of the softmax warp's partial-row loads), the
// largest that still gives one wave of CTAs, else the smallest.
int router_tc_splits(int T, int d) {
  const int tiles = (T + kLtM - 1) / kLtM;
  const int nch = d / kLtKC;
  const int s_min = (d + kLtMaxDS - 1) / kLtMaxDS;
  // with the experts split over up to 8 CTAs as well, the fewest slices (the fewest partial
  // rows for the softmax to add) already give a wave of 128 CTAs
  if (nch % s_min == 0 && tiles * s_min * 8 >= 128) return s_min;
  int best = 0;
  for (int s = s_min; s <= nch && s <= 16; ++s)
    if (nch % s == 0 && (best == 0 || tiles * s <= 152)) best = s;
  if (best == 0)
    for (int s = s_min; s <= nch; ++s)
      if (nch % s == 0) {
        best = s;
        break;
      }
  return best;
}

// Groups of experts per (token tile, slice): with few token tiles the CTAs are split over
// the experts too (N = E / nsplit columns each, a multiple of 32), as far as one wave allows.
int router_tc_nsplit(int T, int E, int splits) {
  const int ctas = ((T + kLtM - 1) / kLtM) * splits;
  int best = 1;
  for (int n = 2; n <= 8; ++n)
    if ((E / 32) % n == 0 && ctas * n <= 152) best = n;
  return best;
}

size_t router_tc_parts_bytes(int d, int E) { return (size_t)3 * E * d * 2; }

cudaError_t launch_router_wsplit(const float* w_r, __nv_bfloat16* parts, int d, int E,
                                 cudaStream_t s) {
  return launch_ex(router_wsplit_kernel, dim3((E + 31) / 32, d / 64), dim3(256), 0, s, true, w_r,
                   parts, d, E);
}

cudaError_t launch_router_tc(const RouterArgs& a, int splits, cudaStream_t s) {
  if (!router_tc_ok(a.T, a.d, a.E) || a.w_parts == nullptr || a.tc_part == nullptr || splits < 1 ||
      (a.d / kLtKC) % splits != 0 || a.d / splits > kLtMaxDS)
    return cudaErrorInvalidValue;
  EncodeFn enc = encode_fn_lt();
  if (enc == nullptr) return cudaErrorInvalidValue;
  const int nsplit = router_tc_nsplit(a.T, a.E, splits);
  const int N = a.E / nsplit;
  LtArgs f{};
  if (!encode_bf16_2d(enc, &f.xmap, a.x, (uint64_t)a.T, (uint64_t)a.d, kLtM) ||
      !encode_bf16_2d(enc, &f.pmap, a.w_parts, 3 * (uint64_t)a.E, (uint64_t)a.d, (uint32_t)N) ||
      !encode_part_3d(enc, &f.omap, a.tc_part, splits, a.T, a.E))
    return cudaErrorInvalidValue;
  f.err = a.err;
  f.shared_pf = a.shared_pf;
  f.T = a.T;
  f.d = a.d;
  f.E = a.E;
  f.ds = a.d / splits;
  f.N = N;
  cudaError_t e = cudaSuccess;
  if (!a.parts_ready) {   // else dmoe_router_prepare wrote this W_r's parts already
    e = launch_router_wsplit(a.w_r, a.w_parts, a.d, a.E, s);
    if (e != cudaSuccess) return e;
  }
  static int mask = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 31 || !(mask & (1 << dev))) {
    e = cudaFuncSetAttribute(router_logits_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)lt_smem_bytes(kMaxExperts));
    if (e != cudaSuccess) return e;
    if (dev < 31) mask |= 1 << dev;
  }
  return launch_ex(router_logits_tc_kernel, dim3((a.T + kLtM - 1) / kLtM, splits, nsplit),
                   dim3(kLtThreads), lt_smem_bytes(N), s, true, f);
}

}  // namespace dmoe

#ifdef DMOE_TRACE
DMOE_KLOG_EXPORT(dmoe_debug_klog_routertc)
extern "C" int dmoe_debug_rtc(void* host) {
  return (int)cudaMemcpyFromSymbol(host, g_rtc, sizeof(g_rtc));
}
extern "C" int dmoe_debug_rtc_clear() {
  static uint64_t zeros[1024 * 16];
  return (int)cudaMemcpyToSymbol(g_rtc, zeros, sizeof(g_rtc));
}
#endif
