// Dispatch kernel: one CTA computes the unique experts of the forward and the
// expert -> (token, slot) lists (see dispatch_impl.cuh for the method).
#include "dispatch_impl.cuh"
#include "dmoe_internal.cuh"
#include "trace_log.cuh"

namespace dmoe {
namespace {

constexpr int kDispatchThreads = 1024;

__global__ void __launch_bounds__(kDispatchThreads)
dispatch_kernel(const int32_t* __restrict__ topk_idx, int T, int E, int k,
                int32_t* __restrict__ n_unique, int32_t* __restrict__ unique_ids,
                int32_t* __restrict__ offsets, int32_t* __restrict__ rows,
                int32_t* __restrict__ pos, DevErrRecord* err) {
  extern __shared__ __align__(16) uint8_t dsm[];
  const int nchunks = (T + 31) / 32;
  uint32_t* bits = reinterpret_cast<uint32_t*>(dsm);                        // [nchunks][E]
  uint16_t* base = reinterpret_cast<uint16_t*>(bits + (size_t)nchunks * E);  // [nchunks][E]
  pdl_launch_dependents();
  pdl_wait();
  KLOG(DMOE_KERNEL_DISPATCH, 0);
  dispatch_cta(topk_idx, T, E, k, n_unique, unique_ids, offsets, rows, pos, err, bits, base);
  KLOG(DMOE_KERNEL_DISPATCH, 1);
}

}  // namespace

size_t dispatch_smem_bytes(int T, int E) {
  const size_t nchunks = (size_t)(T + 31) / 32;
  return nchunks * E * (sizeof(uint32_t) + sizeof(uint16_t));
}

cudaError_t launch_dispatch(const DispatchArgs& a, cudaStream_t s) {
  const size_t smem = dispatch_smem_bytes(a.T, a.E);
  static int attr_dev_mask = 0;  // the dynamic smem limit is a per-device function attribute
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 31 || !(attr_dev_mask & (1 << dev))) {
    cudaError_t e = cudaFuncSetAttribute(dispatch_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         200 * 1024);
    if (e != cudaSuccess) return e;
    if (dev < 31) attr_dev_mask |= 1 << dev;
  }
  prof_begin(DMOE_KERNEL_DISPATCH, s);
  cudaError_t e = launch_ex(dispatch_kernel, dim3(1), dim3(kDispatchThreads), smem, s, true,
                            a.topk_idx, a.T, a.E, a.k, a.n_unique, a.unique_ids, a.offsets,
                            a.rows, a.pos, a.err);
  prof_end(DMOE_KERNEL_DISPATCH, s);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dmoe

#ifdef DMOE_TRACE
DMOE_KLOG_EXPORT(dmoe_debug_klog_dispatch)
#endif
