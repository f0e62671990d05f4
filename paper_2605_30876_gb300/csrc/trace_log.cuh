// Debug builds (-DDMOE_TRACE) only: a log of kernel entries and exits (one record per CTA,
// %globaltimer in ns) for timelines across back-to-back launches. Each translation unit has
// its own log and exports its own reader, named by DMOE_KLOG_EXPORT. Release builds compile
// every KLOG to nothing.
#pragma once

#ifdef DMOE_TRACE
#include <cuda_runtime.h>
#include <stdint.h>

namespace dmoe {
namespace {
struct KLogRec {
  uint32_t tag;  // kernel id * 2 + (1 at exit)
  uint32_t cta;
  uint64_t t;
};
constexpr uint32_t kKLogCap = 32768;
__device__ KLogRec g_klog[kKLogCap];
__device__ uint32_t g_klog_n;
__device__ __forceinline__ void klog(uint32_t tag) {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  const uint32_t i = atomicAdd(&g_klog_n, 1u);
  if (i < kKLogCap) g_klog[i] = KLogRec{tag, blockIdx.x + blockIdx.y * gridDim.x, t};
}
}  // namespace
}  // namespace dmoe
#define KLOG(kid, exit_) \
  do {                   \
    if (threadIdx.x == 0) dmoe::klog((uint32_t)(kid) * 2u + (exit_)); \
  } while (0)
// host reader: copies up to `cap` records, returns the count, then clears the log
#define DMOE_KLOG_EXPORT(name)                                                          \
  extern "C" int name(void* host, unsigned cap) {                                       \
    uint32_t n = 0;                                                                     \
    cudaMemcpyFromSymbol(&n, dmoe::g_klog_n, sizeof(n));                                \
    if (n > dmoe::kKLogCap) n = dmoe::kKLogCap;                                         \
    if (n > cap) n = cap;                                                               \
    if (host != nullptr && n > 0)                                                       \
      cudaMemcpyFromSymbol(host, dmoe::g_klog, n * sizeof(dmoe::KLogRec));              \
    const uint32_t z = 0;                                                               \
    cudaMemcpyToSymbol(dmoe::g_klog_n, &z, sizeof(z));                                  \
    return (int)n;                                                                      \
  }
#else
#define KLOG(kid, exit_) ((void)0)
#endif
