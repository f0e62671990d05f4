// Deterministic CTA-wide reductions and scans (fixed combination order, identical result in
// every thread). Used by the routing and dispatch kernels; blockDim.x must be a multiple of
// 32 and at most 1024.
#pragma once

#include <cuda_runtime.h>

namespace dmoe {

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ int warp_min_i(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// `scratch` holds at least 32 entries; the call synchronises the CTA twice.
__device__ __forceinline__ float block_max(float v, float* scratch) {
  const int nw = blockDim.x >> 5, w = threadIdx.x >> 5;
  v = warp_max(v);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) scratch[w] = v;
  __syncthreads();
  float r = scratch[0];
  for (int i = 1; i < nw; ++i) r = fmaxf(r, scratch[i]);
  return r;
}
__device__ __forceinline__ float block_sum(float v, float* scratch) {
  const int nw = blockDim.x >> 5, w = threadIdx.x >> 5;
  v = warp_sum(v);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) scratch[w] = v;
  __syncthreads();
  float r = scratch[0];
  for (int i = 1; i < nw; ++i) r += scratch[i];
  return r;
}
__device__ __forceinline__ int block_sum_i(int v, int* scratch) {
  const int nw = blockDim.x >> 5, w = threadIdx.x >> 5;
  v = warp_sum_i(v);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) scratch[w] = v;
  __syncthreads();
  int r = 0;
  for (int i = 0; i < nw; ++i) r += scratch[i];
  return r;
}
__device__ __forceinline__ int block_min_i(int v, int* scratch) {
  const int nw = blockDim.x >> 5, w = threadIdx.x >> 5;
  v = warp_min_i(v);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) scratch[w] = v;
  __syncthreads();
  int r = scratch[0];
  for (int i = 1; i < nw; ++i) r = min(r, scratch[i]);
  return r;
}

// Inclusive prefix sum over threads in thread order (fp32: a warp-level Hillis-Steele scan,
// then the warp totals added in warp order).
__device__ __forceinline__ float block_inclusive_scan(float v, float* scratch) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    float u = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += u;
  }
  __syncthreads();
  if (lane == 31) scratch[w] = v;
  __syncthreads();
  float base = 0.f;
  for (int i = 0; i < w; ++i) base += scratch[i];
  return base + v;
}
// Exclusive prefix sum of ints in thread order; *total receives the CTA total.
__device__ __forceinline__ int block_exclusive_scan_i(int v, int* scratch, int* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int u = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += u;
  }
  __syncthreads();
  if (lane == 31) scratch[w] = x;
  __syncthreads();
  int base = 0, all = 0;
  for (int i = 0; i < nw; ++i) {
    if (i < w) base += scratch[i];
    all += scratch[i];
  }
  *total = all;
  return base + x - v;
}

}  // namespace dmoe
