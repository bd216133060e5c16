// Block-wide reductions shared by the PACE kernels.
#pragma once

#include <cuda_runtime.h>

namespace pace {

// Sum of one double per thread with a fixed tree shape (THREADS a power of
// two equal to blockDim.x), so the result is the same on every run.  sh holds
// THREADS doubles.  Every thread of the block must call it.
template <int THREADS>
__device__ double block_sum_fixed(double v, double* sh) {
  sh[threadIdx.x] = v;
  __syncthreads();
  for (int o = THREADS / 2; o > 0; o >>= 1) {
    if (threadIdx.x < o) sh[threadIdx.x] = __dadd_rn(sh[threadIdx.x], sh[threadIdx.x + o]);
    __syncthreads();
  }
  const double r = sh[0];
  __syncthreads();
  return r;
}

// Exclusive scan of one value per thread (blockDim.x a multiple of 32, at most
// 1024); *total, if given, receives the block's sum.  Every thread must call it.
template <typename T>
__device__ T block_exclusive_scan(T v, T* total) {
  __shared__ T warp_sums[32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  T x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const T y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[wid] = x;
  __syncthreads();
  const int nw = blockDim.x >> 5;
  if (wid == 0) {
    T w = lane < nw ? warp_sums[lane] : T(0);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const T y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < nw) warp_sums[lane] = w;  // inclusive
  }
  __syncthreads();
  const T before = wid > 0 ? warp_sums[wid - 1] : T(0);
  if (total) *total = warp_sums[nw - 1];
  __syncthreads();
  return before + x - v;
}

}  // namespace pace
