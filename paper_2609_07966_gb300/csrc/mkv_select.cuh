// Block-level exact top-k by unique 64-bit keys (radix select, 8 bits per
// pass) and block-wide helpers shared by the H2O, SnapKV and RocketKV
// selection kernels.  Every ranking decision of the three methods is a top-k
// under (score desc, index asc); it is made exact by the key
//   key = (order-preserving bits of the fp32 score) << 32 | (0xffffffff - index)
// which is unique per index, so "the k largest keys" is one well-defined set.
#pragma once

#include "mkv_common.cuh"

namespace mkv {

__device__ __forceinline__ uint64_t rank_key(float score, uint32_t index) {
  return ((uint64_t)f32_key(score) << 32) | (uint64_t)(0xffffffffu - index);
}

// Returns (to every thread) the k-th largest of the n keys produced by
// key_of(i), i in [0, n); all keys must be distinct and 1 <= k <= n.
// `hist` is 256 ints of shared memory.  Uses every thread of the block.
template <typename KeyOf>
__device__ uint64_t block_kth_largest(int n, int k, KeyOf key_of, int* hist) {
  __shared__ uint64_t s_prefix;
  __shared__ int s_k;
  if (threadIdx.x == 0) {
    s_prefix = 0;
    s_k = k;
  }
  uint64_t mask = 0;
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    const uint64_t prefix = s_prefix;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      const uint64_t key = key_of(i);
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255], 1);
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      // lane l owns bins 255-8l .. 248-8l (descending); find the bin holding the kr-th key
      const int lane = threadIdx.x, kr = s_k;
      int cnt = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) cnt += hist[255 - 8 * lane - j];
      int incl = cnt;
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const int excl = incl - cnt;
      if (excl < kr && incl >= kr) {       // exactly one lane
        int rem = kr - excl, bin = 255 - 8 * lane;
        for (int j = 0; j < 8; ++j, --bin) {
          if (hist[bin] >= rem) break;
          rem -= hist[bin];
        }
        s_k = rem;
        s_prefix = prefix | ((uint64_t)bin << shift);
      }
    }
    mask |= (uint64_t)255 << shift;
    __syncthreads();
  }
  return s_prefix;
}

// Exclusive block scan of one int per thread over blockDim.x threads
// (blockDim.x a multiple of 32, <= 1024).  Returns the exclusive prefix and
// writes the block total to *total.
__device__ __forceinline__ int block_exclusive_scan(int v, int* warp_sums, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int x = v;
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int s = lane < nw ? warp_sums[lane] : 0;
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    if (lane < nw) warp_sums[lane] = s;
  }
  __syncthreads();
  const int before = (warp > 0 ? warp_sums[warp - 1] : 0) + x - v;
  *total = warp_sums[nw - 1];
  __syncthreads();
  return before;
}

}  // namespace mkv
