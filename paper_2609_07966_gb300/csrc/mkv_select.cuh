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
// key_of(i), i in [0, n); 1 <= k <= n, and the k largest keys must be distinct (equal keys below
// them are allowed).
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

// One radix pass of block_kth_largest_score over 32-bit keys: among the elements with
// (key & mask) == s_pre (and, when `tied`, whose score key equals `score_pre`), the 8-bit digit at
// `shift` of the s_k-th largest is appended to s_pre; s_k and s_cnt become the rank left and the
// count in the chosen bin.  Every thread of the block takes part.
template <typename KeyOf>
__device__ __forceinline__ void radix_pass32(int n, KeyOf key_of, int shift, uint32_t mask, int* hist,
                                             uint32_t& s_pre, int& s_k, int& s_cnt) {
  for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
  __syncthreads();
  const uint32_t prefix = s_pre;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    uint32_t key;
    if (key_of(i, key) && (key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255], 1);
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
    if (excl < kr && incl >= kr) {         // exactly one lane
      int rem = kr - excl, bin = 255 - 8 * lane;
      for (int j = 0; j < 8; ++j, --bin) {
        if (hist[bin] >= rem) break;
        rem -= hist[bin];
      }
      s_k = rem;
      s_cnt = hist[bin];
      s_pre = prefix | ((uint32_t)bin << shift);
    }
  }
  __syncthreads();
}

// The same k-th largest key (score bits << 32 | (0xffffffff - index)) from the fp32 scores
// score_of(i), with fewer and cheaper passes: radix passes over the 32 score-key bits, ended as soon
// as the chosen bin holds a single element; when several elements share the whole score (exact
// ties, common after max-pooling), passes over the low index bits of the tied elements only (an
// index below n < 2^24 fixes the higher bits of 0xffffffff - i).  1 <= k <= n; `hist` is 256 ints
// of shared memory.
template <typename ScoreOf>
__device__ uint64_t block_kth_largest_score(int n, int k, ScoreOf score_of, int* hist) {
  __shared__ uint32_t s_pre, s_ipre, s_full;
  __shared__ int s_k, s_cnt, s_idx;
  if (threadIdx.x == 0) {
    s_pre = 0;
    s_k = k;
    s_cnt = n;
  }
  __syncthreads();
  uint32_t mask = 0;
  for (int shift = 24; shift >= 0; shift -= 8) {
    radix_pass32(n, [&](int i, uint32_t& key) { key = f32_key(score_of(i)); return true; }, shift, mask, hist,
                 s_pre, s_k, s_cnt);
    mask |= 255u << shift;
    if (s_cnt == 1) break;                 // one element has these score bits: it is the k-th
  }
  uint32_t pre = s_pre;
  uint32_t idx_key;                        // 0xffffffff - index of the k-th
  if (s_cnt == 1) {
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      const uint32_t key = f32_key(score_of(i));
      if ((key & mask) == pre) {
        s_idx = i;
        s_full = key;
      }
    }
    __syncthreads();
    idx_key = 0xffffffffu - (uint32_t)s_idx;
    pre = s_full;
  } else {
    // exact ties of the whole score: the s_k-th of them by index ascending = the s_k-th largest of
    // 0xffffffff - i over the tied elements; for i < n the bits above the top digit of n - 1 are ones
    int top = 0;
    while (top < 24 && ((n - 1) >> (top + 8)) != 0) top += 8;   // highest digit holding index bits
    uint32_t imask = (uint32_t)~((1ull << (top + 8)) - 1ull);
    if (threadIdx.x == 0) s_ipre = imask;
    __syncthreads();
    for (int shift = top; shift >= 0; shift -= 8) {
      radix_pass32(n, [&](int i, uint32_t& key) {
        key = 0xffffffffu - (uint32_t)i;
        return f32_key(score_of(i)) == pre;
      }, shift, imask, hist, s_ipre, s_k, s_cnt);
      imask |= 255u << shift;
    }
    idx_key = s_ipre;
  }
  __syncthreads();                         // every thread has read the shared words before reuse
  return ((uint64_t)pre << 32) | (uint64_t)idx_key;
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
