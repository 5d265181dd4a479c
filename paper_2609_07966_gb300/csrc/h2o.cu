// H2O heavy-hitter eviction (Section 2.1, H2O paragraph): initial keep after
// the prompt's accumulated scores, and the per-step score update + eviction.
//
// Keep: the `recent` newest positions, plus the `heavy` best of the rest under
// (score desc, position asc) -- an exact radix top-k on unique 64-bit keys --
// gathered in ascending position into slots 0.. of the cache.
// Step: acc[slot] += sum_h 2^(x_h(slot) - m_h) / l_h for every held slot (the
// softmax probability from the decode call), then, if more than heavy+recent
// tokens are held, evict among all but the `recent` newest positions the one
// that ranks last under (acc desc, position asc): lowest acc, on a tie the
// higher position.  Its slot becomes the next append slot.
#include <math.h>

#include "mkv_common.cuh"
#include "mkv_internal.h"
#include "mkv_h2o.cuh"
#include "mkv_select.cuh"

namespace mkv {

namespace {

constexpr int kSelThreads = 1024;

// One CTA per (batch, kv-head): flags of kept positions -> ascending keep list.
__global__ void __launch_bounds__(kSelThreads) h2o_keep_kernel(const float* __restrict__ score, int64_t T, int H,
                                                               int R, int32_t* __restrict__ keep_out,
                                                               int32_t* __restrict__ n_keep_out) {
  __shared__ int hist[256];
  __shared__ int warp_sums[32];
  const int64_t bh = blockIdx.x;
  const float* s = score + bh * T;
  int32_t* keep = keep_out + bh * T;
  const int64_t n_cand = T > R ? T - R : 0;           // positions 0 .. T-R-1 compete
  const int heavy = (int)(n_cand < (int64_t)H ? n_cand : (int64_t)H);
  uint64_t thr = ~0ull;
  if (heavy > 0) {
    thr = block_kth_largest_score((int)n_cand, heavy, [&](int i) { return s[i]; }, hist);
  }
  // stream compaction in ascending position
  int64_t base = 0;
  for (int64_t i0 = 0; i0 < T; i0 += blockDim.x) {
    const int64_t i = i0 + threadIdx.x;
    int flag = 0;
    if (i < T) flag = (i >= n_cand) || (heavy > 0 && rank_key(s[i], (uint32_t)i) >= thr);
    int total;
    const int before = block_exclusive_scan(flag, warp_sums, &total);
    if (flag) keep[base + before] = (int32_t)i;
    base += total;
  }
  if (threadIdx.x == 0) n_keep_out[bh] = (int32_t)base;
}

// Copy the kept rows into the cache and set pos/acc/slot, T_len.
__global__ void h2o_gather_kernel(const __half* __restrict__ full_k, const __half* __restrict__ full_v,
                                  const float* __restrict__ score, const int32_t* __restrict__ keep,
                                  const int32_t* __restrict__ n_keep, int64_t T, int Hkv, int D, int64_t T_cap,
                                  __half* k, __half* v, int32_t* pos, float* acc, int32_t* slot, int32_t* T_len) {
  const int64_t bh = blockIdx.y;
  const int n = n_keep[bh];
  const int nc = D / 8;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < T_cap * nc; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t sl = e / nc;
    const int col = (int)(e % nc);
    if (sl < n) {
      const int64_t p = keep[bh * T + sl];
      reinterpret_cast<uint4*>(k + (bh * T_cap + sl) * D)[col] = reinterpret_cast<const uint4*>(full_k + (bh * T + p) * D)[col];
      reinterpret_cast<uint4*>(v + (bh * T_cap + sl) * D)[col] = reinterpret_cast<const uint4*>(full_v + (bh * T + p) * D)[col];
      if (col == 0) {
        pos[bh * T_cap + sl] = (int32_t)p;
        acc[bh * T_cap + sl] = score[bh * T + p];
      }
    } else if (col == 0) {
      pos[bh * T_cap + sl] = -1;
      acc[bh * T_cap + sl] = 0.f;
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    slot[bh] = n;            // first free slot
    if (bh % Hkv == 0) T_len[bh / Hkv] = (int32_t)T;
  }
}

// One CTA per (batch, kv-head): score update and eviction (1024 threads: a unit's slots in one round
// of loads).
constexpr int kUpdThreads = 1024;
__global__ void __launch_bounds__(kUpdThreads) h2o_update_kernel(const float* __restrict__ logits, const float* __restrict__ m_tot,
                                                         const float* __restrict__ l_tot, int Hkv, int G, int64_t T_cap,
                                                         int H, int R, const int32_t* __restrict__ T_len,
                                                         int32_t* __restrict__ pos, float* __restrict__ acc,
                                                         int32_t* __restrict__ slot_out) {
  pdl_wait_and_trigger();
  h2o_update_unit(logits, m_tot, l_tot, Hkv, G, T_cap, H, R, T_len, pos, acc, slot_out, blockIdx.x);
}

}  // namespace

cudaError_t launch_h2o_keep(const mkv_config& c, const void* full_k, const void* full_v, int64_t T,
                            const mkv_cache& cache, const PrefillWs& ws, cudaStream_t st) {
  const int units = c.B * c.Hkv;
  int32_t* n_keep = reinterpret_cast<int32_t*>(ws.row_st);   // row stats are dead after scoring
  h2o_keep_kernel<<<units, kSelThreads, 0, st>>>(ws.score, T, c.h2o_heavy, c.h2o_recent, ws.keep, n_keep);
  cudaError_t e = cudaPeekAtLastError();
  if (e != cudaSuccess) return e;
  const int64_t work = cache.T_cap * (c.D / 8);
  const int bx = (int)std::min<int64_t>(ceil_div(work, 256), 64);
  h2o_gather_kernel<<<dim3(bx, units), 256, 0, st>>>(
      static_cast<const __half*>(full_k), static_cast<const __half*>(full_v), ws.score, ws.keep, n_keep, T, c.Hkv,
      c.D, cache.T_cap, static_cast<__half*>(cache.k), static_cast<__half*>(cache.v), cache.pos, cache.acc,
      cache.slot, cache.T_len);
  return cudaPeekAtLastError();
}

cudaError_t launch_h2o_update(const mkv_config& c, const mkv_cache& cache, const DecodeWs& ws, cudaStream_t st) {
  return launch_pdl(h2o_update_kernel, dim3(c.B * c.Hkv), dim3(kUpdThreads), 0, st, (const float*)ws.logits,
                    (const float*)ws.m_tot, (const float*)ws.l_tot, c.Hkv, c.Hq / c.Hkv, cache.T_cap, c.h2o_heavy,
                    c.h2o_recent, (const int32_t*)cache.T_len, cache.pos, cache.acc, cache.slot);
}

}  // namespace mkv
