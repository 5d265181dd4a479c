// Split-KV merge done by the last CTA of each (batch, kv-head) inside the decode
// kernels: every CTA writes its partial (m, l, o) and takes a ticket; the CTA
// that takes the last ticket merges all splits of the group's query heads,
//   out_h = sum_s 2^(m_s - M) o_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s,
// writes the output, and resets the ticket counter to zero for the next call.
#pragma once

#include "mkv_common.cuh"

namespace mkv {

struct MergeArgs {
  const float* part_m;   // [B][Hq][n_split]
  const float* part_l;
  const float* part_o;   // [B][Hq][n_split][D]
  int* counters;         // [B][Hkv], zero between calls
  __half* out;           // [B][Hq][D]
  float* m_tot;          // H2O: [B][Hq] (or null)
  float* l_tot;
  int Hq, G, n_split;
};

template <int D, int NT>
__device__ __forceinline__ void merge_if_last(const MergeArgs& a, int64_t bh, int b, int kvh) {
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int t = atomicAdd(&a.counters[bh], 1);
    s_last = (t == a.n_split - 1);
    if (s_last) a.counters[bh] = 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int e = threadIdx.x; e < a.G * D; e += NT) {
    const int row = e / D, d = e % D;
    const int64_t hq = (int64_t)b * a.Hq + (int64_t)kvh * a.G + row;
    const float* pm = a.part_m + hq * a.n_split;
    const float* pl = a.part_l + hq * a.n_split;
    float M = -INFINITY;
    for (int s = 0; s < a.n_split; ++s) M = fmaxf(M, __ldcg(pm + s));
    float L = 0.f, O = 0.f;
    if (M != -INFINITY) {
      for (int s = 0; s < a.n_split; ++s) {
        const float ms = __ldcg(pm + s);
        if (ms == -INFINITY) continue;
        const float f = exp2f(ms - M);
        L += __ldcg(pl + s) * f;
        O += __ldcg(a.part_o + (hq * a.n_split + s) * D + d) * f;
      }
    }
    a.out[hq * D + d] = __float2half_rn(L > 0.f ? O / L : 0.f);
    if (a.m_tot != nullptr && d == 0) {
      a.m_tot[hq] = M;
      a.l_tot[hq] = L;
    }
  }
}

}  // namespace mkv
