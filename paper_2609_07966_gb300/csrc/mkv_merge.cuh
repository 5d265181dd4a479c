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

// `scratch`: shared memory the caller no longer needs, `cap` floats of it.  `n_parts`: the
// partials of this group (slots 0 .. n_parts-1 of a.n_split; default all).
template <int D, int NT>
__device__ __forceinline__ void merge_if_last(const MergeArgs& a, int64_t bh, int b, int kvh, float* scratch,
                                              int cap, int n_parts = -1) {
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int t = atomicAdd(&a.counters[bh], 1);
    s_last = (t == (n_parts > 0 ? n_parts : a.n_split) - 1);
    if (s_last) a.counters[bh] = 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const int ns = n_parts > 0 ? n_parts : a.n_split, stride = a.n_split, G = a.G;
  const int64_t hq0 = (int64_t)b * a.Hq + (int64_t)kvh * G;
  if (2 * G * ns + 2 * G <= cap) {
    // weights f[row][s] = 2^(m_s - M) and totals, then independent loads of the o partials
    float* f = scratch;                 // [G][ns]
    float* tot = scratch + G * ns;      // [G] M, [G] L
    for (int e = threadIdx.x; e < G * ns; e += NT) f[e] = __ldcg(a.part_m + (hq0 + e / ns) * stride + e % ns);
    __syncthreads();
    if (threadIdx.x < G) {
      const int row = threadIdx.x;
      float M = -INFINITY;
      for (int s = 0; s < ns; ++s) M = fmaxf(M, f[row * ns + s]);
      float L = 0.f;
      for (int s = 0; s < ns; ++s) {
        const float ms = f[row * ns + s];
        const float w = (M == -INFINITY || ms == -INFINITY) ? 0.f : exp2f(ms - M);
        f[row * ns + s] = w;
        L += __ldcg(a.part_l + (hq0 + row) * stride + s) * w;
      }
      tot[row] = M;
      tot[G + row] = L;
    }
    __syncthreads();
    for (int e = threadIdx.x; e < G * D; e += NT) {
      const int row = e / D, d = e % D;
      const float* po = a.part_o + ((hq0 + row) * stride) * D + d;
      const float* fw = f + row * ns;
      float O0 = 0.f, O1 = 0.f, O2 = 0.f, O3 = 0.f;
      int s = 0;
      for (; s + 4 <= ns; s += 4) {
        O0 += __ldcg(po + (int64_t)(s + 0) * D) * fw[s + 0];
        O1 += __ldcg(po + (int64_t)(s + 1) * D) * fw[s + 1];
        O2 += __ldcg(po + (int64_t)(s + 2) * D) * fw[s + 2];
        O3 += __ldcg(po + (int64_t)(s + 3) * D) * fw[s + 3];
      }
      for (; s < ns; ++s) O0 += __ldcg(po + (int64_t)s * D) * fw[s];
      const float O = (O0 + O1) + (O2 + O3);
      const float L = tot[G + row];
      a.out[(hq0 + row) * D + d] = __float2half_rn(L > 0.f ? O / L : 0.f);
      if (a.m_tot != nullptr && d == 0) {
        a.m_tot[hq0 + row] = tot[row];
        a.l_tot[hq0 + row] = L;
      }
    }
    return;
  }
  for (int e = threadIdx.x; e < G * D; e += NT) {      // many splits: direct loop
    const int row = e / D, d = e % D;
    const int64_t hq = hq0 + row;
    const float* pm = a.part_m + hq * stride;
    const float* pl = a.part_l + hq * stride;
    float M = -INFINITY;
    for (int s = 0; s < ns; ++s) M = fmaxf(M, __ldcg(pm + s));
    float L = 0.f, O = 0.f;
    if (M != -INFINITY) {
      for (int s = 0; s < ns; ++s) {
        const float ms = __ldcg(pm + s);
        if (ms == -INFINITY) continue;
        const float w = exp2f(ms - M);
        L += __ldcg(pl + s) * w;
        O += __ldcg(a.part_o + (hq * stride + s) * D + d) * w;
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
