// H2O score update and eviction of one (batch, kv-head) unit (Section 2.1, H2O
// paragraph), run by every thread of one CTA of any size (a multiple of 32, at
// most 1024): acc[slot] += sum_h 2^(x_h(slot) - m_h) / l_h for every held slot,
// then, if more than heavy + recent tokens are held, the lowest-ranked token
// under (acc desc, position asc) among all but the `recent` newest positions is
// evicted and its slot becomes the next append slot; otherwise the first free
// slot is.  Logits are read with L2-coherent loads (the decode CTAs of the
// unit wrote them).  The group's (m, 1 / l) are read once per CTA; 2^x comes from the
// special-function unit's approximation (relative error about 2^-22).
#pragma once

#include "mkv_common.cuh"
#include "mkv_select.cuh"

namespace mkv {

__device__ __forceinline__ float h2o_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void h2o_update_unit(const float* __restrict__ logits, const float* __restrict__ m_tot,
                                                const float* __restrict__ l_tot, int Hkv, int G, int64_t T_cap,
                                                int H, int R, const int32_t* __restrict__ T_len,
                                                int32_t* __restrict__ pos, float* __restrict__ acc,
                                                int32_t* __restrict__ slot_out, int64_t bh) {
  const int b = (int)(bh / Hkv), kvh = (int)(bh % Hkv);
  const int64_t newest = (int64_t)T_len[b] - 1;
  __shared__ float s_m[8], s_il[8];
  if (threadIdx.x < G) {
    const int64_t hq = (int64_t)b * Hkv * G + (int64_t)kvh * G + threadIdx.x;
    s_m[threadIdx.x] = __ldcg(m_tot + hq);
    const float l = __ldcg(l_tot + hq);
    s_il[threadIdx.x] = l > 0.f ? 1.f / l : 0.f;
  }
  __syncthreads();
  float m[8], il[8];                  // G <= 8; unrolled so both stay in registers
#pragma unroll
  for (int h = 0; h < 8; ++h) {
    m[h] = h < G ? s_m[h] : 0.f;
    il[h] = h < G ? s_il[h] : 0.f;
  }
  int held = 0;
  uint64_t best = ~0ull;          // minimum key among candidates -> evicted
  int best_slot = -1, first_free = INT32_MAX;
  // kU slots per thread per pass, their loads issued together so their latencies overlap
  constexpr int kU = 4;
  const int64_t n_slots = min(T_cap, (int64_t)H + R + 1);   // no slot past H + R is ever used
  for (int64_t s0 = threadIdx.x; s0 < n_slots; s0 += (int64_t)kU * blockDim.x) {
    int32_t p[kU];
    float a_old[kU], add[kU];
    // every load of the pass first (a slot's acc and logits are read even when it is empty, so
    // that nothing waits for its position)
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int64_t s = s0 + (int64_t)u * blockDim.x;
      const bool in = s < n_slots;
      p[u] = in ? pos[bh * T_cap + s] : -1;
      a_old[u] = in ? acc[bh * T_cap + s] : 0.f;
      add[u] = 0.f;
      if (in) {
        const float* lg = logits + (bh * T_cap + s) * G;
        if (G == 4) {
          const float4 x = __ldcg(reinterpret_cast<const float4*>(lg));
          add[u] = h2o_ex2(x.x - m[0]) * il[0] + h2o_ex2(x.y - m[1]) * il[1] + h2o_ex2(x.z - m[2]) * il[2] +
                   h2o_ex2(x.w - m[3]) * il[3];
        } else {
#pragma unroll
          for (int h = 0; h < 8; ++h)
            if (h < G) add[u] += h2o_ex2(__ldcg(lg + h) - m[h]) * il[h];
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int64_t s = s0 + (int64_t)u * blockDim.x;
      if (p[u] < 0) {                 // an empty slot (past the end: not a slot)
        if (s < n_slots) first_free = min(first_free, (int)s);
        continue;
      }
      ++held;
      const float a2 = a_old[u] + add[u];
      acc[bh * T_cap + s] = a2;
      if ((int64_t)p[u] <= newest - R) {
        const uint64_t key = rank_key(a2, (uint32_t)p[u]);
        if (key < best) {
          best = key;
          best_slot = (int)s;
        }
      }
    }
  }
  // block reductions: held count, first free slot, min key (with its slot)
  __shared__ int s_held[32], s_free[32];
  __shared__ uint64_t s_key[32];
  __shared__ int s_slot[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int o = 16; o > 0; o >>= 1) {
    held += __shfl_xor_sync(0xffffffffu, held, o);
    first_free = min(first_free, __shfl_xor_sync(0xffffffffu, first_free, o));
    const uint64_t ok = __shfl_xor_sync(0xffffffffu, best, o);
    const int os = __shfl_xor_sync(0xffffffffu, best_slot, o);
    if (ok < best) {
      best = ok;
      best_slot = os;
    }
  }
  if (lane == 0) {
    s_held[warp] = held;
    s_free[warp] = first_free;
    s_key[warp] = best;
    s_slot[warp] = best_slot;
  }
  __syncthreads();
  if (warp == 0) {                    // the warps' results, reduced by warp 0
    const int nw = (int)(blockDim.x >> 5);
    int hsum = lane < nw ? s_held[lane] : 0, ff = lane < nw ? s_free[lane] : INT32_MAX;
    uint64_t bk = lane < nw ? s_key[lane] : ~0ull;
    int bs = lane < nw ? s_slot[lane] : -1;
    for (int o = 16; o > 0; o >>= 1) {
      hsum += __shfl_xor_sync(0xffffffffu, hsum, o);
      ff = min(ff, __shfl_xor_sync(0xffffffffu, ff, o));
      const uint64_t ok = __shfl_xor_sync(0xffffffffu, bk, o);
      const int os = __shfl_xor_sync(0xffffffffu, bs, o);
      if (ok < bk) {
        bk = ok;
        bs = os;
      }
    }
    if (lane != 0) return;
    if (hsum > H + R && bs >= 0) {
      pos[bh * T_cap + bs] = -1;
      slot_out[bh] = bs;
    } else {
      slot_out[bh] = ff == INT32_MAX ? -1 : ff;
    }
  }
}

}  // namespace mkv
