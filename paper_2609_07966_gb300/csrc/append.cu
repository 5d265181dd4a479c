// Per-step append of one token to an FP16, H2O or RocketKV cache, and the
// rotary (cos, sin) table of the KVQuant path.
#include <math.h>

#include "mkv_common.cuh"
#include "mkv_internal.h"

namespace mkv {

namespace {

__device__ uint32_t g_status_append;   // MKV_FLAG_* bits raised by this unit

struct AppendArgs {
  const uint4* k_new;   // [B][Hkv][D] fp16, as 16-byte chunks
  const uint4* v_new;
  uint4* k;             // [B][Hkv][T_cap][D]
  uint4* v;
  int32_t* T_len;
  int32_t* pos;
  float* acc;
  int32_t* slot;
  __half* kmin;         // ROCKET [B][Hkv][D][T_cap/16]
  __half* kmax;
  int64_t T_cap;
  int Hkv, D, mode;     // mode: 0 FP16, 1 H2O, 2 ROCKET
};

// One CTA per batch entry: every kv-head's row, then (ROCKET) the metadata of a
// page the token completes, then T_len[b] += 1.
__global__ void append_kernel(const AppendArgs a) {
  pdl_wait_and_trigger();
  const int b = blockIdx.x;
  const int t = a.T_len[b];
  const int nc = a.D / 8;
  __shared__ int ok;
  if (threadIdx.x == 0) ok = 1;
  __syncthreads();
  // all or nothing per batch entry: if any kv-head has no room, no row is written
  for (int kvh = threadIdx.x; kvh < a.Hkv; kvh += blockDim.x) {
    const int64_t s = a.mode == 1 ? a.slot[(int64_t)b * a.Hkv + kvh] : t;
    if (s < 0 || s >= a.T_cap) ok = 0;
  }
  __syncthreads();
  for (int e = threadIdx.x; ok && e < a.Hkv * nc; e += blockDim.x) {
    const int kvh = e / nc, col = e % nc;
    const int64_t bh = (int64_t)b * a.Hkv + kvh;
    const int64_t s = a.mode == 1 ? a.slot[bh] : t;
    a.k[(bh * a.T_cap + s) * nc + col] = a.k_new[bh * nc + col];
    a.v[(bh * a.T_cap + s) * nc + col] = a.v_new[bh * nc + col];
    if (a.mode == 1 && col == 0) {
      a.pos[bh * a.T_cap + s] = t;
      a.acc[bh * a.T_cap + s] = 0.f;
    }
  }
  __syncthreads();
  if (a.mode == 2 && ok && ((t + 1) % kPage) == 0) {
    const int p = t / kPage;
    const int64_t npc = a.T_cap / kPage;
    const __half* kh = reinterpret_cast<const __half*>(a.k);
    for (int e = threadIdx.x; e < a.Hkv * a.D; e += blockDim.x) {
      const int kvh = e / a.D, d = e % a.D;
      const int64_t bh = (int64_t)b * a.Hkv + kvh;
      __half lo = kh[(bh * a.T_cap + (int64_t)p * kPage) * a.D + d], hi = lo;
      for (int j = 1; j < kPage; ++j) {
        const __half x = kh[(bh * a.T_cap + (int64_t)p * kPage + j) * a.D + d];
        lo = __hlt(x, lo) ? x : lo;
        hi = __hgt(x, hi) ? x : hi;
      }
      a.kmin[(bh * a.D + d) * npc + p] = lo;
      a.kmax[(bh * a.D + d) * npc + p] = hi;
    }
  }
  if (threadIdx.x == 0) {
    if (ok) {
      a.T_len[b] = t + 1;
    } else {
      atomicOr(&g_status_append, MKV_FLAG_CACHE_FULL);
    }
  }
}

// table[p][i] = (cos, sin)(p * theta^(-2i/D)) in fp64, rounded to fp32.
__global__ void rope_table_kernel(int D, double theta, int64_t T_max, float2* table) {
  const int half = D / 2;
  const int64_t n = T_max * half;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t p = e / half;
    const int i = (int)(e % half);
    const double w = pow(theta, -2.0 * (double)i / (double)D);
    double s, c;
    sincos((double)p * w, &s, &c);
    table[e] = make_float2((float)c, (float)s);
  }
}

}  // namespace

cudaError_t launch_append(const mkv_config& c, const void* k_new, const void* v_new,
                          const mkv_cache& cache, cudaStream_t st) {
  AppendArgs a{};
  a.k_new = static_cast<const uint4*>(k_new);
  a.v_new = static_cast<const uint4*>(v_new);
  a.k = static_cast<uint4*>(cache.k);
  a.v = static_cast<uint4*>(cache.v);
  a.T_len = cache.T_len;
  a.pos = cache.pos;
  a.acc = cache.acc;
  a.slot = cache.slot;
  a.kmin = static_cast<__half*>(cache.kmin);
  a.kmax = static_cast<__half*>(cache.kmax);
  a.T_cap = cache.T_cap;
  a.Hkv = c.Hkv;
  a.D = c.D;
  a.mode = c.method == MKV_H2O ? 1 : (c.method == MKV_ROCKET ? 2 : 0);
  return launch_pdl(append_kernel, dim3(c.B), dim3(256), 0, st, a);
}

cudaError_t launch_rope_table(int D, float theta, int64_t T_max, float* table, cudaStream_t st) {
  const int64_t n = T_max * (D / 2);
  const int blocks = (int)std::min<int64_t>(ceil_div(n, 256), 4 * kNumSMs * 8);
  rope_table_kernel<<<blocks, 256, 0, st>>>(D, (double)theta, T_max, reinterpret_cast<float2*>(table));
  return cudaPeekAtLastError();
}

cudaError_t take_status_append(uint32_t* flags, cudaStream_t st) {
  uint32_t zero = 0, v = 0;
  cudaError_t e = cudaMemcpyFromSymbolAsync(&v, g_status_append, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyToSymbolAsync(g_status_append, &zero, sizeof(zero), 0, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  *flags |= v;
  return e;
}

}  // namespace mkv
