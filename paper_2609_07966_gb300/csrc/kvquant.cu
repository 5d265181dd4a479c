// KVQuant-style b-bit KV cache (Section 2.1, KVQuant paragraph): calibration,
// quantization (prefill bulk and per-step append) and the table preparation
// used by the fused-dequant decode kernel (decode_kvq.cu).
//
// Codes are decided with correctly rounded fp32 operations (__fsub_rn,
// __fdiv_rn, __fmul_rn, rintf) so that they are defined bit for bit:
//   uniform: code = clamp(rint((x - lo) / scale), 0, 2^b - 1)
//   NUQ:     code = #{j : x > mu_j},  mu_j = (c_j + c_{j+1}) * 0.5 in fp32
// Key outliers: x < t_lo or x > t_hi (per channel); value outliers: the n_v
// entries of largest |x| per token (ties: lower channel).  Outliers keep the
// code of their clamped value and are stored exactly in fp16 on the side.
#include <math.h>

#include "mkv_common.cuh"
#include "mkv_internal.h"
#include "mkv_quant_token.cuh"

namespace mkv {

namespace {

__device__ uint32_t g_status_kvquant;

// ----------------------------------------------------------------- prepare

// k_dq[h][c][j] = k_lo + j * k_scale (uniform) or the fp16 centroid (NUQ);
// v_tbl[h][c][j] = j (uniform) or the fp16 value centroid (NUQ).
__global__ void prepare_kernel(int n, int K, int nuq, const float* k_lo, const float* k_scale,
                               const uint16_t* k_cb, const uint16_t* v_cb, float* k_dq, uint16_t* v_tbl) {
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < n * K; e += gridDim.x * blockDim.x) {
    const int hc = e / K, j = e % K;
    if (nuq) {
      k_dq[e] = h2f(k_cb[e]);
      v_tbl[e] = v_cb[e];
    } else {
      k_dq[e] = __fadd_rn(k_lo[hc], __fmul_rn((float)j, k_scale[hc]));
      v_tbl[e] = __half_as_ushort(__float2half_rn((float)j));
    }
  }
}

// ----------------------------------------------------------------- quantize

struct QuantArgs {
  const __half* k_pre;   // [B][Hkv][n][D]
  const __half* v;
  int64_t n_tokens;
  int Hkv, D, bits, nuq, n_v;
  const float* t_lo;     // [Hkv][D]
  const float* t_hi;
  const float* k_lo;
  const float* k_scale;
  const uint16_t* k_cb;  // [Hkv][D][K]
  const uint16_t* v_cb;
  int32_t* T_len;
  uint8_t* k_codes;      // [B][Hkv][T_cap][row]
  uint8_t* v_codes;
  float2* v_params;      // [B][Hkv][T_cap]
  uint32_t* v_out;       // [B][Hkv][T_cap][n_v]
  int32_t* k_out_off;    // [B][Hkv][T_cap+1]
  uint32_t* k_out;       // [B][Hkv][k_out_cap]
  int64_t k_out_cap;
  int64_t T_cap;
};

// One CTA per (batch, kv-head), one thread per channel; tokens in order so the
// key-outlier CSR is appended sequentially.  Every CTA reads T_len[b] once; the
// last CTA of batch entry b to finish stores the new length: during the launch
// the top 8 bits of T_len[b] count the finished CTAs (readers mask them off).
__global__ void quantize_kernel(const QuantArgs a) {
  extern __shared__ uint8_t sm[];
  const int D = a.D, K = 1 << a.bits, L = K - 1;
  const int bh = blockIdx.x;
  const int b = bh / a.Hkv, h = bh % a.Hkv;
  const int c = threadIdx.x;   // channel
  uint8_t* kcode = sm;                       // [D]
  uint8_t* vcode = kcode + D;                // [D]
  float* absx = reinterpret_cast<float*>(vcode + D);   // [D] value magnitudes
  uint32_t* words = reinterpret_cast<uint32_t*>(absx + D);   // [2][D*bits/32] packed rows
  __shared__ int s_cnt[32];
  __shared__ float s_lo[32], s_hi[32];
  __shared__ uint32_t s_max[2][32];

  // Every load that does not depend on the length is issued before it: the channel's parameters and
  // codebooks, and the first token's key and value; then the length and the CSR offset it selects.
  const float tlo = a.t_lo[h * D + c], thi = a.t_hi[h * D + c];
  const float klo = a.k_lo ? a.k_lo[h * D + c] : 0.f, ksc = a.k_scale ? a.k_scale[h * D + c] : 0.f;
  uint16_t kr[16], vr[16];                   // all codebook loads in flight at once (K <= 16)
  if (a.nuq) {
    const uint16_t* kc = a.k_cb + ((int64_t)h * D + c) * K;
    const uint16_t* vc = a.v_cb + ((int64_t)h * D + c) * K;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      if (j < K) {
        kr[j] = __ldg(kc + j);
        vr[j] = __ldg(vc + j);
      }
    }
  }
  const int64_t src0 = (int64_t)bh * a.n_tokens * D + c;
  __half xk_next = a.n_tokens > 0 ? a.k_pre[src0] : __ushort_as_half(0);
  __half xv_next = a.n_tokens > 0 ? a.v[src0] : __ushort_as_half(0);
  const int64_t t_base = a.T_len[b] & 0xffffff;
  int32_t* off_row = a.k_out_off + (int64_t)bh * (a.T_cap + 1);
  const bool room = t_base + a.n_tokens <= a.T_cap;
  int32_t off = (t_base == 0 || !room) ? 0 : off_row[t_base];
  // the last CTA of batch entry b stores its new length (after every thread of this CTA read it)
  auto finish = [&](int64_t len) {
    __syncthreads();
    if (c == 0) {
      const unsigned old = atomicAdd(reinterpret_cast<unsigned*>(a.T_len) + b, 1u << 24);
      if ((int)(old >> 24) == a.Hkv - 1) a.T_len[b] = (int32_t)len;
    }
  };
  if (!room) {                            // no room: drop, flag, keep T_len
    if (c == 0 && h == 0) atomicOr(&g_status_kvquant, MKV_FLAG_CACHE_FULL);
    finish(t_base);
    return;
  }
  float kmu[15], vmu[15];
  if (a.nuq) {
#pragma unroll
    for (int j = 0; j < 15; ++j) {
      if (j < L) {
        kmu[j] = fl32_mid(h2f(kr[j]), h2f(kr[j + 1]));
        vmu[j] = fl32_mid(h2f(vr[j]), h2f(vr[j + 1]));
      }
    }
  }
  if (t_base == 0 && c == 0) off_row[0] = 0;
  const QTokDst dst{a.k_out + (int64_t)bh * a.k_out_cap, a.k_out_cap, a.v_out + (int64_t)bh * a.T_cap * a.n_v,
                    a.v_params + (int64_t)bh * a.T_cap, a.k_codes + (int64_t)bh * a.T_cap * (D * a.bits / 8),
                    a.v_codes + (int64_t)bh * a.T_cap * (D * a.bits / 8), off_row};
  const QTokSmem scr{kcode, vcode, absx, words, s_cnt, s_lo, s_hi, &s_max[0][0]};
  for (int64_t i = 0; i < a.n_tokens; ++i) {
    const __half xk = xk_next, xv = xv_next;     // this token's key and value; the next one's in flight
    if (i + 1 < a.n_tokens) {
      xk_next = a.k_pre[src0 + (i + 1) * D];
      xv_next = a.v[src0 + (i + 1) * D];
    }
    off = quantize_token(c, D, a.bits, a.nuq != 0, a.n_v, kmu, vmu, tlo, thi, klo, ksc, xk, xv, t_base + i, off, dst,
                         scr, &g_status_kvquant, [] { __syncthreads(); });
  }
  finish(t_base + a.n_tokens);
}

// ----------------------------------------------------------------- calibrate

// Per (kv-head, calibration token): value-outlier flags and u = (x - lo)/s.
__global__ void calib_values_kernel(const __half* v_cal, int64_t N, int64_t row_stride, int D, int n_v,
                                    float* u_out, uint8_t* vmask) {
  extern __shared__ float absx[];
  const int64_t ht = blockIdx.x;   // h * N + t
  const int64_t h = ht / N, t = ht % N;
  const int c = threadIdx.x, lane = c & 31, warp = c >> 5, nwarp = D >> 5;
  __shared__ float s_lo[32], s_hi[32];
  const __half xv = v_cal[(h * row_stride + t) * D + c];
  const float x = __half2float(xv);
  absx[c] = fabsf(x);
  __syncthreads();
  const float ax = absx[c];
  int rank = 0;
  for (int j = 0; j < D; ++j) {
    const float o = absx[j];
    rank += (o > ax || (o == ax && j < c)) ? 1 : 0;
  }
  const bool out = rank < n_v;
  float lo = out ? INFINITY : x, hi = out ? -INFINITY : x;
  for (int s = 16; s > 0; s >>= 1) {
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, s));
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, s));
  }
  if (lane == 0) {
    s_lo[warp] = lo;
    s_hi[warp] = hi;
  }
  __syncthreads();
  lo = s_lo[0];
  hi = s_hi[0];
  for (int w = 1; w < nwarp; ++w) {
    lo = fminf(lo, s_lo[w]);
    hi = fmaxf(hi, s_hi[w]);
  }
  if (lo > hi) lo = hi = 0.f;
  const float s = __fsub_rn(hi, lo);
  const float u = s == 0.f ? 0.f : __fdiv_rn(__fsub_rn(x, lo), s);
  u_out[(h * N + t) * D + c] = u;
  vmask[(h * N + t) * D + c] = out ? 1 : 0;
}

// Bitonic sort of n <= 4096 floats in shared memory (padded with +inf to a power of two).
__device__ void block_sort(float* s, int n_pow2) {
  for (int k = 2; k <= n_pow2; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n_pow2; i += blockDim.x) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const float a = s[i], b = s[ixj];
          const bool up = (i & k) == 0;
          if ((a > b) == up) {
            s[i] = b;
            s[ixj] = a;
          }
        }
      }
      __syncthreads();
    }
  }
}

__device__ uint16_t fp16_next_up(uint16_t bits) {
  if (bits == 0x8000u || bits == 0u) return 0x0001u;
  return (bits & 0x8000u) ? (uint16_t)(bits - 1u) : (uint16_t)(bits + 1u);
}

// 1-D Lloyd k-means on sorted data x[0..n): quantile start, 25 iterations,
// nearest centroid (ties: lower index), means summed in ascending order in fp64,
// empty clusters keep their centroid; then fp16, sorted, made strictly increasing.
__device__ void lloyd_codebook(const float* x, int n, int K, uint16_t* out, double* cent, uint8_t* asg) {
  const int tid = threadIdx.x;
  if (tid < K) {
    int idx = (int)floor((tid + 0.5) * (double)n / K);
    cent[tid] = n > 0 ? (double)x[min(n - 1, idx)] : 0.0;
  }
  __syncthreads();
  for (int it = 0; it < 25 && n > 0; ++it) {
    for (int i = tid; i < n; i += blockDim.x) {
      const double xv = (double)x[i];
      int best = 0;
      double bd = fabs(xv - cent[0]);
      for (int j = 1; j < K; ++j) {
        const double d = fabs(xv - cent[j]);
        if (d < bd) {
          bd = d;
          best = j;
        }
      }
      asg[i] = (uint8_t)best;
    }
    __syncthreads();
    if (tid < K) {
      double sum = 0.0;
      int cnt = 0;
      for (int i = 0; i < n; ++i) {
        if (asg[i] == tid) {
          sum += (double)x[i];
          ++cnt;
        }
      }
      if (cnt > 0) cent[tid] = sum / (double)cnt;
    }
    __syncthreads();
  }
  if (tid == 0) {
    uint16_t cb[16];
    for (int j = 0; j < K; ++j) cb[j] = __half_as_ushort(__double2half(cent[j]));
    // insertion sort by value (fp16 compare)
    for (int j = 1; j < K; ++j) {
      const uint16_t v = cb[j];
      int m = j - 1;
      while (m >= 0 && __hgt(__ushort_as_half(cb[m]), __ushort_as_half(v))) {
        cb[m + 1] = cb[m];
        --m;
      }
      cb[m + 1] = v;
    }
    for (int j = 1; j < K; ++j) {
      if (__hle(__ushort_as_half(cb[j]), __ushort_as_half(cb[j - 1]))) cb[j] = fp16_next_up(cb[j - 1]);
    }
    for (int j = 0; j < K; ++j) out[j] = cb[j];
  }
  __syncthreads();
}

struct CalibArgs {
  const __half* k_cal;   // [Hkv][row_stride][D]
  const float* u;        // [Hkv][N][D]
  const uint8_t* vmask;  // [Hkv][N][D]
  int64_t N, row_stride;
  int D, bits, nuq, nt, all_out;
  float* t_lo;
  float* t_hi;
  float* k_lo;
  float* k_scale;
  uint16_t* k_cb;
  uint16_t* v_cb;
};

// grid (Hkv*D, 2): y = 0 keys, y = 1 values (NUQ only).
__global__ void calib_channel_kernel(const CalibArgs a) {
  extern __shared__ float s[];   // [n_pow2] data, then fp64 centroids and assignments
  const int hc = blockIdx.x;
  const int h = hc / a.D, c = hc % a.D;
  const bool values = blockIdx.y == 1;
  if (values && !a.nuq) return;
  int n_pow2 = 1;
  while (n_pow2 < a.N) n_pow2 <<= 1;
  double* cent = reinterpret_cast<double*>(s + n_pow2 + (n_pow2 & 1));
  uint8_t* asg = reinterpret_cast<uint8_t*>(cent + 16);
  __shared__ int s_cnt;
  if (threadIdx.x == 0) s_cnt = 0;
  __syncthreads();
  for (int i = threadIdx.x; i < n_pow2; i += blockDim.x) {
    float v = INFINITY;
    if (i < a.N) {
      if (!values) {
        v = __half2float(a.k_cal[((int64_t)h * a.row_stride + i) * a.D + c]);
      } else if (!a.vmask[((int64_t)h * a.N + i) * a.D + c]) {
        v = a.u[((int64_t)h * a.N + i) * a.D + c];
        atomicAdd(&s_cnt, 1);
      }
    }
    s[i] = v;
  }
  __syncthreads();
  block_sort(s, n_pow2);
  const int K = 1 << a.bits, L = K - 1;
  if (!values) {
    const int N = (int)a.N;
    float tl = INFINITY, th = -INFINITY;
    if (!a.all_out) {
      tl = s[a.nt];
      th = s[N - 1 - a.nt];
    }
    if (threadIdx.x == 0) {
      a.t_lo[hc] = tl;
      a.t_hi[hc] = th;
      const float lo = a.all_out ? 0.f : tl, hi = a.all_out ? 0.f : th;
      if (a.k_lo) a.k_lo[hc] = lo;
      if (a.k_scale) a.k_scale[hc] = __fdiv_rn(__fsub_rn(hi, lo), (float)L);
    }
    if (a.nuq) {
      // inliers: the contiguous sorted range with tl <= x <= th
      __shared__ int s_a, s_b;
      if (threadIdx.x == 0) {
        int lo_i = 0, hi_i = 0;
        if (!a.all_out) {
          lo_i = a.nt;
          while (lo_i > 0 && s[lo_i - 1] >= tl) --lo_i;
          hi_i = N - 1 - a.nt;
          while (hi_i + 1 < N && s[hi_i + 1] <= th) ++hi_i;
          hi_i += 1;
        }
        s_a = lo_i;
        s_b = hi_i;
      }
      __syncthreads();
      lloyd_codebook(s + s_a, s_b - s_a, K, a.k_cb + (int64_t)hc * K, cent, asg);
    }
  } else {
    __syncthreads();
    lloyd_codebook(s, s_cnt, K, a.v_cb + (int64_t)hc * K, cent, asg);
  }
}

}  // namespace

cudaError_t launch_quant_prepare(const mkv_config& c, const mkv_quant_params& qp, cudaStream_t st) {
  const int n = c.Hkv * c.D, K = 1 << c.bits;
  prepare_kernel<<<(int)ceil_div((int64_t)n * K, 256), 256, 0, st>>>(
      n, K, c.quant_mode == MKV_QUANT_NUQ, qp.k_lo, qp.k_scale, qp.k_cb, qp.v_cb, qp.k_dq, qp.v_tbl);
  return cudaPeekAtLastError();
}

cudaError_t launch_quantize(const mkv_config& c, const mkv_quant_params& qp, const void* k_pre, const void* v,
                            int64_t n_tokens, const mkv_cache& cache, cudaStream_t st) {
  QuantArgs a{};
  a.k_pre = static_cast<const __half*>(k_pre);
  a.v = static_cast<const __half*>(v);
  a.n_tokens = n_tokens;
  a.Hkv = c.Hkv;
  a.D = c.D;
  a.bits = c.bits;
  a.nuq = c.quant_mode == MKV_QUANT_NUQ;
  a.n_v = std::min(c.D, (int)ceil((double)c.outlier_frac * c.D));
  a.t_lo = qp.t_lo;
  a.t_hi = qp.t_hi;
  a.k_lo = qp.k_lo;
  a.k_scale = qp.k_scale;
  a.k_cb = qp.k_cb;
  a.v_cb = qp.v_cb;
  a.T_len = cache.T_len;
  a.k_codes = cache.k_codes;
  a.v_codes = cache.v_codes;
  a.v_params = reinterpret_cast<float2*>(cache.v_params);
  a.v_out = cache.v_out;
  a.k_out_off = cache.k_out_off;
  a.k_out = cache.k_out;
  a.k_out_cap = cache.k_out_cap;
  a.T_cap = cache.T_cap;
  const int nwords = (c.D * c.bits / 8 + 3) / 4;
  const size_t smem = 2 * c.D + 4 * c.D + 2 * nwords * 4 + 16;
  quantize_kernel<<<c.B * c.Hkv, c.D, smem, st>>>(a);
  return cudaPeekAtLastError();
}

cudaError_t launch_calibrate(const mkv_config& c, const void* k_cal, const void* v_cal, int64_t N,
                             int64_t row_stride, const mkv_quant_params& qp, const CalibWs& ws, cudaStream_t st) {
  const bool nuq = c.quant_mode == MKV_QUANT_NUQ;
  const int n_v = std::min(c.D, (int)ceil((double)c.outlier_frac * c.D));
  if (nuq) {
    calib_values_kernel<<<(unsigned)(c.Hkv * N), c.D, c.D * sizeof(float), st>>>(
        static_cast<const __half*>(v_cal), N, row_stride, c.D, n_v, ws.u, ws.vmask);
    cudaError_t e = cudaPeekAtLastError();
    if (e != cudaSuccess) return e;
  }
  CalibArgs a{};
  a.k_cal = static_cast<const __half*>(k_cal);
  a.u = ws.u;
  a.vmask = ws.vmask;
  a.N = N;
  a.row_stride = row_stride;
  a.D = c.D;
  a.bits = c.bits;
  a.nuq = nuq;
  a.nt = (int)ceil((double)c.outlier_frac / 2.0 * (double)N);
  a.all_out = 2 * a.nt >= N;
  a.t_lo = qp.t_lo;
  a.t_hi = qp.t_hi;
  a.k_lo = qp.k_lo;
  a.k_scale = qp.k_scale;
  a.k_cb = qp.k_cb;
  a.v_cb = qp.v_cb;
  int n_pow2 = 1;
  while (n_pow2 < N) n_pow2 <<= 1;
  const size_t smem = (size_t)(n_pow2 + 2) * sizeof(float) + 16 * sizeof(double) + n_pow2 + 16;
  cudaError_t e = cudaFuncSetAttribute(calib_channel_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  calib_channel_kernel<<<dim3(c.Hkv * c.D, nuq ? 2 : 1), 512, smem, st>>>(a);
  return cudaPeekAtLastError();
}

cudaError_t take_status_kvquant(uint32_t* flags, cudaStream_t st) {
  uint32_t zero = 0, v = 0;
  cudaError_t e = cudaMemcpyFromSymbolAsync(&v, g_status_kvquant, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyToSymbolAsync(g_status_kvquant, &zero, sizeof(zero), 0, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  *flags |= v;
  return e;
}

}  // namespace mkv
