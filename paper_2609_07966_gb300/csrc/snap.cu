// RocketKV (Section 2.1, RocketKV paragraph).
// Stage 1, SnapKV prefill compression: the observation window's aggregated
// scores of the prefix (prefill.cu), max-pooled over |j' - j| <= pool/2,
// the keep - W best prefix positions under (pooled desc, position asc) plus
// the window, gathered in ascending position; per-page key min/max of the
// compact cache.
// Stage 2, page choice at decode: dims = the topq_dims largest sum_h |q_h,i|
// (dim asc on ties), page score = sum_h sum_{i in dims}
// max(q_h,i kmin_i, q_h,i kmax_i) over full pages before the newest token's,
// best topk_pages under (score desc, page asc), listed ascending.
#include <math.h>

#include "mkv_common.cuh"
#include "mkv_internal.h"
#include "mkv_select.cuh"

namespace mkv {

namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelPages = 256;          // page selection: pages whose bounds are prefetched for every dim
constexpr int kSelRow = kSelPages + 8;  // halves per prefetched row (room for the 16-byte alignment offset)
constexpr int kSelChunks = kSelRow / 8; // 16-byte copies per prefetched row

__device__ __forceinline__ float pooled_at(const float* s, int64_t n, int64_t j, int r) {
  float m = -INFINITY;
  const int64_t lo = j - r < 0 ? 0 : j - r, hi = j + r >= n ? n - 1 : j + r;
  for (int64_t i = lo; i <= hi; ++i) m = fmaxf(m, s[i]);
  return m;
}

constexpr int kPooledSmem = 51200;      // pooled scores kept in shared memory up to this many positions

// One CTA per (batch, kv-head): keep list (ascending) of the compressed cache.  The pooled scores
// live in shared memory when they fit (dynamic, n floats), else in the workspace.
__global__ void __launch_bounds__(kSelThreads) snap_keep_kernel(const float* __restrict__ score, int64_t T, int W,
                                                                int pool, int keep, float* __restrict__ pooled_ws,
                                                                int32_t* __restrict__ keep_out) {
  __shared__ int hist[256];
  __shared__ int warp_sums[32];
  extern __shared__ float pooled_sm[];
  const int64_t bh = blockIdx.x;
  const int64_t n = T - W;                        // prefix positions compete
  const float* s = score + bh * T;
  float* pooled = n <= kPooledSmem ? pooled_sm : pooled_ws + bh * T;
  int32_t* out = keep_out + bh * T;
  const int r = pool / 2;
  for (int64_t j = threadIdx.x; j < n; j += blockDim.x) pooled[j] = pooled_at(s, n, j, r);
  __syncthreads();
  const int k = keep - W;
  uint64_t thr = ~0ull;
  if (k > 0) thr = block_kth_largest_score((int)n, k, [&](int i) { return pooled[i]; }, hist);
  int64_t base = 0;
  for (int64_t i0 = 0; i0 < T; i0 += blockDim.x) {
    const int64_t i = i0 + threadIdx.x;
    int flag = 0;
    if (i < T) flag = (i >= n) || (k > 0 && rank_key(pooled[i], (uint32_t)i) >= thr);
    int total;
    const int before = block_exclusive_scan(flag, warp_sums, &total);
    if (flag) out[base + before] = (int32_t)i;
    base += total;
  }
}

// Gather kept rows (keep list, or the identity when keep >= T) into slots 0..n-1.
__global__ void snap_gather_kernel(const __half* __restrict__ full_k, const __half* __restrict__ full_v,
                                   const int32_t* __restrict__ keep, int identity, int64_t T, int64_t n, int Hkv,
                                   int D, int64_t T_cap, __half* k, __half* v, int32_t* kept_pos, int32_t* T_len) {
  const int64_t bh = blockIdx.y;
  const int nc = D / 8;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n * nc; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t sl = e / nc;
    const int col = (int)(e % nc);
    const int64_t p = identity ? sl : keep[bh * T + sl];
    reinterpret_cast<uint4*>(k + (bh * T_cap + sl) * D)[col] = reinterpret_cast<const uint4*>(full_k + (bh * T + p) * D)[col];
    reinterpret_cast<uint4*>(v + (bh * T_cap + sl) * D)[col] = reinterpret_cast<const uint4*>(full_v + (bh * T + p) * D)[col];
    if (col == 0 && kept_pos) kept_pos[bh * n + sl] = (int32_t)p;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0 && bh % Hkv == 0) T_len[bh / Hkv] = (int32_t)n;
}

// kmin/kmax [bh][D][T_cap/16] of every full page among slots 0..n-1.
__global__ void page_meta_kernel(const __half* __restrict__ k, int64_t T_cap, int D, int64_t n, __half* kmin,
                                 __half* kmax) {
  const int64_t bh = blockIdx.y;
  const int64_t npc = T_cap / kPage, np = n / kPage;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < np * D; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t p = e / D;
    const int d = (int)(e % D);
    const __half* base = k + (bh * T_cap + p * kPage) * D + d;
    __half lo = base[0], hi = base[0];
    for (int j = 1; j < kPage; ++j) {
      const __half x = base[(int64_t)j * D];
      lo = __hlt(x, lo) ? x : lo;
      hi = __hgt(x, hi) ? x : hi;
    }
    kmin[(bh * D + d) * npc + p] = lo;
    kmax[(bh * D + d) * npc + p] = hi;
  }
}

// One CTA per (batch, kv-head): dims, page scores, top-k pages.
// Page selection (RocketKV stage 2).  With max(q kmin, q kmax) = q kmax for q >= 0 and q kmin
// otherwise (kmin <= kmax), a page's score over the selected dims t is
//   sum_t (kmax_t P_t + kmin_t N_t),  P_t = sum_h max(q_h,t, 0),  N_t = sum_h min(q_h,t, 0).
// Up to kSelPages candidate pages (the common case) the bounds of every dim are prefetched into
// shared memory while the dims are being chosen; larger caches stage the chosen dims' bounds
// 256 pages at a time.
__global__ void __launch_bounds__(kSelThreads) rocket_select_kernel(const __half* __restrict__ q, const __half* __restrict__ kmin,
                                                                    const __half* __restrict__ kmax,
                                                                    const int32_t* __restrict__ T_len, int Hkv, int G, int D,
                                                                    int64_t T_cap, int kp, int rd, int32_t* __restrict__ out) {
  extern __shared__ __align__(16) float sm[];
  const int64_t npc = T_cap / kPage;
  float* qs = sm;                       // [G][D]
  float* ssc = qs + G * D;              // [npc] page scores
  float* part = ssc + ((npc + 3) & ~3ll);                     // [4][kSelPages] partial scores
  __half* bmn = reinterpret_cast<__half*>(part + 4 * kSelPages);   // fast path: [D][kSelRow]
  __half* bmx = bmn + D * kSelRow;
  __shared__ int hist[256];
  __shared__ int warp_sums[32];
  __shared__ int dims[128];
  __shared__ __align__(16) float a_dim[128];
  __shared__ float pn[2][128];          // P_t, N_t of the selected dims
  const int64_t bh = blockIdx.x;
  const int b = (int)(bh / Hkv), kvh = (int)(bh % Hkv);
  const int n = (int)min((int64_t)T_len[b], T_cap);
  const int ns = n > 0 ? (n - 1) / kPage : 0;
  const bool fast = ns <= kSelPages;
  if (fast && ns > 0) {
    // every dim's bounds of pages [0, ns): 16-byte copies from the row start rounded down to
    // 16 bytes (the first copy may begin in the previous row), the last one cut at the row end
    for (int e = threadIdx.x; e < 2 * D * kSelChunks; e += blockDim.x) {
      const int which = e / (D * kSelChunks), rem = e % (D * kSelChunks);
      const int dim = rem / kSelChunks, ch = rem % kSelChunks;
      const int64_t start = (bh * D + dim) * npc;           // first half of the row
      const int64_t h0 = (start & ~7ll) + ch * 8;
      const int64_t end = start + ns;
      if (h0 < end) {
        const int bytes = (int)min((int64_t)16, (end - h0) * 2);
        cp_async16((which ? bmx : bmn) + dim * kSelRow + ch * 8, (which ? kmax : kmin) + h0, bytes);
      }
    }
    cp_async_commit();
  }
  for (int e = threadIdx.x; e < G * D; e += blockDim.x) qs[e] = __half2float(q[((int64_t)b * Hkv * G + (int64_t)kvh * G) * D + e]);
  __syncthreads();
  if (threadIdx.x < D) {
    float a = 0.f;
    for (int h = 0; h < G; ++h) a += fabsf(qs[h * D + threadIdx.x]);
    a_dim[threadIdx.x] = a;
  }
  __syncthreads();
  if (threadIdx.x < D) {
    // rank under (sum |q| desc, dim asc): four dims per shared-memory read, unrolled so the
    // reads overlap
    const int i = threadIdx.x;
    const float ai = a_dim[i];
    int rank = 0;
#pragma unroll 4
    for (int j = 0; j < D; j += 4) {
      const float4 v = *reinterpret_cast<const float4*>(a_dim + j);
      rank += (v.x > ai || (v.x == ai && j < i)) + (v.y > ai || (v.y == ai && j + 1 < i)) +
              (v.z > ai || (v.z == ai && j + 2 < i)) + (v.w > ai || (v.w == ai && j + 3 < i));
    }
    if (rank < rd) dims[rank] = i;
  }
  __syncthreads();
  if (threadIdx.x < rd) {
    const int d = dims[threadIdx.x];
    float P = 0.f, N = 0.f;
    for (int h = 0; h < G; ++h) {
      const float v = qs[h * D + d];
      P += fmaxf(v, 0.f);
      N += fminf(v, 0.f);
    }
    pn[0][threadIdx.x] = P;
    pn[1][threadIdx.x] = N;
  }
  if (fast) {
    cp_async_wait<0>();
    __syncthreads();
    // thread (page p, slice sl) sums the dims t = sl, sl + 4, ...; the four slices are added after
    const int p = threadIdx.x % kSelPages, sl = threadIdx.x / kSelPages;
    if (sl < 4) {
      float acc = 0.f;
      if (p < ns) {
        for (int t = sl; t < rd; t += 4) {
          const int d = dims[t];
          const int off = (int)(((bh * D + d) * npc) & 7);
          const int i = d * kSelRow + off + p;
          acc += __half2float(bmx[i]) * pn[0][t] + __half2float(bmn[i]) * pn[1][t];
        }
      }
      part[sl * kSelPages + p] = acc;
    }
    __syncthreads();
    if (threadIdx.x < ns)
      ssc[threadIdx.x] = (part[threadIdx.x] + part[kSelPages + threadIdx.x]) +
                         (part[2 * kSelPages + threadIdx.x] + part[3 * kSelPages + threadIdx.x]);
    else if (threadIdx.x < ((ns + 3) & ~3))
      ssc[threadIdx.x] = -INFINITY;       // pads the last group of four; never ranks ahead
    __syncthreads();
  } else {
    __syncthreads();
    // the selected dims' min/max rows staged 256 pages at a time with coalesced loads (dim-major
    // layout), then each thread scores one page from shared memory
    __half* smn = bmn;                                          // [rd][256]
    __half* smx = smn + rd * 256;
    for (int p0 = 0; p0 < ns; p0 += 256) {
      const int np = min(256, ns - p0);
      for (int e = threadIdx.x; e < rd * 256; e += blockDim.x) {
        const int t = e / 256, pp = e % 256;
        if (pp < np) {
          const int64_t src = (bh * D + dims[t]) * npc + p0 + pp;
          smn[e] = kmin[src];
          smx[e] = kmax[src];
        }
      }
      __syncthreads();
      if (threadIdx.x < np) {
        float sc = 0.f;
        for (int t = 0; t < rd; ++t)
          sc += __half2float(smx[t * 256 + threadIdx.x]) * pn[0][t] + __half2float(smn[t * 256 + threadIdx.x]) * pn[1][t];
        ssc[p0 + threadIdx.x] = sc;
      }
      __syncthreads();
    }
  }
  const int k = min(kp, ns);
  int base = 0;
  if (ns <= (int)blockDim.x) {
    // few pages: each thread ranks its page by counting the pages ahead of it under
    // (score desc, page asc)
    const int i = threadIdx.x;
    int flag = 0;
    if (i < ns && k > 0) {
      const float si = ssc[i];
      int rank = 0;
      if (fast) {                         // scores padded to a multiple of four with -inf
#pragma unroll 4
        for (int j = 0; j < ns; j += 4) {
          const float4 v = *reinterpret_cast<const float4*>(ssc + j);
          rank += (v.x > si || (v.x == si && j < i)) + (v.y > si || (v.y == si && j + 1 < i)) +
                  (v.z > si || (v.z == si && j + 2 < i)) + (v.w > si || (v.w == si && j + 3 < i));
        }
      } else {
        for (int j = 0; j < ns; ++j) {
          const float sj = ssc[j];
          rank += (sj > si || (sj == si && j < i)) ? 1 : 0;
        }
      }
      flag = rank < k;
    }
    int total;
    const int before = block_exclusive_scan(flag, warp_sums, &total);
    if (flag) out[bh * kp + before] = i;
    base = total;
  } else {
    uint64_t thr = ~0ull;
    if (k > 0) thr = block_kth_largest_score(ns, k, [&](int i) { return ssc[i]; }, hist);
    for (int i0 = 0; i0 < ns; i0 += blockDim.x) {
      const int i = i0 + threadIdx.x;
      const int flag = (i < ns && k > 0 && rank_key(ssc[i], (uint32_t)i) >= thr) ? 1 : 0;
      int total;
      const int before = block_exclusive_scan(flag, warp_sums, &total);
      if (flag) out[bh * kp + base + before] = i;
      base += total;
    }
  }
  for (int i = base + threadIdx.x; i < kp; i += blockDim.x) out[bh * kp + i] = -1;
}

}  // namespace

cudaError_t launch_snap_keep(const mkv_config& c, const void* full_k, const void* full_v, int64_t T,
                             const mkv_cache& cache, int32_t* kept_pos, const PrefillWs& ws, cudaStream_t st) {
  const int units = c.B * c.Hkv;
  const bool identity = T <= c.snap_keep;
  const int64_t n = identity ? T : c.snap_keep;
  if (!identity) {
    const int64_t n_pre = T - c.snap_window;
    const int smem = n_pre <= kPooledSmem ? (int)(n_pre * sizeof(float)) : 0;
    cudaError_t ea = cudaFuncSetAttribute(snap_keep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (ea != cudaSuccess) return ea;
    snap_keep_kernel<<<units, kSelThreads, smem, st>>>(ws.score, T, c.snap_window, c.snap_pool, c.snap_keep,
                                                    reinterpret_cast<float*>(ws.row_st),
                                                    ws.keep);
    cudaError_t e = cudaPeekAtLastError();
    if (e != cudaSuccess) return e;
  }
  const int bx = (int)std::min<int64_t>(ceil_div(n * (c.D / 8), 256), 128);
  snap_gather_kernel<<<dim3(bx, units), 256, 0, st>>>(
      static_cast<const __half*>(full_k), static_cast<const __half*>(full_v), ws.keep, identity ? 1 : 0, T, n, c.Hkv,
      c.D, cache.T_cap, static_cast<__half*>(cache.k), static_cast<__half*>(cache.v), kept_pos, cache.T_len);
  cudaError_t e = cudaPeekAtLastError();
  if (e != cudaSuccess) return e;
  const int bm = (int)std::min<int64_t>(ceil_div((n / kPage) * c.D, 256), 128);
  if (n >= kPage) {
    page_meta_kernel<<<dim3(bm, units), 256, 0, st>>>(static_cast<const __half*>(cache.k), cache.T_cap, c.D, n,
                                                      static_cast<__half*>(cache.kmin), static_cast<__half*>(cache.kmax));
  }
  return cudaPeekAtLastError();
}

cudaError_t launch_rocket_select(const mkv_config& c, const void* q, const mkv_cache& cache, int32_t* page_idx,
                                 cudaStream_t st) {
  const int G = c.Hq / c.Hkv;
  const int64_t npc = cache.T_cap / kPage;
  const size_t smem = ((size_t)G * c.D + ((npc + 3) & ~3ll) + 4 * kSelPages) * sizeof(float) +
                      std::max<size_t>(2 * (size_t)c.D * kSelRow * 2, 2 * (size_t)c.topq_dims * 256 * 2);
  cudaError_t e = cudaFuncSetAttribute(rocket_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  rocket_select_kernel<<<c.B * c.Hkv, kSelThreads, smem, st>>>(
      static_cast<const __half*>(q), static_cast<const __half*>(cache.kmin), static_cast<const __half*>(cache.kmax),
      cache.T_len, c.Hkv, G, c.D, cache.T_cap, c.topk_pages, c.topq_dims, page_idx);
  return cudaPeekAtLastError();
}

}  // namespace mkv
