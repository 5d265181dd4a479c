// Prefill-side attention scores shared by H2O and SnapKV (Section 2.1):
//   score[j] = sum over the group's query heads h and query rows i whose
//              position p_i >= j of softmax_i(scale q_{h,i} . k)[j]
// -- H2O: every prompt row (p_i = i), the accumulated attention a token
//    receives from later tokens;
// -- SnapKV: the W rows of the observation window (p_i = T - W + i).
// Two tensor-core passes (m16n8k16, fp16 in, fp32 accumulate):
//   pass 1: per query row, running max m_i and sum l_i of 2^(s - m_i) over
//           its causal keys (key range split across CTAs, merged in pass 2);
//   pass 2: per key block, sum of 2^(s - m_i) / l_i over the query rows, the
//           product computed transposed (keys as the M dimension) so each key's
//           column sum stays in the registers of the lanes that own it.
#include <math.h>

#include <algorithm>

#include "mkv_common.cuh"
#include "mkv_internal.h"

namespace mkv {

namespace {

constexpr int kT = 128;   // threads: 4 warps

struct ScoreArgs {
  const __half* q;      // [B][Hq][R][D]
  const __half* k;      // [B][Hkv][T][D]
  int64_t R, T, pos0;   // query rows, keys, position of query row 0
  int Hq, Hkv, G, rpb;  // rpb = rows per block (64 / G)
  int n_ksplit, tiles_per_split;
  float scale_log2;
  float* row_m;         // [B][Hq][R][n_ksplit]
  float* row_l;
  float* score;         // [B][Hkv][T]
};

// query row q in [0, 64) of row block rb -> (head in group, row index)
__device__ __forceinline__ void qrow_map(const ScoreArgs& a, int rb, int q, int& gh, int64_t& i) {
  gh = q / a.rpb;
  i = (int64_t)rb * a.rpb + q % a.rpb;
}

// ---------------------------------------------------------------- pass 1
template <int D>
__global__ void __launch_bounds__(kT) rowstats_kernel(const ScoreArgs a) {
  constexpr int ROWB = D * 2, NC = D / 8, KC = D / 16, TILE = 64 * ROWB;
  extern __shared__ __align__(128) uint8_t smem[];   // [2][64 keys][D] swizzled
  const int ks = blockIdx.x, rb = blockIdx.y;
  const int64_t bh = blockIdx.z;
  const int b = (int)(bh / a.Hkv), kvh = (int)(bh % a.Hkv);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, r = lane & 3;

  // the CTA's rows: positions of its last valid row bound the causal key range
  const int64_t row_lo = (int64_t)rb * a.rpb;
  const int64_t row_hi = std::min<int64_t>(row_lo + a.rpb, a.R);   // exclusive
  const int64_t key_end_causal = a.pos0 + row_hi;                   // keys < this may be attended
  const int64_t k_begin = (int64_t)ks * a.tiles_per_split * 64;
  const int64_t k_end = std::min<int64_t>(std::min<int64_t>(k_begin + (int64_t)a.tiles_per_split * 64, a.T),
                                          key_end_causal);
  const int ntiles = k_end > k_begin ? (int)ceil_div_dev(k_end - k_begin, 64) : 0;

  // A fragments: query rows 16*warp + g and + 8
  uint32_t qa[KC][4];
  int64_t pos_row[2];
  bool valid_row[2];
  int gh_row[2];
  int64_t i_row[2];
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    const int q = 16 * warp + g + 8 * hh;
    qrow_map(a, rb, q, gh_row[hh], i_row[hh]);
    valid_row[hh] = gh_row[hh] < a.G && i_row[hh] < a.R;
    pos_row[hh] = a.pos0 + i_row[hh];
  }
#pragma unroll
  for (int kc = 0; kc < KC; ++kc) {
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      uint32_t lo = 0, hi = 0;
      if (valid_row[hh]) {
        const __half* qr = a.q + (((int64_t)b * a.Hq + (int64_t)kvh * a.G + gh_row[hh]) * a.R + i_row[hh]) * D;
        lo = *reinterpret_cast<const uint32_t*>(qr + kc * 16 + 2 * r);
        hi = *reinterpret_cast<const uint32_t*>(qr + kc * 16 + 2 * r + 8);
      }
      qa[kc][hh] = lo;        // a0 (row g) / a1 (row g+8)
      qa[kc][2 + hh] = hi;    // a2 / a3
    }
  }

  const __half* kbase = a.k + bh * a.T * D;
  auto load_tile = [&](int t, int stage) {
    uint8_t* Ks = smem + stage * TILE;
    const int col = tid % NC;
    for (int rr = tid / NC; rr < 64; rr += kT / NC) {
      const int64_t j = k_begin + (int64_t)t * 64 + rr;
      const bool ok = j < k_end;
      cp_async16(Ks + rr * ROWB + ((col ^ (rr & 7)) << 4), kbase + (ok ? j : 0) * D + col * 8, ok ? 16 : 0);
    }
  };

  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  if (ntiles > 0) load_tile(0, 0);
  cp_async_commit();
  for (int t = 0; t < ntiles; ++t) {
    cp_async_wait<0>();
    __syncthreads();
    if (t + 1 < ntiles) load_tile(t + 1, (t + 1) & 1);
    cp_async_commit();
    const uint8_t* Ks = smem + (t & 1) * TILE;
    float sc[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
    const int mi = lane >> 3, row = lane & 7;
#pragma unroll
    for (int kc = 0; kc < KC; ++kc) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {     // pairs of n-tiles (16 keys)
        uint32_t bk[4];
        const int tok = np * 16 + (mi >> 1) * 8 + row;
        const int ch = kc * 2 + (mi & 1);
        ldsm_x4(bk, Ks + tok * ROWB + ((ch ^ (tok & 7)) << 4));
        mma16816(sc[2 * np], qa[kc][0], qa[kc][1], qa[kc][2], qa[kc][3], bk[0], bk[1]);
        mma16816(sc[2 * np + 1], qa[kc][0], qa[kc][1], qa[kc][2], qa[kc][3], bk[2], bk[3]);
      }
    }
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      float mx = -INFINITY;
      float x[16];
#pragma unroll
      for (int n = 0; n < 8; ++n) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int64_t j = k_begin + (int64_t)t * 64 + n * 8 + 2 * r + e;
          const bool ok = valid_row[hh] && j < k_end && j <= pos_row[hh];
          const float v = ok ? sc[n][2 * hh + e] * a.scale_log2 : -INFINITY;
          x[n * 2 + e] = v;
          mx = fmaxf(mx, v);
        }
      }
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float m_new = fmaxf(m_run[hh], mx);
      if (m_new != -INFINITY) {
        float s = 0.f;
#pragma unroll
        for (int e = 0; e < 16; ++e) s += exp2f(x[e] - m_new);
        l_run[hh] = l_run[hh] * exp2f(m_run[hh] - m_new) + s;
        m_run[hh] = m_new;
      }
    }
  }
  cp_async_wait<0>();
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    float l = l_run[hh];
    l += __shfl_xor_sync(0xffffffffu, l, 1);
    l += __shfl_xor_sync(0xffffffffu, l, 2);
    if (r == 0 && valid_row[hh]) {
      const int64_t idx = (((int64_t)b * a.Hq + (int64_t)kvh * a.G + gh_row[hh]) * a.R + i_row[hh]) * a.n_ksplit + ks;
      a.row_m[idx] = m_run[hh];
      a.row_l[idx] = l;
    }
  }
}

// ---------------------------------------------------------------- pass 2
template <int D>
__global__ void __launch_bounds__(kT) colsum_kernel(const ScoreArgs a) {
  constexpr int ROWB = D * 2, NC = D / 8, KC = D / 16, TILE = 64 * ROWB;
  extern __shared__ __align__(128) uint8_t smem[];   // [2][64 query rows][D], then stats [2][64] (m, 1/l), pos
  float2* stats = reinterpret_cast<float2*>(smem + 2 * TILE);       // [2][64]
  int64_t* qpos = reinterpret_cast<int64_t*>(stats + 128);          // [2][64]
  const int kb = blockIdx.x;
  const int64_t bh = blockIdx.y;
  const int b = (int)(bh / a.Hkv), kvh = (int)(bh % a.Hkv);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, r = lane & 3;
  const int64_t j0 = (int64_t)kb * 64;
  if (j0 >= a.T) return;

  // A fragments: keys j0 + 16*warp + g (+8)
  uint32_t ka[KC][4];
  const __half* kbase = a.k + bh * a.T * D;
#pragma unroll
  for (int kc = 0; kc < KC; ++kc) {
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const int64_t j = j0 + 16 * warp + g + 8 * hh;
      uint32_t lo = 0, hi = 0;
      if (j < a.T) {
        lo = *reinterpret_cast<const uint32_t*>(kbase + j * D + kc * 16 + 2 * r);
        hi = *reinterpret_cast<const uint32_t*>(kbase + j * D + kc * 16 + 2 * r + 8);
      }
      ka[kc][hh] = lo;
      ka[kc][2 + hh] = hi;
    }
  }
  // query-row blocks whose rows can see key j0: rows i with pos0 + i >= j0
  const int64_t first_row = std::max<int64_t>(0, j0 - a.pos0);
  const int rb_begin = (int)(first_row / a.rpb);
  const int rb_end = (int)ceil_div_dev(a.R, a.rpb);
  const int nblk = rb_end - rb_begin;

  auto load_block = [&](int t, int stage) {
    const int rb = rb_begin + t;
    uint8_t* Qs = smem + stage * TILE;
    const int col = tid % NC;
    for (int q = tid / NC; q < 64; q += kT / NC) {
      int gh;
      int64_t i;
      qrow_map(a, rb, q, gh, i);
      const bool ok = gh < a.G && i < a.R;
      const __half* src = a.q + (((int64_t)b * a.Hq + (int64_t)kvh * a.G + (ok ? gh : 0)) * a.R + (ok ? i : 0)) * D;
      cp_async16(Qs + q * ROWB + ((col ^ (q & 7)) << 4), src + col * 8, ok ? 16 : 0);
    }
    if (tid < 64) {
      int gh;
      int64_t i;
      qrow_map(a, rb, tid, gh, i);
      float2 st = make_float2(INFINITY, 0.f);       // (m, 1/l); invalid row -> p = 0
      int64_t p = -1;
      if (gh < a.G && i < a.R) {
        const int64_t idx = (((int64_t)b * a.Hq + (int64_t)kvh * a.G + gh) * a.R + i) * a.n_ksplit;
        float M = -INFINITY;
        for (int s = 0; s < a.n_ksplit; ++s) M = fmaxf(M, a.row_m[idx + s]);
        float L = 0.f;
        for (int s = 0; s < a.n_ksplit; ++s) {
          const float ms = a.row_m[idx + s];
          if (ms != -INFINITY) L += a.row_l[idx + s] * exp2f(ms - M);
        }
        st = make_float2(M, L > 0.f ? 1.f / L : 0.f);
        p = a.pos0 + i;
      }
      stats[stage * 64 + tid] = st;
      qpos[stage * 64 + tid] = p;
    }
  };

  float col[2] = {0.f, 0.f};
  if (nblk > 0) load_block(0, 0);
  cp_async_commit();
  for (int t = 0; t < nblk; ++t) {
    cp_async_wait<0>();
    __syncthreads();
    if (t + 1 < nblk) load_block(t + 1, (t + 1) & 1);
    cp_async_commit();
    const uint8_t* Qs = smem + (t & 1) * TILE;
    const float2* st = stats + (t & 1) * 64;
    const int64_t* qp = qpos + (t & 1) * 64;
    float sc[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
    const int mi = lane >> 3, row = lane & 7;
#pragma unroll
    for (int kc = 0; kc < KC; ++kc) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        uint32_t bq[4];
        const int qq = np * 16 + (mi >> 1) * 8 + row;
        const int ch = kc * 2 + (mi & 1);
        ldsm_x4(bq, Qs + qq * ROWB + ((ch ^ (qq & 7)) << 4));
        mma16816(sc[2 * np], ka[kc][0], ka[kc][1], ka[kc][2], ka[kc][3], bq[0], bq[1]);
        mma16816(sc[2 * np + 1], ka[kc][0], ka[kc][1], ka[kc][2], ka[kc][3], bq[2], bq[3]);
      }
    }
#pragma unroll
    for (int n = 0; n < 8; ++n) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int q = n * 8 + 2 * r + e;
        const float2 s2 = st[q];
        const int64_t pq = qp[q];
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int64_t j = j0 + 16 * warp + g + 8 * hh;
          if (pq >= j) col[hh] += exp2f(sc[n][2 * hh + e] * a.scale_log2 - s2.x) * s2.y;
        }
      }
    }
  }
  cp_async_wait<0>();
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    float v = col[hh];
    v += __shfl_xor_sync(0xffffffffu, v, 1);
    v += __shfl_xor_sync(0xffffffffu, v, 2);
    const int64_t j = j0 + 16 * warp + g + 8 * hh;
    if (r == 0 && j < a.T) a.score[bh * a.T + j] = v;
  }
}

template <int D>
cudaError_t launch_scores_t(const ScoreArgs& a, int rowblocks, int units, int keyblocks, cudaStream_t st) {
  const size_t smem1 = 2 * 64 * D * 2;
  const size_t smem2 = 2 * 64 * D * 2 + 128 * sizeof(float2) + 128 * sizeof(int64_t);
  cudaError_t e = cudaFuncSetAttribute(rowstats_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(colsum_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
  if (e != cudaSuccess) return e;
  rowstats_kernel<D><<<dim3(a.n_ksplit, rowblocks, units), kT, smem1, st>>>(a);
  e = cudaPeekAtLastError();
  if (e != cudaSuccess) return e;
  colsum_kernel<D><<<dim3(keyblocks, units), kT, smem2, st>>>(a);
  return cudaPeekAtLastError();
}

}  // namespace

cudaError_t launch_prefill_scores(const mkv_config& c, const void* q, int64_t q_rows, int64_t T,
                                  const void* full_k, const PrefillWs& ws, cudaStream_t st) {
  ScoreArgs a{};
  a.q = static_cast<const __half*>(q);
  a.k = static_cast<const __half*>(full_k);
  a.R = q_rows;
  a.T = T;
  a.pos0 = T - q_rows;
  a.Hq = c.Hq;
  a.Hkv = c.Hkv;
  a.G = c.Hq / c.Hkv;
  a.rpb = 64 / a.G;
  const float scale = c.softmax_scale > 0.f ? c.softmax_scale : 1.0f / sqrtf((float)c.D);
  a.scale_log2 = scale * kLog2e;
  const int units = c.B * c.Hkv;
  const int rowblocks = (int)ceil_div(q_rows, a.rpb);
  const int64_t tiles = ceil_div(T, 64);
  // split the key range only when there are few row blocks (observation window)
  int64_t ns = std::max<int64_t>(1, ceil_div(4 * kNumSMs, (int64_t)rowblocks * units));
  ns = std::min<int64_t>(ns, std::min<int64_t>(tiles, T / std::max<int64_t>(q_rows, 1)));
  ns = std::max<int64_t>(ns, 1);
  a.tiles_per_split = (int)ceil_div(tiles, ns);
  a.n_ksplit = (int)ceil_div(tiles, a.tiles_per_split);
  a.row_m = ws.row_m;
  a.row_l = ws.row_l;
  a.score = ws.score;
  const int keyblocks = (int)tiles;
  if (c.D == 128) return launch_scores_t<128>(a, rowblocks, units, keyblocks, st);
  return launch_scores_t<64>(a, rowblocks, units, keyblocks, st);
}

}  // namespace mkv
