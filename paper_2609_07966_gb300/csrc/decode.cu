// Decode attention over an fp16 cache: FP16 (all slots), H2O (kept slots,
// with per-slot logits for the score update) and the RocketKV sparse stage
// (selected pages + tail page).  Section 2.1 of the paper; the operation is
//   out_h = sum_t softmax_t(scale q_h . k_t) v_t  over the attended set.
//
// Design (GB300, HBM-bound): one CTA per (batch, kv-head, split) holds all G
// query heads of the group, so every K/V byte is read once.  K and V rows are
// staged by cp.async into XOR-swizzled shared tiles (3-stage pipeline of 64
// tokens), and each warp multiplies its 16 tokens with one m16n8k16 tensor-
// core product per 16 dims (G query rows padded to 16): the contraction costs
// ~5 warp instructions per token, leaving the issue slots to the copies.
// Online softmax runs in the log2 domain on the accumulator fragments; splits
// are merged by the last CTA of each (batch, kv-head) (mkv_merge.cuh).
// mkv_decode_step appends the step's token in the same launch (FP16, H2O).
#include <math.h>

#include <algorithm>

#include <mutex>

#include "mkv_common.cuh"
#include "mkv_internal.h"
#include "mkv_merge.cuh"

namespace mkv {

namespace {

__device__ uint32_t g_status_decode;   // MKV_FLAG_* bits raised by the step's append

constexpr int kStages = 3;
constexpr int kThreads = 128;   // 4 warps x 16 tokens = one 64-token chunk

struct Fp16Args {
  const __half* q;        // [B][Hq][D]
  const __half* k;        // [B][Hkv][T_cap][D]
  const __half* v;
  const int32_t* T_len;   // [B]
  const int32_t* pos;     // H2O [B][Hkv][T_cap]
  const int32_t* page_idx;// ROCKET [B][Hkv][kp]
  int64_t T_cap;
  int64_t n_slots;         // H2O: slots a unit can hold, min(T_cap, H + R + 1)
  int Hq, Hkv, G;
  int chunks_per_split;
  int kp;
  float scale_log2;
  float* part_m;
  float* part_l;
  float* part_o;
  float* logits;          // H2O [B][Hkv][T_cap][G]
  int n_split;
  MergeArgs merge;
  // mkv_decode_step (FP16, H2O): the step's token, appended by this launch (k_new NULL: no append)
  const __half* k_new;    // [B][Hkv][D]
  const __half* v_new;
  __half* k_w;            // the cache rows it is written into
  __half* v_w;
  int32_t* T_len_w;
  int32_t* pos_w;         // H2O: its position and a zero score go to its slot
  float* acc_w;
  const int32_t* slot;    // H2O [B][Hkv]: the slot the token takes
};

constexpr int kMaxSplitPages = 1024;   // ROCKET: page ids of one split, staged in shared memory

// Virtual token v of (b, kv-head) -> cache slot to load, or -1 when nothing is loaded.
// H2O loads every slot and masks it later by its staged position.
template <int MODE>
__device__ __forceinline__ int64_t slot_of(const Fp16Args& a, int64_t v, int n_len, int ns, const int32_t* pages,
                                           int unit0) {
  if (MODE == 0) {                       // FP16: slots 0..T_len-1
    return v < n_len ? v : -1;
  } else if (MODE == 1) {                // H2O: every slot (masked by pos afterwards)
    return v < a.T_cap ? v : -1;
  } else {                               // ROCKET: selected pages, then the tail page
    const int unit = (int)(v / kPage), within = (int)(v % kPage);
    if (unit < a.kp) {
      const int p = pages[unit - unit0];
      return p >= 0 ? (int64_t)p * kPage + within : -1;
    }
    if (unit == a.kp) {
      const int64_t s = (int64_t)ns * kPage + within;
      return s < n_len ? s : -1;
    }
    return -1;
  }
}

template <int D, int MODE>
__global__ void __launch_bounds__(kThreads, 2) decode_fp16_kernel(const Fp16Args a) {
  pdl_wait_and_trigger();
  constexpr int ROWB = D * 2;           // bytes per token row
  constexpr int NC = D / 8;             // 16-byte chunks per row
  constexpr int TILE = kChunk * ROWB;   // one K (or V) tile
  constexpr int KC = D / 16;            // k16 steps of the QK product
  constexpr int ROWS_PER_PASS = kThreads / NC;
  extern __shared__ __align__(128) uint8_t smem[];
  int32_t* slotmap = reinterpret_cast<int32_t*>(smem + kStages * 2 * TILE);   // [kStages][kChunk]
  int32_t* pages = slotmap + kStages * kChunk;                                 // ROCKET [kMaxSplitPages]

  const int split = blockIdx.x;
  const int64_t bh = blockIdx.y;
  const int b = (int)(bh / a.Hkv), kvh = (int)(bh % a.Hkv);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, r = lane & 3;

  // The step's token (mkv_decode_step).  Every CTA takes the cache as holding it: FP16 T_len + 1
  // tokens, H2O the token at position T_len in slot[bh].  The CTA whose range holds its slot writes
  // the row from k_new / v_new (H2O: with its position and a zero score) into the cache before it
  // stages anything; the last CTA of the batch entry stores the new length (meanwhile the top 8 bits of
  // T_len count the finished CTAs, masked off here).  A batch entry with no room (FP16: a full
  // cache; H2O: a slot outside the cache) keeps its length, as mkv_append_kv does.
  const bool step = MODE != 2 && a.k_new != nullptr;
  int t_old = 0;
  bool ok_b = true;
  int64_t s_new = -1;                  // this unit's slot of the new token (-1: none)
  if (step) {
    t_old = a.T_len[b] & 0xffffff;
    if (MODE == 0) {
      ok_b = t_old < a.T_cap;
      s_new = ok_b ? t_old : -1;
    } else {
      for (int h = 0; h < a.Hkv; ++h) {
        const int sh = a.slot[(int64_t)b * a.Hkv + h];
        ok_b = ok_b && sh >= 0 && sh < a.T_cap;
      }
      const int sh = a.slot[bh];
      s_new = ok_b ? sh : -1;          // all or nothing per batch entry, as mkv_append_kv
    }
  }

  int n_len = 0, ns = 0;
  int64_t v_total;
  if (MODE == 0) {
    n_len = step ? (int)min((int64_t)t_old + (ok_b ? 1 : 0), a.T_cap) : (int)min((int64_t)a.T_len[b], a.T_cap);
    v_total = n_len;
  } else if (MODE == 1) {
    v_total = a.n_slots;                 // slots past H + R are never used (H2O slot policy)
  } else {
    n_len = (int)min((int64_t)a.T_len[b], a.T_cap);
    ns = n_len > 0 ? (n_len - 1) / kPage : 0;
    v_total = (int64_t)(a.kp + 1) * kPage;
  }
  const int64_t v_begin = (int64_t)split * a.chunks_per_split * kChunk;
  int64_t v_end = v_begin + (int64_t)a.chunks_per_split * kChunk;
  if (v_end > v_total) v_end = v_total;
  const int nchunks = v_end > v_begin ? (int)ceil_div_dev(v_end - v_begin, kChunk) : 0;

  const __half* kbase = a.k + bh * a.T_cap * D;
  const __half* vbase = a.v + bh * a.T_cap * D;
  const int unit0 = (int)(v_begin / kPage);
  // The CTA holding the new token's slot writes its row (H2O: and position) before anything is
  // staged, fenced, so that the chunk copies below read it like any other row.
  if (step && s_new >= v_begin && s_new < v_end) {
    constexpr int NC16 = D / 8;
    if (tid < NC16) {
      reinterpret_cast<uint4*>(a.k_w + (bh * a.T_cap + s_new) * D)[tid] =
          reinterpret_cast<const uint4*>(a.k_new + bh * D)[tid];
    } else if (tid < 2 * NC16) {
      reinterpret_cast<uint4*>(a.v_w + (bh * a.T_cap + s_new) * D)[tid - NC16] =
          reinterpret_cast<const uint4*>(a.v_new + bh * D)[tid - NC16];
    } else if (MODE == 1 && tid == 2 * NC16) {
      a.pos_w[bh * a.T_cap + s_new] = t_old;
      a.acc_w[bh * a.T_cap + s_new] = 0.f;
    }
    __threadfence();
  }
  if (step) {
    if (!ok_b && split == 0 && kvh == 0 && tid == 0) atomicOr(&g_status_decode, MKV_FLAG_CACHE_FULL);
    __syncthreads();
  }
  if (MODE == 2) {                       // this split's page ids, read once
    int64_t nu64 = ceil_div_dev(v_end, kPage) - unit0;
    if (nu64 > kMaxSplitPages) nu64 = kMaxSplitPages;
    const int nu = (int)nu64;
    for (int u = tid; u < nu; u += kThreads) {
      const int unit = unit0 + u;
      pages[u] = unit < a.kp ? a.page_idx[bh * a.kp + unit] : -1;
    }
    __syncthreads();
  }

  // slotmap holds, per row of a stage: the loaded slot (-1: none), or for H2O the slot's
  // position (-1: empty), staged by cp.async so no load waits on it
  auto load_chunk = [&](int c, int stage) {
    uint8_t* Ks = smem + stage * 2 * TILE;
    uint8_t* Vs = Ks + TILE;
    const int col = tid % NC;
    for (int rr = tid / NC; rr < kChunk; rr += ROWS_PER_PASS) {
      const int64_t v = v_begin + (int64_t)c * kChunk + rr;
      const int64_t s = v < v_end ? slot_of<MODE>(a, v, n_len, ns, pages, unit0) : -1;
      const int64_t ss = s >= 0 ? s : 0;
      const int off = rr * ROWB + ((col ^ (rr & 7)) << 4);
      cp_async16(Ks + off, kbase + ss * D + col * 8, s >= 0 ? 16 : 0);
      cp_async16(Vs + off, vbase + ss * D + col * 8, s >= 0 ? 16 : 0);
      if (col == 0) {
        if (MODE == 1 && s >= 0) {
          cp_async4(&slotmap[stage * kChunk + rr], a.pos + bh * a.T_cap + s, 4);
        } else {
          slotmap[stage * kChunk + rr] = (int32_t)s;
        }
      }
    }
  };

  // query fragments: row g of the 16-row A operand is query head kvh*G + g
  uint32_t qa0[KC], qa2[KC];
  {
    const bool real = g < a.G;
    const __half* qrow = a.q + ((int64_t)b * a.Hq + (int64_t)kvh * a.G + (real ? g : 0)) * D;
#pragma unroll
    for (int kc = 0; kc < KC; ++kc) {
      qa0[kc] = real ? *reinterpret_cast<const uint32_t*>(qrow + kc * 16 + 2 * r) : 0u;
      qa2[kc] = real ? *reinterpret_cast<const uint32_t*>(qrow + kc * 16 + 2 * r + 8) : 0u;
    }
  }

  float o[D / 8][2];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = 0.f;
  float m_run = -INFINITY, l_part = 0.f;

#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    if (s < nchunks) load_chunk(s, s);
    cp_async_commit();
  }

  for (int c = 0; c < nchunks; ++c) {
    cp_async_wait<kStages - 2>();
    __syncthreads();
    {
      const int nc = c + kStages - 1;
      if (nc < nchunks) load_chunk(nc, nc % kStages);
      cp_async_commit();
    }
    const int stage = c % kStages;
    const uint8_t* Ks = smem + stage * 2 * TILE;
    const uint8_t* Vs = Ks + TILE;
    const int32_t* smap = slotmap + stage * kChunk;
    const int t0 = warp * 16;

    float sc[2][4];
#pragma unroll
    for (int i = 0; i < 4; ++i) sc[0][i] = sc[1][i] = 0.f;
    {
      const int mi = lane >> 3, row = lane & 7;
      const int tok = t0 + (mi >> 1) * 8 + row;
      const uint8_t* rowp = Ks + tok * ROWB;
#pragma unroll
      for (int kc = 0; kc < KC; ++kc) {
        uint32_t bk[4];
        const int ch = kc * 2 + (mi & 1);
        ldsm_x4(bk, rowp + ((ch ^ (tok & 7)) << 4));
        mma16816(sc[0], qa0[kc], 0u, qa2[kc], 0u, bk[0], bk[1]);
        mma16816(sc[1], qa0[kc], 0u, qa2[kc], 0u, bk[2], bk[3]);
      }
    }
    // tokens of this lane's four scores
    const int tk[4] = {t0 + 2 * r, t0 + 2 * r + 1, t0 + 8 + 2 * r, t0 + 9 + 2 * r};
    float x[4] = {sc[0][0], sc[0][1], sc[1][0], sc[1][1]};
    float mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int32_t s = smap[tk[i]];
      x[i] = s >= 0 ? x[i] * a.scale_log2 : -INFINITY;
      if (MODE == 1 && g < a.G && s >= 0) {
        const int64_t slot = v_begin + (int64_t)c * kChunk + tk[i];
        a.logits[(bh * a.T_cap + slot) * a.G + g] = x[i];
      }
      mx = fmaxf(mx, x[i]);
    }
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
    const float m_new = fmaxf(m_run, mx);
    float p[4];
    float alpha = 1.f;
    if (m_new == -INFINITY) {
      p[0] = p[1] = p[2] = p[3] = 0.f;
    } else {
      alpha = exp2f(m_run - m_new);
#pragma unroll
      for (int i = 0; i < 4; ++i) p[i] = exp2f(x[i] - m_new);
    }
    l_part = l_part * alpha + (p[0] + p[1]) + (p[2] + p[3]);
    m_run = m_new;
    if (__any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll
      for (int i = 0; i < D / 8; ++i) {
        o[i][0] *= alpha;
        o[i][1] *= alpha;
      }
    }
    const uint32_t pa0 = pack_half2(p[0], p[1]);
    const uint32_t pa2 = pack_half2(p[2], p[3]);
    {
      const int mi = lane >> 3, row = lane & 7;
      const int tok = t0 + (mi & 1) * 8 + row;
      const uint8_t* rowp = Vs + tok * ROWB;
#pragma unroll
      for (int j = 0; j < D / 16; ++j) {
        uint32_t bv[4];
        const int ch = 2 * j + (mi >> 1);
        ldsm_x4_t(bv, rowp + ((ch ^ (tok & 7)) << 4));
        float d0[4] = {o[2 * j][0], o[2 * j][1], 0.f, 0.f};
        float d1[4] = {o[2 * j + 1][0], o[2 * j + 1][1], 0.f, 0.f};
        mma16816(d0, pa0, 0u, pa2, 0u, bv[0], bv[1]);
        mma16816(d1, pa0, 0u, pa2, 0u, bv[2], bv[3]);
        o[2 * j][0] = d0[0];
        o[2 * j][1] = d0[1];
        o[2 * j + 1][0] = d1[0];
        o[2 * j + 1][1] = d1[1];
      }
    }
  }
  cp_async_wait<0>();
  __syncthreads();

  // merge the four warps' (m, l, o) of each query row, then write the split partial
  l_part += __shfl_xor_sync(0xffffffffu, l_part, 1);
  l_part += __shfl_xor_sync(0xffffffffu, l_part, 2);
  float* wm = reinterpret_cast<float*>(smem);          // [4][8]
  float* wl = wm + 32;                                 // [4][8]
  float* wo = wl + 32;                                 // [4][8][D]
  if (g < a.G) {
    if (r == 0) {
      wm[warp * 8 + g] = m_run;
      wl[warp * 8 + g] = l_part;
    }
#pragma unroll
    for (int i = 0; i < D / 8; ++i) {
      wo[(warp * 8 + g) * D + i * 8 + 2 * r] = o[i][0];
      wo[(warp * 8 + g) * D + i * 8 + 2 * r + 1] = o[i][1];
    }
  }
  __syncthreads();
  for (int e = tid; e < a.G * D; e += kThreads) {
    const int row = e / D, d = e % D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, wm[w * 8 + row]);
    float L = 0.f, O = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const float f = exp2f(wm[w * 8 + row] - M);
        L += wl[w * 8 + row] * f;
        O += wo[(w * 8 + row) * D + d] * f;
      }
    }
    const int64_t hq = (int64_t)b * a.Hq + (int64_t)kvh * a.G + row;
    const int64_t pi = hq * a.n_split + split;
    a.part_o[pi * D + d] = O;
    if (d == 0) {
      a.part_m[pi] = M;
      a.part_l[pi] = L;
    }
  }
  __syncthreads();                     // the stage buffers now serve as the merge's scratch
  if (step && tid == 0) {              // every thread of this CTA read T_len before this point
    const unsigned old = atomicAdd(reinterpret_cast<unsigned*>(a.T_len_w) + b, 1u << 24);
    if ((int)(old >> 24) == a.Hkv * (int)gridDim.x - 1) a.T_len_w[b] = ok_b ? t_old + 1 : t_old;
  }
  merge_if_last<D, kThreads>(a.merge, bh, b, kvh, reinterpret_cast<float*>(smem), kStages * 2 * TILE / 4);
}

template <int D, int MODE>
cudaError_t launch_fp16_t(const Fp16Args& a, int n_units, int n_split, cudaStream_t st) {
  constexpr int TILE = kChunk * D * 2;
  const size_t smem = (size_t)kStages * 2 * TILE + (kStages * kChunk + kMaxSplitPages) * sizeof(int32_t);
  cudaError_t e = cudaFuncSetAttribute(decode_fp16_kernel<D, MODE>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(n_split, n_units);
  return launch_pdl(decode_fp16_kernel<D, MODE>, grid, dim3(kThreads), smem, st, a);
}

}  // namespace

MergeArgs merge_args(const mkv_config& c, const DecodeWs& ws, const Split& sp, void* out, bool h2o_stats) {
  MergeArgs m{};
  m.part_m = ws.part_m;
  m.part_l = ws.part_l;
  m.part_o = ws.part_o;
  m.counters = ws.counters;
  m.out = static_cast<__half*>(out);
  m.m_tot = h2o_stats ? ws.m_tot : nullptr;
  m.l_tot = h2o_stats ? ws.l_tot : nullptr;
  m.Hq = c.Hq;
  m.G = c.Hq / c.Hkv;
  m.n_split = sp.n_split;
  return m;
}

cudaError_t take_status_decode(uint32_t* flags, cudaStream_t st) {
  uint32_t v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbolAsync(&v, g_status_decode, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyToSymbolAsync(g_status_decode, &zero, sizeof(zero), 0, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  *flags |= v;
  return e;
}

cudaError_t launch_decode_fp16_family(const mkv_config& c, const void* q, const mkv_cache& cache,
                                      const int32_t* page_idx, void* out, const DecodeWs& ws,
                                      const Split& sp, cudaStream_t st, const void* k_new, const void* v_new) {
  Fp16Args a{};
  a.k_new = static_cast<const __half*>(k_new);
  a.v_new = static_cast<const __half*>(v_new);
  a.k_w = static_cast<__half*>(cache.k);
  a.v_w = static_cast<__half*>(cache.v);
  a.T_len_w = cache.T_len;
  a.pos_w = cache.pos;
  a.acc_w = cache.acc;
  a.slot = cache.slot;
  a.q = static_cast<const __half*>(q);
  a.k = static_cast<const __half*>(cache.k);
  a.v = static_cast<const __half*>(cache.v);
  a.T_len = cache.T_len;
  a.pos = cache.pos;
  a.page_idx = page_idx;
  a.T_cap = cache.T_cap;
  // H2O: the prefill keeps at most H + R tokens in slots 0.., and each step's token goes to the
  // lowest free slot or to the slot its eviction freed, so no slot past H + R is ever used
  a.n_slots = std::min<int64_t>(cache.T_cap, (int64_t)c.h2o_heavy + c.h2o_recent + 1);
  a.Hq = c.Hq;
  a.Hkv = c.Hkv;
  a.G = c.Hq / c.Hkv;
  a.chunks_per_split = sp.chunks_per_split;
  a.kp = c.topk_pages;
  const float scale = c.softmax_scale > 0.f ? c.softmax_scale : 1.0f / sqrtf((float)c.D);
  a.scale_log2 = scale * kLog2e;
  a.part_m = ws.part_m;
  a.part_l = ws.part_l;
  a.part_o = ws.part_o;
  a.logits = ws.logits;
  a.n_split = sp.n_split;
  a.merge = merge_args(c, ws, sp, out, c.method == MKV_H2O);
  const int units = c.B * c.Hkv;
  const int mode = c.method == MKV_H2O ? 1 : (c.method == MKV_ROCKET ? 2 : 0);
  if (c.D == 128) {
    if (mode == 0) return launch_fp16_t<128, 0>(a, units, sp.n_split, st);
    if (mode == 1) return launch_fp16_t<128, 1>(a, units, sp.n_split, st);
    return launch_fp16_t<128, 2>(a, units, sp.n_split, st);
  }
  if (mode == 0) return launch_fp16_t<64, 0>(a, units, sp.n_split, st);
  if (mode == 1) return launch_fp16_t<64, 1>(a, units, sp.n_split, st);
  return launch_fp16_t<64, 2>(a, units, sp.n_split, st);
}


// ---------------------------------------------------------------------------
// FP16 decode without a caller workspace (mkv_decode_attention_noalloc).
//
// The split partials normally live in the caller's `ws`.  Here they live in a
// fixed array compiled into this library, one copy per GPU that loads it, so a
// caller that cannot allocate device memory can still decode.  Host code must
// not hand the array's host-side name to a kernel: the device address is
// looked up once per device with cudaGetSymbolAddress and cached.
constexpr size_t kNoAllocScratchBytes = size_t(8) << 20;   // 8 MiB per GPU
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

namespace {
std::mutex g_noalloc_mu;
constexpr int kMaxDevices = 128;
void* g_noalloc_addr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device (looked up once).
cudaError_t noalloc_scratch(void** addr) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (g_noalloc_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_noalloc_addr[dev] = p;
  }
  *addr = g_noalloc_addr[dev];
  return cudaSuccess;
}
}  // namespace

}  // namespace mkv

extern "C" mkv_status mkv_decode_attention_noalloc(const mkv_config* cfg, const void* q, const mkv_cache* cache,
                                                   void* out, void* stream) {
  using namespace mkv;
  const mkv_status st0 = check_fp16_decode_args(cfg, cache, q, out);
  if (st0 != MKV_OK) return st0;
  const DecodeWs need = decode_ws(*cfg, cache->T_cap, nullptr);
  if (need.bytes > kNoAllocScratchBytes) {
    set_error("this call needs %zu bytes of scratch; the built-in array holds %zu (use mkv_decode_attention "
              "with a workspace)", need.bytes, kNoAllocScratchBytes);
    return MKV_ERR_WORKSPACE;
  }
  void* scratch = nullptr;
  cudaError_t e = noalloc_scratch(&scratch);
  if (e != cudaSuccess) {
    set_error("cudaGetSymbolAddress of the built-in scratch: %s", cudaGetErrorString(e));
    return MKV_ERR_CUDA;
  }
  const DecodeWs w = decode_ws(*cfg, cache->T_cap, scratch);
  const Split sp = decode_split(*cfg, cache->T_cap);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  e = launch_decode_fp16_family(*cfg, q, *cache, nullptr, out, w, sp, st);
  if (e != cudaSuccess) {
    set_error("decode launch: %s", cudaGetErrorString(e));
    return MKV_ERR_CUDA;
  }
  return MKV_OK;
}
