// Fused RocketKV decode (Section 2.1, RocketKV paragraph, stage 2): the page choice and the
// sparse exact attention of one decode step in a single launch.
//
// One thread-block cluster of kCl CTAs per (batch, kv-head):
//  1. each CTA chooses the top-r_d dims of sum_h |q_h,i| (redundantly, it is 128 keys) and
//     scores its 1/kCl share of the candidate pages (the full pages before the newest token's
//     page): score_p = sum_t (kmax_t,p P_t + kmin_t,p N_t) over the chosen dims t, where
//     P_t / N_t are the group's positive / negative query parts (max(q kmin, q kmax) is q kmax
//     for q >= 0, q kmin otherwise, since kmin <= kmax).  Only the chosen dims' bounds are
//     read: they are copied once the dims are known, while the newest page is being staged;
//  2. every score is stored into every CTA of the cluster (distributed shared memory), then a
//     cluster barrier;
//  3. each CTA ranks its own pages against all scores (score desc, page asc), stores their
//     kept flags into every CTA, and after a cluster barrier every CTA lists the kept pages in
//     ascending order; the newest token's partial page is always attended;
//  4. the attended pages are dealt round-robin over the cluster's 64 warps; a warp stages its
//     page's 16 K and V rows by cp.async and runs the tensor-core QK^T, softmax and PV of the
//     group's query heads on them (16 tokens = one mma slab);
//  5. the CTA merges its warps' partials (m, l, o), stores its partial into CTA 0 (distributed
//     shared memory), and after a cluster barrier CTA 0 merges the kCl partials and writes
//     the output.
// No workspace, no global round trip of scores, page ids or partials.
//
// With k_new / v_new (mkv_rocket_step) the launch also appends the step's token first, as
// mkv_append_kv does: every CTA takes the length as T_len + 1, the warp that stages the newest
// page takes the new row from the input and writes it into the cache, completes the page's
// per-dim min/max when the row fills it, and the last CTA of the batch entry to finish stores
// the new length.  During the launch the top 8 bits of T_len[b] count the finished CTAs of
// batch entry b (every reader masks them off); the last one writes the clean length.
#include <math.h>

#include "mkv_common.cuh"
#include "mkv_internal.h"
#include "mkv_select.cuh"

namespace mkv {

__device__ uint32_t g_status_rocket;   // MKV_FLAG_* bits raised by this unit

namespace {

constexpr int kCl = kRocketCluster;  // CTAs per (batch, kv-head)
constexpr int kRfWarps = 8;
constexpr int kRfThreads = kRfWarps * 32;
constexpr int kRfSlices = 8;        // dim slices of the page scoring
static_assert(kCl == 8, "the eight lanes that rank a page store its flag into the eight CTAs");

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
  return r;
}
// every thread of every CTA of the cluster; orders the cluster's shared-memory accesses
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;\n" ::: "memory");
}
// the address of a shared variable of this CTA in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t cluster_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(smem_addr(p)), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_cluster(uint32_t a, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;\n" ::"r"(a), "f"(v) : "memory");
}
__device__ __forceinline__ void st_cluster_u8(uint32_t a, uint32_t v) {
  asm volatile("st.shared::cluster.u8 [%0], %1;\n" ::"r"(a), "r"(v) : "memory");
}

template <int D>
__device__ __forceinline__ int tile_off(int row, int ch) {
  return row * D * 2 + ((ch ^ (row & 7)) << 4);
}

__host__ __device__ constexpr int a16(int x) { return (x + 15) & ~15; }

// Shared-memory layout (bytes); every region 16-byte aligned.  `rs` = halves per bounds row.
struct RfLayout {
  int qs, sc, kf, part, sel, bounds, pages, wpart, cpart, tail, bytes;
  __host__ __device__ RfLayout(int D, int G, int64_t npc, int kp, int rs) {
    qs = 0;                                              // float [G][D]
    sc = a16(qs + G * D * 4);                            // float [npc rounded to 4] page scores
    kf = a16(sc + (int)((npc + 3) & ~3ll) * 4);          // u8 [npc] kept flags
    part = a16(kf + (int)npc);                           // float [kRfSlices][sp] partial scores
    sel = a16(part + kRfSlices * (int)((npc + kCl - 1) / kCl) * 4);   // int [kp + 1] attended pages
    bounds = a16(sel + (kp + 1) * 4);                    // half [2][D][rs] (later: cluster partials)
    const int cp_bytes = kCl * G * (D + 2) * 4;          // CTA 0: float [kCl][G][D + 2]
    pages = a16(bounds + (2 * D * rs * 2 > cp_bytes ? 2 * D * rs * 2 : cp_bytes));
    wpart = pages;                                       // after the attention: warps' partials
    cpart = bounds;
    bytes = pages + kRfWarps * 2 * kPage * D * 2;        // per warp: K and V tiles of one page
    if (wpart + kRfWarps * G * (D + 2) * 4 > bytes) bytes = wpart + kRfWarps * G * (D + 2) * 4;
    tail = a16(bytes);                                   // K and V tiles of the newest token's page
    bytes = tail + 2 * kPage * D * 2;
  }
};

struct RfArgs {
  const __half* q;          // [B][Hq][D]
  __half* k;                // [B][Hkv][T_cap][D]
  __half* v;
  __half* kmin;             // [B][Hkv][D][npc]
  __half* kmax;
  int32_t* T_len;           // low 24 bits: length; top 8: finished CTAs during an appending launch
  const __half* k_new;      // [B][Hkv][D], or null: no append
  const __half* v_new;
  int64_t T_cap, npc;
  int Hq, Hkv, G, kp, rd, rs;
  float scale_log2;
  int32_t* page_idx;        // optional [B][Hkv][kp]
  __half* out;              // [B][Hq][D]
};

template <int D>
__global__ void __cluster_dims__(kCl, 1, 1) __launch_bounds__(kRfThreads, 2) rocket_fused_kernel(const RfArgs a) {
  constexpr int KC = D / 16;
  extern __shared__ __align__(16) uint8_t smem[];
  const int G = a.G;
  const RfLayout L(D, G, a.npc, a.kp, a.rs);
  float* qs = reinterpret_cast<float*>(smem + L.qs);
  float* sc = reinterpret_cast<float*>(smem + L.sc);
  float* part = reinterpret_cast<float*>(smem + L.part);
  uint8_t* kf = smem + L.kf;
  int* sel = reinterpret_cast<int*>(smem + L.sel);
  __half* bmn = reinterpret_cast<__half*>(smem + L.bounds);
  __half* bmx = bmn + D * a.rs;
  __shared__ int warp_sums[32];
  __shared__ int dims[128];
  __shared__ __align__(16) float a_dim[128];
  __shared__ float pn[2][128];
  __shared__ uint32_t qh2[8][64 + 4];   // query as fp16 pairs, rows padded: conflict-free fragments

  const int rank = (int)cluster_rank();
  const int64_t bh = blockIdx.y;
  const int b = (int)(bh / a.Hkv), kvh = (int)(bh % a.Hkv);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // this CTA's share of the pages, fixed by the capacity so the prefetch need not wait for T_len
  const int sp = (int)((a.npc + kCl - 1) / kCl);        // pages per CTA
  const int p0 = min((int)a.npc, rank * sp), npf = min((int)a.npc, p0 + sp) - p0;

  // the group's query (fp16) and the cache length, loaded before the prefetch is issued
  constexpr int kQW = (8 * D / 2 + kRfThreads - 1) / kRfThreads;   // query words per thread (G <= 8)
  const uint32_t* qg = reinterpret_cast<const uint32_t*>(a.q + ((int64_t)b * a.Hq + (int64_t)kvh * G) * D);
  uint32_t qw[kQW];
#pragma unroll
  for (int k = 0; k < kQW; ++k) {
    const int e = tid + k * kRfThreads;
    qw[k] = e < G * (D / 2) ? __ldg(qg + e) : 0u;
  }
  const bool append = a.k_new != nullptr;
  const int n_old = (int)min((int64_t)(a.T_len[b] & 0xffffff), a.T_cap);
  const bool room = append && (int64_t)n_old + 1 <= a.T_cap;
  const int n = room ? n_old + 1 : n_old;              // the step's token included
  // the newest token's page, always attended, is staged now by the warp that attends to it
  const int ns = n > 0 ? (n - 1) / kPage : 0;          // candidate (full) pages; page ns is the newest
  const bool tail_warp = rank == kCl - 1 && warp == kRfWarps - 1 && n > 0;
  const int tail_valid = n - ns * kPage;               // 1 .. 16 rows
  uint8_t* tk = smem + L.tail;
  uint8_t* tv = tk + kPage * D * 2;
  if (tail_warp) {
    const __half* kb = a.k + (bh * a.T_cap + (int64_t)ns * kPage) * D;
    const __half* vb = a.v + (bh * a.T_cap + (int64_t)ns * kPage) * D;
    const int new_row = room ? tail_valid - 1 : kPage;  // the appended token's row (from the input)
    for (int e = lane; e < 2 * kPage * (D / 8); e += 32) {
      const int kv = e / (kPage * (D / 8)), rem = e % (kPage * (D / 8));
      const int row = rem / (D / 8), ch = rem % (D / 8);
      const bool ok = row < tail_valid;
      const __half* src = row == new_row ? (kv ? a.v_new : a.k_new) + bh * D + ch * 8
                                         : (kv ? vb : kb) + (ok ? row : 0) * D + ch * 8;
      cp_async16((kv ? tv : tk) + tile_off<D>(row, ch), src, ok ? 16 : 0);
    }
    if (room) {                                        // the new row into the cache
      for (int e = lane; e < 2 * (D / 8); e += 32) {
        const int kv = e / (D / 8), ch = e % (D / 8);
        const uint4 x = __ldg(reinterpret_cast<const uint4*>((kv ? a.v_new : a.k_new) + bh * D) + ch);
        reinterpret_cast<uint4*>((kv ? a.v : a.k) + (bh * a.T_cap + (int64_t)n_old) * D)[ch] = x;
      }
    }
  }
  cp_async_commit();
  const int np = max(0, min(ns, p0 + sp) - p0);        // of them, this CTA's
#pragma unroll
  for (int k = 0; k < kQW; ++k) {
    const int e = tid + k * kRfThreads;
    if (e < G * (D / 2)) {
      const int row = e / (D / 2), w = e % (D / 2);
      qh2[row][w] = qw[k];
      const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&qw[k]));
      qs[row * D + 2 * w] = f.x;
      qs[row * D + 2 * w + 1] = f.y;
    }
  }
  __syncthreads();
  if (tid < D) {
    float s = 0.f;
    for (int h = 0; h < G; ++h) s += fabsf(qs[h * D + tid]);
    a_dim[tid] = s;
  }
  __syncthreads();
  {                                                    // rank under (sum |q| desc, dim asc)
    const int i = tid >> 1, half = tid & 1;            // two threads per dim, half the dims each
    int rk = 0;
    if (i < D) {
      const float ai = a_dim[i];
#pragma unroll 4
      for (int j = half * (D / 2); j < (half + 1) * (D / 2); j += 4) {
        const float4 v = *reinterpret_cast<const float4*>(a_dim + j);
        rk += (v.x > ai || (v.x == ai && j < i)) + (v.y > ai || (v.y == ai && j + 1 < i)) +
              (v.z > ai || (v.z == ai && j + 2 < i)) + (v.w > ai || (v.w == ai && j + 3 < i));
      }
    }
    rk += __shfl_xor_sync(0xffffffffu, rk, 1);
    if (i < D && half == 0 && rk < a.rd) dims[rk] = i;
  }
  __syncthreads();
  // ---- 1. the chosen dims' bounds of this CTA's pages, row t for the t-th dim (16-byte copies from
  // the row start rounded down to 16 bytes, the last one cut at the end of the pages)
  if (npf > 0) {
    const int nch = (7 + npf + 7) / 8;                 // copies per row (covers the offset)
    for (int e = tid; e < 2 * a.rd * nch; e += kRfThreads) {
      const int which = e / (a.rd * nch), rem = e % (a.rd * nch);
      const int t = rem / nch, ch = rem % nch;
      const int64_t start = (bh * D + dims[t]) * a.npc + p0;
      const int64_t h0 = (start & ~7ll) + ch * 8;
      const int64_t end = start + npf;
      if (h0 < end) {
        const int bytes = (int)min((int64_t)16, (end - h0) * 2);
        cp_async16((which ? bmx : bmn) + t * a.rs + ch * 8, (which ? a.kmax : a.kmin) + h0, bytes);
      }
    }
  }
  cp_async_commit();
  if (tid < a.rd) {
    const int d = dims[tid];
    float P = 0.f, N = 0.f;
    for (int h = 0; h < G; ++h) {
      const float v = qs[h * D + d];
      P += fmaxf(v, 0.f);
      N += fminf(v, 0.f);
    }
    pn[0][tid] = P;
    pn[1][tid] = N;
  }
  cp_async_wait<0>();
  __syncthreads();
  // ---- scores of this CTA's pages: thread (page, slice) sums the dims t = slice (mod kRfSlices)
  for (int e = tid; e < np * kRfSlices; e += kRfThreads) {
    const int pl = e % np, sl = e / np;
    float acc = 0.f;
    for (int t = sl; t < a.rd; t += kRfSlices) {
      const int off = (int)(((bh * D + dims[t]) * a.npc + p0) & 7);
      const int i = t * a.rs + off + pl;
      acc += __half2float(bmx[i]) * pn[0][t] + __half2float(bmn[i]) * pn[1][t];
    }
    part[sl * sp + pl] = acc;
  }
  __syncthreads();
  // ---- 2. every score into every CTA of the cluster (and -inf pads to a multiple of four)
  for (int e = tid; e < np * kCl; e += kRfThreads) {
    const int pl = e % np, dst = e / np;
    float s = 0.f;
#pragma unroll
    for (int sl = 0; sl < kRfSlices; ++sl) s += part[sl * sp + pl];
    st_cluster(cluster_addr(sc + p0 + pl, dst), s);
  }
  for (int p = ns + tid; p < ((ns + 3) & ~3); p += kRfThreads) sc[p] = -INFINITY;   // local pads
  cluster_sync();

  // ---- 3. CTA r ranks the r-th run of ceil(ns / kCl) candidate pages against all scores under
  // (score desc, page asc), eight threads per page each counting over an eighth of the pages,
  // and stores the kept flags into every CTA; then thread t takes a contiguous run of pages so
  // that the kept pages come out in ascending order from one block scan
  const int k = min(a.kp, ns);
  const int seg = ((ns + 7) / 8 + 3) & ~3;              // pages per counting segment (multiple of 4)
  const int rp = (ns + kCl - 1) / kCl;                 // pages ranked per CTA
  const int r0 = rank * rp, nr = max(0, min(ns, r0 + rp) - r0);
  for (int base = 0; base < nr * 8; base += kRfThreads) {   // uniform trip count: shuffles below
    const int task = base + tid;
    const int pl = task >> 3, sg = task & 7;
    int rk = 0;
    if (pl < nr) {
      const int p = r0 + pl;
      const float s = sc[p];
      const int j1 = min(ns, (sg + 1) * seg);
      for (int j = sg * seg; j < j1; j += 4) {        // scores are padded to a multiple of four
        const float4 v = *reinterpret_cast<const float4*>(sc + j);
        rk += (v.x > s || (v.x == s && j < p)) + (v.y > s || (v.y == s && j + 1 < p)) +
              (v.z > s || (v.z == s && j + 2 < p)) + (v.w > s || (v.w == s && j + 3 < p));
      }
    }
    rk += __shfl_xor_sync(0xffffffffu, rk, 1);
    rk += __shfl_xor_sync(0xffffffffu, rk, 2);
    rk += __shfl_xor_sync(0xffffffffu, rk, 4);
    if (pl < nr && sg < kCl) st_cluster_u8(cluster_addr(kf + r0 + pl, sg), rk < k ? 1u : 0u);
  }
  cluster_sync();
  const int ppt = (ns + kRfThreads - 1) / kRfThreads;
  uint32_t keep_bits = 0;
  int cnt = 0;
  for (int u = 0; u < ppt; ++u) {
    const int p = tid * ppt + u;
    if (p < ns && kf[p]) {
      keep_bits |= 1u << u;
      ++cnt;
    }
  }
  int total;
  int pos = block_exclusive_scan(cnt, warp_sums, &total);
  for (int u = 0; u < ppt; ++u)
    if (keep_bits & (1u << u)) sel[pos++] = tid * ppt + u;
  __syncthreads();
  if (rank == 0 && a.page_idx != nullptr)
    for (int i = tid; i < a.kp; i += kRfThreads) a.page_idx[bh * a.kp + i] = i < total ? sel[i] : -1;
  const int n_att = n > 0 ? total : 0;                 // chosen pages attended (and the newest one)

  // ---- 4. attention: page i goes to CTA i % kCl, warp (i / kCl) % kRfWarps
  const int g = lane >> 2, r = lane & 3;
  const bool real = g < G;
  const uint32_t* qrow = qh2[real ? g : 0];           // query fragments: rows = heads
  float o[D / 8][2];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = 0.f;
  float m_run = -INFINITY, l_part = 0.f;
  uint8_t* kt = smem + L.pages + warp * 2 * kPage * D * 2;
  uint8_t* vt = kt + kPage * D * 2;
  const int mi = lane >> 3, rowi = lane & 7;
  const int tokk = (mi >> 1) * 8 + rowi, tokv = (mi & 1) * 8 + rowi;
  const __half* kbase = a.k + bh * a.T_cap * D;
  const __half* vbase = a.v + bh * a.T_cap * D;
  // QK^T, online softmax and PV of the group's heads on one page's K and V tiles (16 rows)
  auto attend = [&](const uint8_t* kt_, const uint8_t* vt_, int valid) {
      float s[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
      for (int kc = 0; kc < KC; ++kc) {
        uint32_t bk[4];
        ldsm_x4(bk, kt_ + tile_off<D>(tokk, kc * 2 + (mi & 1)));
        const uint32_t a0 = real ? qrow[kc * 8 + r] : 0u, a2 = real ? qrow[kc * 8 + 4 + r] : 0u;
        mma16816(s[0], a0, 0u, a2, 0u, bk[0], bk[1]);
        mma16816(s[1], a0, 0u, a2, 0u, bk[2], bk[3]);
      }
      const int tk[4] = {2 * r, 2 * r + 1, 8 + 2 * r, 9 + 2 * r};
      float x[4] = {s[0][0], s[0][1], s[1][0], s[1][1]};
      float mx = -INFINITY;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        x[j] = tk[j] < valid ? x[j] * a.scale_log2 : -INFINITY;
        mx = fmaxf(mx, x[j]);
      }
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float m_new = fmaxf(m_run, mx);
      float p[4] = {0.f, 0.f, 0.f, 0.f};
      float alpha = 1.f;
      if (m_new != -INFINITY) {
        alpha = exp2f(m_run - m_new);
#pragma unroll
        for (int j = 0; j < 4; ++j) p[j] = exp2f(x[j] - m_new);
      }
      l_part = l_part * alpha + (p[0] + p[1]) + (p[2] + p[3]);
      m_run = m_new;
#pragma unroll
      for (int j = 0; j < D / 8; ++j) {
        o[j][0] *= alpha;
        o[j][1] *= alpha;
      }
      const uint32_t pa0 = pack_half2(p[0], p[1]);
      const uint32_t pa2 = pack_half2(p[2], p[3]);
#pragma unroll
      for (int j = 0; j < D / 16; ++j) {
        uint32_t bv[4];
        ldsm_x4_t(bv, vt_ + tile_off<D>(tokv, 2 * j + (mi >> 1)));
        float d0[4] = {o[2 * j][0], o[2 * j][1], 0.f, 0.f};
        float d1[4] = {o[2 * j + 1][0], o[2 * j + 1][1], 0.f, 0.f};
        mma16816(d0, pa0, 0u, pa2, 0u, bv[0], bv[1]);
        mma16816(d1, pa0, 0u, pa2, 0u, bv[2], bv[3]);
        o[2 * j][0] = d0[0];
        o[2 * j][1] = d0[1];
        o[2 * j + 1][0] = d1[0];
        o[2 * j + 1][1] = d1[1];
      }
  };
  // This warp's pages: chosen page i = rank + kCl * warp (+ kCl * kRfWarps ...), and for the
  // designated warp first the newest page, staged at the start, attended while the copies of its
  // first chosen page are in flight.  One call site of attend().
  auto load_page = [&](int i) {
    const int page = sel[i];                           // a full page
    for (int e = lane; e < 2 * kPage * (D / 8); e += 32) {
      const int kv = e / (kPage * (D / 8)), rem = e % (kPage * (D / 8));
      const int row = rem / (D / 8), ch = rem % (D / 8);
      cp_async16((kv ? vt : kt) + tile_off<D>(row, ch), (kv ? vbase : kbase) + ((int64_t)page * kPage + row) * D + ch * 8, 16);
    }
    cp_async_commit();
  };
  int i = rank + kCl * warp;
  if (i < n_att) load_page(i);
  bool tail_left = tail_warp;
  while (tail_left || i < n_att) {
    const bool tail_now = tail_left;
    if (!tail_now) {
      cp_async_wait<0>();
      __syncwarp();
    }
    attend(tail_now ? tk : kt, tail_now ? tv : vt, tail_now ? tail_valid : kPage);
    if (tail_now) {
      tail_left = false;
    } else {
      __syncwarp();                                    // the tiles are reloaded next page
      i += kCl * kRfWarps;
      if (i < n_att) load_page(i);
    }
  }
  __syncthreads();                                     // every warp is done with its tiles

  // ---- 5. merge: warps -> CTA partial -> CTA 0
  float* wm = reinterpret_cast<float*>(smem + L.wpart);   // [warp][G] m, then l, then o [warp][G][D]
  float* wl = wm + kRfWarps * G;
  float* wo = wl + kRfWarps * G;
  l_part += __shfl_xor_sync(0xffffffffu, l_part, 1);
  l_part += __shfl_xor_sync(0xffffffffu, l_part, 2);
  if (real) {
    if (r == 0) {
      wm[warp * G + g] = m_run;
      wl[warp * G + g] = l_part;
    }
#pragma unroll
    for (int j = 0; j < D / 8; ++j) {
      wo[(warp * G + g) * D + j * 8 + 2 * r] = o[j][0];
      wo[(warp * G + g) * D + j * 8 + 2 * r + 1] = o[j][1];
    }
  }
  __syncthreads();
  float* cp = reinterpret_cast<float*>(smem + L.cpart);   // CTA 0: [kCl][G][D + 2]
  const uint32_t cp0 = cluster_addr(cp, 0);
  for (int e = tid; e < G * D; e += kRfThreads) {
    const int row = e / D, d = e % D;
    float M = -INFINITY;
    for (int w = 0; w < kRfWarps; ++w) M = fmaxf(M, wm[w * G + row]);
    float Lsum = 0.f, O = 0.f;
    if (M != -INFINITY) {
      for (int w = 0; w < kRfWarps; ++w) {
        const float f = exp2f(wm[w * G + row] - M);
        Lsum += wl[w * G + row] * f;
        O += wo[(w * G + row) * D + d] * f;
      }
    }
    const uint32_t slot = cp0 + (uint32_t)((rank * G + row) * (D + 2)) * 4u;
    st_cluster(slot + (2 + d) * 4u, O);
    if (d == 0) {
      st_cluster(slot, M);
      st_cluster(slot + 4u, Lsum);
    }
  }
  cluster_sync();
  if (rank == 0) {
    for (int e = tid; e < G * D; e += kRfThreads) {
      const int row = e / D, d = e % D;
      float M = -INFINITY;
      for (int c = 0; c < kCl; ++c) M = fmaxf(M, cp[(c * G + row) * (D + 2)]);
      float Lsum = 0.f, O = 0.f;
      if (M != -INFINITY) {
        for (int c = 0; c < kCl; ++c) {
          const float* slot = cp + (c * G + row) * (D + 2);
          const float f = exp2f(slot[0] - M);
          Lsum += slot[1] * f;
          O += slot[2 + d] * f;
        }
      }
      a.out[((int64_t)b * a.Hq + (int64_t)kvh * G + row) * D + d] = __float2half_rn(Lsum > 0.f ? O / Lsum : 0.f);
    }
  }
  if (!append) return;
  // the appended token filled its page: the page's per-dim min and max, from the staged tiles
  if (tail_warp && room && n % kPage == 0) {
    for (int d = lane; d < D; d += 32) {
      const int off = tile_off<D>(0, d / 8) + (d % 8) * 2;
      __half lo = *reinterpret_cast<const __half*>(tk + off), hi = lo;
      for (int row = 1; row < kPage; ++row) {
        const __half x = *reinterpret_cast<const __half*>(tk + tile_off<D>(row, d / 8) + (d % 8) * 2);
        lo = __hlt(x, lo) ? x : lo;
        hi = __hgt(x, hi) ? x : hi;
      }
      a.kmin[(bh * D + d) * a.npc + ns] = lo;
      a.kmax[(bh * D + d) * a.npc + ns] = hi;
    }
  }
  // every thread of this CTA read T_len before this point; the last CTA of batch entry b (all
  // kCl CTAs of its Hkv clusters) stores the new length and clears the count
  __syncthreads();
  if (tid == 0) {
    const unsigned old = atomicAdd(reinterpret_cast<unsigned*>(a.T_len) + b, 1u << 24);
    if ((int)(old >> 24) == kCl * a.Hkv - 1) a.T_len[b] = n;
    if (!room && rank == 0 && kvh == 0) atomicOr(&g_status_rocket, MKV_FLAG_CACHE_FULL);
  }
}

template <int D>
cudaError_t launch_rf_t(const RfArgs& a, int units, size_t smem, cudaStream_t st) {
  cudaError_t e = cudaFuncSetAttribute(rocket_fused_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  rocket_fused_kernel<D><<<dim3(kCl, units), kRfThreads, smem, st>>>(a);
  return cudaPeekAtLastError();
}

}  // namespace

size_t rocket_fused_smem(const mkv_config& c, int64_t T_cap) {
  const int64_t npc = T_cap / kPage;
  const int sp = (int)((npc + kCl - 1) / kCl);
  const int rs = (sp + 8 + 7) / 8 * 8;
  return (size_t)RfLayout(c.D, c.Hq / c.Hkv, npc, c.topk_pages, rs).bytes;
}

cudaError_t launch_rocket_fused(const mkv_config& c, const void* q, const mkv_cache& cache, int32_t* page_idx,
                                void* out, const void* k_new, const void* v_new, cudaStream_t st) {
  RfArgs a{};
  a.q = static_cast<const __half*>(q);
  a.k = static_cast<__half*>(cache.k);
  a.v = static_cast<__half*>(cache.v);
  a.kmin = static_cast<__half*>(cache.kmin);
  a.kmax = static_cast<__half*>(cache.kmax);
  a.T_len = cache.T_len;
  a.k_new = static_cast<const __half*>(k_new);
  a.v_new = static_cast<const __half*>(v_new);
  a.T_cap = cache.T_cap;
  a.npc = cache.T_cap / kPage;
  a.Hq = c.Hq;
  a.Hkv = c.Hkv;
  a.G = c.Hq / c.Hkv;
  a.kp = c.topk_pages;
  a.rd = c.topq_dims;
  const int sp = (int)((a.npc + kCl - 1) / kCl);
  a.rs = (sp + 8 + 7) / 8 * 8;
  const float scale = c.softmax_scale > 0.f ? c.softmax_scale : 1.0f / sqrtf((float)c.D);
  a.scale_log2 = scale * kLog2e;
  a.page_idx = page_idx;
  a.out = static_cast<__half*>(out);
  const size_t smem = rocket_fused_smem(c, cache.T_cap);
  const int units = c.B * c.Hkv;
  return c.D == 128 ? launch_rf_t<128>(a, units, smem, st) : launch_rf_t<64>(a, units, smem, st);
}

cudaError_t take_status_rocket(uint32_t* flags, cudaStream_t st) {
  uint32_t zero = 0, v = 0;
  cudaError_t e = cudaMemcpyFromSymbolAsync(&v, g_status_rocket, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyToSymbolAsync(g_status_rocket, &zero, sizeof(zero), 0, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  *flags |= v;
  return e;
}

}  // namespace mkv
