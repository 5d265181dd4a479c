// Prefill-side attention scores shared by H2O and SnapKV (Section 2.1):
//   score[j] = sum over the group's query heads h and query rows i whose
//              position p_i >= j of softmax_i(scale q_{h,i} . k)[j]
// -- H2O: every prompt row (p_i = i), the accumulated attention a token
//    receives from later tokens;
// -- SnapKV: the W rows of the observation window (p_i = T - W + i).
//
// Two passes on the 5th-generation tensor cores (tcgen05.mma kind::f16: fp16 operands, fp32
// accumulator in tensor memory), each a stream of 128 x N x D tile products with a softmax epilogue:
//   pass 1 (rows): a CTA holds 128 query rows (the group's G heads, 128 / G rows each) and streams
//           256-key tiles (N = 256: one MMA instruction and one barrier round trip per 256 keys); it
//           keeps per row the running max m and sum l of 2^(s - m) over the causal keys.  When the
//           rows are few (an observation window) the key range is split across CTAs; a small kernel
//           merges the splits into (-m, 1 / l) per row, laid out in the order of pass 2's query blocks;
//   pass 2 (columns): a CTA holds 128 keys and streams the 128-row query blocks that can see them
//           (N = 128, four accumulator buffers: its epilogue is the heavier one), summing
//           2^(s - m_i) / l_i over the rows with p_i >= j for each key j;
//   pass 2 over one query block (colsum_window_kernel): when the window's rows fit one block, a
//           CTA holds that block and streams a run of 128-key tiles instead.
// The held operand is the MMA's A (M = 128 lanes of the accumulator), a streamed tile its B (the
// window kernel swaps them).  Each CTA is warp-specialised, one per SM (all 512 tensor-memory
// columns):
//   warp 0 (one thread) loads operand tiles by TMA (tensor maps with the 128-byte swizzle, the
//           K-major layout the MMA reads) into a ring of stages, and in pass 2 each query block's
//           128 row statistics by a bulk copy beside it;
//   warp 1 (one thread) issues the D / 16 MMAs of tile t into accumulator buffer t % (buffers),
//           then commits to the stage's and the buffer's mbarriers;
//   warps 2..17 read finished accumulators in two groups of eight: group g takes the tiles
//           t = g mod 2, so the groups work a tile apart and one group's exponentials overlap the
//           other's loads and reductions; warp w reads lanes 32 (w % 4) .. + 31 (the lane quarter it
//           may access) and one half of the tile's columns, 64 at a time.
// Loads, products and epilogues of different tiles overlap; nothing in the tile loop waits on a
// CTA-wide barrier.  Every wait is bounded (1 s of the GPU's global timer): on a timeout the role
// raises MKV_FLAG_WAIT_TIMEOUT and sets a flag that ends the other roles' waits; the CTA then waits
// (bounded) for the copies and products it already issued and still frees its tensor memory.
#include <cuda.h>   // CUtensorMap and its enums; the encoder is fetched from the driver at run time
#include <math.h>

#include <algorithm>

#include "mkv_common.cuh"
#include "mkv_internal.h"
#include "mkv_tc.cuh"

namespace mkv {

__device__ uint32_t g_status_prefill;   // MKV_FLAG_* bits raised by the scoring passes

cudaError_t take_status_prefill(uint32_t* flags, cudaStream_t st) {
  uint32_t v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbolAsync(&v, g_status_prefill, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyToSymbolAsync(g_status_prefill, &zero, sizeof(zero), 0, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  *flags |= v;
  return e;
}

namespace {

constexpr int kTM = 128;                 // rows of the held operand (the MMA's M)
constexpr int kBlk = 128;                // a query block (pass 2) / a key block: 128 rows
constexpr int kGroupWarps = 8;           // an epilogue group: four lane quarters x two column halves
constexpr int kEpiWarps = 2 * kGroupWarps;
constexpr int kThr = (2 + kEpiWarps) * 32;
constexpr int kStatBytes = kBlk * 8;     // one query block's (-m, 1 / l)
constexpr uint64_t kWaitNs = 1000000000ull;   // a bounded wait gives up after 1 s

// A streamed tile of TN rows (the MMA's N).  Pass 1 streams 256-key tiles: one MMA instruction and
// one barrier round trip per 256 keys.  Pass 2 streams 128-row query blocks: its heavier epilogue
// gains more from four accumulator buffers, which let the tensor core run further ahead of it.
template <int TN>
struct Tiling {
  static constexpr int kTN = TN;
  static constexpr int kNB = 512 / TN;            // accumulator buffers: all 512 tensor-memory columns
  static constexpr int kS = TN == 256 ? 2 : 4;    // operand stages
  static constexpr int kHalf = TN / 2;            // accumulator columns an epilogue warp reads per tile
  static constexpr int kBlocks = TN / kBlk;       // query blocks per tile (pass 2)
};
constexpr int kTN1 = 256;                // pass 1's tile
constexpr int kTN2 = 128;                // pass 2's tile

struct ScoreArgs {
  int64_t R, T, pos0;   // query rows, keys, position of query row 0
  int Hq, Hkv, G, rpb;  // rpb = rows per head in a 128-row query block (128 / G, a power of two)
  int rowblocks;        // ceil(R / rpb)
  int n_ksplit, tiles_per_split;   // pass 1: key splits and 256-key tiles per split
  float scale_log2;
  float2* row_st;       // [B Hkv][rowblocks][n_ksplit][128]: pass 1's (m, l); merged at split 0 (rowmerge_kernel)
  float* score;         // [B Hkv][T]
};

template <int D, int TN>
struct Layout {
  using C = Tiling<TN>;
  static constexpr int ATOM_A = kTM * 128;                // 128 rows x 64 fp16: one swizzle-atom column
  static constexpr int ATOM_B = TN * 128;                 // TN rows x 64 fp16
  static constexpr int TILE_A = (D / 64) * ATOM_A;
  static constexpr int TILE_B = (D / 64) * ATOM_B;
  static constexpr int A_OFF = 0;
  static constexpr int B_OFF = TILE_A;                    // [kS] streamed tiles
  static constexpr int ST_OFF = B_OFF + C::kS * TILE_B;   // [kS][kBlocks] pass 2: the query blocks' statistics
  static constexpr int MRG_OFF = ST_OFF + C::kS * C::kBlocks * kStatBytes;   // [4][128] (group, half) partials
  static constexpr int CTL_OFF = MRG_OFF + 4 * kTM * 8;
  static constexpr int BYTES = CTL_OFF + 256;
  static constexpr int ALLOC = BYTES + 1024;              // slack to align the base to 1024 B
};

template <int TN>
struct Ctl {
  using C = Tiling<TN>;
  uint64_t full[C::kS];     // stage s loaded (TMA transaction bytes)
  uint64_t empty[C::kS];    // stage s's operand read by the tensor core
  uint64_t sempty[C::kS];   // stage s's row statistics read by its epilogue group (pass 2)
  uint64_t tfull[C::kNB];   // accumulator buffer b holds a finished product
  uint64_t tempty[C::kNB];  // accumulator buffer b read by its epilogue group
  uint64_t abar;         // the held operand loaded
  uint32_t tslot;        // tensor-memory base address
  int fail;              // a wait ran out: every role stops
  int issued;            // tiles whose loads were issued
  int mma_issued;        // tiles whose products were issued
};
static_assert(sizeof(Ctl<kTN1>) <= 256 && sizeof(Ctl<kTN2>) <= 256, "control block");

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return p + ((1024u - (smem_addr(p) & 1023u)) & 1023u);
}

// Bounded wait of one role: false when it ran out after `ns` nanoseconds (the flag is then raised
// and MKV_FLAG_WAIT_TIMEOUT set) or another role did.
__device__ __forceinline__ bool role_wait(uint64_t* bar, uint32_t parity, volatile int* fail, uint64_t ns = kWaitNs) {
  if (tc_mbar_try(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
    if (tc_mbar_try(bar, parity)) return true;
    if (*fail) return false;
    if (globaltimer_ns() - t0 > ns) break;
  }
  *fail = 1;
  atomicOr(&g_status_prefill, MKV_FLAG_WAIT_TIMEOUT);
  return false;
}

// D[tmem] = A (128 rows) x B (TN rows)^T over K = D: D / 16 MMAs, issued by one thread.  `a` and
// `b` are the shared-memory descriptors of the tiles' first K step; a K step adds a compile-time
// offset to the start-address field (no carry: shared addresses stay below 2^18).
template <int D, int TN>
__device__ __forceinline__ void issue_tile(uint32_t d_tmem, uint64_t a, uint64_t b) {
  using L = Layout<D, TN>;
  constexpr uint32_t kId = tc_idesc_f16(kTM, TN);
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    const uint64_t oa = (uint64_t)(((kk >> 2) * L::ATOM_A + (kk & 3) * 32) >> 4);
    const uint64_t ob = (uint64_t)(((kk >> 2) * L::ATOM_B + (kk & 3) * 32) >> 4);
    tc_mma(d_tmem, a + oa, b + ob, kId, kk > 0 ? 1u : 0u);
  }
}

// Barriers and tensor memory of a CTA; returns the tensor-memory base (all 512 columns).
template <int TN>
__device__ __forceinline__ uint32_t cta_setup(Ctl<TN>* ctl) {
  using C = Tiling<TN>;
  if ((threadIdx.x >> 5) == 0) tc_alloc(&ctl->tslot, C::kNB * TN);
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kS; ++s) {
      tc_mbar_init(&ctl->full[s], 1);
      tc_mbar_init(&ctl->empty[s], 1);
      tc_mbar_init(&ctl->sempty[s], kGroupWarps);
    }
    for (int b = 0; b < C::kNB; ++b) {
      tc_mbar_init(&ctl->tfull[b], 1);
      tc_mbar_init(&ctl->tempty[b], kGroupWarps);
    }
    tc_mbar_init(&ctl->abar, 1);
    tc_fence_mbar_init();
    ctl->fail = 0;
    ctl->issued = 0;
    ctl->mma_issued = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  return ctl->tslot;
}

// After every role has returned: on a failure, wait (bounded) for the copies and products already
// issued; then free the tensor memory.
template <int TN>
__device__ __forceinline__ void cta_teardown(Ctl<TN>* ctl, uint32_t tbase) {
  using C = Tiling<TN>;
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && ctl->fail) {
    for (int t = std::max(0, ctl->issued - C::kS); t < ctl->issued; ++t)
      tc_mbar_wait(&ctl->full[t % C::kS], (uint32_t)((t / C::kS) & 1), kWaitNs);
    if (ctl->mma_issued > 0) {
      const int t = ctl->mma_issued - 1;
      tc_mbar_wait(&ctl->tfull[t % C::kNB], (uint32_t)((t / C::kNB) & 1), kWaitNs);
    }
  }
  __syncthreads();
  tc_fence_after();
  if ((threadIdx.x >> 5) == 0) tc_dealloc(tbase, C::kNB * TN);
}

// The three roles over `ntiles` streamed tiles.  issue_a(bar) loads the held operand;
// issue_b(t, s, bar) loads tile t into stage s; epi(t, col, s) reads the thread's half of tile t's
// accumulator (kHalf columns from tensor-memory address col, lane 0) and, with kStats, the
// statistics of stage s.  With kStreamA the streamed tile is the MMA's A operand and the held one its
// B (the accumulator's lanes then follow the streamed rows).
template <int D, int TN, bool kStats, bool kStreamA = false, typename IssueA, typename IssueB, typename Epi>
__device__ __forceinline__ void run_roles(uint8_t* sm, Ctl<TN>* ctl, uint32_t tbase, int ntiles, IssueA issue_a,
                                          IssueB issue_b, Epi epi) {
  using L = Layout<D, TN>;
  using C = Tiling<TN>;
  constexpr int kS = C::kS, kNB = C::kNB, kHalf = C::kHalf;
  volatile int* fail = &ctl->fail;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (ntiles <= 0) return;
  if (warp == 0) {
    if (lane == 0) {                      // producer
      issue_a(&ctl->abar);
      for (int t = 0; t < ntiles; ++t) {
        const int s = t % kS, n = t / kS;
        if (n > 0) {
          if (!role_wait(&ctl->empty[s], (uint32_t)((n - 1) & 1), fail)) break;
          if (kStats && !role_wait(&ctl->sempty[s], (uint32_t)((n - 1) & 1), fail)) break;
        }
        issue_b(t, s, &ctl->full[s]);
        ctl->issued = t + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {                      // MMA issuer
      const uint64_t a_desc = tc_desc_sw128(smem_addr(sm + L::A_OFF));
      const uint64_t b_desc = tc_desc_sw128(smem_addr(sm + L::B_OFF));
      if (role_wait(&ctl->abar, 0, fail)) {
        for (int t = 0; t < ntiles; ++t) {
          const int s = t % kS, bf = t % kNB, u = t / kNB;
          if (!role_wait(&ctl->full[s], (uint32_t)((t / kS) & 1), fail)) break;
          if (u > 0 && !role_wait(&ctl->tempty[bf], (uint32_t)((u - 1) & 1), fail)) break;
          tc_fence_after();
          const uint64_t stage = b_desc + (uint64_t)((s * L::TILE_B) >> 4);
          if (kStreamA)
            issue_tile<D, TN>(tbase + (uint32_t)(bf * TN), stage, a_desc);
          else
            issue_tile<D, TN>(tbase + (uint32_t)(bf * TN), a_desc, stage);
          tc_commit(&ctl->empty[s]);
          tc_commit(&ctl->tfull[bf]);
          ctl->mma_issued = t + 1;
        }
      }
    }
  } else {                                // epilogue warps: group (warp - 2) / 8 takes every other tile
    const int grp = (warp - 2) / kGroupWarps, half = ((warp - 2) >> 2) & 1;
    // the held operand's phase: what came with it (statistics held beside it) is visible after it
    const bool held = role_wait(&ctl->abar, 0, fail);
    if (!__all_sync(0xffffffffu, held)) return;
    for (int t = grp; t < ntiles; t += 2) {
      const int s = t % kS, bf = t % kNB;
      bool ok = role_wait(&ctl->tfull[bf], (uint32_t)((t / kNB) & 1), fail);
      // the statistics came with the stage's operand: their copy completed that phase of full[s]
      if (kStats) ok = ok && role_wait(&ctl->full[s], (uint32_t)((t / kS) & 1), fail);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      epi(t, tbase + (uint32_t)(bf * TN + half * kHalf), s);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        tc_mbar_arrive(&ctl->tempty[bf]);
        if (kStats) tc_mbar_arrive(&ctl->sempty[s]);
      }
    }
  }
}

// ---------------------------------------------------------------- pass 1
template <int D>
__global__ void __launch_bounds__(kThr, 1)
    rowstats_tc_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                       const ScoreArgs a) {
  constexpr int kTN = kTN1, kHalf = Tiling<kTN1>::kHalf;
  using L = Layout<D, kTN1>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = align1024(smem_raw);
  Ctl<kTN1>* ctl = reinterpret_cast<Ctl<kTN1>*>(sm + L::CTL_OFF);
  const int ks = blockIdx.x;
  const int rb = a.rowblocks - 1 - (int)blockIdx.y;      // the row blocks with the most keys first
  const int bh = (int)blockIdx.z;
  const int b = bh / a.Hkv, kvh = bh % a.Hkv;
  const int warp = threadIdx.x >> 5;
  const int lq = warp & 3, cq = (warp - 2) >> 2;         // (epilogue warps) lane quarter; group x half
  const int hf = cq & 1;                                 // column half of the tile
  const int lr = lq * 32 + (threadIdx.x & 31);           // accumulator lane = query row of the block

  // the block's last valid row bounds its causal key range
  const int64_t row_hi = std::min<int64_t>((int64_t)rb * a.rpb + a.rpb, a.R);   // exclusive
  const int64_t k_begin = (int64_t)ks * a.tiles_per_split * kTN;
  const int64_t k_end = std::min<int64_t>(std::min<int64_t>(k_begin + (int64_t)a.tiles_per_split * kTN, a.T),
                                          a.pos0 + row_hi);
  const int ntiles = k_end > k_begin ? (int)ceil_div_dev(k_end - k_begin, kTN) : 0;
  const int64_t irow = (int64_t)rb * a.rpb + (lr & (a.rpb - 1));
  const int64_t lim = irow < a.R ? std::min<int64_t>(k_end - 1, a.pos0 + irow) : -1;   // last key it sees

  const uint32_t tbase = cta_setup(ctl);
  float m_run = -INFINITY, l_run = 0.f;
  run_roles<D, kTN1, false>(
      sm, ctl, tbase, ntiles,
      [&](uint64_t* bar) {                // one box of G heads x rpb rows: head g's rows are tile rows g rpb ..
        tc_mbar_expect_tx(bar, L::TILE_A);
        for (int at = 0; at < D / 64; ++at)
          tma_load_4d(sm + L::A_OFF + at * L::ATOM_A, &qmap, at * 64, rb * a.rpb, kvh * a.G, b, bar);
      },
      [&](int t, int s, uint64_t* bar) {
        tc_mbar_expect_tx(bar, L::TILE_B);
        for (int at = 0; at < D / 64; ++at)
          tma_load_4d(sm + L::B_OFF + s * L::TILE_B + at * L::ATOM_B, &kmap, at * 64,
                      (int)(k_begin + (int64_t)t * kTN), kvh, b, bar);
      },
      [&](int t, uint32_t col, int) {
#pragma unroll 1
        for (int ch = 0; ch < kHalf / 64; ++ch) {
          const int64_t jc = k_begin + (int64_t)t * kTN + hf * kHalf + ch * 64;
          float v[64];
          tc_ld64(col + ((uint32_t)(lq * 32) << 16) + (uint32_t)(ch * 64), v);
          if (jc + 63 > lim) {            // keys past the row's causal limit (or the range) drop out
#pragma unroll
            for (int e = 0; e < 64; ++e) v[e] = jc + e <= lim ? v[e] : -INFINITY;
          }
          float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};   // max of the raw products
#pragma unroll
          for (int q = 0; q < 32; ++q) mx[q & 3] = fmax3(mx[q & 3], v[2 * q], v[2 * q + 1]);
          // the scale is positive: the max of the scaled products is the scaled max
          const float m_new = fmaxf(m_run, fmax3(mx[0], mx[1], fmaxf(mx[2], mx[3])) * a.scale_log2);
          if (m_new != -INFINITY) {
            // 2^(s scale - m) and its sum, two columns per packed instruction
            const uint64_t sc2 = pk2(a.scale_log2, a.scale_log2), nm2 = pk2(-m_new, -m_new);
            uint64_t sp2[2] = {0ull, 0ull};
#pragma unroll
            for (int q = 0; q < 32; ++q) {
              const float2 x = upk2(ffma2(pk2(v[2 * q], v[2 * q + 1]), sc2, nm2));
              sp2[q & 1] = fadd2(sp2[q & 1], pk2(ex2_approx(x.x), ex2_approx(x.y)));
            }
            const float2 s0 = upk2(sp2[0]), s1 = upk2(sp2[1]);
            l_run = l_run * ex2_approx(m_run - m_new) + ((s0.x + s0.y) + (s1.x + s1.y));
            m_run = m_new;
          }
        }
      });
  // the (group, half) partials of each row merged into this split's (m, l)
  float2* mrg = reinterpret_cast<float2*>(sm + L::MRG_OFF);
  if (warp >= 2) mrg[cq * kTM + lr] = make_float2(m_run, l_run);
  __syncthreads();
  if (warp >= 2 && cq == 0) {
    float M = -INFINITY;
#pragma unroll
    for (int q = 0; q < 4; ++q) M = fmaxf(M, mrg[q * kTM + lr].x);
    float l = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 o = mrg[q * kTM + lr];
        l += o.y * ex2_approx(o.x - M);
      }
    }
    a.row_st[(((int64_t)bh * a.rowblocks + rb) * a.n_ksplit + ks) * kTM + lr] = make_float2(M, l);
  }
  cta_teardown(ctl, tbase);
}

// ---------------------------------------------------------------- a row's key splits merged in place:
// (-m, 1 / l) of the whole row into its block's split-0 entries, as float4 {-m_2p, -m_2p+1, 1/l_2p,
// 1/l_2p+1} per row pair p (pass 2 reads a pair's operands as two packed registers); (-inf, 0) for a
// row past the query rows, so that it adds 2^-inf * 0 = 0 in pass 2.  One CTA per (unit, block).
__global__ void __launch_bounds__(kBlk) rowmerge_kernel(float2* __restrict__ row_st, int ns, int rpb, int rowblocks,
                                                        int64_t R) {
  const int64_t blk = blockIdx.x;
  const int c = threadIdx.x;
  const float2* p = row_st + blk * ns * kBlk + c;
  float M = -INFINITY;
  for (int s = 0; s < ns; ++s) M = fmaxf(M, p[s * kBlk].x);
  float Ls = 0.f;
  for (int s = 0; s < ns; ++s) {
    const float2 x = p[s * kBlk];
    if (x.x != -INFINITY) Ls += x.y * exp2f(x.x - M);
  }
  const bool valid = (int64_t)(blk % rowblocks) * rpb + (c & (rpb - 1)) < R && M != -INFINITY && Ls > 0.f;
  __syncthreads();                        // the block's partials are read before split 0 is overwritten
  float* out = reinterpret_cast<float*>(row_st + blk * ns * kBlk);
  out[(c >> 1) * 4 + (c & 1)] = valid ? -M : -INFINITY;
  out[(c >> 1) * 4 + 2 + (c & 1)] = valid ? 1.f / Ls : 0.f;
}

// ---------------------------------------------------------------- pass 2
template <int D>
__global__ void __launch_bounds__(kThr, 1)
    colsum_tc_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                     const ScoreArgs a) {
  using C = Tiling<kTN2>;
  using L = Layout<D, kTN2>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = align1024(smem_raw);
  Ctl<kTN2>* ctl = reinterpret_cast<Ctl<kTN2>*>(sm + L::CTL_OFF);
  const int bh = (int)blockIdx.y;
  const int b = bh / a.Hkv, kvh = bh % a.Hkv;
  const int warp = threadIdx.x >> 5;
  const int lq = warp & 3, cq = (warp - 2) >> 2;         // (epilogue warps) lane quarter; group x half
  const int hf = cq & 1;                                 // column half of the tile
  const int lr = lq * 32 + (threadIdx.x & 31);           // accumulator lane = key of the block
  const int64_t j0 = (int64_t)blockIdx.x * kBlk;
  const int64_t jrel = j0 + lr - a.pos0;                  // rows i >= jrel see this key

  // the query blocks whose rows can see key j0 (rows i with pos0 + i >= j0), kBlocks per tile
  const int64_t first_row = std::max<int64_t>(0, j0 - a.pos0);
  const int rb_begin = (int)(first_row / a.rpb);
  const int ntiles = (int)ceil_div_dev(std::max(0, a.rowblocks - rb_begin), C::kBlocks);
  const float2* stats = a.row_st + (int64_t)bh * a.rowblocks * a.n_ksplit * kTM;

  const uint32_t tbase = cta_setup(ctl);
  float acc = 0.f;
  run_roles<D, kTN2, true>(
      sm, ctl, tbase, ntiles,
      [&](uint64_t* bar) {
        tc_mbar_expect_tx(bar, L::TILE_A);
        for (int at = 0; at < D / 64; ++at)
          tma_load_4d(sm + L::A_OFF + at * L::ATOM_A, &kmap, at * 64, (int)j0, kvh, b, bar);
      },
      [&](int t, int s, uint64_t* bar) {  // the tile's query blocks that exist
        const int rb = rb_begin + C::kBlocks * t;
        const int nb = a.rowblocks - rb < C::kBlocks ? a.rowblocks - rb : C::kBlocks;
        tc_mbar_expect_tx(bar, (uint32_t)nb * (L::TILE_B / C::kBlocks + kStatBytes));
        for (int h = 0; h < nb; ++h) {
          for (int at = 0; at < D / 64; ++at)
            tma_load_4d(sm + L::B_OFF + s * L::TILE_B + at * L::ATOM_B + h * kBlk * 128, &qmap, at * 64,
                        (rb + h) * a.rpb, kvh * a.G, b, bar);
          bulk_load(sm + L::ST_OFF + (s * C::kBlocks + h) * kStatBytes,
                    stats + (int64_t)(rb + h) * a.n_ksplit * kTM, kStatBytes, bar);
        }
      },
      [&](int t, uint32_t col, int s) {
        const uint64_t sc2 = pk2(a.scale_log2, a.scale_log2);
        uint64_t sp2[2] = {0ull, 0ull};
#pragma unroll 1
        for (int ch = 0; ch < C::kHalf / 64; ++ch) {
          const int c0 = hf * C::kHalf + ch * 64;   // the chunk's first column of the tile
          const int h = c0 / kBlk, cin = c0 % kBlk;   // its query block and first column in the block
          const int rb = rb_begin + C::kBlocks * t + h;
          if (rb >= a.rowblocks) break;           // a block past the query rows (warp-uniform)
          const int64_t i0 = (int64_t)rb * a.rpb;   // row index of the block's first row per head
          // row pair p's statistics {-m, -m', 1/l, 1/l'}
          const float4* s4 =
              reinterpret_cast<const float4*>(sm + L::ST_OFF + (s * C::kBlocks + h) * kStatBytes) + cin / 2;
          float v[64];
          tc_ld64(col + ((uint32_t)(lq * 32) << 16) + (uint32_t)(ch * 64), v);
          if (i0 >= j0 + kBlk - 1 - a.pos0) {   // every row sees every key of the CTA: two rows per instruction
#pragma unroll
            for (int q = 0; q < 32; ++q) {
              const float4 w = s4[q];
              const float2 x = upk2(ffma2(pk2(v[2 * q], v[2 * q + 1]), sc2, pk2(w.x, w.y)));
              sp2[q & 1] = ffma2(pk2(ex2_approx(x.x), ex2_approx(x.y)), pk2(w.z, w.w), sp2[q & 1]);
            }
          } else {
#pragma unroll
            for (int q = 0; q < 32; ++q) {
              const float4 w = s4[q];
              const int c = cin + 2 * q;
              const float2 x = upk2(ffma2(pk2(v[2 * q], v[2 * q + 1]), sc2, pk2(w.x, w.y)));
              const float p0 = i0 + (c & (a.rpb - 1)) >= jrel ? ex2_approx(x.x) * w.z : 0.f;
              const float p1 = i0 + ((c + 1) & (a.rpb - 1)) >= jrel ? ex2_approx(x.y) * w.w : 0.f;
              sp2[q & 1] = fadd2(sp2[q & 1], pk2(p0, p1));
            }
          }
        }
        const float2 s0 = upk2(sp2[0]), s1 = upk2(sp2[1]);
        acc += (s0.x + s0.y) + (s1.x + s1.y);
      });
  // the (group, half) partials of each key summed
  float* mrg = reinterpret_cast<float*>(sm + L::MRG_OFF);
  if (warp >= 2) mrg[cq * kTM + lr] = acc;
  __syncthreads();
  if (warp >= 2 && cq == 0 && j0 + lr < a.T)
    a.score[(int64_t)bh * a.T + j0 + lr] = (mrg[lr] + mrg[kTM + lr]) + (mrg[2 * kTM + lr] + mrg[3 * kTM + lr]);
  cta_teardown(ctl, tbase);
}

// ---------------------------------------------------------------- pass 2 over one query block
// When the query rows fit one 128-row block (an observation window of at most 128 / G rows), pass 2's
// CTAs would each meet a single tile; instead a CTA holds the query block and its statistics (the
// MMA's B) and streams a run of 128-key tiles as the MMA's A.  Each key's sum over the block's rows
// comes from the two column halves of the tile and is added to the zeroed score (two float adds onto
// 0, so the result does not depend on their order).
template <int D>
__global__ void __launch_bounds__(kThr, 1)
    colsum_window_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                         const ScoreArgs a, int tiles_per_cta) {
  using L = Layout<D, kTN2>;
  static_assert(L::ATOM_A == L::ATOM_B, "A and B tiles of 128 rows");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = align1024(smem_raw);
  Ctl<kTN2>* ctl = reinterpret_cast<Ctl<kTN2>*>(sm + L::CTL_OFF);
  const int bh = (int)blockIdx.y;
  const int b = bh / a.Hkv, kvh = bh % a.Hkv;
  const int warp = threadIdx.x >> 5;
  const int lq = warp & 3, cq = (warp - 2) >> 2;         // (epilogue warps) lane quarter; group x half
  const int hf = cq & 1;                                 // column half = rows hf * 64 .. of the block
  const int lr = lq * 32 + (threadIdx.x & 31);           // accumulator lane = key of the tile
  const int64_t t_begin = (int64_t)blockIdx.x * tiles_per_cta;
  const int ntiles = (int)std::max<int64_t>(0, std::min<int64_t>(ceil_div_dev(a.T, kBlk) - t_begin, tiles_per_cta));
  const float2* stats = a.row_st + (int64_t)bh * a.n_ksplit * kTM;   // the unit's one block, split 0

  const uint32_t tbase = cta_setup(ctl);
  run_roles<D, kTN2, false, true>(
      sm, ctl, tbase, ntiles,
      [&](uint64_t* bar) {                // the query block and its statistics
        tc_mbar_expect_tx(bar, L::TILE_A + kStatBytes);
        for (int at = 0; at < D / 64; ++at)
          tma_load_4d(sm + L::A_OFF + at * L::ATOM_A, &qmap, at * 64, 0, kvh * a.G, b, bar);
        bulk_load(sm + L::ST_OFF, stats, kStatBytes, bar);
      },
      [&](int t, int s, uint64_t* bar) {  // 128 keys
        tc_mbar_expect_tx(bar, L::TILE_B);
        for (int at = 0; at < D / 64; ++at)
          tma_load_4d(sm + L::B_OFF + s * L::TILE_B + at * L::ATOM_B, &kmap, at * 64, (int)((t_begin + t) * kBlk),
                      kvh, b, bar);
      },
      [&](int t, uint32_t col, int) {
        const int64_t jt = (t_begin + t) * kBlk;
        const int64_t jrel = jt + lr - a.pos0;   // rows i >= jrel see this key
        const float4* s4 = reinterpret_cast<const float4*>(sm + L::ST_OFF) + hf * 32;
        const uint64_t sc2 = pk2(a.scale_log2, a.scale_log2);
        uint64_t sp2[2] = {0ull, 0ull};
        float v[64];
        tc_ld64(col + ((uint32_t)(lq * 32) << 16), v);
        if (0 >= jt + kBlk - 1 - a.pos0) {   // every row of the window sees every key of the tile
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            const float4 w = s4[q];
            const float2 x = upk2(ffma2(pk2(v[2 * q], v[2 * q + 1]), sc2, pk2(w.x, w.y)));
            sp2[q & 1] = ffma2(pk2(ex2_approx(x.x), ex2_approx(x.y)), pk2(w.z, w.w), sp2[q & 1]);
          }
        } else {
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            const float4 w = s4[q];
            const int c = hf * 64 + 2 * q;
            const float2 x = upk2(ffma2(pk2(v[2 * q], v[2 * q + 1]), sc2, pk2(w.x, w.y)));
            const float p0 = (c & (a.rpb - 1)) >= jrel ? ex2_approx(x.x) * w.z : 0.f;
            const float p1 = ((c + 1) & (a.rpb - 1)) >= jrel ? ex2_approx(x.y) * w.w : 0.f;
            sp2[q & 1] = fadd2(sp2[q & 1], pk2(p0, p1));
          }
        }
        const float2 s0 = upk2(sp2[0]), s1 = upk2(sp2[1]);
        if (jt + lr < a.T) atomicAdd(a.score + (int64_t)bh * a.T + jt + lr, (s0.x + s0.y) + (s1.x + s1.y));
      });
  cta_teardown(ctl, tbase);
}

// ---------------------------------------------------------------- host side
using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                 const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encoder() {
  static const EncodeTiled fn = []() -> EncodeTiled {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return nullptr;
    return reinterpret_cast<EncodeTiled>(p);
  }();
  return fn;
}

// fp16 [n3][n2][rows][D] read in boxes of 64 x box_rows x box2 x 1 with the 128-byte swizzle (a box's
// 128-byte rows land in shared memory in order: row, then dimension 2); rows past the end read as zero
cudaError_t make_map(CUtensorMap* m, const void* base, int D, int64_t rows, int64_t n2, int64_t n3, int box_rows,
                     int box2) {
  const EncodeTiled enc = encoder();
  if (enc == nullptr) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)rows, (cuuint64_t)n2, (cuuint64_t)n3};
  const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)rows * D * 2, (cuuint64_t)n2 * rows * D * 2};
  const cuuint32_t box[4] = {64, (cuuint32_t)box_rows, (cuuint32_t)box2, 1};
  const cuuint32_t es[4] = {1, 1, 1, 1};
  const CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <int D>
cudaError_t launch_scores_t(const CUtensorMap& qm, const CUtensorMap& k256, const CUtensorMap& k128,
                            const ScoreArgs& a, int units, int keyblocks, cudaStream_t st) {
  // one CTA per SM (it takes all 512 tensor-memory columns), so no allocation waits
  constexpr int smem1 = std::max(Layout<D, kTN1>::ALLOC, 116 * 1024);
  constexpr int smem2 = std::max(Layout<D, kTN2>::ALLOC, 116 * 1024);
  static_assert(smem1 <= 227 * 1024 && smem2 <= 227 * 1024, "shared memory");
  cudaError_t e = cudaFuncSetAttribute(rowstats_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem1);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(colsum_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem2);
  if (e != cudaSuccess) return e;
  rowstats_tc_kernel<D><<<dim3(a.n_ksplit, a.rowblocks, units), kThr, smem1, st>>>(qm, k256, a);
  e = cudaPeekAtLastError();
  if (e != cudaSuccess) return e;
  rowmerge_kernel<<<(unsigned)((int64_t)units * a.rowblocks), kBlk, 0, st>>>(a.row_st, a.n_ksplit, a.rpb,
                                                                            a.rowblocks, a.R);
  e = cudaPeekAtLastError();
  if (e != cudaSuccess) return e;
  if (a.rowblocks == 1) {                 // one query block: hold it, stream runs of key tiles
    e = cudaFuncSetAttribute(colsum_window_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem2);
    if (e == cudaSuccess) e = cudaMemsetAsync(a.score, 0, (size_t)units * a.T * sizeof(float), st);
    if (e != cudaSuccess) return e;
    const int64_t per = ceil_div((int64_t)keyblocks, ceil_div(kNumSMs, (int64_t)units));
    colsum_window_kernel<D><<<dim3((unsigned)ceil_div((int64_t)keyblocks, per), units), kThr, smem2, st>>>(
        qm, k128, a, (int)per);
    return cudaPeekAtLastError();
  }
  colsum_tc_kernel<D><<<dim3(keyblocks, units), kThr, smem2, st>>>(qm, k128, a);
  return cudaPeekAtLastError();
}

// The timeout path of role_wait, exercised without a fault: an mbarrier that nothing arrives on
__global__ void wait_selftest_kernel(uint64_t ns) {
  __shared__ uint64_t bar;
  __shared__ int fail;
  if (threadIdx.x == 0) {
    tc_mbar_init(&bar, 1);
    tc_fence_mbar_init();
    fail = 0;
  }
  __syncthreads();
  if (threadIdx.x == 0) role_wait(&bar, 0, &fail, ns);
}

}  // namespace

cudaError_t launch_wait_selftest(int ms, cudaStream_t st) {
  wait_selftest_kernel<<<1, 32, 0, st>>>((uint64_t)ms * 1000000ull);
  return cudaPeekAtLastError();
}

cudaError_t launch_prefill_scores(const mkv_config& c, const void* q, int64_t q_rows, int64_t T,
                                  const void* full_k, const PrefillWs& ws, cudaStream_t st) {
  if (q_rows <= 0 || T <= 0) return cudaSuccess;
  ScoreArgs a{};
  a.R = q_rows;
  a.T = T;
  a.pos0 = T - q_rows;
  a.Hq = c.Hq;
  a.Hkv = c.Hkv;
  a.G = c.Hq / c.Hkv;
  a.rpb = kTM / a.G;
  a.rowblocks = (int)ceil_div(q_rows, a.rpb);
  const float scale = c.softmax_scale > 0.f ? c.softmax_scale : 1.0f / sqrtf((float)c.D);
  a.scale_log2 = scale * kLog2e;
  const int units = c.B * c.Hkv;
  const int64_t tiles = ceil_div(T, kTN1);               // pass 1's key tiles
  if (a.rowblocks > 65535 || T > INT32_MAX - kTN1) return cudaErrorInvalidConfiguration;
  // split the key range only when the row blocks are fewer than the SMs (an observation window);
  // the splits' partials stay within the row-statistics workspace of B Hq (T + 128) entries
  int64_t ns = ceil_div(kNumSMs, (int64_t)a.rowblocks * units);
  ns = std::min<int64_t>(ns, std::min<int64_t>(tiles, (T + kTM) / ((int64_t)a.rowblocks * a.rpb)));
  ns = std::max<int64_t>(ns, 1);
  a.tiles_per_split = (int)ceil_div(tiles, ns);
  a.n_ksplit = (int)ceil_div(tiles, a.tiles_per_split);
  a.row_st = ws.row_st;
  a.score = ws.score;
  CUtensorMap qm, k256, k128;
  // q [B][Hq][R][D] in boxes of G heads x rpb rows; k [B][Hkv][T][D] in 256- and 128-key boxes
  cudaError_t e = make_map(&qm, q, c.D, q_rows, c.Hq, c.B, a.rpb, a.G);
  if (e == cudaSuccess) e = make_map(&k256, full_k, c.D, T, c.Hkv, c.B, kTN1, 1);
  if (e == cudaSuccess) e = make_map(&k128, full_k, c.D, T, c.Hkv, c.B, kBlk, 1);
  if (e != cudaSuccess) return e;
  const int keyblocks = (int)ceil_div(T, kBlk);         // pass 2: one CTA per 128 keys
  if (c.D == 128) return launch_scores_t<128>(qm, k256, k128, a, units, keyblocks, st);
  return launch_scores_t<64>(qm, k256, k128, a, units, keyblocks, st);
}

}  // namespace mkv
