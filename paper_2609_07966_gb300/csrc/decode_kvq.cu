// KVQuant decode attention with dequantization fused into QK^T / softmax / PV
// (Section 2.1, KVQuant paragraph: keys quantized per channel before the
// rotary embedding, values per token, outliers kept in fp16).
//
// For each token t of the cache and each query head h of the group:
//   k_t = rope_t(dq_K(t)) with outliers restored before the rotation,
//   v_t = lo_t + scale_t * tbl[code] with outliers restored,
//   out_h = softmax_t(scale q_h . k_t) v_t.
//
// GB300 design: one CTA (8 warps) per (batch, kv-head, split); packed codes are
// staged by cp.async (double buffer, 64 tokens per chunk).  Phase 1: each
// thread dequantizes half of one token's key or value row from shared tables
// (all lanes of a warp read the same channel's table -> conflict-free), rotates
// key pairs (i, i + D/2) by the token's offset delta from its 32-token base,
// and writes fp16 tiles (keys as hi + lo halves so the tensor-core product
// keeps fp32 accuracy).  The base rotation R(tb) is applied to the query
// instead (q . R(tb+d) k = (R(tb)^T q) . (R(d) k)), so only the 32-entry delta
// table is needed.  Phase 2: tensor-core QK^T (hi*hi + hi*lo + lo*hi), online
// softmax and PV as in the fp16 kernel.  Tile columns hold pair i at columns
// (2i, 2i+1) = channels (i, i + D/2); the output is un-permuted at the end.
#include <math.h>

#include "mkv_common.cuh"
#include "mkv_internal.h"
#include "mkv_merge.cuh"

namespace mkv {

namespace {

constexpr int kThr = 256;

struct KvqArgs {
  const __half* q;        // [B][Hq][D]
  const uint8_t* k_codes; // [B][Hkv][T_cap][row]
  const uint8_t* v_codes;
  const float2* v_params; // [B][Hkv][T_cap]
  const uint32_t* v_out;  // [B][Hkv][T_cap][n_v]
  const int32_t* k_out_off;
  const uint32_t* k_out;
  const float* k_dq;      // [Hkv][D][K]
  const uint16_t* v_tbl;  // [Hkv][D][K]
  const float2* rope;     // [rope_len][D/2]
  int64_t rope_len;
  const int32_t* T_len;
  int64_t T_cap, k_out_cap;
  int Hq, Hkv, G, log2G, n_v;
  int chunks_per_split, n_split;
  float scale_log2;
  float* part_m;
  float* part_l;
  float* part_o;
  MergeArgs merge;
};

template <int D, int BITS>
struct KvqLayout {
  static constexpr int NP = D / 2;
  static constexpr int K = 1 << BITS;
  static constexpr int ROWB = D * BITS / 8;                  // packed bytes per token row
  static constexpr int CP = (ROWB % 16 == 0) ? 16 : 8;       // cp.async granularity
  static constexpr int SROW0 = (ROWB + 15) / 16 * 16;
  static constexpr int SROW = ((SROW0 / 16) % 2 == 0) ? SROW0 + 16 : SROW0;   // odd # of 16B
  static constexpr int TILE = kChunk * D * 2;                // fp16 tile bytes
  static constexpr int NVS = 4;                              // value outliers staged per token (<=)
  static constexpr int KE_CAP = 128;                         // key outliers staged per chunk (<=)
  // one pipeline stage: codes, then the chunk's per-token side data
  static constexpr int S_KC = 0;                             // [64][SROW] key codes
  static constexpr int S_VC = S_KC + kChunk * SROW;          // [64][SROW] value codes
  static constexpr int S_VP = S_VC + kChunk * SROW;          // [64] float2 (lo, scale)
  static constexpr int S_KE = S_VP + kChunk * 8;             // [KE_CAP] uint32 key outliers of the chunk
  static constexpr int S_VO = S_KE + KE_CAP * 4;             // [64][NVS] uint32 value outliers
  static constexpr int STAGE = S_VO + kChunk * NVS * 4;
  // byte offsets
  static constexpr int DTAB = 0;                             // [NP][32] float2
  static constexpr int KDQ = DTAB + NP * 32 * 8;             // [D][K] float
  static constexpr int VTB = KDQ + D * K * 4;                // [D][K] float
  static constexpr int QHI = VTB + D * K * 4;                // [2 bases][8][NP] half2 (rotated query, hi)
  static constexpr int QLO = QHI + 2 * 8 * NP * 4;           // [2][8][NP] half2 (lo)
  static constexpr int KOFF = QLO + 2 * 8 * NP * 4;          // [3 chunks][68] int32 key-outlier CSR offsets
  static constexpr int STG = KOFF + 3 * 68 * 4;              // [2 stages][STAGE]
  static constexpr int KHI = STG + 2 * STAGE;
  static constexpr int KLO = KHI + TILE;
  static constexpr int VT = KLO + TILE;
  static constexpr int BYTES = VT + TILE;
};

// the `bits`-wide code of channel-in-pair `which` for pair j of a thread's word array
template <int BITS, int NW>
__device__ __forceinline__ void pair_codes(const uint32_t (&w)[NW], int j, int& lo, int& hi) {
  const int bit = 2 * BITS * j;
  const int wi = bit >> 5, sh = bit & 31;
  uint32_t x = w[wi] >> sh;
  if (sh + 2 * BITS > 32 && wi + 1 < NW) x |= w[wi + 1] << (32 - sh);
  lo = (int)(x & ((1u << BITS) - 1u));
  hi = (int)((x >> BITS) & ((1u << BITS) - 1u));
}

// pair j's codes read from a packed row in shared memory (any j)
template <int BITS>
__device__ __forceinline__ void pair_codes_row(const uint8_t* row, int j, int& lo, int& hi) {
  const int bit = 2 * BITS * j;
  const int wi = bit >> 5, sh = bit & 31;
  const uint32_t w0 = reinterpret_cast<const uint32_t*>(row)[wi];
  const uint32_t w1 = reinterpret_cast<const uint32_t*>(row)[wi + 1];
  const uint32_t x = __funnelshift_r(w0, w1, sh);
  lo = (int)(x & ((1u << BITS) - 1u));
  hi = (int)((x >> BITS) & ((1u << BITS) - 1u));
}

__device__ __forceinline__ void split_hi_lo(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(a, b);
  const float2 hf = __half22float2(h);
  const __half2 l = __floats2half2_rn(a - hf.x, b - hf.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// D(16x8 f32) += A(16x8 f16, row) * B(8x8 f16, col)
__device__ __forceinline__ void mma1688(float c[4], uint32_t a0, uint32_t a1, uint32_t b0) {
  asm volatile(
      "mma.sync.aligned.m16n8k8.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5}, {%6}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(b0));
}

// byte offset of (row, 16B chunk) in a swizzled fp16 tile of D columns
template <int D>
__device__ __forceinline__ int tile_off(int row, int ch) {
  return row * D * 2 + ((ch ^ (row & 7)) << 4);
}

template <int D, int BITS>
__global__ void __launch_bounds__(kThr, 2) decode_kvq_kernel(const KvqArgs a) {
  using Lay = KvqLayout<D, BITS>;
  constexpr int NP = Lay::NP, K = Lay::K, ROWB = Lay::ROWB, SROW = Lay::SROW;
  constexpr int KC = D / 16;
  // Phase 1 splits each row's pairs into GROUPS groups of whole 32-bit words.
  constexpr int GROUPS = ((NP / 4) * 2 * BITS) % 32 == 0 ? 4 : 2;
  constexpr int QP = NP / GROUPS;                         // pairs per group
  constexpr int NWQ = QP * 2 * BITS / 32;                 // code words per group
  constexpr bool SPLIT_KV = GROUPS == 2;                  // then a thread does K or V, not both
  extern __shared__ __align__(128) uint8_t smem[];
  float2* dtab = reinterpret_cast<float2*>(smem + Lay::DTAB);
  float* kdq = reinterpret_cast<float*>(smem + Lay::KDQ);
  float* vtb = reinterpret_cast<float*>(smem + Lay::VTB);
  uint32_t* qhi = reinterpret_cast<uint32_t*>(smem + Lay::QHI);
  uint32_t* qlo = reinterpret_cast<uint32_t*>(smem + Lay::QLO);
  uint8_t* stg = smem + Lay::STG;
  int32_t* kring = reinterpret_cast<int32_t*>(smem + Lay::KOFF);
  uint8_t* khi_t = smem + Lay::KHI;
  uint8_t* klo_t = smem + Lay::KLO;
  uint8_t* v_t = smem + Lay::VT;

  const int split = blockIdx.x;
  const int64_t bh = blockIdx.y;
  const int b = (int)(bh / a.Hkv), kvh = (int)(bh % a.Hkv);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, r = lane & 3;
  const int n_len = (int)min((int64_t)a.T_len[b], a.T_cap);
  const int64_t v_begin = (int64_t)split * a.chunks_per_split * kChunk;
  int64_t v_end = v_begin + (int64_t)a.chunks_per_split * kChunk;
  if (v_end > n_len) v_end = n_len;
  const int nchunks = v_end > v_begin ? (int)ceil_div_dev(v_end - v_begin, kChunk) : 0;

  const uint8_t* kc_base = a.k_codes + bh * a.T_cap * ROWB;
  const uint8_t* vc_base = a.v_codes + bh * a.T_cap * ROWB;

  const bool stage_vout = a.n_v <= Lay::NVS;
  auto load_chunk = [&](int c, int stage) {
    uint8_t* dst = stg + stage * Lay::STAGE;
    const int64_t c0 = v_begin + (int64_t)c * kChunk;
    constexpr int PER_ROW = ROWB / Lay::CP;
    for (int e = tid; e < 2 * kChunk * PER_ROW; e += kThr) {
      const int kv = e / (kChunk * PER_ROW);
      const int rem = e % (kChunk * PER_ROW);
      const int row = rem / PER_ROW, piece = rem % PER_ROW;
      const int64_t s = c0 + row;
      const bool ok = s < n_len;
      const uint8_t* src = (kv ? vc_base : kc_base) + (ok ? s : 0) * ROWB + piece * Lay::CP;
      uint8_t* d = dst + (kv ? Lay::S_VC : Lay::S_KC) + row * SROW + piece * Lay::CP;
      if (Lay::CP == 16) {
        cp_async16(d, src, ok ? 16 : 0);
      } else {
        cp_async8(d, src, ok ? 8 : 0);
      }
    }
    if (tid < kChunk) {                          // value (lo, scale)
      const int64_t s = c0 + tid;
      const bool ok = s < n_len;
      cp_async8(dst + Lay::S_VP + tid * 8, a.v_params + bh * a.T_cap + (ok ? s : 0), ok ? 8 : 0);
    }
    if (stage_vout && a.n_v > 0) {
      for (int e = tid; e < kChunk * a.n_v; e += kThr) {
        const int row = e / a.n_v, k = e % a.n_v;
        const int64_t s = c0 + row;
        const bool ok = s < n_len;
        cp_async4(dst + Lay::S_VO + (row * Lay::NVS + k) * 4, a.v_out + (bh * a.T_cap + (ok ? s : 0)) * a.n_v + k,
                  ok ? 4 : 0);
      }
    }
  };

  // key-outlier CSR offsets run one chunk ahead of the codes so that each
  // chunk's outlier entries can be staged together with its codes
  auto load_koff = [&](int c) {
    if (tid <= kChunk) {
      const int64_t s = min(v_begin + (int64_t)c * kChunk + tid, (int64_t)n_len);
      cp_async4(kring + (c % 3) * 68 + tid, a.k_out_off + bh * (a.T_cap + 1) + s, 4);
    }
  };
  auto load_kents = [&](int c, int stage) {      // needs chunk c's offsets in kring
    const int32_t* ko = kring + (c % 3) * 68;
    const int e0 = ko[0];
    const int n = min((int)min((int64_t)ko[kChunk], a.k_out_cap) - e0, Lay::KE_CAP);
    for (int e = tid; e < n; e += kThr)
      cp_async4(stg + stage * Lay::STAGE + Lay::S_KE + e * 4, a.k_out + bh * a.k_out_cap + e0 + e, 4);
  };
  if (nchunks > 0) {
    load_koff(0);
    if (nchunks > 1) load_koff(1);
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
    load_chunk(0, 0);
    load_kents(0, 0);
    if (nchunks > 2) load_koff(2);
    cp_async_commit();
  }
  // CTA-resident tables: rotations by delta in [0, 32), dequant tables of this kv-head
  for (int e = tid; e < NP * 32; e += kThr) {      // coalesced read of rows 0..31, transposed
    const int d = e / NP, i = e % NP;
    dtab[i * 32 + d] = a.rope[(int64_t)d * NP + i];
  }
  for (int e = tid; e < D * K; e += kThr) {
    kdq[e] = a.k_dq[(int64_t)kvh * D * K + e];
    vtb[e] = __half2float(__ushort_as_half(a.v_tbl[(int64_t)kvh * D * K + e]));
  }
  // This thread's fixed share of the rotated-query table: element e = (base, head, pair) for
  // e = tid + k*kThr.  Its raw query pair is loaded once; the rotation of its base is
  // prefetched one chunk ahead.
  constexpr int kQE = 2 * 8 * NP / kThr;                   // at most G = 8
  float qx[kQE], qy[kQE];
  float2 qcs[kQE];
  const int nqe = 2 * a.G * NP;
#pragma unroll
  for (int k = 0; k < kQE; ++k) {
    const int e = tid + k * kThr;
    qx[k] = qy[k] = 0.f;
    qcs[k] = make_float2(1.f, 0.f);
    if (e < nqe) {
      const int t = e / NP, i = e % NP;
      const int gg = t & (a.G - 1), base = t >> a.log2G;
      const __half* qr = a.q + ((int64_t)b * a.Hq + (int64_t)kvh * a.G + gg) * D;
      qx[k] = __half2float(qr[i]);
      qy[k] = __half2float(qr[i + NP]);
      if (nchunks > 0) qcs[k] = a.rope[min(v_begin + 32 * base, a.rope_len - 1) * NP + i];
    }
  }

  float o[D / 8][2];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = 0.f;
  float m_run = -INFINITY, l_part = 0.f;
  const int t4 = warp & 3;                 // phase 1: pair group (or K/V role) of this warp
  const int tok = (warp >> 2) * 32 + lane; // phase 1: this thread's token in the chunk
  const int dl = tok & 31;                 // its offset from its 32-token base

  for (int c = 0; c < nchunks; ++c) {
    cp_async_wait<0>();
    __syncthreads();
    if (c + 1 < nchunks) {
      load_chunk(c + 1, (c + 1) & 1);
      load_kents(c + 1, (c + 1) & 1);
    }
    if (c + 2 < nchunks) load_koff(c + 2);
    cp_async_commit();
    const int64_t t0 = v_begin + (int64_t)c * kChunk;      // position of the chunk's first token
    const uint8_t* st = stg + (c & 1) * Lay::STAGE;
    const float2* vpar = reinterpret_cast<const float2*>(st + Lay::S_VP);
    const int32_t* koff = kring + (c % 3) * 68;
    const uint32_t* kents = reinterpret_cast<const uint32_t*>(st + Lay::S_KE);
    const int kbase = koff[0];
    const int kstaged = min((int)min((int64_t)koff[kChunk], a.k_out_cap) - kbase, Lay::KE_CAP);
    const uint32_t* vouts = reinterpret_cast<const uint32_t*>(st + Lay::S_VO);

    // ---- query rotated back by each 32-token base tb: R(tb)^T q as hi/lo fp16 pairs, stored in
    //      the order the mma fragments read: pair i = kc*8 + 4*hf + r at word kc*8 + 2*r + hf
#pragma unroll
    for (int k = 0; k < kQE; ++k) {
      const int e = tid + k * kThr;
      if (e < nqe) {
        const int t = e / NP, i = e % NP;
        const int gg = t & (a.G - 1), base = t >> a.log2G;
        const float x = qx[k], y = qy[k];
        const float2 cs = qcs[k];
        const int wpos = (i / 8) * 8 + (i % 4) * 2 + ((i % 8) / 4);
        split_hi_lo(x * cs.x + y * cs.y, y * cs.x - x * cs.y, qhi[(base * 8 + gg) * NP + wpos],
                    qlo[(base * 8 + gg) * NP + wpos]);
        if (c + 1 < nchunks) qcs[k] = a.rope[min(t0 + kChunk + 32 * base, a.rope_len - 1) * NP + i];
      }
    }

    // ---- phase 1: dequantize one pair group of the thread's token (keys and/or values)
    {
      const int64_t slot = t0 + tok;
      const bool valid = slot < n_len;
      const bool do_k = SPLIT_KV ? (t4 < 2) : true;
      const bool do_v = SPLIT_KV ? (t4 >= 2) : true;
      const int grp = SPLIT_KV ? (t4 & 1) : t4;
      if (do_k) {
        const uint8_t* rowfull = st + Lay::S_KC + tok * SROW;
        uint32_t w[NWQ];
#pragma unroll
        for (int k = 0; k < NWQ; ++k) w[k] = reinterpret_cast<const uint32_t*>(rowfull)[grp * NWQ + k];
#pragma unroll
        for (int jj = 0; jj < QP; jj += 4) {
          uint32_t ph[4], pl[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int j = jj + u, i = grp * QP + j;
            int clo, chi;
            pair_codes<BITS, NWQ>(w, j, clo, chi);
            // rows past the cache end were zero-filled: finite keys, masked in phase 2
            const float x = kdq[i * K + clo];
            const float y = kdq[(i + NP) * K + chi];
            const float2 cs = dtab[i * 32 + dl];
            split_hi_lo(x * cs.x - y * cs.y, y * cs.x + x * cs.y, ph[u], pl[u]);
          }
          const int ch = (grp * QP + jj) / 4;
          *reinterpret_cast<uint4*>(khi_t + tile_off<D>(tok, ch)) = make_uint4(ph[0], ph[1], ph[2], ph[3]);
          *reinterpret_cast<uint4*>(klo_t + tile_off<D>(tok, ch)) = make_uint4(pl[0], pl[1], pl[2], pl[3]);
        }
        // key outliers of this token in this group: recompute their pair exactly
        if (valid) {
          const int e0 = koff[tok], e1 = (int)min((int64_t)koff[tok + 1], a.k_out_cap);
          const uint32_t* gents = a.k_out + bh * a.k_out_cap;
          auto ent = [&](int e) { return e - kbase < kstaged ? kents[e - kbase] : gents[e]; };
          for (int e = e0; e < e1; ++e) {
            const int chn = (int)(ent(e) >> 16);
            const int i = chn % NP;
            if (i / QP != grp) continue;
            int clo, chi;
            pair_codes_row<BITS>(rowfull, i, clo, chi);
            float x = kdq[i * K + clo], y = kdq[(i + NP) * K + chi];
            for (int f = e0; f < e1; ++f) {
              const uint32_t ef = ent(f);
              const int cf = (int)(ef >> 16);
              if (cf == i) x = h2f((uint16_t)(ef & 0xffffu));
              if (cf == i + NP) y = h2f((uint16_t)(ef & 0xffffu));
            }
            const float2 cs = dtab[i * 32 + dl];
            uint32_t ph, pl;
            split_hi_lo(x * cs.x - y * cs.y, y * cs.x + x * cs.y, ph, pl);
            const int byte = tile_off<D>(tok, i / 4) + (i % 4) * 4;
            *reinterpret_cast<uint32_t*>(khi_t + byte) = ph;
            *reinterpret_cast<uint32_t*>(klo_t + byte) = pl;
          }
        }
      }
      if (do_v) {
        const uint8_t* rowfull = st + Lay::S_VC + tok * SROW;
        uint32_t w[NWQ];
#pragma unroll
        for (int k = 0; k < NWQ; ++k) w[k] = reinterpret_cast<const uint32_t*>(rowfull)[grp * NWQ + k];
        const float2 lp = vpar[tok];
#pragma unroll
        for (int jj = 0; jj < QP; jj += 4) {
          uint32_t pv[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int j = jj + u, i = grp * QP + j;
            int clo, chi;
            pair_codes<BITS, NWQ>(w, j, clo, chi);
            // rows past the cache end have lo = scale = 0 (zero-filled): value 0
            const float x = fmaf(lp.y, vtb[i * K + clo], lp.x);
            const float y = fmaf(lp.y, vtb[(i + NP) * K + chi], lp.x);
            pv[u] = pack_half2(x, y);
          }
          const int ch = (grp * QP + jj) / 4;
          *reinterpret_cast<uint4*>(v_t + tile_off<D>(tok, ch)) = make_uint4(pv[0], pv[1], pv[2], pv[3]);
        }
        if (valid) {
          const uint32_t* ents = stage_vout ? vouts + tok * Lay::NVS : a.v_out + (bh * a.T_cap + slot) * a.n_v;
          for (int e = 0; e < a.n_v; ++e) {
            const uint32_t ev = ents[e];
            const int chn = (int)(ev >> 16);
            const int i = chn % NP;
            if (i / QP != grp) continue;
            const int col = chn < NP ? 2 * chn : 2 * (chn - NP) + 1;
            *reinterpret_cast<uint16_t*>(v_t + tile_off<D>(tok, col / 8) + (col % 8) * 2) =
                (uint16_t)(ev & 0xffffu);
          }
        }
      }
    }
    __syncthreads();

    // ---- phase 2: warps 0-3 each own 16 tokens of the chunk and every output dim
    if (warp < 4) {
      const bool real = g < a.G;
      const int base = warp >> 1;                            // tokens 0-31: base t0, 32-63: t0 + 32
      const uint2* qh2 = reinterpret_cast<const uint2*>(qhi + (base * 8 + (real ? g : 0)) * NP);
      const uint2* ql2 = reinterpret_cast<const uint2*>(qlo + (base * 8 + (real ? g : 0)) * NP);
      float sc[2][4];
#pragma unroll
      for (int i = 0; i < 4; ++i) sc[0][i] = sc[1][i] = 0.f;
      const int mi = lane >> 3, rowi = lane & 7;
      const int t0w = warp * 16;
      const int tokk = t0w + (mi >> 1) * 8 + rowi;
#pragma unroll
      for (int kc = 0; kc < KC; ++kc) {
        const uint2 ah = real ? qh2[kc * 4 + r] : make_uint2(0u, 0u);
        const uint2 al = real ? ql2[kc * 4 + r] : make_uint2(0u, 0u);
        uint32_t bh[4], bl[4];
        const int ch = kc * 2 + (mi & 1);
        ldsm_x4(bh, khi_t + tile_off<D>(tokk, ch));
        ldsm_x4(bl, klo_t + tile_off<D>(tokk, ch));
        mma16816(sc[0], ah.x, 0u, ah.y, 0u, bh[0], bh[1]);
        mma16816(sc[1], ah.x, 0u, ah.y, 0u, bh[2], bh[3]);
        mma16816(sc[0], ah.x, 0u, ah.y, 0u, bl[0], bl[1]);
        mma16816(sc[1], ah.x, 0u, ah.y, 0u, bl[2], bl[3]);
        mma16816(sc[0], al.x, 0u, al.y, 0u, bh[0], bh[1]);
        mma16816(sc[1], al.x, 0u, al.y, 0u, bh[2], bh[3]);
      }
      const int tk[4] = {t0w + 2 * r, t0w + 2 * r + 1, t0w + 8 + 2 * r, t0w + 9 + 2 * r};
      float x[4] = {sc[0][0], sc[0][1], sc[1][0], sc[1][1]};
      float mx = -INFINITY;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        x[i] = (t0 + tk[i] < n_len) ? x[i] * a.scale_log2 : -INFINITY;
        mx = fmaxf(mx, x[i]);
      }
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float m_new = fmaxf(m_run, mx);
      float p[4] = {0.f, 0.f, 0.f, 0.f};
      float alpha = 1.f;
      if (m_new != -INFINITY) {
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
      const int tokv = t0w + (mi & 1) * 8 + rowi;
#pragma unroll
      for (int j = 0; j < D / 16; ++j) {
        uint32_t bv[4];
        ldsm_x4_t(bv, v_t + tile_off<D>(tokv, 2 * j + (mi >> 1)));
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

  // ---- merge the eight warps' (m, l, o) per query row; o is in the permuted column order
  l_part += __shfl_xor_sync(0xffffffffu, l_part, 1);
  l_part += __shfl_xor_sync(0xffffffffu, l_part, 2);
  float* wm = reinterpret_cast<float*>(khi_t);              // [8 warps][8 rows]
  float* wl = wm + 64;                                       // [8][8]
  float* wo = wl + 64;                                       // [8][8][D]  natural channel order
  if (g < a.G) {
    if (r == 0) {
      wm[warp * 8 + g] = m_run;
      wl[warp * 8 + g] = l_part;
    }
#pragma unroll
    for (int dt = 0; dt < D / 8; ++dt) {
      const int chn = dt * 4 + r;                            // column dt*8 + 2r -> channel dt*4 + r
      wo[(warp * 8 + g) * D + chn] = o[dt][0];
      wo[(warp * 8 + g) * D + chn + NP] = o[dt][1];
    }
  }
  __syncthreads();
  for (int e = tid; e < a.G * D; e += kThr) {
    const int row = e / D, d = e % D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 8; ++w) M = fmaxf(M, wm[w * 8 + row]);
    float L = 0.f, O = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < 8; ++w) {
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
  merge_if_last<D, kThr>(a.merge, bh, b, kvh, reinterpret_cast<float*>(stg), 2 * Lay::STAGE / 4);
}

template <int D, int BITS>
cudaError_t launch_kvq_t(const KvqArgs& a, int units, int n_split, cudaStream_t st) {
  using Lay = KvqLayout<D, BITS>;
  static_assert(Lay::BYTES <= 113 * 1024, "two CTAs per SM");
  cudaError_t e = cudaFuncSetAttribute(decode_kvq_kernel<D, BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Lay::BYTES);
  if (e != cudaSuccess) return e;
  decode_kvq_kernel<D, BITS><<<dim3(n_split, units), kThr, Lay::BYTES, st>>>(a);
  return cudaPeekAtLastError();
}

}  // namespace

cudaError_t launch_decode_kvquant(const mkv_config& c, const void* q, const mkv_cache& cache,
                                  const mkv_quant_params& qp, void* out, const DecodeWs& ws, const Split& sp,
                                  cudaStream_t st) {
  KvqArgs a{};
  a.q = static_cast<const __half*>(q);
  a.k_codes = cache.k_codes;
  a.v_codes = cache.v_codes;
  a.v_params = reinterpret_cast<const float2*>(cache.v_params);
  a.v_out = cache.v_out;
  a.k_out_off = cache.k_out_off;
  a.k_out = cache.k_out;
  a.k_dq = qp.k_dq;
  a.v_tbl = qp.v_tbl;
  a.rope = reinterpret_cast<const float2*>(qp.rope);
  a.rope_len = qp.rope_len;
  a.T_len = cache.T_len;
  a.T_cap = cache.T_cap;
  a.k_out_cap = cache.k_out_cap;
  a.Hq = c.Hq;
  a.Hkv = c.Hkv;
  a.G = c.Hq / c.Hkv;
  a.log2G = a.G == 8 ? 3 : (a.G == 4 ? 2 : (a.G == 2 ? 1 : 0));
  a.n_v = std::min(c.D, (int)ceil((double)c.outlier_frac * c.D));
  a.chunks_per_split = sp.chunks_per_split;
  a.n_split = sp.n_split;
  const float scale = c.softmax_scale > 0.f ? c.softmax_scale : 1.0f / sqrtf((float)c.D);
  a.scale_log2 = scale * kLog2e;
  a.part_m = ws.part_m;
  a.part_l = ws.part_l;
  a.part_o = ws.part_o;
  a.merge = merge_args(c, ws, sp, out, false);
  const int units = c.B * c.Hkv;
  if (c.D == 128) {
    if (c.bits == 4) return launch_kvq_t<128, 4>(a, units, sp.n_split, st);
    if (c.bits == 3) return launch_kvq_t<128, 3>(a, units, sp.n_split, st);
    return launch_kvq_t<128, 2>(a, units, sp.n_split, st);
  }
  if (c.bits == 4) return launch_kvq_t<64, 4>(a, units, sp.n_split, st);
  if (c.bits == 3) return launch_kvq_t<64, 3>(a, units, sp.n_split, st);
  return launch_kvq_t<64, 2>(a, units, sp.n_split, st);
}

}  // namespace mkv
