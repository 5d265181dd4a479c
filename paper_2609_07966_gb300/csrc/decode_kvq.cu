// KVQuant decode attention with dequantization fused into QK^T / softmax / PV
// (Section 2.1, KVQuant paragraph: keys quantized per channel before the
// rotary embedding, values per token, outliers kept in fp16).
//
// For each token t of the cache and each query head h of the group:
//   k_t = rope_t(dq_K(t)) with outliers restored before the rotation,
//   v_t = lo_t + scale_t * tbl[code] with outliers restored,
//   out_h = softmax_t(scale q_h . k_t) v_t.
//
// GB300 design: one CTA of 20 warps per (batch, kv-head, split), one CTA per
// SM, warp-specialised.  Sixteen producer warps stage packed codes by cp.async
// (three 64-token chunks in flight) and dequantize chunk c into one of two
// fp16 tile buffers while four consumer warps run the tensor-core attention on
// the previous chunk from the other; named barriers (FULL / EMPTY per buffer)
// hand the buffers over.
//
// Producers: thread (token row tok, pair group g) dequantizes QP = D/16 pairs
// (i, i + D/2) of its token's key and value rows from shared per-channel tables
// (all lanes of a warp read the same channel's table -> conflict-free).  Each
// key pair is rotated by the token's offset d = tok from the chunk start with
// a rotation held in registers for the whole kernel (the chunk start's own
// rotation R(t0) is applied to the query instead:
// q . R(t0 + d) k = (R(t0)^T q) . (R(d) k)) and written as fp16 hi plus the
// negated fp16 remainder, so the tensor-core product keeps fp32 accuracy.
// Dense-and-sparse outliers are restored by the consumers before the
// attention, one thread per outlier entry (key entries are read one chunk
// ahead): a value outlier overwrites its tile entry; for a key outlier the
// pair before the rotation is recovered from the tile, the fp16 value(s) put
// in, and the pair rotated and split again.  Consumers: QK^T = q_hi k_hi - q_hi nk_lo + q_lo k_hi, online
// softmax and PV on 16-token slabs.  Tile columns hold pair i at columns
// (2i, 2i+1) = channels (i, i + D/2); the output is un-permuted at the end.
#include <math.h>

#include "mkv_common.cuh"
#include "mkv_internal.h"
#include "mkv_merge.cuh"

namespace mkv {

namespace {

constexpr int kProdWarps = 16;                         // dequantize chunk c (+ stage loads)
constexpr int kConsWarps = 4;                          // attention on chunk c-1 (tensor cores)
constexpr int kProdThr = kProdWarps * 32;
constexpr int kThr = (kProdWarps + kConsWarps) * 32;
constexpr int kGroups = 8;                             // pair groups of a token row
constexpr int kEntCap = kProdThr;                      // key-outlier entries of a chunk kept in smem
// named barriers (0 is __syncthreads)
constexpr int kBarProd = 1;                            // producers only
constexpr int kBarFull = 2;                            // + buffer: tiles of a chunk are ready
constexpr int kBarEmpty = 4;                           // + buffer: tiles may be overwritten
constexpr int kBarCons = 6;                            // consumers only
// Register split: the kernel is compiled for (and launched with) kRegLaunch registers a
// thread; producer warpgroups give registers back, the consumer warpgroup takes them.
constexpr int kRegLaunch = 96, kRegProd = 88, kRegCons = 128;
static_assert(kProdThr * kRegProd + (kThr - kProdThr) * kRegCons == kThr * kRegLaunch,
              "the register split must add up to the launch allocation");
static_assert(kProdThr % 128 == 0 && (kThr - kProdThr) % 128 == 0, "roles are whole warpgroups");

// bar.sync / bar.arrive are warp-aligned: reconverge the warp first
__device__ __forceinline__ void bar_sync(int id, int n) {
  __syncwarp();
  asm volatile("bar.sync %0, %1;\n" ::"r"(id), "r"(n) : "memory");
}
__device__ __forceinline__ void bar_arrive(int id, int n) {
  __syncwarp();
  asm volatile("bar.arrive %0, %1;\n" ::"r"(id), "r"(n) : "memory");
}

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
  int Hq, Hkv, G, n_v;
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
  static constexpr int ROWW = D * BITS / 32;                 // packed words per token row
  static constexpr int SROWW = ROWW + 1;                     // staged row stride (odd: conflict-free)
  static constexpr int QP = NP / kGroups;                    // pairs per producer thread
  static constexpr int NWG = (QP * 2 * BITS + 31) / 32;      // words holding one group's codes
  static constexpr int TILE = kChunk * D * 2;                // fp16 tile bytes
  static constexpr int NVS = 4;                              // value outliers staged per token (<=)
  static constexpr int NS = 4;                               // staged chunks (two in flight ahead)
  static constexpr int QROW = NP + 8;                        // u32 per query row (padded)
  // one pipeline stage: codes (row-major, odd word stride), then per-token side data
  static constexpr int S_KC = 0;                             // [64][SROWW] u32 key codes
  static constexpr int S_VC = S_KC + ((kChunk * SROWW * 4 + 15) / 16) * 16;
  static constexpr int S_VP = S_VC + ((kChunk * SROWW * 4 + 15) / 16) * 16;   // [64] float2
  static constexpr int S_KO = S_VP + kChunk * 8;             // [65] int32 key-outlier CSR offsets
  static constexpr int S_VO = S_KO + 68 * 4;                 // [NVS][64] u32 value outliers
  static constexpr int STAGE = S_VO + NVS * kChunk * 4;
  // one tile buffer: keys (hi, negated lo), values, and the rotated query
  static constexpr int B_KHI = 0;
  static constexpr int B_KLO = B_KHI + TILE;
  static constexpr int B_VT = B_KLO + TILE;
  static constexpr int B_QH = B_VT + TILE;                   // [8][QROW] q_hi pairs, fragment order
  static constexpr int B_QN = B_QH + 8 * QROW * 4;           // -q_hi
  static constexpr int B_QL = B_QN + 8 * QROW * 4;           // q_lo
  static constexpr int B_ENT = B_QL + 8 * QROW * 4;          // [kEntCap] u32 key-outlier entries
  static constexpr int B_KO = B_ENT + kEntCap * 4;           // [68] int32 their CSR offsets
  static constexpr int B_OWN = B_KO + 68 * 4;                // [kEntCap] u8 token of each entry
  static constexpr int B_VO = B_OWN + kEntCap;               // [NVS][64] u32 value outliers
  static constexpr int BUF = B_VO + NVS * kChunk * 4;
  // CTA layout
  static constexpr int DTAB = 0;                             // [NP][64] float2 rotation by delta
  static constexpr int KDQ = DTAB + NP * kChunk * 8;         // [D][K] float
  static constexpr int VTB = KDQ + D * K * 4;                // [D][K] float
  static constexpr int STG = VTB + D * K * 4;                // [NS][STAGE]
  static constexpr int BUFS = STG + NS * STAGE;              // [2][BUF]
  static constexpr int BYTES = BUFS + 2 * BUF;
};

// pair j's two `BITS`-wide codes from a group's realigned code words (j compile-time)
template <int BITS, int NW>
__device__ __forceinline__ void pair_codes(const uint32_t (&w)[NW], int j, int& lo, int& hi) {
  const int bit = 2 * BITS * j;
  const int wi = bit >> 5, sh = bit & 31;
  uint32_t x = w[wi] >> sh;
  if (sh + 2 * BITS > 32 && wi + 1 < NW) x |= w[wi + 1] << (32 - sh);
  lo = (int)(x & ((1u << BITS) - 1u));
  hi = (int)((x >> BITS) & ((1u << BITS) - 1u));
}

// pair i's codes read from a packed row in shared memory (any i; the row has a pad word)
template <int BITS>
__device__ __forceinline__ void pair_codes_row(const uint32_t* row, int i, int& lo, int& hi) {
  const int bit = 2 * BITS * i;
  const int wi = bit >> 5, sh = bit & 31;
  const uint32_t x = __funnelshift_r(row[wi], row[wi + 1], sh);
  lo = (int)(x & ((1u << BITS) - 1u));
  hi = (int)((x >> BITS) & ((1u << BITS) - 1u));
}

// the code words of pair group g of a staged row, shifted so the group starts at bit 0
template <int BITS, int QP, int NW>
__device__ __forceinline__ void group_words(const uint32_t* row, int g, uint32_t (&w)[NW]) {
  const int bit0 = g * QP * 2 * BITS;
  const int w0 = bit0 >> 5, sh = bit0 & 31;
  if ((QP * 2 * BITS) % 32 == 0) {         // groups are word-aligned
#pragma unroll
    for (int k = 0; k < NW; ++k) w[k] = row[w0 + k];
  } else {
    uint32_t raw[NW + 1];
#pragma unroll
    for (int k = 0; k <= NW; ++k) raw[k] = row[w0 + k];
#pragma unroll
    for (int k = 0; k < NW; ++k) w[k] = __funnelshift_r(raw[k], raw[k + 1], sh);
  }
}

// (a, b) as fp16 hi and the negated fp16 remainder (hi - x), exact in fp32
__device__ __forceinline__ void split_hi_nlo(float a, float b, uint32_t& hi, uint32_t& nlo) {
  uint32_t h;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(h) : "f"(b), "f"(a));
  float d0, d1;
  asm("{.reg .f16 l, u;\n mov.b32 {l, u}, %2;\n sub.rn.f32.f16 %0, l, %3;\n sub.rn.f32.f16 %1, u, %4;\n}"
      : "=f"(d0), "=f"(d1)
      : "r"(h), "f"(a), "f"(b));
  hi = h;
  nlo = pack_half2(d0, d1);
}

__device__ __forceinline__ void cp_async4s(uint32_t saddr, const void* gmem, int src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(saddr), "l"(gmem), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async8s(uint32_t saddr, const void* gmem, int src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;\n" ::"r"(saddr), "l"(gmem), "r"(src_bytes));
}

// byte offset of (row, 16B chunk) in a swizzled fp16 tile of D columns
template <int D>
__device__ __forceinline__ int tile_off(int row, int ch) {
  return row * D * 2 + ((ch ^ (row & 7)) << 4);
}

template <int D, int BITS>
__global__ void __launch_bounds__(kThr, 1) decode_kvq_kernel(const KvqArgs a) {
  using Lay = KvqLayout<D, BITS>;
  constexpr int NP = Lay::NP, K = Lay::K, ROWW = Lay::ROWW, SROWW = Lay::SROWW, QP = Lay::QP;
  constexpr int NWG = Lay::NWG, NS = Lay::NS, QROW = Lay::QROW;
  constexpr int KC = D / 16;
  extern __shared__ __align__(128) uint8_t smem[];
  float2* dtab = reinterpret_cast<float2*>(smem + Lay::DTAB);
  float* kdq = reinterpret_cast<float*>(smem + Lay::KDQ);
  float* vtb = reinterpret_cast<float*>(smem + Lay::VTB);
  uint8_t* stg = smem + Lay::STG;
  uint8_t* bufs = smem + Lay::BUFS;

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

  // CTA-resident tables: rotations by delta in [0, 64), dequant tables of this kv-head
  for (int e = tid; e < NP * kChunk; e += kThr) {  // coalesced read of rope rows 0..63, transposed
    const int d = e / NP, i = e % NP;
    dtab[i * kChunk + d] = a.rope[(int64_t)min((int64_t)d, a.rope_len - 1) * NP + i];
  }
  for (int e = tid; e < D * K; e += kThr) {
    kdq[e] = a.k_dq[(int64_t)kvh * D * K + e];
    vtb[e] = __half2float(__ushort_as_half(a.v_tbl[(int64_t)kvh * D * K + e]));
  }
  __syncthreads();

  // the four attention warps' (m, l, o) per query row, merged after both roles finish
  float* wm = reinterpret_cast<float*>(stg);                // [4 warps][8 rows]
  float* wl = wm + 32;                                       // [4][8]
  float* wo = wl + 32;                                       // [4][8][D]  natural channel order

  if (warp < kProdWarps) {
    // ======================= producers: stage, dequantize, rotate =======================
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(kRegProd) : "memory");
    const int ptid = tid;
    const int tok = (warp & 1) * 32 + lane;   // this thread's token row in every chunk
    const int grp = warp >> 1;                // its pairs: grp * QP .. grp * QP + QP - 1
    const uint32_t* kc_base = reinterpret_cast<const uint32_t*>(a.k_codes) + bh * a.T_cap * ROWW;
    const uint32_t* vc_base = reinterpret_cast<const uint32_t*>(a.v_codes) + bh * a.T_cap * ROWW;
    const uint32_t* gents = a.k_out + bh * a.k_out_cap;
    const bool stage_vout = a.n_v <= Lay::NVS;

    const int64_t off_base = bh * (a.T_cap + 1);

    const uint32_t stg_s = smem_addr(stg);
    constexpr int NCW = kChunk * ROWW;                       // code words per chunk (keys or values)
    constexpr int NIT = (NCW + kProdThr - 1) / kProdThr;
    auto load_chunk = [&](int c, int stage) {
      const uint32_t dst = stg_s + stage * Lay::STAGE;
      const int64_t c0 = v_begin + (int64_t)c * kChunk;     // < n_len: the chunk has a first row
      const int lim = (int)min((int64_t)kChunk, (int64_t)n_len - c0);
      const uint32_t* kc = kc_base + c0 * ROWW;
      const uint32_t* vc = vc_base + c0 * ROWW;
#pragma unroll
      for (int k = 0; k < NIT; ++k) {                        // row-contiguous: coalesced
        const int e = ptid + k * kProdThr;
        if (NCW % kProdThr == 0 || e < NCW) {
          const int row = e / ROWW, w = e % ROWW;
          const bool ok = row < lim;
          const int src = ok ? e : 0;
          const uint32_t d = dst + (row * SROWW + w) * 4;
          cp_async4s(d + Lay::S_KC, kc + src, ok ? 4 : 0);
          cp_async4s(d + Lay::S_VC, vc + src, ok ? 4 : 0);
        }
      }
      if (ptid < kChunk) {                                          // value (lo, scale)
        const bool ok = ptid < lim;
        cp_async8s(dst + Lay::S_VP + ptid * 8, a.v_params + bh * a.T_cap + c0 + (ok ? ptid : 0), ok ? 8 : 0);
      } else if (ptid <= 2 * kChunk) {                              // key-outlier offsets c0 .. c0+64
        const int i = ptid - kChunk;
        cp_async4s(dst + Lay::S_KO + i * 4, a.k_out_off + off_base + c0 + min(i, lim), 4);
      } else if (stage_vout && ptid >= 3 * kChunk && ptid < (3 + Lay::NVS) * kChunk) {
        const int k = (ptid - 3 * kChunk) / kChunk, row = ptid % kChunk;
        if (k < a.n_v) {
          const bool ok = row < lim;
          cp_async4s(dst + Lay::S_VO + (k * kChunk + row) * 4, a.v_out + (bh * a.T_cap + c0 + (ok ? row : 0)) * a.n_v + k,
                     ok ? 4 : 0);
        }
      }
    };
    // this thread's key rotations R(tok) for its pairs: the same in every chunk
    float2 rot[QP];
#pragma unroll
    for (int j = 0; j < QP; ++j) rot[j] = dtab[(grp * QP + j) * kChunk + tok];

    // this thread's element of the rotated-query table (head qg, pair qi)
    const int nq = a.G * NP;
    const int qg = ptid / NP, qi = ptid % NP;
    float qx = 0.f, qy = 0.f;
    float2 qcs = make_float2(1.f, 0.f);
    if (ptid < nq) {
      const __half* qr = a.q + ((int64_t)b * a.Hq + (int64_t)kvh * a.G + qg) * D;
      qx = __half2float(qr[qi]);
      qy = __half2float(qr[qi + NP]);
      if (nchunks > 0) qcs = a.rope[min(v_begin, a.rope_len - 1) * NP + qi];
    }
    const int qpos = qg * QROW + (qi / 8) * 8 + (qi % 4) * 2 + ((qi % 8) / 4);

    // key-outlier entries are fetched one chunk ahead, one per thread
    uint32_t kent = 0u;
    if (nchunks > 0) {
      const int64_t e0 = __ldg(a.k_out_off + off_base + min(v_begin, (int64_t)n_len));
      const int64_t e1 = min((int64_t)__ldg(a.k_out_off + off_base + min(v_begin + kChunk, (int64_t)n_len)),
                             a.k_out_cap);
      if (e0 + ptid < e1) kent = __ldg(gents + e0 + ptid);
    }

#pragma unroll
    for (int s = 0; s < NS - 1; ++s) {
      if (s < nchunks) load_chunk(s, s);
      cp_async_commit();
    }
    for (int c = 0; c < nchunks; ++c) {
      cp_async_wait<NS - 3>();                // this thread's copies of chunks c and c+1 landed
      bar_sync(kBarProd, kProdThr);           // everyone's landed; the stage of chunk c-1 is free
      if (c + NS - 1 < nchunks) load_chunk(c + NS - 1, (c + NS - 1) % NS);
      cp_async_commit();
      // read ahead: this thread's key-outlier entry of chunk c+1 (its offsets are staged)
      uint32_t kent_n = 0u;
      if (c + 1 < nchunks) {
        const int32_t* koff_n = reinterpret_cast<const int32_t*>(stg + ((c + 1) % NS) * Lay::STAGE + Lay::S_KO);
        const int e = koff_n[0] + ptid;
        if (e < min((int64_t)koff_n[kChunk], a.k_out_cap)) kent_n = __ldg(gents + e);
      }

      const uint8_t* st = stg + (c % NS) * Lay::STAGE;
      const int32_t* koff = reinterpret_cast<const int32_t*>(st + Lay::S_KO);
      const int buf = c & 1;
      if (c >= 2) bar_sync(kBarEmpty + buf, kThr);   // attention on chunk c-2 released the buffer
      uint8_t* B_ = bufs + buf * Lay::BUF;
      uint8_t* khi_t = B_ + Lay::B_KHI;
      uint8_t* klo_t = B_ + Lay::B_KLO;
      uint8_t* v_t = B_ + Lay::B_VT;
      const int64_t t0 = v_begin + (int64_t)c * kChunk;

      // hand the chunk's key-outlier entries, their offsets and owners to the consumers
      reinterpret_cast<uint32_t*>(B_ + Lay::B_ENT)[ptid] = kent;
      if (ptid <= kChunk) reinterpret_cast<int32_t*>(B_ + Lay::B_KO)[ptid] = koff[ptid];
      if (stage_vout && ptid < kChunk * a.n_v)
        reinterpret_cast<uint32_t*>(B_ + Lay::B_VO)[ptid] = reinterpret_cast<const uint32_t*>(st + Lay::S_VO)[ptid];
      if (ptid < kChunk) {
        const int E0 = koff[0];
        const int e_hi = min((int)min((int64_t)koff[ptid + 1], a.k_out_cap), E0 + kEntCap);
        for (int e = koff[ptid]; e < e_hi; ++e) (B_ + Lay::B_OWN)[e - E0] = (uint8_t)ptid;
      }

      // query rotated back by the chunk start: R(t0)^T q as hi, -hi and lo fp16 pairs, stored in
      // the order the mma fragments read (pair i = kc*8 + 4*hf + r at word kc*8 + 2*r + hf)
      if (ptid < nq) {
        const float xr = qx * qcs.x + qy * qcs.y, yr = qy * qcs.x - qx * qcs.y;
        const uint32_t h = pack_half2(xr, yr);
        const float2 hf = __half22float2(*reinterpret_cast<const __half2*>(&h));
        reinterpret_cast<uint32_t*>(B_ + Lay::B_QH)[qpos] = h;
        reinterpret_cast<uint32_t*>(B_ + Lay::B_QN)[qpos] = h ^ 0x80008000u;
        reinterpret_cast<uint32_t*>(B_ + Lay::B_QL)[qpos] = pack_half2(xr - hf.x, yr - hf.y);
        if (c + 1 < nchunks) qcs = a.rope[min(t0 + kChunk, a.rope_len - 1) * NP + qi];
      }

      // keys: dequantize, rotate by R(tok), split; rows past the cache end were zero-filled
      // (finite keys, masked in the attention)
      const uint32_t* krow = reinterpret_cast<const uint32_t*>(st + Lay::S_KC) + tok * SROWW;
      {
        uint32_t w[NWG];
        group_words<BITS, QP, NWG>(krow, grp, w);
        const float* kq = kdq + grp * QP * K;
#pragma unroll
        for (int jj = 0; jj < QP; jj += 4) {
          uint32_t ph[4], pl[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int j = jj + u;
            int clo, chi;
            pair_codes<BITS, NWG>(w, j, clo, chi);
            const float x = kq[j * K + clo];
            const float y = kq[(j + NP) * K + chi];
            split_hi_nlo(x * rot[j].x - y * rot[j].y, y * rot[j].x + x * rot[j].y, ph[u], pl[u]);
          }
          const int ch = (grp * QP + jj) / 4;
          *reinterpret_cast<uint4*>(khi_t + tile_off<D>(tok, ch)) = make_uint4(ph[0], ph[1], ph[2], ph[3]);
          *reinterpret_cast<uint4*>(klo_t + tile_off<D>(tok, ch)) = make_uint4(pl[0], pl[1], pl[2], pl[3]);
        }
      }
      // values: rows past the cache end have lo = scale = 0 (zero-filled): value 0
      {
        const uint32_t* row = reinterpret_cast<const uint32_t*>(st + Lay::S_VC) + tok * SROWW;
        uint32_t w[NWG];
        group_words<BITS, QP, NWG>(row, grp, w);
        const float2 lp = reinterpret_cast<const float2*>(st + Lay::S_VP)[tok];
        const float* vq = vtb + grp * QP * K;
#pragma unroll
        for (int jj = 0; jj < QP; jj += 4) {
          uint32_t pv[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int j = jj + u;
            int clo, chi;
            pair_codes<BITS, NWG>(w, j, clo, chi);
            pv[u] = pack_half2(fmaf(lp.y, vq[j * K + clo], lp.x), fmaf(lp.y, vq[(j + NP) * K + chi], lp.x));
          }
          const int ch = (grp * QP + jj) / 4;
          *reinterpret_cast<uint4*>(v_t + tile_off<D>(tok, ch)) = make_uint4(pv[0], pv[1], pv[2], pv[3]);
        }
      }
      kent = kent_n;
      bar_arrive(kBarFull + buf, kThr);       // chunk c's tiles are ready
    }
    cp_async_wait<0>();
  } else {
    // ======================= consumers: tensor-core attention =======================
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;\n" ::"n"(kRegCons) : "memory");
    const int cw = warp - kProdWarps;        // tokens 16*cw .. 16*cw + 15 of each chunk
    const bool real = g < a.G;
    const int mi = lane >> 3, rowi = lane & 7;
    const int t0w = cw * 16;
    const int tokk = t0w + (mi >> 1) * 8 + rowi;
    const int tokv = t0w + (mi & 1) * 8 + rowi;
    float o[D / 8][2];
#pragma unroll
    for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = 0.f;
    float m_run = -INFINITY, l_part = 0.f;
    for (int c = 0; c < nchunks; ++c) {
      const int buf = c & 1;
      bar_sync(kBarFull + buf, kThr);
      uint8_t* B_ = bufs + buf * Lay::BUF;
      uint8_t* khi_t = B_ + Lay::B_KHI;
      uint8_t* klo_t = B_ + Lay::B_KLO;
      uint8_t* v_t = B_ + Lay::B_VT;
      const int64_t t0 = v_begin + (int64_t)c * kChunk;
      // key outliers: the thread of entry e recovers its pair before the rotation from the
      // tile (hi - nlo, then R(d)^T), puts in the fp16 value(s), rotates and splits again
      {
        const int32_t* ko = reinterpret_cast<const int32_t*>(B_ + Lay::B_KO);
        const uint32_t* ents = reinterpret_cast<const uint32_t*>(B_ + Lay::B_ENT);
        const uint8_t* own = B_ + Lay::B_OWN;
        const uint32_t* gents = a.k_out + bh * a.k_out_cap;
        const int E0 = ko[0];
        const int E1 = (int)min((int64_t)ko[kChunk], a.k_out_cap);
        for (int idx = E0 + (tid - kProdThr); idx < E1; idx += kThr - kProdThr) {
          const bool staged = idx - E0 < kEntCap;
          const uint32_t ev = staged ? ents[idx - E0] : __ldg(gents + idx);
          int t;
          if (staged) {
            t = own[idx - E0];
          } else {                            // beyond the staged entries: search the offsets
            t = 0;
#pragma unroll
            for (int step = kChunk / 2; step >= 1; step >>= 1)
              if (ko[t + step] <= idx) t += step;
          }
          const int ch = (int)(ev >> 16);
          if (ch >= D) continue;              // not a channel (never written by the quantizer)
          const int i = ch < NP ? ch : ch - NP;
          const int partner = ch < NP ? ch + NP : ch - NP;
          const int f_hi = min(ko[t + 1], E1);
          bool has_p = false;
          float pval = 0.f;
          for (int f = ko[t]; f < f_hi; ++f) {
            const uint32_t ef = f - E0 < kEntCap ? ents[f - E0] : __ldg(gents + f);
            if ((int)(ef >> 16) == partner) {
              has_p = true;
              pval = h2f((uint16_t)(ef & 0xffffu));
            }
          }
          if (has_p && ch >= NP) continue;    // handled with its partner entry
          const int byte = tile_off<D>(t, i / 4) + (i % 4) * 4;
          const float2 hf = __half22float2(*reinterpret_cast<const __half2*>(khi_t + byte));
          const float2 nf = __half22float2(*reinterpret_cast<const __half2*>(klo_t + byte));
          const float kx = hf.x - nf.x, ky = hf.y - nf.y;
          const float2 cs = dtab[i * kChunk + t];
          float x = kx * cs.x + ky * cs.y, y = ky * cs.x - kx * cs.y;
          const float val = h2f((uint16_t)(ev & 0xffffu));
          if (ch < NP) {
            x = val;
            if (has_p) y = pval;
          } else {
            y = val;
          }
          uint32_t ph, pl;
          split_hi_nlo(x * cs.x - y * cs.y, y * cs.x + x * cs.y, ph, pl);
          *reinterpret_cast<uint32_t*>(khi_t + byte) = ph;
          *reinterpret_cast<uint32_t*>(klo_t + byte) = pl;
        }
        // value outliers: exact fp16 values over the dequantized ones
        const bool stage_vout = a.n_v <= Lay::NVS;
        const uint32_t* vo = reinterpret_cast<const uint32_t*>(B_ + Lay::B_VO);
        for (int e = tid - kProdThr; e < kChunk * a.n_v; e += kThr - kProdThr) {
          const int k = e / kChunk, t = e % kChunk;
          if (t0 + t >= n_len) continue;
          const uint32_t ev = stage_vout ? vo[e] : __ldg(a.v_out + (bh * a.T_cap + t0 + t) * a.n_v + k);
          const int chn = (int)(ev >> 16);
          if (chn >= D) continue;
          const int col = chn < NP ? 2 * chn : 2 * (chn - NP) + 1;
          *reinterpret_cast<uint16_t*>(v_t + tile_off<D>(t, col / 8) + (col % 8) * 2) = (uint16_t)(ev & 0xffffu);
        }
        bar_sync(kBarCons, kThr - kProdThr);  // every consumer warp reads every row
      }
      const int qrow = (real ? g : 0) * (QROW / 2);
      const uint2* qh2 = reinterpret_cast<const uint2*>(B_ + Lay::B_QH) + qrow;
      const uint2* qn2 = reinterpret_cast<const uint2*>(B_ + Lay::B_QN) + qrow;
      const uint2* ql2 = reinterpret_cast<const uint2*>(B_ + Lay::B_QL) + qrow;
      float sc[2][4];
#pragma unroll
      for (int i = 0; i < 4; ++i) sc[0][i] = sc[1][i] = 0.f;
#pragma unroll
      for (int kc = 0; kc < KC; ++kc) {
        const uint2 ah = real ? qh2[kc * 4 + r] : make_uint2(0u, 0u);
        const uint2 an = real ? qn2[kc * 4 + r] : make_uint2(0u, 0u);
        const uint2 al = real ? ql2[kc * 4 + r] : make_uint2(0u, 0u);
        uint32_t bhi[4], bnl[4];
        const int ch = kc * 2 + (mi & 1);
        ldsm_x4(bhi, khi_t + tile_off<D>(tokk, ch));
        ldsm_x4(bnl, klo_t + tile_off<D>(tokk, ch));
        mma16816(sc[0], ah.x, 0u, ah.y, 0u, bhi[0], bhi[1]);
        mma16816(sc[1], ah.x, 0u, ah.y, 0u, bhi[2], bhi[3]);
        mma16816(sc[0], an.x, 0u, an.y, 0u, bnl[0], bnl[1]);
        mma16816(sc[1], an.x, 0u, an.y, 0u, bnl[2], bnl[3]);
        mma16816(sc[0], al.x, 0u, al.y, 0u, bhi[0], bhi[1]);
        mma16816(sc[1], al.x, 0u, al.y, 0u, bhi[2], bhi[3]);
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
      if (c + 2 < nchunks) bar_arrive(kBarEmpty + buf, kThr);   // producers may refill the buffer
    }
    // The producers are done with every stage once the last chunk was handed over (and no
    // stage was filled when there are no chunks), so the stage area takes the partials.
    l_part += __shfl_xor_sync(0xffffffffu, l_part, 1);
    l_part += __shfl_xor_sync(0xffffffffu, l_part, 2);
    if (g < a.G) {
      if (r == 0) {
        wm[cw * 8 + g] = m_run;
        wl[cw * 8 + g] = l_part;
      }
#pragma unroll
      for (int dt = 0; dt < D / 8; ++dt) {
        const int chn = dt * 4 + r;                          // column dt*8 + 2r -> channel dt*4 + r
        wo[(cw * 8 + g) * D + chn] = o[dt][0];
        wo[(cw * 8 + g) * D + chn + NP] = o[dt][1];
      }
    }
  }
  __syncthreads();
  for (int e = tid; e < a.G * D; e += kThr) {
    const int row = e / D, d = e % D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kConsWarps; ++w) M = fmaxf(M, wm[w * 8 + row]);
    float L = 0.f, O = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < kConsWarps; ++w) {
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
  merge_if_last<D, kThr>(a.merge, bh, b, kvh, reinterpret_cast<float*>(stg), Lay::NS * Lay::STAGE / 4);
}

template <int D, int BITS>
cudaError_t launch_kvq_t(const KvqArgs& a, int units, int n_split, cudaStream_t st) {
  using Lay = KvqLayout<D, BITS>;
  static_assert(Lay::BYTES <= 227 * 1024, "one CTA per SM");
  static int checked = 0;                 // 1: attributes set and register count verified
  if (!checked) {
    cudaFuncAttributes attr;
    cudaError_t e = cudaFuncGetAttributes(&attr, decode_kvq_kernel<D, BITS>);
    if (e != cudaSuccess) return e;
    // the register split above assumes exactly kRegLaunch registers a thread at launch
    if (attr.numRegs != kRegLaunch) return cudaErrorInvalidConfiguration;
    e = cudaFuncSetAttribute(decode_kvq_kernel<D, BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize, Lay::BYTES);
    if (e != cudaSuccess) return e;
    checked = 1;
  }
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
