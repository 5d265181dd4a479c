// KVQuant decode attention with dequantization fused into QK^T / softmax / PV
// (Section 2.1, KVQuant paragraph: keys quantized per channel before the
// rotary embedding, values per token, outliers kept in fp16).
//
// For each token t of the cache and each query head h of the group:
//   k_t = rope_t(dq_K(t)) with outliers restored before the rotation,
//   v_t = lo_t + scale_t * tbl[code] with outliers restored,
//   out_h = softmax_t(scale q_h . k_t) v_t.
//
// GB300 design: one CTA of 20 warps per SM (at most 152), warp-specialised.
// The 64-token chunks of all (batch, kv-head) units, laid end to end, are cut
// into equal ranges, one per CTA; a CTA runs its range unit by unit, writes one
// partial (m, l, o) per unit into its slot, and the last CTA of a unit merges
// the unit's partials.  Sixteen producer warps stage packed codes by cp.async
// (three chunks in flight) and dequantize chunk c into one of two fp16 tile
// buffers while four consumer warps run the tensor-core attention on the
// previous chunk from the other; named barriers (FULL / EMPTY per buffer) hand
// the buffers over.
//
// Producers: thread (token row tok, pair group g) dequantizes QP = D/16 pairs
// (i, i + D/2) of its token's key and value rows from shared per-channel tables
// (all lanes of a warp read the same channel's table -> conflict-free).  Each
// key pair is rotated by the token's offset d = tok from the chunk start with
// a rotation held in registers for the whole kernel (the chunk start's own
// rotation R(t0) is applied to the query instead:
// q . R(t0 + d) k = (R(t0)^T q) . (R(d) k)), computed on the paired fp32 pipe
// from key tables stored as (v, v) pairs, and written as fp16 hi plus the
// fp16 remainder lo, so the tensor-core product keeps fp32 accuracy.
// Consumers: each of the four attention warps owns 16 token rows of a chunk and
// first restores their outliers (only this warp reads those rows, so __syncwarp
// orders it): a key outlier x at channel ch adds (x - k_dense[ch]) R(d) e_ch to
// the rotated pair, which is split again (x-channels before y-channels, so the
// two entries of a pair never write one word at once); a value outlier
// overwrites its value tile entry with the exact fp16 value.  The warp then
// computes S^T (tokens x heads) = K_hi q_hi + K_lo q_hi + K_hi q_lo, the
// online softmax, and O^T (dims x heads) += V^T P^T with P^T transposed in
// registers (movmatrix).  Tile columns hold pair i at columns (2i, 2i+1) =
// channels (i, i + D/2); the output is un-permuted at the end.
//
// Fused step (mkv_kvquant_step, the kStep instantiation): the same launch first
// appends the step's token to every unit.  Each CTA reads the lengths of the
// batch entries it touches with a ticket in the top 8 bits of T_len[b] (the
// last of them stores the new length) and takes every cache as holding the
// token.  The CTA whose range holds a unit's new chunk row has its attention
// warps quantize the token (the quantize kernel's routine, so the bits match)
// before they attend to anything, while the producers stage the first chunks.
// Every copy made after the producers' first wait for a released tile buffer,
// or in a later segment, therefore reads the new rows; only a new token in one
// of the first segment's first NS + 2 chunks makes the producers wait for the
// quantizer (one named barrier) before they copy anything.
#include <math.h>

#include "mkv_common.cuh"
#include "mkv_internal.h"
#include "mkv_merge.cuh"
#include "mkv_quant_token.cuh"

namespace mkv {

namespace {

constexpr int kProdWarps = 16;                         // dequantize chunk c (+ stage loads)
constexpr int kConsWarps = 4;                          // attention on chunk c-1 (tensor cores)
constexpr int kProdThr = kProdWarps * 32;
constexpr int kThr = (kProdWarps + kConsWarps) * 32;
constexpr int kGroups = 8;                             // pair groups of a token row
constexpr int kEnt = 256;                              // key-outlier entries of a chunk staged
// named barriers (0 is __syncthreads)
constexpr int kBarProd = 1;                            // producers only
constexpr int kBarFull = 2;                            // + buffer: tiles of a chunk are ready
constexpr int kBarEmpty = 4;                           // + buffer: tiles may be overwritten
constexpr int kBarQDone = 6;                           // fused step: the CTA's new tokens are quantized
constexpr int kBarQGrp = 7;                            // fused step: the attention warps' quantizer
constexpr int kMaxUnitsCta = 32;                      // units a CTA's range may touch (tables by unit & 31)
constexpr int kNewTok = 1 << 30;                       // length flag: the step appended a token
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

__device__ uint32_t g_status_kvq;   // MKV_FLAG_* bits raised by the fused step

// Fused step: what the quantizer of the step's token writes and reads.
struct KvqStep {
  const __half* k_new;    // [B][Hkv][D] pre-rotation key of the step's token
  const __half* v_new;    // [B][Hkv][D]
  int32_t* T_len;
  uint8_t* k_codes;
  uint8_t* v_codes;
  float2* v_params;
  uint32_t* v_out;
  int32_t* k_out_off;
  uint32_t* k_out;
  const float* t_lo;      // [Hkv][D]
  const float* t_hi;
  const float* k_lo;
  const float* k_scale;
  const uint16_t* k_cb;   // [Hkv][D][K]
  const uint16_t* v_cb;
  int nuq;
};

// A load of cache data the kernel does not write, or (fused step) may have written: then coherent.
template <bool kCoherent, typename T>
__device__ __forceinline__ T ld_cache(const T* p) {
  if constexpr (kCoherent) return __ldcg(p);
  else return __ldg(p);
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
  int n_split;             // partial slots per (batch, kv-head)
  int n_cta;               // CTA i covers virtual chunks [i * c_tot / n_cta, (i + 1) * c_tot / n_cta)
  int64_t cpu, c_tot;      // virtual chunks per (batch, kv-head), and of all of them
  float scale_log2;
  float* part_m;
  float* part_l;
  float* part_o;
  MergeArgs merge;
  int step;                // 1: fused step (append the token, then attend)
  KvqStep st;
};

template <int D, int BITS>
struct KvqLayout {
  static constexpr int NP = D / 2;
  static constexpr int K = 1 << BITS;
  static constexpr int ROWW = D * BITS / 32;                 // packed words per token row
  // Rows of whole 16-byte pieces are staged by 16-byte copies that bypass L1, at a stride of
  // 4 mod 8 words (at most 4 rows share a bank); other rows by 4-byte copies at an odd stride.
  static constexpr bool CG = ROWW % 4 == 0;
  static constexpr int SROWW = CG ? ((ROWW + 4) % 8 == 4 ? ROWW + 4 : ROWW + 8) : ROWW + 1;
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
  static constexpr int S_ENT = S_VO + NVS * kChunk * 4;      // [kEnt] u32 first key-outlier entries
  static constexpr int S_RT = S_ENT + kEnt * 4;          // [NP] float2 rotation of the chunk start
  static constexpr int STAGE = S_RT + NP * 8;
  // one tile buffer: keys (hi, lo), values, the rotated query and the chunk's key outliers
  static constexpr int B_KHI = 0;
  static constexpr int B_KLO = B_KHI + TILE;
  static constexpr int B_VT = B_KLO + TILE;
  static constexpr int B_QH = B_VT + TILE;                   // [8][QROW] q_hi pairs, fragment order
  static constexpr int B_QL = B_QH + 8 * QROW * 4;           // q_lo
  static constexpr int B_ENT = B_QL + 8 * QROW * 4;          // [kEnt] u32 first key-outlier entries
  static constexpr int B_KO = B_ENT + kEnt * 4;              // [68] int32 CSR offsets of the chunk
  static constexpr int B_VO = B_KO + 68 * 4;                 // [NVS][64] u32 value outliers
  static constexpr int BUF = B_VO + NVS * kChunk * 4;
  // CTA layout
  static constexpr int DTAB = 0;                             // [NP][64] float2 rotation by delta
  static constexpr int KDQ = DTAB + NP * kChunk * 8;         // [D][K] float pairs (v, v)
  static constexpr int VTB = KDQ + D * K * 8;                // [D][K] float
  static constexpr int QS = VTB + D * K * 4;                 // [8][D] f32 query (as given, rotated)
  static constexpr int STG = QS + 8 * D * 4;                 // [NS][STAGE]
  static constexpr int BUFS = STG + NS * STAGE;              // [2][BUF]
  // fused step: the attention warps' quantizer scratch, and the lengths of the CTA's batch entries
  static constexpr int NWQ = (D * BITS / 8 + 3) / 4;         // packed words of a code row
  static constexpr int QT_KC = BUFS + 2 * BUF;               // [D] u8 key codes
  static constexpr int QT_VC = QT_KC + D;                    // [D] u8 value codes
  static constexpr int QT_ABS = QT_VC + D;                   // [D] f32
  static constexpr int QT_W = QT_ABS + 4 * D;                // [2][NWQ] u32
  static constexpr int QT_CNT = QT_W + 8 * NWQ;              // [4] int, then lo [4], hi [4]
  static constexpr int QT_MX = QT_CNT + 48;                  // [2][32] u32
  static constexpr int BLEN = QT_MX + 256;                   // [32] int per batch entry
  static constexpr int ULEN = BLEN + 32 * 4;                 // [32] int per unit (unit & 31)
  static constexpr int UCQ = ULEN + 32 * 4;                  // [32] int per unit (unit & 31)
  static constexpr int BYTES = UCQ + 32 * 4;
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

// packed fp32 pairs (two lanes of one 64-bit register; Blackwell's paired fp32 pipe)
__device__ __forceinline__ uint64_t f2_pack(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t r, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}

// (a, b) as fp16 hi and the fp16 remainder lo = x - hi (exact in fp32 before its rounding)
__device__ __forceinline__ void split_hi_lo(float a, float b, uint32_t& hi, uint32_t& lo) {
  uint32_t h;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(h) : "f"(b), "f"(a));
  float d0, d1;
  asm("{.reg .f16 l, u;\n mov.b32 {l, u}, %2;\n sub.rn.f32.f16 %0, l, %3;\n sub.rn.f32.f16 %1, u, %4;\n}"
      : "=f"(d0), "=f"(d1)
      : "r"(h), "f"(a), "f"(b));
  hi = h;
  lo = pack_half2(-d0, -d1);
}

__device__ __forceinline__ void cp_async4s(uint32_t saddr, const void* gmem, int src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(saddr), "l"(gmem), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async16s(uint32_t saddr, const void* gmem, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(saddr), "l"(gmem), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async8s(uint32_t saddr, const void* gmem, int src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;\n" ::"r"(saddr), "l"(gmem), "r"(src_bytes));
}

// byte offset of (row, 16B chunk) in a swizzled fp16 tile of D columns
template <int D>
__device__ __forceinline__ int tile_off(int row, int ch) {
  return row * D * 2 + ((ch ^ (row & 7)) << 4);
}

// S^T fragment of P transposed in registers: an 8x8 b16 matrix held as the rows of an mma
// accumulator becomes the column-major operand of the next mma
__device__ __forceinline__ uint32_t movm_trans(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;\n" : "=r"(y) : "r"(x));
  return y;
}

// Fused step: the step's token of every unit whose new chunk row this CTA holds, quantized by the
// attention warps with one thread per channel c (Section 2.1, KVQuant paragraph); then the producers
// may copy those chunks.
template <int D, int BITS>
__device__ __forceinline__ void quantize_new_tokens(const KvqArgs& a, int64_t x0, int64_t x1, uint8_t* smem, int c) {
  using Lay = KvqLayout<D, BITS>;
  constexpr int K = 1 << BITS;
  const int* s_ulen = reinterpret_cast<const int*>(smem + Lay::ULEN);
  const int cc = min(c, D - 1);            // threads c >= D only take part in the barriers
  const QTokSmem scr{smem + Lay::QT_KC, smem + Lay::QT_VC, reinterpret_cast<float*>(smem + Lay::QT_ABS),
                     reinterpret_cast<uint32_t*>(smem + Lay::QT_W), reinterpret_cast<int*>(smem + Lay::QT_CNT),
                     reinterpret_cast<float*>(smem + Lay::QT_CNT + 16), reinterpret_cast<float*>(smem + Lay::QT_CNT + 32),
                     reinterpret_cast<uint32_t*>(smem + Lay::QT_MX)};
  bool any = false;
  const int64_t u_lo = x0 / a.cpu;
  for (int64_t u = u_lo; u <= (x1 - 1) / a.cpu; ++u) {
    const int lv = s_ulen[u & 31];
    if (!(lv & kNewTok)) continue;
    const int64_t p = (lv & (kNewTok - 1)) - 1, xc = u * a.cpu + p / kChunk;
    if (xc < x0 || xc >= x1) continue;       // another CTA holds this unit's new token
    any = true;
    const int64_t hc = (u % a.Hkv) * D + cc;
    const float tlo = a.st.t_lo[hc], thi = a.st.t_hi[hc];
    const float klo = a.st.k_lo ? a.st.k_lo[hc] : 0.f, ksc = a.st.k_scale ? a.st.k_scale[hc] : 0.f;
    const __half xk = a.st.k_new[u * D + cc], xv = a.st.v_new[u * D + cc];
    float kmu[15], vmu[15];
#pragma unroll
    for (int j = 0; j < 15; ++j) kmu[j] = vmu[j] = 0.f;
    if (a.st.nuq) {
      uint16_t kr[K], vr[K];
#pragma unroll
      for (int j = 0; j < K; ++j) {
        kr[j] = a.st.k_cb[hc * K + j];
        vr[j] = a.st.v_cb[hc * K + j];
      }
#pragma unroll
      for (int j = 0; j + 1 < K; ++j) {
        kmu[j] = fl32_mid(h2f(kr[j]), h2f(kr[j + 1]));
        vmu[j] = fl32_mid(h2f(vr[j]), h2f(vr[j + 1]));
      }
    }
    int32_t* off_row = a.st.k_out_off + u * (a.T_cap + 1);
    const int32_t off = p == 0 ? 0 : __ldcg(off_row + p);
    if (p == 0 && c == 0) off_row[0] = 0;
    constexpr int RB = D * BITS / 8;
    const QTokDst dst{a.st.k_out + u * a.k_out_cap, a.k_out_cap, a.st.v_out + u * a.T_cap * a.n_v,
                      a.st.v_params + u * a.T_cap, a.st.k_codes + u * a.T_cap * RB, a.st.v_codes + u * a.T_cap * RB,
                      off_row};
    quantize_token(c, D, BITS, a.st.nuq != 0, a.n_v, kmu, vmu, tlo, thi, klo, ksc, xk, xv, p, off, dst, scr,
                   &g_status_kvq, [] { bar_sync(kBarQGrp, kThr - kProdThr); });
  }
  if (any) __threadfence_block();          // the cache rows before the producers' copies
  const int cq0 = reinterpret_cast<const int*>(smem + Lay::UCQ)[u_lo & 31];
  if (cq0 >= 0 && cq0 < Lay::NS + 2) bar_arrive(kBarQDone, kThr);   // the producers wait for it
}

// kStep: the fused step (the step's token quantized by the launch); otherwise the cache as it is.
template <int D, int BITS, bool kStep>
__global__ void __launch_bounds__(kThr, 1) decode_kvq_kernel(const KvqArgs a) {
  using Lay = KvqLayout<D, BITS>;
  constexpr int NP = Lay::NP, K = Lay::K, ROWW = Lay::ROWW, SROWW = Lay::SROWW, QP = Lay::QP;
  constexpr int NWG = Lay::NWG, NS = Lay::NS, QROW = Lay::QROW;
  constexpr int KC = D / 16;
  extern __shared__ __align__(128) uint8_t smem[];
  float2* dtab = reinterpret_cast<float2*>(smem + Lay::DTAB);
  uint64_t* kdq = reinterpret_cast<uint64_t*>(smem + Lay::KDQ);
  float* vtb = reinterpret_cast<float*>(smem + Lay::VTB);
  float* qs = reinterpret_cast<float*>(smem + Lay::QS);
  uint8_t* stg = smem + Lay::STG;
  uint8_t* bufs = smem + Lay::BUFS;

  const int cta = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, r = lane & 3;
  // this CTA's virtual chunks of the concatenated (batch, kv-head) units: one segment per unit
  const int64_t x0 = (int64_t)cta * a.c_tot / a.n_cta, x1 = ((int64_t)cta + 1) * a.c_tot / a.n_cta;

  // Fused step: each CTA that touches batch entry b takes a ticket in the top 8 bits of T_len[b] as
  // it reads the length (one thread per batch entry); the last one stores the new length, and the
  // cache is taken as holding the step's token (kNewTok marks it).  The lengths then go to per-unit
  // tables (unit & 31: a CTA's range spans at most 28 units) with the segment-relative chunk of the
  // CTA's first new token (-1 elsewhere), so the roles' loops keep no extra registers for them.
  int* s_blen = reinterpret_cast<int*>(smem + Lay::BLEN);
  const int* s_ulen = reinterpret_cast<const int*>(smem + Lay::ULEN);
  const int* s_ucq = reinterpret_cast<const int*>(smem + Lay::UCQ);
  if (kStep) {
    const int64_t b_lo = x0 / a.cpu / a.Hkv, nb = (x1 - 1) / a.cpu / a.Hkv - b_lo + 1;
    if (tid < nb) {
      const int64_t bb = b_lo + tid;
      const unsigned old = atomicAdd(reinterpret_cast<unsigned*>(a.st.T_len) + bb, 1u << 24);
      const int64_t f = cta_of_chunk(bb * a.Hkv * a.cpu, a.c_tot, a.n_cta);
      const int64_t l = cta_of_chunk((bb + 1) * a.Hkv * a.cpu - 1, a.c_tot, a.n_cta);
      const int64_t n0 = old & 0xffffffu;
      const bool room = n0 < a.T_cap;
      if ((int64_t)(old >> 24) == l - f) {            // the last reader of bb
        a.st.T_len[bb] = (int32_t)(room ? n0 + 1 : n0);
        if (!room) atomicOr(&g_status_kvq, MKV_FLAG_CACHE_FULL);
      }
      s_blen[tid] = room ? (int)(n0 + 1) | kNewTok : (int)min(n0, a.T_cap);
    }
  }

  // CTA-resident rotations by delta in [0, 64): coalesced reads of rope rows 0..63, all issued
  // before the transposed stores
  {
    constexpr int NE = (NP * kChunk + kThr - 1) / kThr;
    float2 v[NE];
#pragma unroll
    for (int k = 0; k < NE; ++k) {
      const int e = tid + k * kThr;
      const int d = e / NP, i = e % NP;
      if (e < NP * kChunk) v[k] = __ldg(a.rope + (int64_t)min((int64_t)d, a.rope_len - 1) * NP + i);
    }
#pragma unroll
    for (int k = 0; k < NE; ++k) {
      const int e = tid + k * kThr;
      if (e < NP * kChunk) dtab[(e % NP) * kChunk + e / NP] = v[k];
    }
  }
  __syncthreads();
  if (kStep && warp == 0) {                // the per-unit tables (read after the first begin_unit)
    const int64_t u_lo = x0 / a.cpu, b_lo = u_lo / a.Hkv;
    const int64_t u = u_lo + lane;
    const bool in = u <= (x1 - 1) / a.cpu;
    int lv = 0, cq = -1;
    if (in) {
      lv = s_blen[(int)(u / a.Hkv - b_lo)];
      if (lv & kNewTok) {
        const int64_t xc = u * a.cpu + ((lv & (kNewTok - 1)) - 1) / kChunk;   // the new token's chunk
        if (xc >= x0 && xc < x1) cq = (int)(xc - max(x0, u * a.cpu));
      }
    }
    const unsigned own = __ballot_sync(0xffffffffu, cq >= 0);
    if (in) {
      reinterpret_cast<int*>(smem + Lay::ULEN)[u & 31] = lv;
      reinterpret_cast<int*>(smem + Lay::UCQ)[u & 31] = own && lane == __ffs(own) - 1 ? cq : -1;
    }
  }

  // the four attention warps' (m, l, o) per query row, merged after both roles finish a segment
  float* wm = reinterpret_cast<float*>(stg);                // [4 warps][8 rows]
  float* wl = wm + 32;                                       // [4][8]
  float* wo = wl + 32;                                       // [4][8][D]  natural channel order

  // Both roles run the same segments; these steps take every thread of the CTA.
  // Start of a segment of unit bh: dequant tables of its kv-head, its group's queries in fp32.
  auto begin_unit = [&](int64_t bh) {
    const int b = (int)(bh / a.Hkv), kvh = (int)(bh % a.Hkv);
    constexpr int NT = (D * K + kThr - 1) / kThr;           // all loads in flight, then the stores
    float kv[NT];
    uint16_t vv[NT];
#pragma unroll
    for (int k = 0; k < NT; ++k) {
      const int e = tid + k * kThr;
      if (e < D * K) {
        kv[k] = __ldg(a.k_dq + (int64_t)kvh * D * K + e);
        vv[k] = __ldg(a.v_tbl + (int64_t)kvh * D * K + e);
      }
    }
    constexpr int NQ = (8 * D + kThr - 1) / kThr;
    __half qv[NQ];
#pragma unroll
    for (int k = 0; k < NQ; ++k) {
      const int e = tid + k * kThr;
      if (e < a.G * D) qv[k] = a.q[((int64_t)b * a.Hq + (int64_t)kvh * a.G) * D + e];
    }
#pragma unroll
    for (int k = 0; k < NT; ++k) {
      const int e = tid + k * kThr;
      if (e < D * K) {
        kdq[e] = f2_pack(kv[k], kv[k]);
        vtb[e] = __half2float(__ushort_as_half(vv[k]));
      }
    }
#pragma unroll
    for (int k = 0; k < NQ; ++k) {
      const int e = tid + k * kThr;
      if (e < a.G * D) qs[e] = __half2float(qv[k]);
    }
    __syncthreads();
  };
  // End of a segment: the warps' partials merged into this CTA's partial slot of the unit, and
  // the unit's last CTA merges all of them.
  auto end_unit = [&](int64_t bh) {
    const int b = (int)(bh / a.Hkv), kvh = (int)(bh % a.Hkv);
    const int64_t first = cta_of_chunk(bh * a.cpu, a.c_tot, a.n_cta);
    const int slot = (int)(cta - first);
    const int parts = (int)(cta_of_chunk((bh + 1) * a.cpu - 1, a.c_tot, a.n_cta) - first + 1);
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
      const int64_t pi = hq * a.n_split + slot;
      a.part_o[pi * D + d] = O;
      if (d == 0) {
        a.part_m[pi] = M;
        a.part_l[pi] = L;
      }
    }
    __syncthreads();                   // the stage buffers now serve as the merge's scratch
    merge_if_last<D, kThr>(a.merge, bh, b, kvh, reinterpret_cast<float*>(stg), Lay::NS * Lay::STAGE / 4, parts);
    __syncthreads();                   // before the next segment's copies into the stages
  };

  if (warp < kProdWarps) {
    // ======================= producers: stage, dequantize, rotate =======================
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(kRegProd) : "memory");
    const int ptid = tid;
    const int tok = (warp & 1) * 32 + lane;   // this thread's token row in every chunk
    const int grp = warp >> 1;                // its pairs: grp * QP .. grp * QP + QP - 1
    for (int64_t x = x0; x < x1;) {
      const int64_t bh = x / a.cpu;                           // this segment's unit
      const int64_t xe = min(x1, (bh + 1) * a.cpu);
      begin_unit(bh);
      const int b = (int)(bh / a.Hkv);
      const int n_len = kStep ? s_ulen[bh & 31] & (kNewTok - 1) : (int)min((int64_t)a.T_len[b], a.T_cap);
      const int64_t v_begin = (x - bh * a.cpu) * kChunk;
      const int64_t v_end = min((xe - bh * a.cpu) * kChunk, (int64_t)n_len);
      const int nchunks = v_end > v_begin ? (int)ceil_div_dev(v_end - v_begin, kChunk) : 0;
      // Fused step: the attention warps quantize the CTA's new tokens before they attend to anything,
      // so every copy made after the producers' first wait for a released buffer (chunk NS + 2 of the
      // first segment on) or in a later segment (after a CTA barrier) reads the new rows.  A new token
      // in one of the first segment's earlier chunks makes the producers wait for the quantizer here.
      if (kStep && x == x0) {
        const int cq = s_ucq[bh & 31];
        if (cq >= 0 && cq < NS + 2) bar_sync(kBarQDone, kThr);
      }
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
      if constexpr (Lay::CG) {
        constexpr int PR = ROWW / 4;                         // 16-byte pieces per row
        constexpr int NPC = kChunk * PR;                     // pieces per chunk (keys or values)
#pragma unroll
        for (int k = 0; k < (2 * NPC + kProdThr - 1) / kProdThr; ++k) {
          const int e = ptid + k * kProdThr;                 // key pieces, then value pieces
          if ((2 * NPC) % kProdThr == 0 || e < 2 * NPC) {
            const bool vals = e >= NPC;
            const int pe = vals ? e - NPC : e;
            const int row = pe / PR, q = pe % PR;
            const bool ok = row < lim;
            cp_async16s(dst + (vals ? Lay::S_VC : Lay::S_KC) + (row * SROWW + q * 4) * 4,
                        (vals ? vc : kc) + (ok ? pe * 4 : 0), ok ? 16 : 0);
          }
        }
      } else {
#pragma unroll
        for (int k = 0; k < NIT; ++k) {                      // row-contiguous: coalesced
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
      }
      if (ptid < kChunk) {                                          // value (lo, scale)
        const bool ok = ptid < lim;
        cp_async8s(dst + Lay::S_VP + ptid * 8, a.v_params + bh * a.T_cap + c0 + (ok ? ptid : 0), ok ? 8 : 0);
      } else if (ptid <= 2 * kChunk) {                              // key-outlier offsets c0 .. c0+64
        const int i = ptid - kChunk;
        cp_async4s(dst + Lay::S_KO + i * 4, a.k_out_off + off_base + c0 + min(i, lim), 4);
      } else if (ptid >= kProdThr - NP) {                            // rotation of the chunk start
        const int i = ptid - (kProdThr - NP);
        cp_async8s(dst + Lay::S_RT + i * 8, a.rope + min(c0, a.rope_len - 1) * NP + i, 8);
      } else if (stage_vout && ptid >= 3 * kChunk && ptid < (3 + Lay::NVS) * kChunk) {
        const int k = (ptid - 3 * kChunk) / kChunk, row = ptid % kChunk;
        if (k < a.n_v) {
          const bool ok = row < lim;
          cp_async4s(dst + Lay::S_VO + (k * kChunk + row) * 4, a.v_out + (bh * a.T_cap + c0 + (ok ? row : 0)) * a.n_v + k,
                     ok ? 4 : 0);
        }
      }
    };
    // this thread's key rotations R(tok) = [c -s; s c] for its pairs, the same in every chunk, as
    // the packed columns (c, s) and (-s, c)
    uint64_t rc0[QP], rc1[QP];
#pragma unroll
    for (int j = 0; j < QP; ++j) {
      const float2 cs = dtab[(grp * QP + j) * kChunk + tok];
      rc0[j] = f2_pack(cs.x, cs.y);
      rc1[j] = f2_pack(-cs.y, cs.x);
    }

    // this thread's element of the rotated-query table (head qg, pair qi)
    const int nq = a.G * NP;
    const int qg = ptid / NP, qi = ptid % NP;
    float qx = 0.f, qy = 0.f;
    if (ptid < nq) {
      qx = qs[qg * D + qi];
      qy = qs[qg * D + qi + NP];
    }
    const int qpos = qg * QROW + (qi / 8) * 8 + (qi % 4) * 2 + ((qi % 8) / 4);

    // The first kEnt key-outlier entries of a chunk are staged by cp.async one chunk ahead
    // (once the chunk's offsets have landed), one per thread, in a commit group of their own
    // ahead of that iteration's chunk copies; those of chunk 0 with chunk 0.
    // (threads ptid < kEnt, whole warps; entry indices fit in 32 bits, checked by the host)
    auto load_entries = [&](int stage, int e0, int e1) {
      const int e = e0 + ptid;
      const bool ok = e >= 0 && e < e1;       // offsets of a corrupted cache stay harmless
      cp_async4s(stg_s + stage * Lay::STAGE + Lay::S_ENT + ptid * 4, gents + (ok ? e : 0), ok ? 4 : 0);
    };
#pragma unroll
    for (int s = 0; s < NS - 1; ++s) {
      if (s < nchunks) {
        load_chunk(s, s);
        if (s == 0 && ptid < kEnt) {
          const int e0 = ld_cache<kStep>(a.k_out_off + off_base + v_begin);
          const int e1 = min(ld_cache<kStep>(a.k_out_off + off_base + min(v_begin + kChunk, (int64_t)n_len)),
                             (int)a.k_out_cap);
          load_entries(0, e0, e1);
        }
      }
      cp_async_commit();
    }
    for (int c = 0; c < nchunks; ++c) {
      cp_async_wait<NS - 3>();                // this thread's copies of chunks c, c+1 and entries of c landed
      bar_sync(kBarProd, kProdThr);           // everyone's landed; the stage of chunk c-1 is free
      if (c + 1 < nchunks && ptid < kEnt) {   // chunk c+1's offsets landed with the wait above
        const int32_t* ko1 = reinterpret_cast<const int32_t*>(stg + ((c + 1) % NS) * Lay::STAGE + Lay::S_KO);
        load_entries((c + 1) % NS, ko1[0], min(ko1[kChunk], (int)a.k_out_cap));
      }
      cp_async_commit();
      if (c + NS - 1 < nchunks) load_chunk(c + NS - 1, (c + NS - 1) % NS);
      cp_async_commit();

      const uint8_t* st = stg + (c % NS) * Lay::STAGE;
      const int32_t* koff = reinterpret_cast<const int32_t*>(st + Lay::S_KO);
      const uint32_t* kcodes = reinterpret_cast<const uint32_t*>(st + Lay::S_KC);
      const int buf = c & 1;
      // staged words this thread hands on or uses late, read before the wait for the buffer: its
      // key-outlier entry and offset for the consumers, its part of the chunk-start rotation, and
      // its token's value outliers
      const uint32_t my_ent = ptid < kEnt ? reinterpret_cast<const uint32_t*>(st + Lay::S_ENT)[ptid] : 0u;
      const int32_t my_ko = ptid <= kChunk ? koff[ptid] : 0;
      const float2 qcs = reinterpret_cast<const float2*>(st + Lay::S_RT)[qi];
      const bool my_vo_in = stage_vout && ptid < kChunk * a.n_v;
      const uint32_t my_vo = my_vo_in ? reinterpret_cast<const uint32_t*>(st + Lay::S_VO)[ptid] : 0u;
      if (c >= 2) bar_sync(kBarEmpty + buf, kThr);   // attention on chunk c-2 released the buffer
      uint8_t* B_ = bufs + buf * Lay::BUF;
      uint8_t* khi_t = B_ + Lay::B_KHI;
      uint8_t* klo_t = B_ + Lay::B_KLO;
      uint8_t* v_t = B_ + Lay::B_VT;

      // query rotated back by the chunk start: R(t0)^T q as hi, -hi and lo fp16 pairs, stored in
      // the order the mma fragments read (pair i = kc*8 + 4*hf + r at word kc*8 + 2*r + hf)
      if (ptid < nq) {
        const float xr = qx * qcs.x + qy * qcs.y, yr = qy * qcs.x - qx * qcs.y;
        const uint32_t h = pack_half2(xr, yr);
        const float2 hf = __half22float2(*reinterpret_cast<const __half2*>(&h));
        reinterpret_cast<uint32_t*>(B_ + Lay::B_QH)[qpos] = h;
        reinterpret_cast<uint32_t*>(B_ + Lay::B_QL)[qpos] = pack_half2(xr - hf.x, yr - hf.y);
      }

      // the chunk's outlier entries for the consumers, who restore them
      if (ptid < kEnt) reinterpret_cast<uint32_t*>(B_ + Lay::B_ENT)[ptid] = my_ent;
      if (ptid <= kChunk) reinterpret_cast<int32_t*>(B_ + Lay::B_KO)[ptid] = my_ko;
      if (my_vo_in) reinterpret_cast<uint32_t*>(B_ + Lay::B_VO)[ptid] = my_vo;

      // keys: dequantize, rotate by R(tok), split; rows past the cache end were zero-filled
      // (finite keys, masked in the attention)
      const uint32_t* krow = kcodes + tok * SROWW;
      {
        uint32_t w[NWG];
        group_words<BITS, QP, NWG>(krow, grp, w);
        const uint64_t* kq = kdq + grp * QP * K;
#pragma unroll
        for (int jj = 0; jj < QP; jj += 4) {
          uint32_t ph[4], pl[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int j = jj + u;
            int clo, chi;
            pair_codes<BITS, NWG>(w, j, clo, chi);
            // (x, x) (c, s) + (y, y) (-s, c) = R(tok) (x, y); as scalars for 3-bit codes, whose
            // word-straddling extraction schedules worse around the paired ops (measured)
            float xr, yr;
            if constexpr (BITS != 3) {
              f2_unpack(f2_fma(kq[(j + NP) * K + chi], rc1[j], f2_mul(kq[j * K + clo], rc0[j])), xr, yr);
            } else {
              float x, y, c, sn, unused0, unused1;
              f2_unpack(kq[j * K + clo], x, unused0);
              f2_unpack(kq[(j + NP) * K + chi], y, unused1);
              f2_unpack(rc0[j], c, sn);
              xr = x * c - y * sn;
              yr = y * c + x * sn;
            }
            split_hi_lo(xr, yr, ph[u], pl[u]);
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
      bar_arrive(kBarFull + buf, kThr);       // chunk c's tiles are ready
    }
    cp_async_wait<0>();
    end_unit(bh);
    x = xe;
    }
  } else {
    // ======================= consumers: tensor-core attention =======================
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;\n" ::"n"(kRegCons) : "memory");
    const int cw = warp - kProdWarps;        // tokens 16*cw .. 16*cw + 15 of each chunk
    const bool real = g < a.G;               // this lane's column of the q operand is a head
    const int mi = lane >> 3, rowi = lane & 7;
    const int t0w = cw * 16;
    const int tokA = t0w + (mi & 1) * 8 + rowi, chA = mi >> 1;   // K slab as the A operand
    const int tokV = t0w + (mi >> 1) * 8 + rowi, chV = mi & 1;   // V^T slab as the A operand
    bool q_todo = kStep;                     // fused step: quantize the CTA's new tokens first
    for (int64_t x = x0; x < x1;) {
      const int64_t bh = x / a.cpu;                           // this segment's unit
      const int64_t xe = min(x1, (bh + 1) * a.cpu);
      begin_unit(bh);
      if (q_todo) {
        quantize_new_tokens<D, BITS>(a, x0, x1, smem, tid - kProdThr);
        q_todo = false;
      }
      const int b = (int)(bh / a.Hkv);
      const int n_len = kStep ? s_ulen[bh & 31] & (kNewTok - 1) : (int)min((int64_t)a.T_len[b], a.T_cap);
      const int64_t v_begin = (x - bh * a.cpu) * kChunk;
      const int64_t v_end = min((xe - bh * a.cpu) * kChunk, (int64_t)n_len);
      const int nchunks = v_end > v_begin ? (int)ceil_div_dev(v_end - v_begin, kChunk) : 0;
    // o[j] = O^T rows (tile columns) 16j + g and 16j + g + 8, heads 2r and 2r + 1
    float o[D / 16][4];
#pragma unroll
    for (int j = 0; j < D / 16; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
    float m_run[2] = {-INFINITY, -INFINITY}, l_part[2] = {0.f, 0.f};
    for (int c = 0; c < nchunks; ++c) {
      const int buf = c & 1;
      bar_sync(kBarFull + buf, kThr);
      uint8_t* B_ = bufs + buf * Lay::BUF;
      uint8_t* khi_t = B_ + Lay::B_KHI;
      uint8_t* klo_t = B_ + Lay::B_KLO;
      uint8_t* v_t = B_ + Lay::B_VT;
      const int64_t t0 = v_begin + (int64_t)c * kChunk;
      // Key outliers of this warp's 16 tokens, restored in the rows of the key tiles that only this
      // warp reads (ordered by __syncwarp).  An outlier x at channel ch of token t adds
      // (x - k_dense[ch]) R(d) e_ch to the rotated pair in the tile (k_dense = R(d)^T (k_hi + k_lo)),
      // which is then split again; channels i < D/2 first, then i + D/2, so that the two entries of
      // one pair never write the same word at once.  Each entry carries its token within the chunk.
      {
        const int32_t* ko = reinterpret_cast<const int32_t*>(B_ + Lay::B_KO);
        const uint32_t* ents = reinterpret_cast<const uint32_t*>(B_ + Lay::B_ENT);
        const uint32_t* gents = a.k_out + bh * a.k_out_cap;
        const int E0 = ko[0];
        const int e_lo = ko[t0w], e_hi = (int)min((int64_t)ko[t0w + 16], a.k_out_cap);
        auto fetch = [&](int e) -> uint32_t {
          if (e < 0 || e >= e_hi) return 0xffff0000u;  // no entry: not a channel
          if (e - E0 < kEnt) return ents[e - E0];
          return ld_cache<kStep>(gents + e);  // beyond the staged entries
        };
        auto fix = [&](uint32_t ev, int pass) {
          const int ch = (int)((ev >> 16) & 0xffu);
          if (ch >= D || (ch >= NP) != (pass == 1)) return;
          const int t = (int)(ev >> 24) & (kChunk - 1);
          const int i = ch < NP ? ch : ch - NP;
          const int byte = tile_off<D>(t, i / 4) + (i % 4) * 4;
          const float2 hf = __half22float2(*reinterpret_cast<const __half2*>(khi_t + byte));
          const float2 lf = __half22float2(*reinterpret_cast<const __half2*>(klo_t + byte));
          float kx = hf.x + lf.x, ky = hf.y + lf.y;
          const float2 cs = dtab[i * kChunk + t];
          const float val = h2f((uint16_t)(ev & 0xffffu));
          if (pass == 0) {
            const float dk = val - (kx * cs.x + ky * cs.y);
            kx = fmaf(dk, cs.x, kx);
            ky = fmaf(dk, cs.y, ky);
          } else {
            const float dk = val - (ky * cs.x - kx * cs.y);
            kx = fmaf(-dk, cs.y, kx);
            ky = fmaf(dk, cs.x, ky);
          }
          uint32_t ph, pl;
          split_hi_lo(kx, ky, ph, pl);
          *reinterpret_cast<uint32_t*>(khi_t + byte) = ph;
          *reinterpret_cast<uint32_t*>(klo_t + byte) = pl;
        };
        const uint32_t ea = fetch(e_lo + lane), eb = fetch(e_lo + 32 + lane);
        fix(ea, 0);
        fix(eb, 0);
        for (int e = e_lo + 64 + lane; e < e_hi; e += 32) fix(fetch(e), 0);
        __syncwarp();
        fix(ea, 1);
        fix(eb, 1);
        for (int e = e_lo + 64 + lane; e < e_hi; e += 32) fix(fetch(e), 1);
        // value outliers of the warp's rows: the exact fp16 value over the dense one, one lane per entry
        for (int e = lane; e < 16 * a.n_v; e += 32) {
          const int t = t0w + (e & 15), k = e >> 4;
          if (t0 + t >= n_len) continue;
          const uint32_t ev = a.n_v <= Lay::NVS ? reinterpret_cast<const uint32_t*>(B_ + Lay::B_VO)[k * kChunk + t]
                                                : ld_cache<kStep>(a.v_out + (bh * a.T_cap + t0 + t) * a.n_v + k);
          const int chn = (int)(ev >> 16);
          if (chn >= D) continue;
          const int col = chn < NP ? 2 * chn : 2 * (chn - NP) + 1;
          *reinterpret_cast<uint16_t*>(v_t + tile_off<D>(t, col / 8) + (col % 8) * 2) = (uint16_t)(ev & 0xffffu);
        }
        __syncwarp();
      }
      const int qrow = (real ? g : 0) * (QROW / 2);
      const uint2* qh2 = reinterpret_cast<const uint2*>(B_ + Lay::B_QH) + qrow;
      const uint2* ql2 = reinterpret_cast<const uint2*>(B_ + Lay::B_QL) + qrow;
      // S^T = K_hi q_hi + K_lo q_hi + K_hi q_lo on 16 tokens x 8 heads, two independent accumulators
      // (even / odd kc)
      float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int kc = 0; kc < KC; ++kc) {
        const uint2 bhq = real ? qh2[kc * 4 + r] : make_uint2(0u, 0u);
        const uint2 blq = real ? ql2[kc * 4 + r] : make_uint2(0u, 0u);
        uint32_t ahi[4], alo[4];
        ldsm_x4(ahi, khi_t + tile_off<D>(tokA, 2 * kc + chA));
        ldsm_x4(alo, klo_t + tile_off<D>(tokA, 2 * kc + chA));
        float* acc = (kc & 1) ? sb : sa;
        mma16816(acc, ahi[0], ahi[1], ahi[2], ahi[3], bhq.x, bhq.y);
        mma16816(acc, alo[0], alo[1], alo[2], alo[3], bhq.x, bhq.y);
        mma16816(acc, ahi[0], ahi[1], ahi[2], ahi[3], blq.x, blq.y);
      }
      // x[e][u]: head 2r + e, token g + 8u of the slab
      const bool ok0 = t0 + t0w + g < n_len, ok1 = t0 + t0w + g + 8 < n_len;
      float x[2][2];
      x[0][0] = ok0 ? (sa[0] + sb[0]) * a.scale_log2 : -INFINITY;
      x[1][0] = ok0 ? (sa[1] + sb[1]) * a.scale_log2 : -INFINITY;
      x[0][1] = ok1 ? (sa[2] + sb[2]) * a.scale_log2 : -INFINITY;
      x[1][1] = ok1 ? (sa[3] + sb[3]) * a.scale_log2 : -INFINITY;
      float p[2][2];
      // the running maxima move only when a score exceeds them: then (rarely, after the first
      // chunks) reduce the slab's maxima across the lanes of each head and rescale
      if (__any_sync(0xffffffffu, fmaxf(x[0][0], x[0][1]) > m_run[0] || fmaxf(x[1][0], x[1][1]) > m_run[1])) {
        float alpha[2] = {1.f, 1.f};
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          float mx = fmaxf(x[e][0], x[e][1]);
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
          const float m_new = fmaxf(m_run[e], mx);
          if (m_new != -INFINITY) alpha[e] = exp2f(m_run[e] - m_new);
          l_part[e] *= alpha[e];
          m_run[e] = m_new;
        }
#pragma unroll
        for (int j = 0; j < D / 16; ++j) {
          o[j][0] *= alpha[0];
          o[j][1] *= alpha[1];
          o[j][2] *= alpha[0];
          o[j][3] *= alpha[1];
        }
      }
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        // exp2(-inf - m) = 0 for masked tokens; a head with no score yet (m = -inf) has none
        p[e][0] = m_run[e] != -INFINITY ? exp2f(x[e][0] - m_run[e]) : 0.f;
        p[e][1] = m_run[e] != -INFINITY ? exp2f(x[e][1] - m_run[e]) : 0.f;
        l_part[e] += p[e][0] + p[e][1];
      }
      // P as two 8x8 (token x head) fp16 matrices, transposed into the B operand (tokens x heads)
      const uint32_t pb0 = movm_trans(pack_half2(p[0][0], p[1][0]));
      const uint32_t pb1 = movm_trans(pack_half2(p[0][1], p[1][1]));
#pragma unroll
      for (int j = 0; j < D / 16; ++j) {
        uint32_t av[4];
        ldsm_x4_t(av, v_t + tile_off<D>(tokV, 2 * j + chV));
        mma16816(o[j], av[0], av[1], av[2], av[3], pb0, pb1);
      }
      if (c + 2 < nchunks) bar_arrive(kBarEmpty + buf, kThr);   // producers may refill the buffer
    }
    // The producers are done with every stage once the last chunk was handed over (and no
    // stage was filled when there are no chunks), so the stage area takes the partials.
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      l_part[e] += __shfl_xor_sync(0xffffffffu, l_part[e], 4);
      l_part[e] += __shfl_xor_sync(0xffffffffu, l_part[e], 8);
      l_part[e] += __shfl_xor_sync(0xffffffffu, l_part[e], 16);
      const int hh = 2 * r + e;
      if (hh < a.G) {
        if (g == 0) {
          wm[cw * 8 + hh] = m_run[e];
          wl[cw * 8 + hh] = l_part[e];
        }
#pragma unroll
        for (int j = 0; j < D / 16; ++j) {
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int col = 16 * j + g + 8 * u;                  // tile column -> channel
            wo[(cw * 8 + hh) * D + (col >> 1) + (col & 1) * NP] = o[j][2 * u + e];
          }
        }
      }
    }
    end_unit(bh);
    x = xe;
    }
  }
}

template <int D, int BITS, bool kStep>
cudaError_t launch_kvq_s(const KvqArgs& a, cudaStream_t st) {
  using Lay = KvqLayout<D, BITS>;
  static_assert(Lay::BYTES <= 227 * 1024, "one CTA per SM");
  static int checked = 0;                 // 1: attributes set and register count verified
  if (!checked) {
    cudaFuncAttributes attr;
    cudaError_t e = cudaFuncGetAttributes(&attr, decode_kvq_kernel<D, BITS, kStep>);
    if (e != cudaSuccess) return e;
    // the register split above assumes exactly kRegLaunch registers a thread at launch
    if (attr.numRegs != kRegLaunch) return cudaErrorInvalidConfiguration;
    e = cudaFuncSetAttribute(decode_kvq_kernel<D, BITS, kStep>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             Lay::BYTES);
    if (e != cudaSuccess) return e;
    checked = 1;
  }
  decode_kvq_kernel<D, BITS, kStep><<<a.n_cta, kThr, Lay::BYTES, st>>>(a);
  return cudaPeekAtLastError();
}

template <int D, int BITS>
cudaError_t launch_kvq_t(const KvqArgs& a, cudaStream_t st) {
  return a.step ? launch_kvq_s<D, BITS, true>(a, st) : launch_kvq_s<D, BITS, false>(a, st);
}

}  // namespace

int kvquant_step_max_units_per_cta() { return kMaxUnitsCta; }

cudaError_t take_status_kvq_step(uint32_t* flags, cudaStream_t st) {
  uint32_t zero = 0, v = 0;
  cudaError_t e = cudaMemcpyFromSymbolAsync(&v, g_status_kvq, sizeof(v), 0, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyToSymbolAsync(g_status_kvq, &zero, sizeof(zero), 0, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  *flags |= v;
  return e;
}

cudaError_t launch_decode_kvquant(const mkv_config& c, const void* q, const mkv_cache& cache,
                                  const mkv_quant_params& qp, void* out, const DecodeWs& ws, const Split& sp,
                                  cudaStream_t st, const void* k_new, const void* v_new) {
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
  a.n_split = sp.n_split;
  a.n_cta = sp.n_cta;
  a.cpu = sp.chunks_per_unit;
  a.c_tot = sp.chunks_per_unit * c.B * c.Hkv;
  const float scale = c.softmax_scale > 0.f ? c.softmax_scale : 1.0f / sqrtf((float)c.D);
  a.scale_log2 = scale * kLog2e;
  a.part_m = ws.part_m;
  a.part_l = ws.part_l;
  a.part_o = ws.part_o;
  a.merge = merge_args(c, ws, sp, out, false);
  if (k_new) {
    a.step = 1;
    a.st.k_new = static_cast<const __half*>(k_new);
    a.st.v_new = static_cast<const __half*>(v_new);
    a.st.T_len = cache.T_len;
    a.st.k_codes = cache.k_codes;
    a.st.v_codes = cache.v_codes;
    a.st.v_params = reinterpret_cast<float2*>(cache.v_params);
    a.st.v_out = cache.v_out;
    a.st.k_out_off = cache.k_out_off;
    a.st.k_out = cache.k_out;
    a.st.t_lo = qp.t_lo;
    a.st.t_hi = qp.t_hi;
    a.st.k_lo = qp.k_lo;
    a.st.k_scale = qp.k_scale;
    a.st.k_cb = qp.k_cb;
    a.st.v_cb = qp.v_cb;
    a.st.nuq = c.quant_mode == MKV_QUANT_NUQ;
  }
  if (c.D == 128) {
    if (c.bits == 4) return launch_kvq_t<128, 4>(a, st);
    if (c.bits == 3) return launch_kvq_t<128, 3>(a, st);
    return launch_kvq_t<128, 2>(a, st);
  }
  if (c.bits == 4) return launch_kvq_t<64, 4>(a, st);
  if (c.bits == 3) return launch_kvq_t<64, 3>(a, st);
  return launch_kvq_t<64, 2>(a, st);
}

}  // namespace mkv
