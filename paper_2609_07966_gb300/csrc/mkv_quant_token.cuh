// One token of one (batch, kv-head) quantized into the KVQuant cache (Section 2.1,
// KVQuant paragraph): per-channel key codes (pre-rotation), the key outliers as
// CSR entries, the token's value outliers, its value range and value codes.
// Shared by the quantize kernel (one CTA per unit, one thread per channel) and
// the fused decode step (the attention warps of the CTA that owns the token's
// chunk), so both write the same bits.
//
// Codes are decided with correctly rounded fp32 operations (__fsub_rn, __fdiv_rn,
// __fmul_rn, rintf):
//   uniform: code = clamp(rint((x - lo) / scale), 0, 2^b - 1)
//   NUQ:     code = #{j : x > mu_j},  mu_j = (c_j + c_{j+1}) * 0.5 in fp32
// Key outliers: x < t_lo or x > t_hi (per channel); value outliers: the n_v
// entries of largest |x| of the token (ties: lower channel).  Outliers keep the
// code of their clamped value and are stored exactly in fp16 on the side.
#pragma once

#include "mkv_common.cuh"

namespace mkv {

__device__ __forceinline__ float fl32_mid(float a, float b) { return __fmul_rn(__fadd_rn(a, b), 0.5f); }

__device__ __forceinline__ int uniform_code(float x, float lo, float scale, int L) {
  if (scale == 0.f) return 0;
  const float r = rintf(__fdiv_rn(__fsub_rn(x, lo), scale));
  return (int)fminf(fmaxf(r, 0.f), (float)L);
}

// The cache rows of one (batch, kv-head) unit.
struct QTokDst {
  uint32_t* k_out;      // [k_out_cap] key-outlier entries
  int64_t k_out_cap;
  uint32_t* v_out;      // [T_cap][n_v] value outliers
  float2* v_params;     // [T_cap] value (lo, scale)
  uint8_t* k_codes;     // [T_cap][D * bits / 8]
  uint8_t* v_codes;
  int32_t* off_row;     // [T_cap + 1] CSR offsets of the key outliers
};

// Shared scratch of the thread group (D >= 32 channels, one warp per 32 of them).
struct QTokSmem {
  uint8_t* kcode;       // [D]
  uint8_t* vcode;       // [D]
  float* absx;          // [D]
  uint32_t* words;      // [2][nwords] packed key and value rows
  int* cnt;             // [warps] key outliers per warp
  float* lo;            // [warps]
  float* hi;            // [warps]
  uint32_t* mx;         // [2][32] per-warp maxima of the value-outlier rounds
};

// Quantizes the token at position t, whose key-outlier entries start at `off`; thread c owns
// channel c (threads c >= D take part in the group's barriers only).  kmu / vmu are the channel's
// NUQ midpoints, (tlo, thi) its key-outlier thresholds, (klo, ksc) its uniform key grid.  `sync`
// is a barrier over the whole group, called the same number of times by every thread.  Returns the
// offset after the token's entries (the value stored at off_row[t + 1]).  Entries beyond k_out_cap
// are dropped and raise MKV_FLAG_K_OUTLIER_OVERFLOW in *status.
template <typename Sync>
__device__ __forceinline__ int32_t quantize_token(int c, int D, int bits, bool nuq, int n_v, const float (&kmu)[15],
                                                  const float (&vmu)[15], float tlo, float thi, float klo, float ksc,
                                                  __half xk, __half xv, int64_t t, int32_t off, const QTokDst& o,
                                                  const QTokSmem& s, uint32_t* status, Sync sync) {
  const int K = 1 << bits, L = K - 1, NP = D / 2;
  const bool act = c < D;
  const int warp = c >> 5, lane = c & 31, nwarp = D >> 5;
  const int rowb = D * bits / 8;
  const int nwords = (rowb + 3) / 4;
  // ---- keys
  const float x = __half2float(xk);
  const bool kout = act && ((x < tlo) || (x > thi));
  int code;
  if (nuq) {
    code = 0;
#pragma unroll
    for (int j = 0; j < 15; ++j) code += (j < L && x > kmu[j]) ? 1 : 0;   // registers, no local array
  } else {
    code = uniform_code(x, klo, ksc, L);
  }
  if (act) s.kcode[c] = (uint8_t)code;
  // rank of this outlier among the token's outliers (channel order)
  const unsigned bal = __ballot_sync(0xffffffffu, kout);
  if (lane == 0) s.cnt[warp] = __popc(bal);
  // ---- values: rank by (|x| desc, channel asc).  With few value outliers the ranks 0..n_v-1 are
  // taken by group-wide maxima of key = (|x| as fp16 magnitude bits << 8) | (255 - c), which orders
  // like (|x| desc, channel asc) for finite values and is unique; the first round shares this
  // barrier.  Otherwise each thread counts the channels ahead of it.
  const float vx = __half2float(xv);
  const bool few = n_v <= 8;
  uint32_t vkey = act ? (((uint32_t)(__half_as_ushort(xv) & 0x7fffu) << 8) | (uint32_t)(255 - c)) : 0u;
  if (few) {
    const uint32_t wmax = __reduce_max_sync(0xffffffffu, vkey);
    if (lane == 0 && n_v > 0) s.mx[warp] = wmax;
  } else if (act) {
    s.absx[c] = fabsf(vx);
  }
  sync();
  int before = 0, total = 0;
  for (int w = 0; w < nwarp; ++w) {
    before += (w < warp) ? s.cnt[w] : 0;
    total += s.cnt[w];
  }
  if (kout) {
    const int64_t e = (int64_t)off + before + __popc(bal & ((1u << lane) - 1u));
    if (e < o.k_out_cap) {
      // (token position within its 64-token block << 24) | (channel << 16) | fp16 bits
      o.k_out[e] = ((uint32_t)(t & 63) << 24) | ((uint32_t)c << 16) | __half_as_ushort(xk);
    } else {
      atomicOr(status, MKV_FLAG_K_OUTLIER_OVERFLOW);
    }
  }
  int rank = 0;
  if (few) {
    rank = n_v;                        // not among the n_v largest unless a round picks it
    for (int r = 0; r < n_v; ++r) {
      if (r > 0) {
        const uint32_t wmax = __reduce_max_sync(0xffffffffu, vkey);
        if (lane == 0) s.mx[(r & 1) * 32 + warp] = wmax;
        sync();
      }
      uint32_t m = s.mx[(r & 1) * 32];
      for (int w = 1; w < nwarp; ++w) m = max(m, s.mx[(r & 1) * 32 + w]);
      if (vkey == m) {                 // every live key is >= 128, the idle threads' 0 never matches
        rank = r;
        vkey = 0u;                     // out of the later rounds
      }
    }
  } else if (act) {
    const float ax = s.absx[c];
    for (int j = 0; j < D; ++j) {
      const float oj = s.absx[j];
      rank += (oj > ax || (oj == ax && j < c)) ? 1 : 0;
    }
  }
  const bool vout = act && rank < n_v;
  // inlier range of the token's values
  float lo = (vout || !act) ? INFINITY : vx, hi = (vout || !act) ? -INFINITY : vx;
  for (int sh = 16; sh > 0; sh >>= 1) {
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, sh));
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, sh));
  }
  if (lane == 0) {
    s.lo[warp] = lo;
    s.hi[warp] = hi;
  }
  sync();
  lo = s.lo[0];
  hi = s.hi[0];
  for (int w = 1; w < nwarp; ++w) {
    lo = fminf(lo, s.lo[w]);
    hi = fmaxf(hi, s.hi[w]);
  }
  if (lo > hi) lo = hi = 0.f;   // no inlier
  float scale;
  int vc;
  if (nuq) {
    scale = __fsub_rn(hi, lo);
    const float u = scale == 0.f ? 0.f : __fdiv_rn(__fsub_rn(vx, lo), scale);
    vc = 0;
#pragma unroll
    for (int j = 0; j < 15; ++j) vc += (j < L && u > vmu[j]) ? 1 : 0;
  } else {
    scale = __fdiv_rn(__fsub_rn(hi, lo), (float)L);
    vc = uniform_code(vx, lo, scale, L);
  }
  if (act) s.vcode[c] = (uint8_t)vc;
  if (vout) o.v_out[t * n_v + rank] = ((uint32_t)c << 16) | __half_as_ushort(xv);
  if (c == 0) o.v_params[t] = make_float2(lo, scale);
  if (act)
    for (int wi = c; wi < 2 * nwords; wi += D) s.words[wi] = 0u;
  sync();
  // pack pair i = channels (i, i + D/2) at bits [2*bits*i, 2*bits*(i+1))
  if (c < NP) {
    const uint32_t pk = (uint32_t)s.kcode[c] | ((uint32_t)s.kcode[c + NP] << bits);
    const uint32_t pv = (uint32_t)s.vcode[c] | ((uint32_t)s.vcode[c + NP] << bits);
    const int bit = 2 * bits * c;
    const int w0 = bit >> 5, sh = bit & 31;
    atomicOr(&s.words[w0], pk << sh);
    atomicOr(&s.words[nwords + w0], pv << sh);
    if (sh + 2 * bits > 32) {
      atomicOr(&s.words[w0 + 1], pk >> (32 - sh));
      atomicOr(&s.words[nwords + w0 + 1], pv >> (32 - sh));
    }
  }
  sync();
  if (act) {
    for (int by = c; by < rowb; by += D) {
      o.k_codes[t * rowb + by] = reinterpret_cast<const uint8_t*>(s.words)[by];
      o.v_codes[t * rowb + by] = reinterpret_cast<const uint8_t*>(s.words + nwords)[by];
    }
  }
  const int32_t next = off + total;
  if (c == 0) o.off_row[t + 1] = next;
  sync();                              // the scratch may be reused for the next token
  return next;
}

}  // namespace mkv
