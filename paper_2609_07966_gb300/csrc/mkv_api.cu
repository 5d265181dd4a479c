// C ABI layer of libmkv: argument validation, workspace carve-up, dispatch.
// Every entry point validates on the host and launches nothing on a bad
// argument; launch failures map to MKV_ERR_CUDA (see include/mkv.h).
#include <math.h>
#include <stdarg.h>
#include <stdio.h>

#include <algorithm>

#include "mkv_common.cuh"
#include "mkv_internal.h"

namespace mkv {

namespace {
thread_local char g_err[512] = "no error";
}

void set_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
}

Split decode_split(const mkv_config& c, int64_t T_cap) {
  Split s{};
  s.v_tokens = c.method == MKV_ROCKET ? (int64_t)(c.topk_pages + 1) * kPage
              : c.method == MKV_H2O  ? std::min<int64_t>(T_cap, (int64_t)c.h2o_heavy + c.h2o_recent + 1)
                                     : T_cap;
  const int64_t chunks = std::max<int64_t>(1, ceil_div(s.v_tokens, kChunk));
  const int64_t units = (int64_t)c.B * c.Hkv;
  // The fp16-family decode kernels keep two CTAs resident per SM, the KVQuant
  // kernel one.  Pick the split count that minimises (waves of CTAs) x
  // (chunks per CTA), i.e. the time of the busiest SM; among equals prefer
  // fewer splits (smaller partials).
  const int64_t slots = (c.method == MKV_KVQUANT ? 1 : 2) * kNumSMs;
  int64_t best_n = 1, best_cost = INT64_MAX;
  for (int64_t n = 1; n <= std::min<int64_t>(chunks, 1024); ++n) {
    const int64_t cps = ceil_div(chunks, n);
    if (ceil_div(chunks, cps) != n) continue;      // n is not the split count of any cps
    // + 6: a CTA's fixed cost (query and table loads, pipeline fill and drain, merge) in chunk
    // units, fitted to measured split sweeps of the FP16 and KVQuant kernels
    const int64_t cost = ceil_div(units * n, slots) * (cps + 6);
    if (cost < best_cost) {
      best_cost = cost;
      best_n = n;
    }
  }
  s.chunks_per_split = (int)ceil_div(chunks, best_n);
  s.n_split = (int)ceil_div(chunks, s.chunks_per_split);
  if (c.method == MKV_KVQUANT) {
    // one CTA per SM, each over an equal range of all units' chunks (at most a few units per
    // CTA); a unit's partial slots are the CTAs that cover part of it
    const int64_t c_tot = units * chunks;
    s.chunks_per_unit = chunks;
    s.n_cta = (int)std::min<int64_t>(kNumSMs, c_tot);
    int64_t slots_max = 1;
    for (int64_t u = 0; u < units; ++u) {
      const int64_t n = cta_of_chunk((u + 1) * chunks - 1, c_tot, s.n_cta) - cta_of_chunk(u * chunks, c_tot, s.n_cta) + 1;
      slots_max = std::max(slots_max, n);
    }
    s.n_split = (int)slots_max;
    s.chunks_per_split = (int)chunks;
  }
  return s;
}

DecodeWs decode_ws(const mkv_config& c, int64_t T_cap, void* base) {
  const Split sp = decode_split(c, T_cap);
  const size_t hq = (size_t)c.B * c.Hq;
  uint8_t* p = static_cast<uint8_t*>(base);
  size_t off = kCounterBytes;
  DecodeWs w{};
  auto take = [&](size_t bytes) -> float* {
    float* r = base ? reinterpret_cast<float*>(p + off) : nullptr;
    off += align256(bytes);
    return r;
  };
  w.part_m = take(hq * sp.n_split * 4);
  w.part_l = take(hq * sp.n_split * 4);
  w.part_o = take(hq * sp.n_split * c.D * 4);
  w.counters = base ? static_cast<int*>(base) : nullptr;
  if (c.method == MKV_H2O) {
    w.logits = take((size_t)c.B * c.Hkv * T_cap * (c.Hq / c.Hkv) * 4);
    w.m_tot = take(hq * 4);
    w.l_tot = take(hq * 4);
  }
  w.bytes = off;
  return w;
}

PrefillWs prefill_ws(const mkv_config& c, int64_t T, void* base) {
  uint8_t* p = static_cast<uint8_t*>(base);
  size_t off = kCounterBytes;
  auto take = [&](size_t bytes) -> void* {
    void* r = base ? p + off : nullptr;
    off += align256(bytes);
    return r;
  };
  PrefillWs w{};
  w.row_st = static_cast<float2*>(take((size_t)c.B * c.Hq * (T + 128) * 8));
  w.score = static_cast<float*>(take((size_t)c.B * c.Hkv * T * 4));
  w.keep = static_cast<int32_t*>(take((size_t)c.B * c.Hkv * T * 4));
  w.bytes = off;
  return w;
}

CalibWs calib_ws(const mkv_config& c, int64_t N, void* base) {
  uint8_t* p = static_cast<uint8_t*>(base);
  size_t off = kCounterBytes;
  auto take = [&](size_t bytes) -> void* {
    void* r = base ? p + off : nullptr;
    off += align256(bytes);
    return r;
  };
  CalibWs w{};
  w.sorted = static_cast<float*>(take((size_t)c.Hkv * c.D * N * 4));
  w.u = static_cast<float*>(take((size_t)c.Hkv * N * c.D * 4));
  w.vmask = static_cast<uint8_t*>(take((size_t)c.Hkv * N * c.D));
  w.bytes = off;
  return w;
}

}  // namespace mkv

using namespace mkv;

namespace {

#define MKV_CUDA(expr)                                                          \
  do {                                                                          \
    cudaError_t e_ = (expr);                                                    \
    if (e_ != cudaSuccess) {                                                    \
      set_error("%s: %s", #expr, cudaGetErrorString(e_));                       \
      return MKV_ERR_CUDA;                                                      \
    }                                                                           \
  } while (0)

#define MKV_REQUIRE(cond, code, ...) \
  do {                               \
    if (!(cond)) {                   \
      set_error(__VA_ARGS__);        \
      return code;                   \
    }                                \
  } while (0)

inline cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

mkv_status check_config(const mkv_config* c) {
  MKV_REQUIRE(c != nullptr, MKV_ERR_INVALID_ARG, "config is NULL");
  MKV_REQUIRE(c->abi_version == MKV_ABI_VERSION, MKV_ERR_INVALID_ARG, "abi_version %u != %u",
              c->abi_version, MKV_ABI_VERSION);
  MKV_REQUIRE(c->method >= MKV_FP16 && c->method <= MKV_ROCKET, MKV_ERR_INVALID_ARG,
              "unknown method %d", c->method);
  MKV_REQUIRE(c->B >= 1 && c->Hq >= 1 && c->Hkv >= 1 && c->D >= 1, MKV_ERR_INVALID_ARG,
              "B, Hq, Hkv, D must be positive");
  MKV_REQUIRE(c->Hq % c->Hkv == 0, MKV_ERR_INVALID_ARG, "Hq %% Hkv != 0");
  MKV_REQUIRE((int64_t)c->B * c->Hkv <= kMaxUnits, MKV_ERR_UNSUPPORTED, "B * Hkv = %lld above %d",
              (long long)c->B * c->Hkv, kMaxUnits);
  const int G = c->Hq / c->Hkv;
  MKV_REQUIRE(G == 1 || G == 2 || G == 4 || G == 8, MKV_ERR_UNSUPPORTED, "G = %d not built", G);
  MKV_REQUIRE(c->D == 64 || c->D == 128, MKV_ERR_UNSUPPORTED, "D = %d not built", c->D);
  MKV_REQUIRE(c->softmax_scale >= 0.f && isfinite(c->softmax_scale), MKV_ERR_INVALID_ARG,
              "softmax_scale must be >= 0");
  if (c->method == MKV_KVQUANT) {
    MKV_REQUIRE(c->bits >= 2 && c->bits <= 4, MKV_ERR_UNSUPPORTED, "bits = %d not built", c->bits);
    MKV_REQUIRE(c->quant_mode == MKV_QUANT_UNIFORM || c->quant_mode == MKV_QUANT_NUQ,
                MKV_ERR_INVALID_ARG, "unknown quant_mode %d", c->quant_mode);
    MKV_REQUIRE(c->outlier_frac >= 0.f && c->outlier_frac <= 1.f, MKV_ERR_INVALID_ARG,
                "outlier_frac outside [0, 1]");
    MKV_REQUIRE(c->rope_theta > 0.f, MKV_ERR_INVALID_ARG, "rope_theta must be > 0");
  }
  if (c->method == MKV_H2O) {
    MKV_REQUIRE(c->h2o_heavy >= 0 && c->h2o_recent >= 0 && c->h2o_heavy + c->h2o_recent >= 1,
                MKV_ERR_INVALID_ARG, "H2O budget must be >= 1");
  }
  if (c->method == MKV_ROCKET) {
    MKV_REQUIRE(c->page_size == kPage, MKV_ERR_UNSUPPORTED, "page_size %d not built", c->page_size);
    MKV_REQUIRE(c->topk_pages >= 1, MKV_ERR_INVALID_ARG, "topk_pages must be >= 1");
    MKV_REQUIRE(c->topq_dims >= 1 && c->topq_dims <= c->D, MKV_ERR_INVALID_ARG,
                "topq_dims outside [1, D]");
    MKV_REQUIRE(c->snap_window >= 1 && c->snap_keep >= c->snap_window, MKV_ERR_INVALID_ARG,
                "snap_window/snap_keep invalid");
    MKV_REQUIRE(c->snap_pool >= 1 && (c->snap_pool & 1), MKV_ERR_INVALID_ARG,
                "snap_pool must be odd");
  }
  return MKV_OK;
}

int n_value_outliers(const mkv_config* c) {
  return std::min(c->D, (int)ceil((double)c->outlier_frac * c->D));
}

mkv_status check_cache(const mkv_config* c, const mkv_cache* k) {
  MKV_REQUIRE(k != nullptr, MKV_ERR_INVALID_ARG, "cache is NULL");
  MKV_REQUIRE(k->T_cap >= 1 && k->T_len != nullptr, MKV_ERR_INVALID_ARG, "cache T_cap/T_len invalid");
  switch (c->method) {
    case MKV_FP16:
      MKV_REQUIRE(k->k && k->v, MKV_ERR_INVALID_ARG, "FP16 cache needs k and v");
      break;
    case MKV_H2O:
      MKV_REQUIRE(k->k && k->v && k->pos && k->acc && k->slot, MKV_ERR_INVALID_ARG,
                  "H2O cache needs k, v, pos, acc, slot");
      MKV_REQUIRE(k->T_cap >= (int64_t)c->h2o_heavy + c->h2o_recent + 1, MKV_ERR_INVALID_ARG,
                  "H2O cache needs T_cap >= heavy + recent + 1");
      break;
    case MKV_ROCKET:
      MKV_REQUIRE(k->k && k->v && k->kmin && k->kmax, MKV_ERR_INVALID_ARG,
                  "ROCKET cache needs k, v, kmin, kmax");
      MKV_REQUIRE(k->T_cap % kPage == 0, MKV_ERR_INVALID_ARG, "ROCKET T_cap must be a multiple of 16");
      MKV_REQUIRE(((uintptr_t)k->kmin & 15) == 0 && ((uintptr_t)k->kmax & 15) == 0, MKV_ERR_INVALID_ARG,
                  "ROCKET kmin/kmax must be 16-byte aligned");
      break;
    case MKV_KVQUANT:
      MKV_REQUIRE(k->k_codes && k->v_codes && k->v_params && k->k_out_off && k->k_out &&
                      k->k_out_cap >= 0 && (n_value_outliers(c) == 0 || k->v_out),
                  MKV_ERR_INVALID_ARG, "KVQUANT cache needs codes, params and outlier stores");
      break;
  }
  return MKV_OK;
}

mkv_status check_qparams(const mkv_config* c, const mkv_quant_params* p, bool need_tables) {
  MKV_REQUIRE(p != nullptr, MKV_ERR_INVALID_ARG, "quant params are NULL");
  MKV_REQUIRE(p->t_lo && p->t_hi, MKV_ERR_INVALID_ARG, "quant params need t_lo, t_hi");
  if (c->quant_mode == MKV_QUANT_UNIFORM) {
    MKV_REQUIRE(p->k_lo && p->k_scale, MKV_ERR_INVALID_ARG, "uniform mode needs k_lo, k_scale");
  } else {
    MKV_REQUIRE(p->k_cb && p->v_cb, MKV_ERR_INVALID_ARG, "NUQ mode needs k_cb, v_cb");
  }
  if (need_tables) {
    MKV_REQUIRE(p->k_dq && p->v_tbl, MKV_ERR_INVALID_ARG, "quant params need k_dq, v_tbl");
  }
  return MKV_OK;
}

#define MKV_TRY(expr)              \
  do {                             \
    mkv_status s_ = (expr);        \
    if (s_ != MKV_OK) return s_;   \
  } while (0)

size_t workspace_bytes(const mkv_config* c, int64_t T_cap) {
  size_t b = decode_ws(*c, T_cap, nullptr).bytes;
  if (c->method == MKV_H2O || c->method == MKV_ROCKET) b = std::max(b, prefill_ws(*c, T_cap, nullptr).bytes);
  if (c->method == MKV_KVQUANT) b = std::max(b, calib_ws(*c, std::min<int64_t>(T_cap, 4096), nullptr).bytes);
  return b;
}

}  // namespace

mkv_status mkv::check_fp16_decode_args(const mkv_config* cfg, const mkv_cache* cache, const void* q,
                                       const void* out) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_FP16, MKV_ERR_UNSUPPORTED, "this entry point serves FP16 caches only");
  MKV_TRY(check_cache(cfg, cache));
  MKV_REQUIRE(q && out, MKV_ERR_INVALID_ARG, "q/out NULL");
  return MKV_OK;
}

extern "C" {

const char* mkv_last_error(void) { return mkv::g_err; }

mkv_status mkv_workspace_size(const mkv_config* cfg, int64_t T_cap, size_t* bytes) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(bytes != nullptr && T_cap >= 1, MKV_ERR_INVALID_ARG, "bytes NULL or T_cap < 1");
  *bytes = workspace_bytes(cfg, T_cap);
  return MKV_OK;
}

mkv_status mkv_cache_bytes(const mkv_config* c, int64_t T, size_t* resident, size_t* peak) {
  MKV_TRY(check_config(c));
  MKV_REQUIRE(resident && peak && T >= 0, MKV_ERR_INVALID_ARG, "resident/peak NULL or T < 0");
  const size_t units = (size_t)c->B * c->Hkv;
  const size_t fp16_tok = (size_t)c->D * 2 * 2;    // K and V rows
  const size_t prompt = units * (size_t)T * fp16_tok;
  size_t res = 0;
  switch (c->method) {
    case MKV_FP16:
      res = prompt;
      *resident = res;
      *peak = res;
      return MKV_OK;
    case MKV_KVQUANT: {
      const size_t codes = (size_t)c->D * c->bits / 8 * 2;
      const size_t k_out = (size_t)ceil((double)c->outlier_frac * c->D) * 4;   // expected key outliers
      res = units * (size_t)T * (codes + 8 + (size_t)n_value_outliers(c) * 4 + 4 + k_out) + units * 4;
      break;
    }
    case MKV_H2O:
      res = units * std::min<size_t>(T, (size_t)c->h2o_heavy + c->h2o_recent) * (fp16_tok + 8);
      break;
    case MKV_ROCKET: {
      const size_t kept = std::min<size_t>(T, (size_t)c->snap_keep);
      res = units * kept * fp16_tok + units * 2 * (size_t)c->D * ((kept + kPage - 1) / kPage) * 2;
      break;
    }
  }
  *resident = res;
  *peak = res + prompt;
  return MKV_OK;
}

mkv_status mkv_rope_table(int32_t D, float theta, int64_t T_max, float* table, void* stream) {
  MKV_REQUIRE(D == 64 || D == 128, MKV_ERR_UNSUPPORTED, "D = %d not built", D);
  MKV_REQUIRE(theta > 0.f && T_max >= 1 && table != nullptr, MKV_ERR_INVALID_ARG,
              "theta <= 0, T_max < 1 or table NULL");
  MKV_CUDA(launch_rope_table(D, theta, T_max, table, as_stream(stream)));
  return MKV_OK;
}

mkv_status mkv_wait_timeout_selftest(int32_t ms, void* stream) {
  MKV_REQUIRE(ms >= 1 && ms <= 1000, MKV_ERR_INVALID_ARG, "ms = %d outside [1, 1000]", ms);
  MKV_CUDA(launch_wait_selftest(ms, as_stream(stream)));
  return MKV_OK;
}

mkv_status mkv_get_status(void* stream, uint32_t* flags) {
  MKV_REQUIRE(flags != nullptr, MKV_ERR_INVALID_ARG, "flags is NULL");
  *flags = 0;
  MKV_CUDA(take_status_append(flags, as_stream(stream)));
  MKV_CUDA(take_status_kvquant(flags, as_stream(stream)));
  MKV_CUDA(take_status_rocket(flags, as_stream(stream)));
  MKV_CUDA(take_status_decode(flags, as_stream(stream)));
  MKV_CUDA(take_status_prefill(flags, as_stream(stream)));
  MKV_CUDA(take_status_kvq_step(flags, as_stream(stream)));
  if (*flags & MKV_FLAG_WAIT_TIMEOUT) {
    set_error("device status flags 0x%x (a bounded wait ran out)", *flags);
    return MKV_ERR_TIMEOUT;
  }
  if (*flags != 0) {
    set_error("device status flags 0x%x", *flags);
    return MKV_ERR_CAPACITY;
  }
  return MKV_OK;
}

mkv_status mkv_append_kv(const mkv_config* cfg, const void* k_new, const void* v_new, mkv_cache* cache,
                         void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method != MKV_KVQUANT, MKV_ERR_INVALID_ARG,
              "KVQUANT caches append through mkv_quantize_kv");
  MKV_TRY(check_cache(cfg, cache));
  MKV_REQUIRE(k_new && v_new, MKV_ERR_INVALID_ARG, "k_new/v_new NULL");
  MKV_CUDA(launch_append(*cfg, k_new, v_new, *cache, as_stream(stream)));
  return MKV_OK;
}

mkv_status mkv_decode_attention(const mkv_config* cfg, const void* q, const mkv_cache* cache,
                                const mkv_quant_params* qparams, const int32_t* page_idx, void* out,
                                void* ws, size_t ws_bytes, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_TRY(check_cache(cfg, cache));
  MKV_REQUIRE(q && out, MKV_ERR_INVALID_ARG, "q/out NULL");
  if (cfg->method == MKV_ROCKET) MKV_REQUIRE(page_idx != nullptr, MKV_ERR_INVALID_ARG, "ROCKET needs page_idx");
  if (cfg->method == MKV_KVQUANT) {
    MKV_TRY(check_qparams(cfg, qparams, true));
    MKV_REQUIRE(qparams->rope && qparams->rope_len >= std::max<int64_t>(cache->T_cap, 64), MKV_ERR_INVALID_ARG,
                "KVQUANT decode needs a rope table with rope_len >= max(T_cap, 64)");
    MKV_REQUIRE(((uintptr_t)cache->k_codes | (uintptr_t)cache->v_codes) % 16 == 0, MKV_ERR_INVALID_ARG,
                "KVQUANT decode stages k_codes / v_codes in 16-byte pieces: both must be 16-byte aligned");
    MKV_REQUIRE(cache->k_out_cap <= INT32_MAX && cache->T_cap < INT32_MAX, MKV_ERR_UNSUPPORTED,
                "KVQUANT decode indexes key outliers and tokens with 32 bits (k_out_cap %lld, T_cap %lld)",
                (long long)cache->k_out_cap, (long long)cache->T_cap);
  }
  const DecodeWs need = decode_ws(*cfg, cache->T_cap, nullptr);
  MKV_REQUIRE(ws != nullptr && ws_bytes >= need.bytes, MKV_ERR_WORKSPACE,
              "workspace %zu bytes < %zu needed", ws_bytes, need.bytes);
  const DecodeWs w = decode_ws(*cfg, cache->T_cap, ws);
  const Split sp = decode_split(*cfg, cache->T_cap);
  MKV_REQUIRE(cfg->method != MKV_ROCKET || (int64_t)sp.chunks_per_split * (kChunk / kPage) + 1 <= 1024,
              MKV_ERR_UNSUPPORTED, "topk_pages too large for one decode split");
  cudaStream_t st = as_stream(stream);
  if (cfg->method == MKV_KVQUANT) {
    MKV_CUDA(launch_decode_kvquant(*cfg, q, *cache, *qparams, out, w, sp, st));
  } else {
    MKV_CUDA(launch_decode_fp16_family(*cfg, q, *cache, page_idx, out, w, sp, st));
  }
  return MKV_OK;
}

mkv_status mkv_decode_step(const mkv_config* cfg, const void* q, const void* k_new, const void* v_new,
                           mkv_cache* cache, void* out, void* ws, size_t ws_bytes, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_FP16 || cfg->method == MKV_H2O, MKV_ERR_INVALID_ARG,
              "decode_step is for FP16 and H2O (KVQUANT: mkv_kvquant_step; ROCKET: mkv_rocket_step)");
  MKV_TRY(check_cache(cfg, cache));
  MKV_REQUIRE(q && out && k_new && v_new, MKV_ERR_INVALID_ARG, "q/out/k_new/v_new NULL");
  MKV_REQUIRE(((uintptr_t)k_new | (uintptr_t)v_new) % 16 == 0, MKV_ERR_INVALID_ARG,
              "k_new/v_new must be 16-byte aligned (the step reads them in 16-byte pieces)");
  const DecodeWs need = decode_ws(*cfg, cache->T_cap, nullptr);
  MKV_REQUIRE(ws != nullptr && ws_bytes >= need.bytes, MKV_ERR_WORKSPACE,
              "workspace %zu bytes < %zu needed", ws_bytes, need.bytes);
  const Split sp = decode_split(*cfg, cache->T_cap);
  // the launch counts its finished CTAs per batch entry (Hkv x splits) in the top 8 bits of T_len[b]
  MKV_REQUIRE(cache->T_cap < (1 << 24) && (int64_t)cfg->Hkv * sp.n_split <= 255, MKV_ERR_UNSUPPORTED,
              "decode_step needs T_cap < 2^24 and Hkv * splits <= 255 (T_cap %lld, Hkv %d, splits %d); use "
              "mkv_append_kv + mkv_decode_attention",
              (long long)cache->T_cap, cfg->Hkv, sp.n_split);
  MKV_CUDA(launch_decode_fp16_family(*cfg, q, *cache, nullptr, out, decode_ws(*cfg, cache->T_cap, ws), sp,
                                     as_stream(stream), k_new, v_new));
  return MKV_OK;
}

mkv_status mkv_kvquant_step(const mkv_config* cfg, const mkv_quant_params* qparams, const void* q,
                            const void* k_new, const void* v_new, mkv_cache* cache, void* out, void* ws,
                            size_t ws_bytes, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_KVQUANT, MKV_ERR_INVALID_ARG, "kvquant_step is for KVQUANT");
  MKV_TRY(check_cache(cfg, cache));
  MKV_TRY(check_qparams(cfg, qparams, true));
  MKV_REQUIRE(q && out && k_new && v_new, MKV_ERR_INVALID_ARG, "q/out/k_new/v_new NULL");
  MKV_REQUIRE(qparams->rope && qparams->rope_len >= std::max<int64_t>(cache->T_cap, 64), MKV_ERR_INVALID_ARG,
              "KVQUANT decode needs a rope table with rope_len >= max(T_cap, 64)");
  MKV_REQUIRE(((uintptr_t)cache->k_codes | (uintptr_t)cache->v_codes) % 16 == 0, MKV_ERR_INVALID_ARG,
              "KVQUANT decode stages k_codes / v_codes in 16-byte pieces: both must be 16-byte aligned");
  MKV_REQUIRE(cache->k_out_cap <= INT32_MAX && cache->T_cap < INT32_MAX, MKV_ERR_UNSUPPORTED,
              "KVQUANT decode indexes key outliers and tokens with 32 bits (k_out_cap %lld, T_cap %lld)",
              (long long)cache->k_out_cap, (long long)cache->T_cap);
  const DecodeWs need = decode_ws(*cfg, cache->T_cap, nullptr);
  MKV_REQUIRE(ws != nullptr && ws_bytes >= need.bytes, MKV_ERR_WORKSPACE,
              "workspace %zu bytes < %zu needed", ws_bytes, need.bytes);
  const Split sp = decode_split(*cfg, cache->T_cap);
  // Each CTA that touches batch entry b takes one ticket in the top 8 bits of T_len[b] (at most
  // n_cta <= 152 of them, within the 8 bits); a CTA keeps its units' lengths in 32-entry tables (it
  // spans at most 28 of the <= 4096 units).
  const int64_t units = (int64_t)cfg->B * cfg->Hkv, cpu = sp.chunks_per_unit, c_tot = cpu * units;
  const int64_t span = (ceil_div(c_tot, (int64_t)sp.n_cta) - 1) / cpu + 2;
  MKV_REQUIRE(sp.n_cta <= 255 && span <= kvquant_step_max_units_per_cta(), MKV_ERR_UNSUPPORTED,
              "kvquant_step: %d CTAs read one batch entry's length (at most 255) or a CTA spans %lld units "
              "(at most %d); use mkv_quantize_kv + mkv_decode_attention",
              sp.n_cta, (long long)span, kvquant_step_max_units_per_cta());
  MKV_REQUIRE(cache->T_cap < (1 << 24), MKV_ERR_UNSUPPORTED,
              "kvquant_step needs T_cap < 2^24 (T_cap %lld); use mkv_quantize_kv + mkv_decode_attention",
              (long long)cache->T_cap);
  MKV_CUDA(launch_decode_kvquant(*cfg, q, *cache, *qparams, out, decode_ws(*cfg, cache->T_cap, ws), sp,
                                 as_stream(stream), k_new, v_new));
  return MKV_OK;
}

mkv_status mkv_kvquant_calibrate(const mkv_config* cfg, const void* k_cal, const void* v_cal, int64_t N_cal,
                                 int64_t row_stride, mkv_quant_params* qparams, void* ws, size_t ws_bytes,
                                 void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_KVQUANT, MKV_ERR_INVALID_ARG, "calibration is for KVQUANT");
  MKV_REQUIRE(k_cal && v_cal && N_cal >= 1 && N_cal <= 4096 && row_stride >= N_cal, MKV_ERR_INVALID_ARG,
              "k_cal/v_cal NULL, N_cal outside [1, 4096] or row_stride < N_cal");
  MKV_TRY(check_qparams(cfg, qparams, true));
  const CalibWs need = calib_ws(*cfg, N_cal, nullptr);
  MKV_REQUIRE(ws != nullptr && ws_bytes >= need.bytes, MKV_ERR_WORKSPACE,
              "workspace %zu bytes < %zu needed", ws_bytes, need.bytes);
  MKV_CUDA(launch_calibrate(*cfg, k_cal, v_cal, N_cal, row_stride, *qparams, calib_ws(*cfg, N_cal, ws),
                            as_stream(stream)));
  MKV_CUDA(launch_quant_prepare(*cfg, *qparams, as_stream(stream)));
  return MKV_OK;
}

mkv_status mkv_quant_prepare(const mkv_config* cfg, mkv_quant_params* qparams, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_KVQUANT, MKV_ERR_INVALID_ARG, "quant_prepare is for KVQUANT");
  MKV_TRY(check_qparams(cfg, qparams, true));
  MKV_CUDA(launch_quant_prepare(*cfg, *qparams, as_stream(stream)));
  return MKV_OK;
}

mkv_status mkv_quantize_kv(const mkv_config* cfg, const mkv_quant_params* qparams, const void* k_pre,
                           const void* v, int64_t n_tokens, mkv_cache* cache, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_KVQUANT, MKV_ERR_INVALID_ARG, "quantize is for KVQUANT");
  MKV_TRY(check_cache(cfg, cache));
  MKV_TRY(check_qparams(cfg, qparams, false));
  MKV_REQUIRE(k_pre && v && n_tokens >= 1 && n_tokens <= cache->T_cap, MKV_ERR_INVALID_ARG,
              "k_pre/v NULL or n_tokens outside [1, T_cap]");
  // the launch counts its finished CTAs per batch entry in the top 8 bits of T_len[b]
  MKV_REQUIRE(cache->T_cap < (1 << 24) && cfg->Hkv <= 256, MKV_ERR_UNSUPPORTED,
              "quantize needs T_cap < 2^24 and Hkv <= 256 (T_cap %lld, Hkv %d)", (long long)cache->T_cap, cfg->Hkv);
  MKV_CUDA(launch_quantize(*cfg, *qparams, k_pre, v, n_tokens, *cache, as_stream(stream)));
  return MKV_OK;
}

mkv_status mkv_h2o_prefill(const mkv_config* cfg, const void* q_prompt, const void* full_k, const void* full_v,
                           int64_t T, mkv_cache* cache, void* ws, size_t ws_bytes, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_H2O, MKV_ERR_INVALID_ARG, "h2o_prefill is for H2O");
  MKV_TRY(check_cache(cfg, cache));
  MKV_REQUIRE(q_prompt && full_k && full_v && T >= 1, MKV_ERR_INVALID_ARG, "prompt tensors NULL or T < 1");
  MKV_REQUIRE((((uintptr_t)q_prompt | (uintptr_t)full_k) & 15) == 0, MKV_ERR_INVALID_ARG,
              "q_prompt and full_k must be 16-byte aligned (tensor-core scoring reads them by TMA)");
  const PrefillWs need = prefill_ws(*cfg, T, nullptr);
  MKV_REQUIRE(ws != nullptr && ws_bytes >= need.bytes, MKV_ERR_WORKSPACE,
              "workspace %zu bytes < %zu needed", ws_bytes, need.bytes);
  const PrefillWs w = prefill_ws(*cfg, T, ws);
  cudaStream_t st = as_stream(stream);
  MKV_CUDA(launch_prefill_scores(*cfg, q_prompt, T, T, full_k, w, st));
  MKV_CUDA(launch_h2o_keep(*cfg, full_k, full_v, T, *cache, w, st));
  return MKV_OK;
}

mkv_status mkv_h2o_update(const mkv_config* cfg, mkv_cache* cache, void* ws, size_t ws_bytes, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_H2O, MKV_ERR_INVALID_ARG, "h2o_update is for H2O");
  MKV_TRY(check_cache(cfg, cache));
  const DecodeWs need = decode_ws(*cfg, cache->T_cap, nullptr);
  MKV_REQUIRE(ws != nullptr && ws_bytes >= need.bytes, MKV_ERR_WORKSPACE,
              "workspace %zu bytes < %zu needed", ws_bytes, need.bytes);
  MKV_CUDA(launch_h2o_update(*cfg, *cache, decode_ws(*cfg, cache->T_cap, ws), as_stream(stream)));
  return MKV_OK;
}

mkv_status mkv_snap_compress(const mkv_config* cfg, const void* q_window, const void* full_k,
                             const void* full_v, int64_t T, mkv_cache* cache, int32_t* kept_pos, void* ws,
                             size_t ws_bytes, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_ROCKET, MKV_ERR_INVALID_ARG, "snap_compress is for ROCKET");
  MKV_TRY(check_cache(cfg, cache));
  MKV_REQUIRE(q_window && full_k && full_v && T >= cfg->snap_window, MKV_ERR_INVALID_ARG,
              "prompt tensors NULL or T < snap_window");
  MKV_REQUIRE((((uintptr_t)q_window | (uintptr_t)full_k) & 15) == 0, MKV_ERR_INVALID_ARG,
              "q_window and full_k must be 16-byte aligned (tensor-core scoring reads them by TMA)");
  MKV_REQUIRE(cache->T_cap >= std::min<int64_t>(T, cfg->snap_keep), MKV_ERR_INVALID_ARG,
              "cache T_cap below the kept tokens");
  const PrefillWs need = prefill_ws(*cfg, T, nullptr);
  MKV_REQUIRE(ws != nullptr && ws_bytes >= need.bytes, MKV_ERR_WORKSPACE,
              "workspace %zu bytes < %zu needed", ws_bytes, need.bytes);
  const PrefillWs w = prefill_ws(*cfg, T, ws);
  cudaStream_t st = as_stream(stream);
  if (T > cfg->snap_keep) MKV_CUDA(launch_prefill_scores(*cfg, q_window, cfg->snap_window, T, full_k, w, st));
  MKV_CUDA(launch_snap_keep(*cfg, full_k, full_v, T, *cache, kept_pos, w, st));
  return MKV_OK;
}

mkv_status mkv_rocket_select(const mkv_config* cfg, const void* q, const mkv_cache* cache, int32_t* page_idx_out,
                             void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_ROCKET, MKV_ERR_INVALID_ARG, "rocket_select is for ROCKET");
  MKV_TRY(check_cache(cfg, cache));
  MKV_REQUIRE(q && page_idx_out, MKV_ERR_INVALID_ARG, "q/page_idx_out NULL");
  MKV_CUDA(launch_rocket_select(*cfg, q, *cache, page_idx_out, as_stream(stream)));
  return MKV_OK;
}

mkv_status mkv_rocket_decode(const mkv_config* cfg, const void* q, const mkv_cache* cache, int32_t* page_idx_out,
                             void* out, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_ROCKET, MKV_ERR_INVALID_ARG, "rocket_decode is for ROCKET");
  MKV_TRY(check_cache(cfg, cache));
  MKV_REQUIRE(q && out, MKV_ERR_INVALID_ARG, "q/out NULL");
  MKV_REQUIRE(rocket_fused_smem(*cfg, cache->T_cap) <= 227 * 1024, MKV_ERR_UNSUPPORTED,
              "T_cap = %lld is too long for the fused step; use mkv_rocket_select + mkv_decode_attention",
              (long long)cache->T_cap);
  MKV_CUDA(launch_rocket_fused(*cfg, q, *cache, page_idx_out, out, nullptr, nullptr, as_stream(stream)));
  return MKV_OK;
}

mkv_status mkv_rocket_step(const mkv_config* cfg, const void* q, const void* k_new, const void* v_new,
                           mkv_cache* cache, int32_t* page_idx_out, void* out, void* stream) {
  MKV_TRY(check_config(cfg));
  MKV_REQUIRE(cfg->method == MKV_ROCKET, MKV_ERR_INVALID_ARG, "rocket_step is for ROCKET");
  MKV_TRY(check_cache(cfg, cache));
  MKV_REQUIRE(q && out && k_new && v_new, MKV_ERR_INVALID_ARG, "q/out/k_new/v_new NULL");
  MKV_REQUIRE(((uintptr_t)k_new | (uintptr_t)v_new) % 16 == 0, MKV_ERR_INVALID_ARG,
              "k_new/v_new must be 16-byte aligned (the step reads them in 16-byte pieces)");
  MKV_REQUIRE(rocket_fused_smem(*cfg, cache->T_cap) <= 227 * 1024, MKV_ERR_UNSUPPORTED,
              "T_cap = %lld is too long for the fused step; use the separate calls", (long long)cache->T_cap);
  // the launch counts its finished CTAs per batch entry in the top 8 bits of T_len[b]
  MKV_REQUIRE(cache->T_cap < (1 << 24) && (int64_t)kRocketCluster * cfg->Hkv <= 256, MKV_ERR_UNSUPPORTED,
              "rocket_step needs T_cap < 2^24 and 8 * Hkv <= 256 (T_cap %lld, Hkv %d)", (long long)cache->T_cap,
              cfg->Hkv);
  MKV_CUDA(launch_rocket_fused(*cfg, q, *cache, page_idx_out, out, k_new, v_new, as_stream(stream)));
  return MKV_OK;
}

}  // extern "C"
