// Host-side interfaces between the C ABI layer (mkv_api.cu) and the kernel
// translation units.  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <utility>

#include "mkv.h"

namespace mkv {

constexpr int kChunk = 64;       // tokens per decode pipeline chunk
constexpr int kPage = 16;        // ROCKET page size (the only one built)

void set_error(const char* fmt, ...);

inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Every workspace starts with this many bytes of split tickets (one int per
// (batch, kv-head)); they must be zero before first use and every call leaves
// them zero.  Nothing else is ever written there, whatever the config.
constexpr size_t kCounterBytes = 16384;
constexpr int kMaxUnits = (int)(kCounterBytes / 4);
inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Work split of a decode call: `n_split` CTAs per (batch, kv-head), each over
// `chunks_per_split` chunks of kChunk virtual tokens (KVQuant: a balanced range per CTA).
struct Split {
  int n_split;           // partial slots per (batch, kv-head)
  int chunks_per_split;
  int64_t v_tokens;      // virtual tokens per (batch, kv-head)
  // KVQuant: one CTA per SM over the concatenated chunks of all (batch, kv-head) units; CTA i
  // takes chunks [i * c_tot / n_cta, (i + 1) * c_tot / n_cta)
  int n_cta;
  int64_t chunks_per_unit;
};
Split decode_split(const mkv_config& c, int64_t T_cap);
// The balanced KVQuant split: CTA of virtual chunk x, first and last CTA of unit u.
#ifdef __CUDACC__
__host__ __device__
#endif
inline int64_t cta_of_chunk(int64_t x, int64_t c_tot, int64_t n_cta) { return ((x + 1) * n_cta - 1) / c_tot; }

// Workspace carve-up (all float32).  Offsets are 256-byte aligned.
struct DecodeWs {
  float* part_m;   // [B][Hq][n_split]   running max (log2 domain)
  float* part_l;   // [B][Hq][n_split]   sum of 2^(x - m)
  float* part_o;   // [B][Hq][n_split][D] unnormalized output
  float* logits;   // H2O: [B][Hkv][T_cap][G] scaled logits (log2 domain)
  float* m_tot;    // H2O: [B][Hq]
  float* l_tot;    // H2O: [B][Hq]
  int* counters;   // [B][Hkv] split tickets; zero between calls
  size_t bytes;
};
DecodeWs decode_ws(const mkv_config& c, int64_t T_cap, void* base);

// Prefill workspace (H2O prefill, SnapKV compression): scores and selection.
struct PrefillWs {
  float2* row_st;  // [B][Hq][T + 128] per-query-row (max, sum) partials, then merged (-max, 1 / sum)
  float* score;    // [B][Hkv][T] accumulated column sums
  int32_t* keep;   // [B][Hkv][T] kept positions (ascending)
  size_t bytes;
};
PrefillWs prefill_ws(const mkv_config& c, int64_t T, void* base);

// Calibration workspace (KVQuant).
struct CalibWs {
  float* sorted;   // [Hkv][D][N] sorted calibration values (keys or u)
  float* u;        // [Hkv][N][D] normalized values
  uint8_t* vmask;  // [Hkv][N][D] value-outlier flags
  size_t bytes;
};
CalibWs calib_ws(const mkv_config& c, int64_t N, void* base);

struct MergeArgs;
MergeArgs merge_args(const mkv_config& c, const DecodeWs& ws, const Split& sp, void* out, bool h2o_stats);

// Launch of a decode-step kernel with the programmatic stream-serialization attribute (the kernel
// calls pdl_wait_and_trigger() before its first global access).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args&&... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
  return e != cudaSuccess ? e : cudaPeekAtLastError();
}

// ---- launchers (return the launch status; arguments already validated) ----
// k_new / v_new (FP16, H2O): the step's token, appended by the same launch (null: no append).
cudaError_t launch_decode_fp16_family(const mkv_config& c, const void* q, const mkv_cache& cache,
                                      const int32_t* page_idx, void* out, const DecodeWs& ws,
                                      const Split& sp, cudaStream_t st, const void* k_new = nullptr,
                                      const void* v_new = nullptr);
// k_new / v_new (KVQUANT fused step): the step's token, quantized and appended by the same launch.
cudaError_t launch_decode_kvquant(const mkv_config& c, const void* q, const mkv_cache& cache,
                                  const mkv_quant_params& qp, void* out,
                                  const DecodeWs& ws, const Split& sp, cudaStream_t st,
                                  const void* k_new = nullptr, const void* v_new = nullptr);
// Units one CTA of the fused KVQuant step may touch (its length tables).
int kvquant_step_max_units_per_cta();
cudaError_t launch_append(const mkv_config& c, const void* k_new, const void* v_new,
                          const mkv_cache& cache, cudaStream_t st);
cudaError_t launch_rope_table(int D, float theta, int64_t T_max, float* table, cudaStream_t st);

cudaError_t launch_quant_prepare(const mkv_config& c, const mkv_quant_params& qp, cudaStream_t st);
cudaError_t launch_calibrate(const mkv_config& c, const void* k_cal, const void* v_cal, int64_t N,
                             int64_t row_stride, const mkv_quant_params& qp, const CalibWs& ws,
                             cudaStream_t st);
cudaError_t launch_quantize(const mkv_config& c, const mkv_quant_params& qp, const void* k_pre,
                            const void* v, int64_t n_tokens, const mkv_cache& cache, cudaStream_t st);

cudaError_t launch_h2o_update(const mkv_config& c, const mkv_cache& cache, const DecodeWs& ws,
                              cudaStream_t st);
cudaError_t launch_prefill_scores(const mkv_config& c, const void* q, int64_t q_rows, int64_t T,
                                  const void* full_k, const PrefillWs& ws, cudaStream_t st);
cudaError_t launch_h2o_keep(const mkv_config& c, const void* full_k, const void* full_v, int64_t T,
                            const mkv_cache& cache, const PrefillWs& ws, cudaStream_t st);
cudaError_t launch_snap_keep(const mkv_config& c, const void* full_k, const void* full_v, int64_t T,
                             const mkv_cache& cache, int32_t* kept_pos, const PrefillWs& ws,
                             cudaStream_t st);
cudaError_t launch_rocket_select(const mkv_config& c, const void* q, const mkv_cache& cache,
                                 int32_t* page_idx, cudaStream_t st);
// Fused RocketKV step (page choice + sparse attention, one cluster per (batch, kv-head)).
size_t rocket_fused_smem(const mkv_config& c, int64_t T_cap);
// k_new / v_new: the step's token, appended by the same launch (null: no append).
cudaError_t launch_rocket_fused(const mkv_config& c, const void* q, const mkv_cache& cache, int32_t* page_idx,
                                void* out, const void* k_new, const void* v_new, cudaStream_t st);
constexpr int kRocketCluster = 8;   // CTAs of the fused step per (batch, kv-head)

// Host-side argument checks of an FP16 decode call (config, cache, q/out pointers).
mkv_status check_fp16_decode_args(const mkv_config* cfg, const mkv_cache* cache, const void* q, const void* out);

// Status word accessors (one per translation unit that can set a flag).
cudaError_t take_status_kvquant(uint32_t* flags, cudaStream_t st);
cudaError_t take_status_append(uint32_t* flags, cudaStream_t st);
cudaError_t take_status_rocket(uint32_t* flags, cudaStream_t st);
cudaError_t take_status_decode(uint32_t* flags, cudaStream_t st);
cudaError_t take_status_prefill(uint32_t* flags, cudaStream_t st);
cudaError_t take_status_kvq_step(uint32_t* flags, cudaStream_t st);
cudaError_t launch_wait_selftest(int ms, cudaStream_t st);

}  // namespace mkv
