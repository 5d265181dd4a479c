/*
 * mkv.h -- C ABI of libmkv: decode-step attention over a compressed KV cache
 * on one GB300 GPU (sm_103a).
 *
 * The paper (MetaKV) chooses, per prompt, one of ten KV-cache configurations
 * (Table 1): uncompressed FP16, KVQuant b-bit (b = 2, 3, 4), H2O p%
 * (p = 20, 40, 60) and RocketKV rx (r = 8, 16, 32).  Section 2.1 describes the
 * three compression methods; Section 2.3 states the problem this library
 * serves: run configuration c on a prompt and report its latency and peak
 * KV memory.  This library is the hot path of that problem -- one decode step
 * of attention over the compressed cache, plus the prefill-side compression
 * that builds each cache.
 *
 * Conventions (every entry point):
 *  - All tensor arguments are DEVICE pointers to caller-allocated memory
 *    unless a parameter says "host".  The library never allocates or frees
 *    device memory; scratch space is the caller's `ws` buffer, sized by
 *    mkv_workspace_size().  The first 16 KiB of a workspace hold counters
 *    that must be zero before the first call that uses it (allocate it
 *    zero-filled); every call leaves them zero again.  Calls that share a
 *    workspace must not overlap on the GPU.  Nothing is retained between
 *    calls except the library's status word (see mkv_get_status).
 *  - B * Hkv is at most 4096.
 *  - fp16 means IEEE binary16 stored as uint16 bits; fp32 is IEEE binary32.
 *  - Calls are asynchronous on `stream` (a cudaStream_t passed as void*;
 *    NULL is the legacy default stream).  Arguments are validated on the host
 *    before anything is launched: a bad argument returns an error code and
 *    launches nothing.  A launch failure returns MKV_ERR_CUDA.  A condition
 *    only the device can see (outlier storage full, a bounded wait that ran
 *    out) sets a bit of the status
 *    word that mkv_get_status() reports.  No call aborts or throws.
 *  - mkv_last_error() returns a thread-local text for the last failure.
 *  - Shapes: B batch entries, Hq query heads, Hkv key/value heads,
 *    G = Hq/Hkv query heads per group, D head dimension.  Supported:
 *    D in {64, 128}; G in {1, 2, 4, 8}; bits in {2, 3, 4}; page_size 16.
 *    Anything else returns MKV_ERR_UNSUPPORTED.
 *  - Layouts are row-major with the last index fastest:
 *      q            [B][Hq][D] fp16 (already rotated by the query position)
 *      out          [B][Hq][D] fp16
 *      K, V cache   [B][Hkv][T_cap][D] fp16 (FP16, H2O, ROCKET)
 *  - One call handles one layer; the caller owns the layer loop (and may
 *    capture it in a CUDA graph: every length lives on the device).
 */
#ifndef MKV_H
#define MKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define MKV_ABI_VERSION 1u

typedef enum {
  MKV_OK = 0,
  MKV_ERR_INVALID_ARG = 1,  /* null pointer, bad size, inconsistent config  */
  MKV_ERR_UNSUPPORTED = 2,  /* valid but not built (e.g. D = 96)             */
  MKV_ERR_CUDA = 3,         /* a CUDA call or launch failed                  */
  MKV_ERR_CAPACITY = 4,     /* a device-side store ran out of room           */
  MKV_ERR_WORKSPACE = 5,    /* ws is NULL or ws_bytes below the required size */
  MKV_ERR_TIMEOUT = 6       /* a bounded device-side wait ran out            */
} mkv_status;

typedef enum { MKV_FP16 = 0, MKV_KVQUANT = 1, MKV_H2O = 2, MKV_ROCKET = 3 } mkv_method;
typedef enum { MKV_QUANT_UNIFORM = 0, MKV_QUANT_NUQ = 1 } mkv_quant_mode;

/* Status-word bits (mkv_get_status). */
#define MKV_FLAG_K_OUTLIER_OVERFLOW 0x1u  /* a key-outlier CSR region is full */
#define MKV_FLAG_CACHE_FULL 0x2u          /* an append found no free slot; dropped */
#define MKV_FLAG_WAIT_TIMEOUT 0x4u        /* a prefill-scoring CTA gave up waiting on the
                                             tensor core; that call's scores are invalid */

/* One configuration (a row of Table 1, with its parameters).  Host POD. */
typedef struct {
  uint32_t abi_version;   /* must equal MKV_ABI_VERSION                      */
  int32_t method;         /* mkv_method                                      */
  int32_t B, Hq, Hkv, D;
  float softmax_scale;    /* 0 -> 1/sqrt(D)                                  */
  float rope_theta;       /* rotary base (KVQUANT rotates keys after dequant) */
  /* KVQUANT (Section 2.1, KVQuant paragraph) */
  int32_t bits;           /* 2, 3 or 4                                       */
  int32_t quant_mode;     /* mkv_quant_mode                                  */
  float outlier_frac;     /* fraction kept as fp16 outliers, e.g. 0.01       */
  /* H2O (Section 2.1, H2O paragraph): budget = heavy + recent tokens */
  int32_t h2o_heavy, h2o_recent;
  /* ROCKET (Section 2.1, RocketKV paragraph) */
  int32_t snap_window;    /* W: observation window at the end of the prompt  */
  int32_t snap_pool;      /* max-pool kernel (odd)                            */
  int32_t snap_keep;      /* tokens kept per kv-head after prefill           */
  int32_t page_size;      /* tokens per page (16)                            */
  int32_t topk_pages;     /* k_p pages attended per step (+ the tail page)   */
  int32_t topq_dims;      /* r_d dims used for approximate page scores       */
} mkv_config;

/* The cache of one layer.  All pointers are device memory owned by the
 * caller; fields a method does not use may be NULL.
 *
 *  T_cap   slots per (batch entry, kv-head).
 *  T_len   int32 [B]: tokens written so far per batch entry.  FP16, KVQUANT
 *          and ROCKET store token t in slot t; H2O uses it as the position of
 *          the next token.  Appends advance it on the device.
 *
 *  FP16 / ROCKET: k, v fp16 [B][Hkv][T_cap][D], rows 0..T_len-1 valid.
 *  H2O:   k, v fp16 [B][Hkv][T_cap][D] with T_cap >= heavy + recent + 1;
 *         only slots 0..heavy+recent are ever used (the prefill fills slots
 *         from 0 and each step writes the lowest free slot or the one its
 *         eviction freed), and the decode and the update read only those;
 *         pos int32 [B][Hkv][T_cap] (position held by each slot, -1 = empty);
 *         acc fp32 [B][Hkv][T_cap] accumulated attention score;
 *         slot int32 [B][Hkv] the slot the next append writes.
 *  ROCKET: kmin, kmax fp16 [B][Hkv][D][T_cap/page_size] (16-byte aligned) per-page per-dim key
 *         min/max (dim-major), valid for every completed page.
 *  KVQUANT (keys stored before rotation; Section 2.1, KVQuant paragraph):
 *         k_codes, v_codes uint8 [B][Hkv][T_cap][D*bits/8]: per token, the
 *           D/2 "pair codes" of channels (i, i + D/2) as a little-endian
 *           bitstream; pair i occupies bits [2*bits*i, 2*bits*(i+1)), channel
 *           i in the low `bits` bits.
 *         v_params fp32 [B][Hkv][T_cap][2]: per token (lo, scale); a value
 *           dequantizes to lo + scale * v_tbl[channel][code].
 *         v_out uint32 [B][Hkv][T_cap][n_v], n_v = ceil(outlier_frac * D):
 *           value outliers, (channel << 16) | fp16 bits.
 *         k_out_off int32 [B][Hkv][T_cap + 1]: CSR offsets of key outliers
 *           per token (k_out_off[..][0] = 0).
 *         k_out uint32 [B][Hkv][k_out_cap]: key outliers of token t at
 *           [k_out_off[t], k_out_off[t+1]), in channel order, each
 *           ((t mod 64) << 24) | (channel << 16) | fp16 bits.
 */
typedef struct {
  int64_t T_cap;
  int32_t* T_len;
  void* k;
  void* v;
  int32_t* pos;
  float* acc;
  int32_t* slot;
  void* kmin;
  void* kmax;
  uint8_t* k_codes;
  uint8_t* v_codes;
  float* v_params;
  uint32_t* v_out;
  int32_t* k_out_off;
  uint32_t* k_out;
  int64_t k_out_cap;
} mkv_cache;

/* KVQuant calibration of one layer (device memory, caller-owned).  Per
 * kv-head h and channel c (index [h][c], or [h][c][j] for tables):
 *   t_lo, t_hi fp32 [Hkv][D]   key inlier range; x < t_lo or x > t_hi is an
 *                              outlier
 *   k_lo, k_scale fp32 [Hkv][D] uniform-mode key offset and step
 *   k_cb fp16 [Hkv][D][2^bits]  NUQ key centroids (ascending)
 *   v_cb fp16 [Hkv][D][2^bits]  NUQ value centroids on u in [0, 1]
 *   k_dq fp32 [Hkv][D][2^bits]  dequantized key per code (filled by
 *                               mkv_quant_prepare)
 *   v_tbl fp16 [Hkv][D][2^bits] value table per code: the NUQ centroid, or j
 *                               in uniform mode (filled by mkv_quant_prepare)
 *   rope fp32 [rope_len][D/2][2] (cos, sin) table from mkv_rope_table, with
 *                               rope_len >= max(the cache's T_cap, 64); decode rotates
 *                               each dequantized key by its position
 */
typedef struct {
  float* t_lo;
  float* t_hi;
  float* k_lo;
  float* k_scale;
  uint16_t* k_cb;
  uint16_t* v_cb;
  float* k_dq;
  uint16_t* v_tbl;
  float* rope;
  int64_t rope_len;
} mkv_quant_params;

/* ---------------------------------------------------------------- sizing */

/* Bytes of workspace the calls of this config need for caches of T_cap
 * slots (the maximum over all calls).  Host only. */
mkv_status mkv_workspace_size(const mkv_config* cfg, int64_t T_cap, size_t* bytes);

/* KV-cache bytes of one layer: `resident` for a cache holding T tokens after
 * compression (what decode reads and keeps), `peak` including the prefill
 * transient (the uncompressed prompt that compression reads).  This is the
 * peak-memory figure the paper's selector predicts (Section 2.3).  Host only. */
mkv_status mkv_cache_bytes(const mkv_config* cfg, int64_t T, size_t* resident, size_t* peak);

/* ------------------------------------------------------------ selector */

/* One candidate configuration for mkv_select_config: its method, its level
 * of compression within the method (larger = less compressed: KVQuant bits,
 * H2O budget percent, RocketKV minus its compression ratio), and its
 * predicted end-to-end latency, peak memory and probability of a correct
 * answer.  Latency and memory use the units of the budgets they are compared
 * with. */
typedef struct {
  int32_t method;   /* mkv_method */
  int32_t level;
  double latency;
  double memory;
  double accuracy;
} mkv_candidate;

/* The configuration choice of MetaKV (Section 2.3), fed by measured or
 * predicted costs: keep the candidates with latency <= L_max and memory <=
 * M_max; if FP16 is among them choose it (the first FP16 candidate); else
 * keep the least compressed candidate of each method (largest level, ties:
 * lower index) and choose it if it is alone, otherwise the one with the
 * highest accuracy (ties: lower index).  If no candidate is within both
 * budgets, choose the smallest violation v_c = latency/L_max +
 * memory/M_max (ties: higher accuracy, then lower index).  *chosen gets the
 * index into `cands`, *within_budget 1 or 0 for the fallback.  Host only;
 * MKV_ERR_INVALID_ARG for n < 1, a budget <= 0, a non-finite or negative
 * cost, or a method out of range. */
mkv_status mkv_select_config(const mkv_candidate* cands, int32_t n, double L_max, double M_max,
                             int32_t* chosen, int32_t* within_budget);

/* ------------------------------------------------------------ utilities */

/* table fp32 [T_max][D/2][2]: (cos, sin) of p * theta^(-2i/D), computed in
 * fp64 on the device and rounded; the rotary embedding of the KVQuant path
 * (keys are rotated after dequantization). */
mkv_status mkv_rope_table(int32_t D, float theta, int64_t T_max, float* table, void* stream);

/* Synchronizes `stream`, then returns the status word in *flags (host) and
 * clears it.  MKV_ERR_TIMEOUT if MKV_FLAG_WAIT_TIMEOUT was set, else
 * MKV_ERR_CAPACITY if any bit was set. */
mkv_status mkv_get_status(void* stream, uint32_t* flags);

/* Diagnostic of the device wait-timeout path (no counterpart in the paper):
 * launches one CTA whose bounded mbarrier wait, the routine the prefill
 * scoring's waits use, can never complete (nothing arrives on its barrier);
 * after about `ms` milliseconds (1..1000, else MKV_ERR_INVALID_ARG) it gives
 * up and sets MKV_FLAG_WAIT_TIMEOUT, so the next mkv_get_status returns
 * MKV_ERR_TIMEOUT with that bit, and the context stays usable.  Asynchronous
 * on `stream`; it reads and writes no caller memory. */
mkv_status mkv_wait_timeout_selftest(int32_t ms, void* stream);

/* Thread-local description of the last error (never NULL). */
const char* mkv_last_error(void);

/* ---------------------------------------------------------------- FP16 */

/* Append one token per (batch entry, kv-head) to an FP16, H2O or ROCKET cache:
 * the decode step's new key and value join the cache before attention (the
 * per-step cache growth of every configuration of Table 1, Section 2.1; the
 * H2O slot reuse follows the H2O paragraph, the page bounds the RocketKV
 * paragraph's second stage).  k_new, v_new fp16 [B][Hkv][D] (keys already rotated).  FP16/ROCKET write
 * slot T_len[b]; H2O writes slot[b][h] and sets pos = T_len[b], acc = 0.
 * ROCKET also fills kmin/kmax of a page the token completes.  T_len[b] += 1.
 * A batch entry where any kv-head has no room (FP16/ROCKET: T_len = T_cap;
 * H2O: a slot outside [0, T_cap)) gets no row in any kv-head, keeps T_len and
 * sets MKV_FLAG_CACHE_FULL.
 * Errors: MKV_ERR_INVALID_ARG for a null field the method needs. */
mkv_status mkv_append_kv(const mkv_config* cfg, const void* k_new, const void* v_new,
                         mkv_cache* cache, void* stream);

/* Decode attention (every method).  Each query head h of q attends, with a
 * softmax over the attended set, to the cached tokens of kv-head h / G
 * (the decode step of every configuration of Table 1; the attended set of
 * each method is Section 2.1's):
 *   FP16, KVQUANT: slots 0..T_len[b]-1 (KVQUANT dequantizes keys, restores
 *                  outliers, rotates keys by their position, dequantizes
 *                  values -- all fused; Section 2.1 KVQuant paragraph);
 *   H2O:           every slot among 0..heavy+recent with pos >= 0;
 *   ROCKET:        the pages listed in page_idx [B][Hkv][topk_pages] (int32,
 *                  -1 = unused) plus the tail page that holds the newest
 *                  token (Section 2.1, RocketKV paragraph, second stage).
 * out fp16 [B][Hq][D].  For H2O the call also leaves, in ws, the per-slot
 * logits and per-head softmax statistics that mkv_h2o_update reads.
 * qparams: KVQUANT only (else NULL).  ws/ws_bytes: workspace.
 * KVQUANT also requires 16-byte aligned k_codes and v_codes (MKV_ERR_INVALID_ARG
 * otherwise), and k_out_cap <= INT32_MAX and T_cap < INT32_MAX
 * (MKV_ERR_UNSUPPORTED otherwise). */
mkv_status mkv_decode_attention(const mkv_config* cfg, const void* q, const mkv_cache* cache,
                                const mkv_quant_params* qparams, const int32_t* page_idx,
                                void* out, void* ws, size_t ws_bytes, void* stream);

/* FP16 decode attention that allocates nothing and takes no workspace.
 * No counterpart in the paper: it exists for callers that cannot call
 * cudaMalloc or hand this library a scratch buffer -- for instance code that
 * runs inside a host framework owning every device allocation, or an existing
 * C interface with no place to pass a workspace.  It computes exactly what
 * mkv_decode_attention computes for an FP16 cache (same kernels, same
 * result); only the split partials live elsewhere: in one array of 8 MiB
 * compiled into the library, which every GPU that loads the library keeps
 * until the process exits.
 *  - cfg->method must be MKV_FP16 (else MKV_ERR_UNSUPPORTED).
 *  - The call needs exactly the bytes mkv_workspace_size reports for this
 *    config and T_cap (16 KiB of merge tickets, then the partials m, l and o
 *    of B*Hq*n_split, B*Hq*n_split and B*Hq*n_split*D floats, each part
 *    rounded up to 256 bytes); that must be at most 8 MiB, else
 *    MKV_ERR_WORKSPACE and nothing is launched.
 *  - The first call on each device looks up the array's device address
 *    (cudaGetSymbolAddress) and caches it for the process; make that first
 *    call before any stream capture.  A cudaDeviceReset (or anything else
 *    that destroys and recreates the device's primary context) invalidates
 *    the cached address, and the library does not notice: do not call this
 *    entry point on a device after resetting it.
 *  - All calls share the one array per device: calls whose kernels overlap on
 *    the GPU (different streams, or a second call before the first finished
 *    on another stream) race and corrupt each other's result.  Calls in order
 *    on one stream are safe; every partial is rewritten before it is read, so
 *    nothing has to be cleared between calls.
 * q, out fp16 [B][Hq][D]; cache as for mkv_decode_attention. */
mkv_status mkv_decode_attention_noalloc(const mkv_config* cfg, const void* q, const mkv_cache* cache,
                                        void* out, void* stream);

/* ------------------------------------------------------------- KVQuant */

/* Learn one layer's calibration from the first N_cal tokens of the prompt:
 * k_cal (keys before rotation), v_cal fp16 [Hkv][N_cal][D] with row stride
 * `row_stride` tokens between kv-heads (so a [B][Hkv][T][D] prompt's batch
 * entry 0 can be passed with row_stride = T).  Fills t_lo, t_hi, k_lo,
 * k_scale and, in NUQ mode, k_cb and v_cb (1-D Lloyd k-means, 25 iterations,
 * quantile start), then k_dq and v_tbl.  Needs ws. */
mkv_status mkv_kvquant_calibrate(const mkv_config* cfg, const void* k_cal, const void* v_cal,
                                 int64_t N_cal, int64_t row_stride, mkv_quant_params* qparams,
                                 void* ws, size_t ws_bytes, void* stream);

/* Derive k_dq and v_tbl from t_lo/t_hi/k_lo/k_scale/k_cb/v_cb (for
 * calibrations computed elsewhere). */
mkv_status mkv_quant_prepare(const mkv_config* cfg, mkv_quant_params* qparams, void* stream);

/* KVQuant quantization (Section 2.1, KVQuant paragraph: keys per channel,
 * values per token, outliers kept in fp16; Table 1's 2/3/4-bit settings).
 * Quantize n_tokens tokens per (batch entry, kv-head) into the KVQUANT cache
 * at slots T_len[b]..T_len[b]+n_tokens-1 (n_tokens = T at prefill, 1 per
 * decode step): key outliers by the per-channel range, value outliers as the
 * n_v largest |x| per token, codes by correctly rounded fp32 arithmetic.
 * k_pre (keys before rotation), v fp16 [B][Hkv][n_tokens][D].  T_len += n,
 * stored by the launch's last CTA of each batch entry: while it runs, the
 * top 8 bits of T_len[b] count its finished CTAs, so nothing else may read
 * or write T_len of this cache during the call (MKV_ERR_UNSUPPORTED when
 * T_cap >= 2^24 or Hkv > 256).  A full cache sets MKV_FLAG_CACHE_FULL and
 * keeps T_len.  A full key-outlier region sets MKV_FLAG_K_OUTLIER_OVERFLOW
 * (entries past k_out_cap are dropped). */
mkv_status mkv_quantize_kv(const mkv_config* cfg, const mkv_quant_params* qparams,
                           const void* k_pre, const void* v, int64_t n_tokens,
                           mkv_cache* cache, void* stream);

/* ----------------------------------------------------------------- H2O */

/* Build an H2O cache from a prompt (Section 2.1, H2O paragraph).  q_prompt
 * fp16 [B][Hq][T][D], full_k, full_v fp16 [B][Hkv][T][D] (post-rotation).
 * Scores acc0[j] = sum over the group's heads and prompt rows i >= j of the
 * causal softmax probability of key j; keeps the h2o_recent newest positions
 * and the h2o_heavy best others (acc desc, position asc), compacted in
 * ascending position into slots 0..; sets pos, acc, slot and T_len[b] = T.
 * q_prompt and full_k must be 16-byte aligned (MKV_ERR_INVALID_ARG).
 * Needs ws (mkv_workspace_size with T_cap >= T).  A scoring CTA whose bounded
 * wait on the tensor core ran out sets MKV_FLAG_WAIT_TIMEOUT. */
mkv_status mkv_h2o_prefill(const mkv_config* cfg, const void* q_prompt, const void* full_k,
                           const void* full_v, int64_t T, mkv_cache* cache, void* ws,
                           size_t ws_bytes, void* stream);

/* H2O's per-step score update and eviction (Section 2.1, H2O paragraph: tokens
 * are scored by the attention they receive, and the lowest-scored are evicted
 * to keep the budget).  The softmax probabilities it adds are the logits and
 * per-head (m, l) that mkv_decode_attention left in `ws` (so they are not
 * arguments).  After mkv_decode_attention on an H2O cache: add each slot's softmax
 * probability summed over the group's heads to acc, then, if the cache holds
 * more than heavy + recent tokens, evict among all but the `recent` newest
 * positions the lowest-acc token (exact tie: the higher position) and make
 * its slot the next append slot. */
mkv_status mkv_h2o_update(const mkv_config* cfg, mkv_cache* cache, void* ws, size_t ws_bytes,
                          void* stream);

/* -------------------------------------------------------------- ROCKET */

/* SnapKV prefill compression (RocketKV first stage).  q_window fp16
 * [B][Hq][W][D] are the last W prompt queries; full_k, full_v fp16
 * [B][Hkv][T][D].  Scores prefix keys by the window's causal softmax mass
 * (summed over the group), max-pools them (kernel snap_pool, stride 1), keeps
 * the snap_keep - W best (score desc, position asc) plus the window, gathers
 * them in ascending position into slots 0..keep-1 of `cache`, fills kmin/kmax
 * of every full page and sets T_len[b] = keep.  keep >= T copies everything.
 * kept_pos (optional, int32 [B][Hkv][keep]) receives the kept positions.
 * q_window and full_k must be 16-byte aligned (MKV_ERR_INVALID_ARG); a
 * scoring wait that ran out sets MKV_FLAG_WAIT_TIMEOUT as for H2O. */
mkv_status mkv_snap_compress(const mkv_config* cfg, const void* q_window, const void* full_k,
                             const void* full_v, int64_t T, mkv_cache* cache, int32_t* kept_pos,
                             void* ws, size_t ws_bytes, void* stream);

/* RocketKV second stage, page choice (Section 2.1, RocketKV paragraph: at each
 * decode step attention reads a subset of the earlier tokens chosen by an
 * approximate score).  For the current query: dims = the
 * topq_dims largest sum_h |q_h,i| (ties: lower dim); page score = sum_h
 * sum_{i in dims} max(q_h,i * kmin_i, q_h,i * kmax_i) over the full pages
 * before the newest token's page; page_idx_out int32 [B][Hkv][topk_pages]
 * gets the best pages (score desc, page asc) in ascending order, -1 padded. */
mkv_status mkv_rocket_select(const mkv_config* cfg, const void* q, const mkv_cache* cache,
                             int32_t* page_idx_out, void* stream);

/* RocketKV decode step in one launch: the page choice of mkv_rocket_select
 * and the sparse exact attention of mkv_decode_attention over the chosen
 * pages plus the newest token's page (Section 2.1, RocketKV paragraph, stage
 * 2).  One cluster of 8 CTAs per (batch, kv-head) exchanges page scores and
 * attention partials through distributed shared memory, so no workspace is
 * needed.  q fp16 [B][Hq][D]; out fp16 [B][Hq][D]; page_idx_out (optional,
 * NULL to skip) int32 [B][Hkv][topk_pages] as mkv_rocket_select writes it.
 * The page scores are the same sums in another fp32 order, so a near-tie
 * may pick another page than mkv_rocket_select.  MKV_ERR_UNSUPPORTED when
 * T_cap is too long for the step's shared memory (about 32K slots at D=128);
 * use the two calls then. */
mkv_status mkv_rocket_decode(const mkv_config* cfg, const void* q, const mkv_cache* cache,
                             int32_t* page_idx_out, void* out, void* stream);

/* A whole FP16 or H2O decode step's attention in one launch: mkv_append_kv of
 * the step's token followed by mkv_decode_attention, with the same cache
 * contents and output (Section 2.1; H2O's score update stays a separate
 * mkv_h2o_update).  k_new, v_new fp16 [B][Hkv][D], 16-byte aligned
 * (MKV_ERR_INVALID_ARG otherwise); q, out, ws as mkv_decode_attention.
 * The split of the decode whose range holds the token's slot (FP16: T_len,
 * H2O: slot[b][kv-head]) stages the row from k_new / v_new and writes it
 * (H2O: with position T_len and a zero score).  While the launch runs, the
 * top 8 bits of T_len[b] count its finished CTAs (the last one stores the new
 * length), so nothing else may read or write T_len of this cache during the
 * call.  A batch entry with no room in some kv-head is not appended in any
 * (MKV_FLAG_CACHE_FULL, read by mkv_get_status) and attends to its existing tokens.  MKV_ERR_UNSUPPORTED
 * when T_cap >= 2^24 or Hkv x (the decode's splits) > 255: use the two calls
 * then. */
mkv_status mkv_decode_step(const mkv_config* cfg, const void* q, const void* k_new, const void* v_new,
                           mkv_cache* cache, void* out, void* ws, size_t ws_bytes, void* stream);

/* A whole KVQuant decode step in one launch: mkv_quantize_kv of the step's
 * token (n_tokens = 1) followed by mkv_decode_attention, with the same cache
 * contents (codes, key-outlier CSR, value outliers and ranges, T_len) and the
 * same output bits (Section 2.1, KVQuant paragraph: the token's key is
 * quantized per channel before the rotary embedding, its value per token,
 * with fp16 outliers).  k_new fp16 [B][Hkv][D] is the token's pre-rotation
 * key, v_new fp16 [B][Hkv][D] its value; q, out, qparams, ws as
 * mkv_decode_attention.  The decode CTA whose range holds a unit's new token
 * quantizes it before it stages that chunk.  While the launch runs, the top 8
 * bits of T_len[b] count the CTAs that read it (the last one stores the new
 * length), so nothing else may read or write T_len of this cache during the
 * call.  A batch entry whose cache is full is not appended
 * (MKV_FLAG_CACHE_FULL) and attends to its existing tokens; key-outlier
 * entries beyond k_out_cap raise MKV_FLAG_K_OUTLIER_OVERFLOW as in
 * mkv_quantize_kv (both read by mkv_get_status).  MKV_ERR_UNSUPPORTED when
 * T_cap >= 2^24: use the two calls then. */
mkv_status mkv_kvquant_step(const mkv_config* cfg, const mkv_quant_params* qparams, const void* q,
                            const void* k_new, const void* v_new, mkv_cache* cache, void* out, void* ws,
                            size_t ws_bytes, void* stream);

/* A whole RocketKV decode step in one launch: mkv_append_kv of the step's
 * token followed by mkv_rocket_decode, with the same cache contents, page
 * choice and output.  k_new, v_new fp16 [B][Hkv][D] (post-rotation keys),
 * 16-byte aligned (MKV_ERR_INVALID_ARG otherwise).
 * While the launch runs, the top 8 bits of T_len[b] count its finished CTAs
 * (the last one stores the new length), so nothing else may read or write
 * T_len of this cache during the call.  A batch entry whose cache is full is
 * not appended (MKV_FLAG_CACHE_FULL, read by mkv_get_status) and attends to
 * its existing tokens.  MKV_ERR_UNSUPPORTED as mkv_rocket_decode, and when
 * T_cap >= 2^24 or 8 * Hkv > 256. */
mkv_status mkv_rocket_step(const mkv_config* cfg, const void* q, const void* k_new, const void* v_new,
                           mkv_cache* cache, int32_t* page_idx_out, void* out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* MKV_H */
