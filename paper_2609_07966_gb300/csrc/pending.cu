// Launchers of the paths still under construction: they report
// cudaErrorNotSupported, which the ABI maps to MKV_ERR_CUDA.
#include "mkv_common.cuh"
#include "mkv_internal.h"

namespace mkv {
cudaError_t launch_h2o_update(const mkv_config&, const mkv_cache&, const DecodeWs&, cudaStream_t) { return cudaErrorNotSupported; }
cudaError_t launch_prefill_scores(const mkv_config&, const void*, int64_t, int64_t, const void*, const PrefillWs&,
                                  cudaStream_t) { return cudaErrorNotSupported; }
cudaError_t launch_h2o_keep(const mkv_config&, const void*, const void*, int64_t, const mkv_cache&, const PrefillWs&,
                            cudaStream_t) { return cudaErrorNotSupported; }
cudaError_t launch_snap_keep(const mkv_config&, const void*, const void*, int64_t, const mkv_cache&, int32_t*,
                             const PrefillWs&, cudaStream_t) { return cudaErrorNotSupported; }
cudaError_t launch_rocket_select(const mkv_config&, const void*, const mkv_cache&, int32_t*, cudaStream_t) {
  return cudaErrorNotSupported;
}
}  // namespace mkv
