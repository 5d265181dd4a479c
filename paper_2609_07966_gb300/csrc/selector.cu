// MetaKV's configuration choice (Section 2.3): budget filter, the FP16-first
// hierarchy with the least compressed setting of each method, the accuracy
// tie-break, and the relative-violation fallback when no candidate fits.
// Host only; fed by measured or predicted latency and memory (for example the
// bench's per-configuration step times and mkv_cache_bytes).
#include <math.h>

#include "mkv_internal.h"

extern "C" mkv_status mkv_select_config(const mkv_candidate* cands, int32_t n, double L_max, double M_max,
                                        int32_t* chosen, int32_t* within_budget) {
  using mkv::set_error;
  if (cands == nullptr || chosen == nullptr || within_budget == nullptr || n < 1) {
    set_error("cands/chosen/within_budget NULL or n < 1");
    return MKV_ERR_INVALID_ARG;
  }
  if (!(L_max > 0.0) || !(M_max > 0.0) || !isfinite(L_max) || !isfinite(M_max)) {
    set_error("budgets must be finite and > 0");
    return MKV_ERR_INVALID_ARG;
  }
  for (int32_t i = 0; i < n; ++i) {
    const mkv_candidate& c = cands[i];
    if (c.method < MKV_FP16 || c.method > MKV_ROCKET || !isfinite(c.latency) || !isfinite(c.memory) ||
        !isfinite(c.accuracy) || c.latency < 0.0 || c.memory < 0.0) {
      set_error("candidate %d: method out of range or a non-finite / negative cost", (int)i);
      return MKV_ERR_INVALID_ARG;
    }
  }
  // budget filter
  bool any = false;
  for (int32_t i = 0; i < n; ++i) any = any || (cands[i].latency <= L_max && cands[i].memory <= M_max);
  if (!any) {
    // smallest relative violation; ties: higher accuracy, then lower index
    int32_t best = 0;
    double bv = cands[0].latency / L_max + cands[0].memory / M_max;
    for (int32_t i = 1; i < n; ++i) {
      const double v = cands[i].latency / L_max + cands[i].memory / M_max;
      if (v < bv || (v == bv && cands[i].accuracy > cands[best].accuracy)) {
        best = i;
        bv = v;
      }
    }
    *chosen = best;
    *within_budget = 0;
    return MKV_OK;
  }
  *within_budget = 1;
  for (int32_t i = 0; i < n; ++i) {           // FP16 within budget: chosen at once
    if (cands[i].method == MKV_FP16 && cands[i].latency <= L_max && cands[i].memory <= M_max) {
      *chosen = i;
      return MKV_OK;
    }
  }
  // the least compressed survivor of each method (largest level; ties: lower index)
  int32_t keep[4] = {-1, -1, -1, -1};
  for (int32_t i = 0; i < n; ++i) {
    const mkv_candidate& c = cands[i];
    if (!(c.latency <= L_max && c.memory <= M_max)) continue;
    int32_t& k = keep[c.method];
    if (k < 0 || c.level > cands[k].level) k = i;
  }
  int32_t best = -1;
  for (int m = 0; m < 4; ++m) {
    if (keep[m] < 0) continue;
    // highest accuracy; ties: lower index
    if (best < 0 || cands[keep[m]].accuracy > cands[best].accuracy ||
        (cands[keep[m]].accuracy == cands[best].accuracy && keep[m] < best))
      best = keep[m];
  }
  *chosen = best;                              // a single survivor is its own best
  return MKV_OK;
}
