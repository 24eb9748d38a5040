// Host-side controllers of the admission layer (Sec. 4.1), outside the batched GPU path:
//
//  * overload pressure: per instance, the hit-rate gap G_w = max(0, h*_w - h_w) against a
//    reference learned from recent healthy windows, filtered by confirmation and slope
//    checks, together with a persistent-waiting-queue signal, contracts the operational
//    cap K_w below its base and lets it recover gradually.  Its output is the
//    cap_contraction input of misat_set_instance_state.
//  * grouped-rollout recheck delays: a held request is re-evaluated sooner the more
//    siblings of its prompt group the scheduler sees.
//
// The paper states the signals and their roles but no thresholds, window lengths or step
// sizes; every such number here is this library's choice and is a configuration field.
// Integer arithmetic only (hit rates in parts per million), so results are exact and the
// same on every host.
#include <stdint.h>

#include <algorithm>
#include <new>
#include <unordered_map>
#include <vector>

#include "../../include/misat.h"

namespace {

constexpr int64_t kPpm = 1000000;

struct InstState {
  std::vector<int64_t> ref;  // hit rates (ppm) of the last healthy windows (ring)
  int head = 0, count = 0;
  int64_t prev_h = -1;       // hit rate of the previous observed window
  int32_t sig_run = 0;       // consecutive signalling windows
  int32_t ok_run = 0;        // consecutive windows without a signal
  int64_t contraction = 0;
};

bool valid(const misat_overload_config& c) {
  return c.ref_windows >= 1 && c.ref_windows <= 64 && c.min_ref >= 1 && c.min_ref <= c.ref_windows &&
         c.gap_ppm >= 0 && c.gap_ppm <= kPpm && c.confirm >= 1 && c.confirm <= 1000 && c.queue_thresh >= 0 &&
         c.recover_after >= 1 && c.recover_after <= 1000 && c.max_contraction_pct >= 0 &&
         c.max_contraction_pct <= 100;
}

}  // namespace

struct misat_overload {
  int32_t W = 0;
  misat_overload_config cfg{};
  std::vector<InstState> inst;
};

extern "C" {

void misat_overload_default_config(misat_overload_config* c) {
  if (!c) return;
  c->ref_windows = 8;
  c->min_ref = 3;
  c->gap_ppm = 100000;  // 10 points of hit rate below the healthy reference
  c->confirm = 2;
  c->queue_thresh = 64;
  c->recover_after = 2;
  c->max_contraction_pct = 50;
}

int misat_overload_create(int32_t n_instances, const misat_overload_config* cfg, misat_overload** out) {
  if (!out) return MISAT_ERR_INVALID_ARG;
  *out = nullptr;
  if (n_instances < 1 || n_instances > 1024 || !cfg || !valid(*cfg)) return MISAT_ERR_INVALID_ARG;
  misat_overload* ov = new (std::nothrow) misat_overload();
  if (!ov) return MISAT_ERR_OOM;
  ov->W = n_instances;
  ov->cfg = *cfg;
  ov->inst.resize(n_instances);
  for (auto& s : ov->inst) s.ref.assign(cfg->ref_windows, 0);
  *out = ov;
  return MISAT_OK;
}

int misat_overload_destroy(misat_overload* ov) {
  if (!ov) return MISAT_ERR_INVALID_ARG;
  delete ov;
  return MISAT_OK;
}

int misat_overload_observe(misat_overload* ov, const int64_t* hit_tokens, const int64_t* query_tokens,
                           const int64_t* waiting, const int64_t* k_base, int32_t* contraction_out) {
  if (!ov || !hit_tokens || !query_tokens || !waiting || !k_base) return MISAT_ERR_INVALID_ARG;
  const int64_t kMaxTok = (int64_t)1 << 40;
  for (int w = 0; w < ov->W; ++w) {
    if (hit_tokens[w] < 0 || query_tokens[w] < 0 || query_tokens[w] > kMaxTok || hit_tokens[w] > query_tokens[w] ||
        waiting[w] < 0 || k_base[w] < 0 || k_base[w] > ((int64_t)1 << 31))
      return MISAT_ERR_INVALID_ARG;
  }
  const misat_overload_config& c = ov->cfg;
  for (int w = 0; w < ov->W; ++w) {
    InstState& s = ov->inst[w];
    // observed hit rate of the window (none without queries)
    const int64_t h = query_tokens[w] > 0 ? hit_tokens[w] * kPpm / query_tokens[w] : -1;
    // reference h*: the best hit rate of the recent healthy windows
    int64_t href = -1;
    if (s.count >= c.min_ref)
      for (int i = 0; i < s.count; ++i) href = std::max(href, s.ref[i]);
    const int64_t gap = (h >= 0 && href >= 0) ? std::max<int64_t>(0, href - h) : 0;
    // a degradation counts only while the hit rate is not already recovering
    const bool hit_sig = gap > c.gap_ppm && (s.prev_h < 0 || h <= s.prev_h);
    const bool queue_sig = waiting[w] > c.queue_thresh;
    const bool signal = hit_sig || queue_sig;
    if (signal) {
      s.sig_run += 1;
      s.ok_run = 0;
    } else {
      s.sig_run = 0;
      s.ok_run += 1;
    }
    if (signal && s.sig_run >= c.confirm) {
      int64_t step = 0;
      if (hit_sig) step = std::max<int64_t>(step, std::max<int64_t>(1, k_base[w] * gap / kPpm));
      if (queue_sig) step = std::max<int64_t>(step, std::max<int64_t>(1, k_base[w] / 8));
      s.contraction += step;
    } else if (!signal && s.ok_run >= c.recover_after && s.contraction > 0) {
      s.contraction -= 1;  // gradual recovery: one session per recover_after healthy windows
      s.ok_run = 0;
    }
    const int64_t max_c = k_base[w] * c.max_contraction_pct / 100;
    s.contraction = std::min(std::max<int64_t>(s.contraction, 0), max_c);
    // a healthy window (observed, within the gap, no queue) joins the reference
    if (h >= 0 && gap <= c.gap_ppm && !queue_sig) {
      s.ref[s.head] = h;
      s.head = (s.head + 1) % c.ref_windows;
      s.count = std::min(s.count + 1, c.ref_windows);
    }
    if (h >= 0) s.prev_h = h;
    if (contraction_out) contraction_out[w] = (int32_t)s.contraction;
  }
  return MISAT_OK;
}

int misat_recheck_delays(int32_t n, const uint64_t* group, const uint8_t* held, int64_t base_delay_us,
                         int64_t min_delay_us, int64_t* delay_out) {
  if (n < 0 || base_delay_us < 0 || min_delay_us < 0 || min_delay_us > base_delay_us) return MISAT_ERR_INVALID_ARG;
  if (n == 0) return MISAT_OK;
  if (!group || !held || !delay_out) return MISAT_ERR_INVALID_ARG;
  std::unordered_map<uint64_t, int64_t> visible;
  visible.reserve((size_t)n * 2);
  for (int i = 0; i < n; ++i)
    if (group[i] != 0) visible[group[i]] += 1;
  for (int i = 0; i < n; ++i) {
    if (!held[i]) {
      delay_out[i] = 0;
    } else if (group[i] == 0) {
      delay_out[i] = base_delay_us;
    } else {
      delay_out[i] = std::max(min_delay_us, base_delay_us / visible[group[i]]);
    }
  }
  return MISAT_OK;
}

}  // extern "C"
