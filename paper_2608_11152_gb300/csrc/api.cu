// C ABI of the MISA-T routing library: context, orchestration of the kernels, class
// histories (host), table growth and state dumps.  See include/misat.h.
#include <algorithm>
#include <array>
#include <cstdlib>
#include <cstring>
#include <deque>
#include <memory>
#include <new>
#include <unordered_set>
#include <vector>

#include "common.cuh"
#include "envelope.cuh"
#include "kernels.h"

using namespace misat;

namespace {


// Small device block copied to the host in one transfer after each route / commit.
// Layout (8-byte words): stats[32] | U[W] | size[W] | sess_used | err | cand[3] | work | n_hits
struct MetaLayout {
  size_t stats = 0, U = 0, size = 0, sess_used = 0, err = 0, cand = 0, work = 0, n_hits = 0, g_used = 0, words = 0;
  void init(int W) {
    stats = 0;
    U = 32;
    size = U + W;
    sess_used = size + W;
    err = sess_used + 1;
    cand = err + 1;
    work = cand + 3;
    n_hits = work + 1;
    g_used = n_hits + 1;
    words = g_used + 1;
  }
};

inline int ceil_log2(uint64_t x) {
  int l = 0;
  while ((1ull << l) < x) ++l;
  return l;
}

// Eviction work buffers of one instance table (sized with the table).
struct InstBufs {
  uint32_t* bitmap = nullptr;  // fullness, 1 bit per bucket
  uint32_t* dmask = nullptr;   // deleted slots, 4 bits per bucket
  uint4* ca = nullptr;         // collected candidates (meta, key)
  uint4* cb = nullptr;         // narrowing work lists
  uint4* cc = nullptr;
  uint32_t* slots = nullptr;   // slot of each collected candidate
  uint32_t* dslots = nullptr;  // slots certainly evicted
};

void free_bufs(InstBufs& b) {
  cudaFree(b.bitmap);
  cudaFree(b.dmask);
  cudaFree(b.ca);
  cudaFree(b.cb);
  cudaFree(b.cc);
  cudaFree(b.slots);
  cudaFree(b.dslots);
  b = InstBufs{};
}

}  // namespace

struct misat_ctx {
  int device = 0, num_sms = 1;
  cudaStream_t stream = nullptr;
  // configuration
  int32_t W = 0, pf_q16 = 0, mode = 0, max_batch = 0, max_sessions = 0, hist_window = 256,
          min_obs = 8;
  int64_t max_tokens = 0, hold_delay_q = 0, prior_kbar[3] = {1, 1, 1}, prior_T = 0;
  uint64_t seed = kGold;
  double table_load = 0.75;
  std::vector<int64_t> cap;
  // host state
  std::deque<int64_t> hist_blocks[3], hist_res[3];
  uint32_t rho[3] = {333334, 333333, 333333};
  uint64_t seq = 0;
  bool routed = false;
  int32_t last_n = 0;
  int64_t last_ntok = 0;
  int64_t kbar_b[3] = {0, 0, 0}, T_b[3] = {0, 0, 0};
  // instance tables
  std::vector<InstDesc> h_desc;
  std::vector<InstBufs> h_bufs;
  InstDesc* d_desc = nullptr;
  uint32_t** d_bitmap = nullptr;
  uint32_t** d_dmask = nullptr;
  uint4** d_ca = nullptr;
  uint4** d_cb = nullptr;
  uint4** d_cc = nullptr;
  uint32_t** d_slots = nullptr;
  uint32_t** d_dslots = nullptr;
  unsigned* d_ncand = nullptr;
  unsigned* d_nd = nullptr;
  unsigned long long* d_thr = nullptr;  // [2W] bracket lo | hi
  // per-instance inputs and state
  int64_t* d_backlog = nullptr;
  int64_t* d_tokcost = nullptr;
  int32_t* d_contraction = nullptr;
  int32_t* d_prot = nullptr;
  unsigned long long* d_theta = nullptr;
  int32_t* d_active = nullptr;
  int32_t* d_act = nullptr;      // instances over capacity in the current eviction
  unsigned* d_nact = nullptr;
  int32_t* d_onew = nullptr;
  InstArrays ia{};
  // sessions
  SessTable sess{};
  // per-request scratch
  ReqArrays rq{};
  uint64_t* d_keys = nullptr;
  // global prefix index (MISAT_PREFIX_GLOBAL); its arrays are reallocated by rebuilds
  bool use_gix = false;
  GIndex gix{};
  int4* d_units = nullptr;      // insert work list (two int4 per unit)
  unsigned* d_units_n = nullptr;
  ulonglong2* d_gnew = nullptr; // keys new to a table during a commit (global index pass)
  unsigned* d_gnew_n = nullptr;
  int64_t units_cap = 0;
  int64_t keys_cap = 0;
  uint16_t* d_H = nullptr;
  int2* d_hits = nullptr;
  int64_t hits_cap = 0;
  unsigned long long* d_bm_key = nullptr;
  int32_t* d_bm_val = nullptr;
  int4* d_sel_rec = nullptr;     // per-request records of the selection
  uint8_t* d_onhull = nullptr;   // initial envelopes of the selection [3W]
  int32_t* d_rank = nullptr;     // slope order of the instances [W]
  int32_t* d_rank_a = nullptr;   // (d_w, w) order of the instances [W]
  int32_t* d_sel_list = nullptr; // [3 max_batch] each class's leaders per block of 256 requests
  int32_t* d_sel_cnt = nullptr;  // [3 * blocks] leaders per class and block
  int32_t* d_sel_x = nullptr;    // [W + 2] admissions per instance, ticket, coupled flag
  ulonglong2* d_grp = nullptr;   // (first key, instance) groups of a route's admitted requests
  GIndex fb{};                   // per-instance layout: batch-local index of the distinct block-0 keys
  int32_t* d_fb_list = nullptr;  // [max_batch] its claimed slots
  uint32_t grp_log2 = 1;
  int32_t* d_skip = nullptr;     // [max_batch] leading blocks a later request of the group inserts
  // every d_w and every 1/mu_w below 2^25: the selection's envelope arithmetic fits in 64 bits
  bool bk_small = true, tc_small = true;
  int32_t* d_chain_max = nullptr;  // per-chain insert limits of misat_load_chains
  // one small block of counters, mirrored to pinned host memory
  MetaLayout ml;
  unsigned long long* d_meta = nullptr;
  unsigned long long* h_meta = nullptr;
  cudaEvent_t ev_meta = nullptr;
  // staging of misat_route_host and of host-array calls
  int32_t* d_stage_tok = nullptr;
  int64_t* d_stage_off = nullptr;
  uint8_t* d_stage_cls = nullptr;
  uint64_t* d_stage_ses = nullptr;
  // completion events: two pinned host copies (so that the caller's arrays are free when
  // misat_complete returns), read by the completion kernel in place, and the event after the
  // kernel that last read each
  struct CompBuf {
    uint64_t* h_ses = nullptr;   // mapped pinned host memory
    uint8_t* h_done = nullptr;
    uint64_t* d_ses = nullptr;   // the same memory as the device addresses it
    uint8_t* d_done = nullptr;
    cudaEvent_t ev = nullptr;
  } comp[2];
  int comp_turn = 0;
  int32_t* d_out_inst = nullptr;
  uint8_t* d_out_reason = nullptr;
  int32_t* d_out_hit = nullptr;
  // pipelined host path (misat_stage_host / misat_route_staged): two device slots, filled on
  // a copy stream while the context's stream routes the other one; allocated on first use
  struct StageSlot {
    int32_t* tok = nullptr;
    int64_t* off = nullptr;
    uint8_t* cls = nullptr;
    uint64_t* ses = nullptr;
    int32_t n = 0;
    int64_t n_tokens = 0;
    bool staged = false;
    cudaEvent_t ev_copied = nullptr;  // the slot's H2D copies are done
    cudaEvent_t ev_free = nullptr;    // the last route that read the slot is done
    // delta-encoded batches (misat_stage_host_delta), allocated on first use
    int32_t* dbase = nullptr;
    int64_t* doff = nullptr;
    int32_t* dtok = nullptr;
    int64_t* h_off = nullptr;  // pinned: full offsets computed on the host
  } slot[2];
  std::vector<int64_t> delta_len;  // host scratch of misat_stage_host_delta
  std::vector<uint8_t> delta_depth;
  cudaStream_t copy_stream = nullptr;
  std::vector<void*> owned;  // fixed allocations freed in destroy
  // launch sequences replayed as CUDA graphs (captured on a private stream, which never
  // runs work, and launched on the context's stream)
  cudaStream_t cap_stream = nullptr;
  struct GraphCache {
    static constexpr size_t kEntries = 4;  // execs kept (least recently used dropped first)
    struct Entry {
      std::vector<uint64_t> key;
      cudaGraphExec_t exec = nullptr;
    };
    std::vector<Entry> entries;                   // most recently used last
    std::vector<std::vector<uint64_t>> pending;   // keys seen once (captured when they come again)
    bool failed = false;                          // a capture or instantiation failed: launch directly
    void clear() {
      for (auto& e : entries)
        if (e.exec) cudaGraphExecDestroy(e.exec);
      entries.clear();
      pending.clear();
    }
  } g_evict, g_evict_apply, g_route;
  int64_t* d_params = nullptr;  // [9] per-route class parameters (caps)
  // the commit's global-index pass runs on a side stream, beside the session update and
  // the read-only half of the eviction, and joins before the deletions
  cudaStream_t side_stream = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  // phase timing: events 0..7 bracket the route phases, 8..11 the commit phases
  bool timing = false;
  cudaEvent_t ev[17] = {};

  void mark(int i) {
    if (timing) cudaEventRecord(ev[i], stream);
  }
  void mark(int i, cudaStream_t s) {
    if (timing) cudaEventRecord(ev[i], s);
  }

  long long* size_ptr() { return reinterpret_cast<long long*>(d_meta + ml.size); }
  long long* U_ptr() { return reinterpret_cast<long long*>(d_meta + ml.U); }
  int32_t* err_ptr() { return reinterpret_cast<int32_t*>(d_meta + ml.err); }
  long long* cand_ptr() { return reinterpret_cast<long long*>(d_meta + ml.cand); }
  unsigned* work_ptr() { return reinterpret_cast<unsigned*>(d_meta + ml.work); }
  unsigned* nhits_ptr() { return reinterpret_cast<unsigned*>(d_meta + ml.n_hits); }
  unsigned long long* stats_ptr() { return d_meta + ml.stats; }
  long long h_size(int w) const { return reinterpret_cast<const long long*>(h_meta + ml.size)[w]; }
  long long h_U(int w) const { return reinterpret_cast<const long long*>(h_meta + ml.U)[w]; }
  int32_t h_err() const { return *reinterpret_cast<const int32_t*>(h_meta + ml.err); }
};

namespace {

#define CK(x)                                    \
  do {                                           \
    if ((x) != cudaSuccess) return MISAT_ERR_CUDA; \
  } while (0)

// Launch a fixed sequence through a cached CUDA graph: `launch(stream)` enqueues the
// sequence; it is captured once per key (the values its kernel arguments depend on) and
// replayed with one graph launch; the cache keeps the graphs of the four most recently used
// keys.  When the context's stream is itself being captured by the caller, or capture is
// unavailable, the sequence is launched directly.
template <class F>
int run_graph(misat_ctx* c, misat_ctx::GraphCache& gc, const std::vector<uint64_t>& key, F&& launch) {
  cudaStream_t st = c->stream;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  // direct launches while phase timing is on (events inside a graph do not time), after a
  // failed capture, and while the caller captures the stream itself
  if (c->timing || gc.failed || !c->cap_stream || cudaStreamIsCapturing(st, &cs) != cudaSuccess ||
      cs != cudaStreamCaptureStatusNone) {
    cudaGetLastError();
    launch(st);
    return cudaGetLastError() == cudaSuccess ? MISAT_OK : MISAT_ERR_CUDA;
  }
  for (size_t i = 0; i < gc.entries.size(); ++i) {
    if (gc.entries[i].key != key) continue;
    // replay; the entry becomes the most recently used
    misat_ctx::GraphCache::Entry hit = std::move(gc.entries[i]);
    gc.entries.erase(gc.entries.begin() + i);
    gc.entries.push_back(std::move(hit));
    CK(cudaGraphLaunch(gc.entries.back().exec, st));
    return MISAT_OK;
  }
  // a sequence is captured only when its key repeats: a caller that changes buffers on every
  // call is served by direct launches instead of a capture per call.  A few keys are
  // remembered, so that callers alternating between buffer sets (double-buffered staging)
  // are replayed from graphs too.
  bool seen = false;
  for (size_t i = 0; i < gc.pending.size(); ++i)
    if (gc.pending[i] == key) {
      gc.pending.erase(gc.pending.begin() + i);
      seen = true;
      break;
    }
  if (!seen) {
    if (gc.pending.size() >= misat_ctx::GraphCache::kEntries) gc.pending.erase(gc.pending.begin());
    gc.pending.push_back(key);
    launch(st);
    return cudaGetLastError() == cudaSuccess ? MISAT_OK : MISAT_ERR_CUDA;
  }
  cudaGraphExec_t exec = nullptr;
  cudaGraph_t g = nullptr;
  cudaError_t e = cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal);
  if (e == cudaSuccess) {
    launch(c->cap_stream);
    e = cudaStreamEndCapture(c->cap_stream, &g);
  }
  if (e == cudaSuccess && g) e = cudaGraphInstantiate(&exec, g, 0);
  if (g) cudaGraphDestroy(g);
  if (e != cudaSuccess || !exec) {
    // nothing was launched by the failed capture: run the sequence directly, now and later
    cudaGetLastError();
    if (exec) cudaGraphExecDestroy(exec);
    gc.clear();
    gc.failed = true;
    launch(st);
    return cudaGetLastError() == cudaSuccess ? MISAT_OK : MISAT_ERR_CUDA;
  }
  if (gc.entries.size() >= misat_ctx::GraphCache::kEntries) {
    // the stream may still run the oldest exec: destroying it is deferred by CUDA until then
    cudaGraphExecDestroy(gc.entries.front().exec);
    gc.entries.erase(gc.entries.begin());
  }
  gc.entries.push_back({key, exec});
  CK(cudaGraphLaunch(exec, st));
  return MISAT_OK;
}

int dalloc(misat_ctx* c, void** p, size_t bytes) {
  *p = nullptr;
  if (bytes == 0) bytes = 16;
  if (cudaMalloc(p, bytes) != cudaSuccess) {
    cudaGetLastError();
    return MISAT_ERR_OOM;
  }
  if (cudaMemset(*p, 0, bytes) != cudaSuccess) return MISAT_ERR_CUDA;
  c->owned.push_back(*p);
  return MISAT_OK;
}

template <typename T>
int dalloc_n(misat_ctx* c, T** p, size_t n) {
  return dalloc(c, reinterpret_cast<void**>(p), n * sizeof(T));
}

// Allocate instance w's table (zeroed) and its eviction buffers for 2^lg buckets.
int alloc_instance(misat_ctx* c, int w, uint32_t lg, InstDesc* out, InstBufs* bufs) {
  const size_t nb = (size_t)1 << lg;
  void* t = nullptr;
  InstBufs b;
  if (cudaMalloc(&t, nb * sizeof(Bucket)) != cudaSuccess ||
      cudaMalloc((void**)&b.bitmap, (nb / 32 + 1) * 4) != cudaSuccess ||
      cudaMalloc((void**)&b.dmask, (nb / 8 + 1) * 4) != cudaSuccess ||
      cudaMalloc((void**)&b.ca, nb * 4 * sizeof(uint4)) != cudaSuccess ||
      cudaMalloc((void**)&b.cb, nb * 4 * sizeof(uint4)) != cudaSuccess ||
      cudaMalloc((void**)&b.cc, nb * 4 * sizeof(uint4)) != cudaSuccess ||
      cudaMalloc((void**)&b.slots, nb * 4 * sizeof(uint32_t)) != cudaSuccess ||
      cudaMalloc((void**)&b.dslots, nb * 4 * sizeof(uint32_t)) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(t);
    free_bufs(b);
    return MISAT_ERR_OOM;
  }
  CK(cudaMemsetAsync(t, 0, nb * sizeof(Bucket), c->stream));
  CK(cudaMemsetAsync(b.bitmap, 0, (nb / 32 + 1) * 4, c->stream));
  CK(cudaMemsetAsync(b.dmask, 0, (nb / 8 + 1) * 4, c->stream));
  out->tab = (Bucket*)t;
  out->log2nb = lg;
  out->pad = 0;
  out->cap = c->cap[w];
  *bufs = b;
  return MISAT_OK;
}

int push_desc(misat_ctx* c, int w) {
  cudaStream_t st = c->stream;
  const InstBufs& b = c->h_bufs[w];
  CK(cudaMemcpyAsync(c->d_desc + w, &c->h_desc[w], sizeof(InstDesc), cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->d_bitmap + w, &b.bitmap, sizeof(void*), cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->d_dmask + w, &b.dmask, sizeof(void*), cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->d_ca + w, &b.ca, sizeof(void*), cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->d_cb + w, &b.cb, sizeof(void*), cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->d_cc + w, &b.cc, sizeof(void*), cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->d_slots + w, &b.slots, sizeof(void*), cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->d_dslots + w, &b.dslots, sizeof(void*), cudaMemcpyHostToDevice, st));
  return MISAT_OK;
}

// Replace instance w's table and buffers (the old ones are freed after the stream drains).
int swap_instance(misat_ctx* c, int w, const InstDesc& nd, const InstBufs& nb) {
  CK(cudaStreamSynchronize(c->stream));
  cudaFree(c->h_desc[w].tab);
  free_bufs(c->h_bufs[w]);
  c->h_desc[w] = nd;
  c->h_bufs[w] = nb;
  return push_desc(c, w);
}

uint32_t buckets_log2_for(int64_t entries, double load) {
  // smallest power-of-two bucket count whose slots hold `entries` at `load`
  const double slots = (double)entries / load;
  uint32_t lg = 1;
  while ((double)((uint64_t)4 << lg) < slots) ++lg;
  return lg;
}

// Grow instance w so that `need` entries fit at half load; entries are re-inserted.
int grow_instance(misat_ctx* c, int w, int64_t need) {
  const uint32_t lg = std::max(buckets_log2_for(need, 0.5), c->h_desc[w].log2nb + 1);
  InstDesc nd;
  InstBufs nb;
  int rc = alloc_instance(c, w, lg, &nd, &nb);
  if (rc) return rc;
  RehashArgs ra{c->h_desc[w], nd, c->err_ptr()};
  launch_rehash(ra, c->stream);
  CK(cudaGetLastError());
  return swap_instance(c, w, nd, nb);
}

// Make room for `add[w]` more entries on every instance (current sizes must be on the host).
int ensure_capacity(misat_ctx* c, const std::vector<int64_t>& sizes, const std::vector<int64_t>& add) {
  for (int w = 0; w < c->W; ++w) {
    const int64_t need = sizes[w] + add[w];
    const double slots = (double)((uint64_t)4 << c->h_desc[w].log2nb);
    if ((double)need > c->table_load * slots) {
      int rc = grow_instance(c, w, need);
      if (rc) return rc;
    }
  }
  return MISAT_OK;
}

// ---- global prefix index ----
constexpr double kGixLoad = 0.35;  // load after a rebuild
constexpr double kGixMax = 0.7;    // claimed slots that trigger a rebuild

size_t gix_slots(const misat_ctx* c) { return (size_t)4 << c->gix.log2nb; }

// Replace the index arrays by zeroed ones of 2^lg buckets (waits for the stream).
int gix_alloc(misat_ctx* c, uint32_t lg) {
  const size_t slots = (size_t)4 << lg;
  unsigned long long *k = nullptr, *m = nullptr;
  if (cudaMalloc(&k, slots * 8) != cudaSuccess || cudaMalloc(&m, slots * c->gix.mw * 8) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(k);
    return MISAT_ERR_OOM;
  }
  CK(cudaStreamSynchronize(c->stream));
  cudaFree(c->gix.keys);
  cudaFree(c->gix.masks);
  c->gix.keys = k;
  c->gix.masks = m;
  c->gix.log2nb = lg;
  CK(cudaMemsetAsync(k, 0, slots * 8, c->stream));
  CK(cudaMemsetAsync(m, 0, slots * c->gix.mw * 8, c->stream));
  return MISAT_OK;
}

// Rebuild the index from the instance tables, growing it so that `live` keys fill at
// most kGixLoad of it.
int gix_rebuild(misat_ctx* c, int64_t live) {
  const uint32_t lg = std::max(c->gix.log2nb, buckets_log2_for(std::max<int64_t>(live, 1024), kGixLoad));
  if (lg != c->gix.log2nb) {
    int rc = gix_alloc(c, lg);
    if (rc) return rc;
  } else {
    CK(cudaMemsetAsync(c->gix.keys, 0, gix_slots(c) * 8, c->stream));
    CK(cudaMemsetAsync(c->gix.masks, 0, gix_slots(c) * c->gix.mw * 8, c->stream));
  }
  CK(cudaMemsetAsync(c->d_meta + c->ml.g_used, 0, 8, c->stream));
  c->h_meta[c->ml.g_used] = 0;
  uint32_t maxlg = 1;
  for (auto& d : c->h_desc) maxlg = std::max(maxlg, d.log2nb);
  launch_gix_build(c->d_desc, c->W, maxlg, c->gix, c->err_ptr(), c->stream);
  CK(cudaGetLastError());
  return MISAT_OK;
}

// Before up to `add` keys enter the tables (claimed-slot count must be on the host).
int gix_ensure(misat_ctx* c, const std::vector<int64_t>& sizes, int64_t add) {
  if (!c->use_gix) return MISAT_OK;
  const uint64_t used = c->h_meta[c->ml.g_used];
  if ((double)(used + (uint64_t)add) <= kGixMax * (double)gix_slots(c)) return MISAT_OK;
  int64_t live = add;
  for (int64_t x : sizes) live += x;
  return gix_rebuild(c, live);
}

GIndex gix_or_null(const misat_ctx* c) { return c->use_gix ? c->gix : GIndex{}; }

// Read the counters block (sync).
int read_meta(misat_ctx* c) {
  CK(cudaMemcpyAsync(c->h_meta, c->d_meta, c->ml.words * 8, cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  return MISAT_OK;
}

int enqueue_meta(misat_ctx* c) {
  CK(cudaMemcpyAsync(c->h_meta, c->d_meta, c->ml.words * 8, cudaMemcpyDeviceToHost, c->stream));
  CK(cudaEventRecord(c->ev_meta, c->stream));
  return MISAT_OK;
}

// Session table rebuild when claimed slots (live + finished) pass 70% of it.
int maybe_rebuild_sessions(misat_ctx* c, int64_t incoming) {
  const uint64_t used = c->h_meta[c->ml.sess_used];
  const uint64_t capn = 1ull << c->sess.log2n;
  if ((double)(used + incoming) <= 0.7 * (double)capn) return MISAT_OK;
  // count live sessions on the host from a copy (rare path)
  std::vector<SessSlot> hs(capn);
  CK(cudaMemcpyAsync(hs.data(), c->sess.slots, capn * sizeof(SessSlot), cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  uint64_t live = 0;
  for (auto& s : hs)
    if (s.key && (sess_state(s.val) == kSessProtected || sess_state(s.val) == kSessReleased)) ++live;
  const uint64_t want = std::max<uint64_t>(2 * (uint64_t)c->max_sessions, 2 * (live + (uint64_t)incoming));
  const uint32_t lg = (uint32_t)std::max(4, ceil_log2(want));
  SessSlot* ns = nullptr;
  if (cudaMalloc(&ns, ((size_t)1 << lg) * sizeof(SessSlot)) != cudaSuccess) {
    cudaGetLastError();
    return MISAT_ERR_OOM;
  }
  CK(cudaMemsetAsync(ns, 0, ((size_t)1 << lg) * sizeof(SessSlot), c->stream));
  CK(cudaMemsetAsync(c->d_meta + c->ml.sess_used, 0, 8, c->stream));
  SessTable to{ns, lg, c->d_meta + c->ml.sess_used};
  SessRehashArgs a{c->sess, to, c->err_ptr()};
  launch_sess_rehash(a, c->stream);
  CK(cudaGetLastError());
  CK(cudaStreamSynchronize(c->stream));
  cudaFree(c->sess.slots);
  c->sess = to;
  return read_meta(c);
}

void estimate_classes(misat_ctx* c) {
  for (int b = 0; b < 3; ++b) {
    const auto& h = c->hist_blocks[b];
    if (h.empty()) {
      c->kbar_b[b] = c->prior_kbar[b];
    } else {
      std::vector<int64_t> v(h.begin(), h.end());
      std::sort(v.begin(), v.end());
      const int64_t m = (int64_t)v.size();
      const int64_t rank = (9 * m + 9) / 10;  // nearest-rank 90th percentile
      c->kbar_b[b] = std::max(c->prior_kbar[b], v[rank - 1]);
    }
    const auto& t = c->hist_res[b];
    if ((int64_t)t.size() < c->min_obs) {
      c->T_b[b] = c->prior_T;
    } else {
      int64_t s = 0;
      for (int64_t x : t) s += x;
      c->T_b[b] = s / (int64_t)t.size();
    }
  }
}

EvictArgs evict_args(misat_ctx* c, unsigned long long* evicted_counter) {
  EvictArgs ev{};
  ev.desc = c->d_desc;
  ev.W = c->W;
  ev.only_w = nullptr;
  ev.size = c->size_ptr();
  ev.bitmaps = c->d_bitmap;
  ev.cand_a = c->d_ca;
  ev.cand_b = c->d_cb;
  ev.cand_c = c->d_cc;
  ev.slots = c->d_slots;
  ev.dslots = c->d_dslots;
  ev.dmask = c->d_dmask;
  ev.n_cand = c->d_ncand;
  ev.n_d = c->d_nd;
  ev.thr_lo = c->d_thr;
  ev.thr_hi = c->d_thr + c->W;
  ev.theta = c->d_theta;
  ev.active = c->d_active;
  ev.act = c->d_act;
  ev.n_act = c->d_nact;
  ev.evicted = evicted_counter;
  ev.err = c->err_ptr();
  ev.gix = gix_or_null(c);
  return ev;
}

// Eviction of every instance above capacity; `join` (may be NULL) is waited for between the
// read-only half and the deletions.
int evict_all(misat_ctx* c, unsigned long long* evicted_counter, cudaEvent_t join = nullptr) {
  const EvictArgs ev = evict_args(c, evicted_counter);
  // streaming CTAs per instance: about 4 buckets per thread, at most 256 CTAs of 256
  uint32_t maxlg = 1;
  for (auto& d : c->h_desc) maxlg = std::max(maxlg, d.log2nb);
  const int chunks = (int)std::min<uint64_t>(256, std::max<uint64_t>(1, ((uint64_t)1 << maxlg) / (4 * 256)));
  const std::vector<uint64_t> key{(uint64_t)chunks, reinterpret_cast<uint64_t>(ev.gix.keys),
                                  (uint64_t)ev.gix.log2nb, reinterpret_cast<uint64_t>(evicted_counter)};
  // with phase timing the kernels are launched directly with an event after each
  const cudaEvent_t* marks = c->timing ? c->ev + 12 : nullptr;
  int rc = run_graph(c, c->g_evict, key,
                     [&](cudaStream_t s) { launch_evict_select(ev, chunks, c->num_sms, s, marks); });
  if (rc) return rc;
  if (join) CK(cudaStreamWaitEvent(c->stream, join, 0));
  return run_graph(c, c->g_evict_apply, key,
                   [&](cudaStream_t s) { launch_evict_apply(ev, c->num_sms, s, marks ? marks + 3 : nullptr); });
}

CapsArgs caps_args(misat_ctx* c) {
  CapsArgs ca{};
  ca.W = c->W;
  ca.desc = c->d_desc;
  ca.prot = c->d_prot;
  ca.cand = c->cand_ptr();
  ca.params = c->d_params;
  ca.pf_q16 = c->pf_q16;
  ca.mode = c->mode;
  ca.contraction = c->d_contraction;
  ca.ia = c->ia;
  ca.err = c->err_ptr();
  return ca;
}

// The device work of one route (n > 0), enqueued on stream st: counters reset, prologue,
// block hash, caps, probes, serial selection, finalize.  Captured into the route graph, or
// launched directly while the caller captures the context's stream.
void enqueue_route(misat_ctx* c, const misat_batch* b, misat_decisions* out, cudaStream_t st) {
  const int32_t n = b->n;
  // reset the per-batch counters: stats, U, cand, work, n_hits (size and sess_used persist)
  cudaMemsetAsync(c->d_meta + c->ml.stats, 0, 32 * 8, st);
  cudaMemsetAsync(c->d_meta + c->ml.U, 0, c->W * 8, st);
  cudaMemsetAsync(c->d_meta + c->ml.cand, 0, 5 * 8, st);
  const int bm_log2 = std::max(1, ceil_log2(2 * (uint64_t)n));
  cudaMemsetAsync(c->d_bm_key, 0, ((size_t)1 << bm_log2) * 8, st);
  cudaMemsetAsync(c->d_bm_val, 0x7f, ((size_t)1 << bm_log2) * 4, st);
  cudaMemsetAsync(c->d_grp, 0, ((size_t)1 << bm_log2) * sizeof(ulonglong2), st);
  GIndex fb{};
  if (c->fb.keys) {
    fb = c->fb;
    fb.log2nb = (uint32_t)std::max(0, bm_log2 - 2);
    cudaMemsetAsync(fb.keys, 0, ((size_t)4 << fb.log2nb) * 8, st);
  }

  c->mark(0, st);
  PrologueArgs pa{};
  pa.n = n;
  pa.n_tokens = b->n_tokens;
  pa.cls = b->cls;
  pa.session = b->session;
  pa.tok_off = b->tok_off;
  pa.rq = c->rq;
  pa.st = c->sess;
  pa.bm_key = c->d_bm_key;
  pa.bm_val = c->d_bm_val;
  pa.bm_log2 = (uint32_t)bm_log2;
  pa.cand = c->cand_ptr();
  pa.err = c->err_ptr();
  launch_prologue(pa, st);
  c->mark(1, st);

  HashArgs ha{};
  ha.tok_off = b->tok_off;
  ha.tokens = b->tokens;
  ha.n_tokens = b->n_tokens;
  ha.n = n;
  ha.seed = c->seed;
  ha.keys = c->d_keys;
  ha.keys_cap = c->keys_cap;
  ha.work = c->work_ptr();
  ha.err = c->err_ptr();
  launch_block_hash(ha, c->num_sms, st);
  c->mark(2, st);
  launch_caps(caps_args(c), st);
  c->mark(3, st);

  ProbeArgs pr{};
  pr.desc = c->d_desc;
  pr.W = c->W;
  pr.n = n;
  pr.nb = c->rq.nb;
  pr.kbase = c->rq.kbase;
  pr.keys = c->d_keys;
  pr.H = c->d_H;
  pr.hits = c->d_hits;
  pr.hbest = c->rq.hbest;
  pr.n_hits = c->nhits_ptr();
  pr.hits_cap = c->hits_cap;
  pr.stats = c->stats_ptr() + 16;
  pr.stats_search = c->stats_ptr() + 22;
  pr.err = c->err_ptr();
  pr.gix = gix_or_null(c);
  pr.fb = fb;
  pr.fb_list = c->d_fb_list;
  pr.fb_count = c->stats_ptr() + 26;
  pr.stats_fb = c->stats_ptr() + 27;
  launch_probe_first(pr, c->num_sms, st);
  c->mark(4, st);
  launch_probe_search(pr, c->num_sms, st);
  c->mark(5, st);
  if (b->out_H)
    cudaMemcpyAsync(b->out_H, c->d_H, (size_t)n * c->W * sizeof(uint16_t), cudaMemcpyDeviceToDevice, st);

  SelectPrepArgs sp{};
  sp.n = n;
  sp.W = c->W;
  sp.rq = c->rq;
  sp.H = c->d_H;
  sp.rec = c->d_sel_rec;
  sp.adm = c->d_sel_x;
  sp.ticket = reinterpret_cast<unsigned*>(c->d_sel_x + c->W);
  sp.coupled = c->d_sel_x + c->W + 1;
  sp.seg = c->d_sel_list;
  sp.segcnt = c->d_sel_cnt;
  sp.err = c->err_ptr();
  launch_select_prep(sp, st);
  EnvInitArgs ei{};
  ei.W = c->W;
  ei.backlog = c->d_backlog;
  ei.tokcost = c->d_tokcost;
  ei.gh = c->ia.gh;
  ei.ch = c->ia.ch;
  ei.onhull = c->d_onhull;
  ei.rank = c->d_rank;
  ei.rank_a = c->d_rank_a;
  ei.small = c->bk_small && c->tc_small;
  ei.err = c->err_ptr();
  launch_env_init(ei, st);
  SelectClassArgs sc{};
  sc.n = n;
  sc.W = c->W;
  sc.rec = c->d_sel_rec;
  sc.rq = c->rq;
  sc.gh = c->ia.gh;
  sc.ch = c->ia.ch;
  sc.backlog = c->d_backlog;
  sc.tokcost = c->d_tokcost;
  sc.onhull = c->d_onhull;
  sc.rank = c->d_rank;
  sc.rank_a = c->d_rank_a;
  sc.H = c->d_H;
  sc.hold_delay_q = c->hold_delay_q;
  sc.small = c->bk_small && c->tc_small;
  sc.seg = c->d_sel_list;
  sc.segcnt = c->d_sel_cnt;
  sc.adm = c->d_sel_x;
  sc.ticket = reinterpret_cast<unsigned*>(c->d_sel_x + c->W);
  sc.coupled = c->d_sel_x + c->W + 1;
  sc.stats = c->stats_ptr();
  sc.err = c->err_ptr();
  launch_select_class(sc, st);
  SelectArgs sa{};
  sa.n = n;
  sa.W = c->W;
  sa.rec = c->d_sel_rec;
  sa.rq = c->rq;
  sa.gh = c->ia.gh;
  sa.ch = c->ia.ch;
  sa.backlog = c->d_backlog;
  sa.tokcost = c->d_tokcost;
  sa.onhull = c->d_onhull;
  sa.rank = c->d_rank;
  sa.rank_a = c->d_rank_a;
  sa.small = c->bk_small && c->tc_small;
  sa.H = c->d_H;
  sa.hold_delay_q = c->hold_delay_q;
  sa.coupled = c->d_sel_x + c->W + 1;
  sa.err = c->err_ptr();
  launch_select(sa, st);
  c->mark(6, st);

  FinalizeArgs fa{};
  fa.n = n;
  fa.W = c->W;
  fa.rq = c->rq;
  fa.H = c->d_H;
  fa.out_inst = out->inst;
  fa.out_reason = out->reason;
  fa.out_hit = out->hit_blocks;
  fa.U = c->U_ptr();
  fa.stats = c->stats_ptr();
  fa.grp = c->d_grp;
  fa.grp_log2 = (uint32_t)bm_log2;
  fa.keys = c->d_keys;
  fa.err = c->err_ptr();
  launch_finalize(fa, st);
  c->mark(7, st);
}


}  // namespace

extern "C" {

const char* misat_strerror(int code) {
  switch (code) {
    case MISAT_OK: return "ok";
    case MISAT_ERR_INVALID_ARG: return "invalid argument";
    case MISAT_ERR_OOM: return "out of memory";
    case MISAT_ERR_CUDA: return "CUDA runtime error";
    case MISAT_ERR_STATE: return "call not valid in this state";
    case MISAT_ERR_TABLE_FULL: return "table full";
    case MISAT_ERR_BATCH_TOO_LARGE: return "batch exceeds max_batch or max_tokens";
    case MISAT_ERR_INTERNAL: return "global prefix index out of step with the instance tables";
    default: return "unknown error";
  }
}

int misat_destroy(misat_ctx* c) {
  if (!c) return MISAT_ERR_INVALID_ARG;
  cudaStreamSynchronize(c->stream);
  c->g_evict.clear();
  c->g_evict_apply.clear();
  c->g_route.clear();
  if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
  if (c->side_stream) {
    cudaStreamSynchronize(c->side_stream);
    cudaStreamDestroy(c->side_stream);
  }
  if (c->copy_stream) {
    cudaStreamSynchronize(c->copy_stream);
    cudaStreamDestroy(c->copy_stream);
  }
  for (auto& cb : c->comp) {
    if (cb.ev) cudaEventDestroy(cb.ev);
    if (cb.h_ses) cudaFreeHost(cb.h_ses);
    if (cb.h_done) cudaFreeHost(cb.h_done);
  }
  for (auto& sl : c->slot) {
    if (sl.ev_copied) cudaEventDestroy(sl.ev_copied);
    if (sl.ev_free) cudaEventDestroy(sl.ev_free);
    if (sl.h_off) cudaFreeHost(sl.h_off);
  }
  if (c->ev_fork) cudaEventDestroy(c->ev_fork);
  if (c->ev_join) cudaEventDestroy(c->ev_join);
  for (size_t w = 0; w < c->h_desc.size(); ++w) {
    cudaFree(c->h_desc[w].tab);
    if (w < c->h_bufs.size()) free_bufs(c->h_bufs[w]);
  }
  cudaFree(c->sess.slots);
  cudaFree(c->gix.keys);
  cudaFree(c->gix.masks);
  for (void* p : c->owned) cudaFree(p);
  if (c->h_meta) cudaFreeHost(c->h_meta);
  if (c->ev_meta) cudaEventDestroy(c->ev_meta);
  for (auto& e : c->ev)
    if (e) cudaEventDestroy(e);
  delete c;
  return MISAT_OK;
}

int misat_create(const misat_config* cfg, void* cuda_stream, misat_ctx** out) {
  if (!cfg || !out || !cfg->cap_blocks) return MISAT_ERR_INVALID_ARG;
  *out = nullptr;
  const int W = cfg->n_instances;
  if (W < 1 || W > kMaxW) return MISAT_ERR_INVALID_ARG;
  for (int w = 0; w < W; ++w)
    if (cfg->cap_blocks[w] < 1 || cfg->cap_blocks[w] > ((int64_t)1 << 26)) return MISAT_ERR_INVALID_ARG;
  if (cfg->protected_frac_q16 < 1 || cfg->protected_frac_q16 > 65536) return MISAT_ERR_INVALID_ARG;
  if (cfg->mode < 0 || cfg->mode > 3) return MISAT_ERR_INVALID_ARG;
  if (cfg->max_batch < 1 || cfg->max_batch > (1 << 20)) return MISAT_ERR_INVALID_ARG;
  if (cfg->max_tokens < 16 || cfg->max_tokens > ((int64_t)1 << 36)) return MISAT_ERR_INVALID_ARG;
  if (cfg->max_sessions < 1 || cfg->max_sessions > (1 << 28)) return MISAT_ERR_INVALID_ARG;
  if (cfg->hist_window < 1 || cfg->hist_window > 4096 || cfg->min_obs < 1) return MISAT_ERR_INVALID_ARG;
  if (cfg->hold_delay_q < 0 || cfg->hold_delay_q > kBacklogMax) return MISAT_ERR_INVALID_ARG;
  for (int b = 0; b < 3; ++b)
    if (cfg->prior_kbar_blocks[b] < 1 || cfg->prior_kbar_blocks[b] > ((int64_t)1 << 30)) return MISAT_ERR_INVALID_ARG;
  if (cfg->prior_T_us < 0 || cfg->prior_T_us > ((int64_t)1 << 40)) return MISAT_ERR_INVALID_ARG;
  if (!(cfg->table_load >= 0.25 && cfg->table_load <= 0.9)) return MISAT_ERR_INVALID_ARG;
  if (cfg->prefix_index != MISAT_PREFIX_GLOBAL && cfg->prefix_index != MISAT_PREFIX_PER_INSTANCE)
    return MISAT_ERR_INVALID_ARG;

  misat_ctx* c = new (std::nothrow) misat_ctx();
  if (!c) return MISAT_ERR_OOM;
  int rc = MISAT_OK;
  auto fail = [&](int code) {
    misat_destroy(c);
    return code;
  };
  if (cudaGetDevice(&c->device) != cudaSuccess) return fail(MISAT_ERR_CUDA);
  if (cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device) != cudaSuccess)
    return fail(MISAT_ERR_CUDA);
  if (select_configure() != cudaSuccess || select_class_configure() != cudaSuccess) return fail(MISAT_ERR_CUDA);
  c->stream = (cudaStream_t)cuda_stream;
  c->W = W;
  c->cap.assign(cfg->cap_blocks, cfg->cap_blocks + W);
  c->pf_q16 = cfg->protected_frac_q16;
  c->mode = cfg->mode;
  c->max_batch = cfg->max_batch;
  c->max_tokens = cfg->max_tokens;
  c->max_sessions = cfg->max_sessions;
  c->hist_window = cfg->hist_window;
  c->min_obs = cfg->min_obs;
  c->hold_delay_q = cfg->hold_delay_q;
  for (int b = 0; b < 3; ++b) c->prior_kbar[b] = cfg->prior_kbar_blocks[b];
  c->prior_T = cfg->prior_T_us;
  c->seed = cfg->hash_seed;
  c->table_load = cfg->table_load;
  c->ml.init(W);
  if (cudaEventCreateWithFlags(&c->ev_meta, cudaEventDisableTiming) != cudaSuccess) return fail(MISAT_ERR_CUDA);
  if (cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking) != cudaSuccess) {
    cudaGetLastError();
    c->cap_stream = nullptr;  // sequences are then launched directly
  }
  if (cudaStreamCreateWithFlags(&c->side_stream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&c->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&c->ev_join, cudaEventDisableTiming) != cudaSuccess) {
    cudaGetLastError();
    if (c->side_stream) cudaStreamDestroy(c->side_stream);
    c->side_stream = nullptr;  // the global-index pass then runs on the context's stream
  }
  if (cudaMallocHost(&c->h_meta, c->ml.words * 8) != cudaSuccess) return fail(MISAT_ERR_OOM);
  std::memset(c->h_meta, 0, c->ml.words * 8);

  const size_t NB = (size_t)c->max_batch, Ws = (size_t)W;
  c->keys_cap = c->max_tokens / 16 + 1;
  c->units_cap = (int64_t)NB + c->keys_cap / 128 + 1;  // one unit per 128 blocks of a request
  c->hits_cap = (int64_t)std::min<size_t>(NB * Ws, (size_t)1 << 27);
  const int bm_log2 = std::max(1, ceil_log2(2 * NB));
  if ((rc = dalloc_n(c, &c->d_meta, c->ml.words)) || (rc = dalloc_n(c, &c->d_keys, (size_t)c->keys_cap)) ||
      (rc = dalloc_n(c, &c->d_units, 2 * (size_t)c->units_cap)) || (rc = dalloc_n(c, &c->d_units_n, 1)) ||
      (rc = dalloc_n(c, &c->d_H, NB * Ws)) || (rc = dalloc_n(c, &c->d_hits, (size_t)c->hits_cap)) ||
      (rc = dalloc_n(c, &c->d_bm_key, (size_t)1 << bm_log2)) ||
      (rc = dalloc_n(c, &c->d_bm_val, (size_t)1 << bm_log2)) || (rc = dalloc_n(c, &c->d_sel_rec, 2 * NB)) ||
      (rc = dalloc_n(c, &c->d_onhull, 3 * Ws)) || (rc = dalloc_n(c, &c->d_rank, Ws)) ||
      (rc = dalloc_n(c, &c->d_rank_a, Ws)) || (rc = dalloc_n(c, &c->d_sel_list, 3 * NB)) ||
      (rc = dalloc_n(c, &c->d_sel_cnt, 3 * ((NB + 255) / 256))) ||
      (rc = dalloc_n(c, &c->d_sel_x, Ws + 2)) || (rc = dalloc_n(c, &c->d_skip, NB)) ||
      (rc = dalloc_n(c, &c->d_grp, (size_t)1 << bm_log2)) ||
      (rc = dalloc_n(c, &c->rq.nb, NB)) || (rc = dalloc_n(c, &c->rq.kbase, NB)) || (rc = dalloc_n(c, &c->rq.L, NB)) ||
      (rc = dalloc_n(c, &c->rq.cls, NB)) || (rc = dalloc_n(c, &c->rq.session, NB)) ||
      (rc = dalloc_n(c, &c->rq.sst, NB)) || (rc = dalloc_n(c, &c->rq.sinst, NB)) ||
      (rc = dalloc_n(c, &c->rq.leader, NB)) || (rc = dalloc_n(c, &c->rq.status, NB)) ||
      (rc = dalloc_n(c, &c->d_chain_max, NB)) || (rc = dalloc_n(c, &c->rq.last_reason, NB)) ||
      (rc = dalloc_n(c, &c->rq.inst, NB)) || (rc = dalloc_n(c, &c->rq.reason, NB)) ||
      (rc = dalloc_n(c, &c->rq.hbest, NB)) ||
      (rc = dalloc_n(c, &c->ia.K_w, Ws)) || (rc = dalloc_n(c, &c->ia.K_wb, 3 * Ws)) ||
      (rc = dalloc_n(c, &c->ia.N_wb, 3 * Ws)) || (rc = dalloc_n(c, &c->ia.kbar_w, Ws)) ||
      (rc = dalloc_n(c, &c->ia.tot, Ws)) || (rc = dalloc_n(c, &c->ia.gh, Ws)) || (rc = dalloc_n(c, &c->ia.ch, 3 * Ws)) ||
      (rc = dalloc_n(c, &c->d_params, 9)) ||
      (rc = dalloc_n(c, &c->d_backlog, Ws)) ||
      (rc = dalloc_n(c, &c->d_tokcost, Ws)) || (rc = dalloc_n(c, &c->d_contraction, Ws)) ||
      (rc = dalloc_n(c, &c->d_prot, 3 * Ws)) || (rc = dalloc_n(c, &c->d_theta, 2 * Ws)) ||
      (rc = dalloc_n(c, &c->d_active, Ws)) || (rc = dalloc_n(c, &c->d_onew, 1)) ||
      (rc = dalloc_n(c, &c->d_act, Ws)) || (rc = dalloc_n(c, &c->d_nact, 1)) ||
      (rc = dalloc_n(c, &c->d_desc, Ws)) || (rc = dalloc_n(c, &c->d_bitmap, Ws)) || (rc = dalloc_n(c, &c->d_ca, Ws)) ||
      (rc = dalloc_n(c, &c->d_cb, Ws)) || (rc = dalloc_n(c, &c->d_cc, Ws)) || (rc = dalloc_n(c, &c->d_slots, Ws)) ||
      (rc = dalloc_n(c, &c->d_dmask, Ws)) || (rc = dalloc_n(c, &c->d_ncand, Ws)) ||
      (rc = dalloc_n(c, &c->d_dslots, Ws)) || (rc = dalloc_n(c, &c->d_nd, Ws)) ||
      (rc = dalloc_n(c, &c->d_thr, 2 * Ws)) ||
      (rc = dalloc_n(c, &c->d_stage_tok, (size_t)c->max_tokens + 8)) ||
      (rc = dalloc_n(c, &c->d_stage_off, NB + 1)) || (rc = dalloc_n(c, &c->d_stage_cls, NB)) ||
      (rc = dalloc_n(c, &c->d_stage_ses, NB)) || (rc = dalloc_n(c, &c->d_out_inst, NB)) ||
      (rc = dalloc_n(c, &c->d_out_reason, NB)) || (rc = dalloc_n(c, &c->d_out_hit, NB)))
    return fail(rc);
  c->ia.U = c->U_ptr();
  // instance tables: at most half full after eviction
  c->h_desc.resize(W);
  c->h_bufs.resize(W);
  for (int w = 0; w < W; ++w) {
    if ((rc = alloc_instance(c, w, buckets_log2_for(c->cap[w], 0.5), &c->h_desc[w], &c->h_bufs[w])))
      return fail(rc);
    if ((rc = push_desc(c, w))) return fail(rc);
  }
  // session table
  {
    const uint32_t lg = (uint32_t)std::max(4, ceil_log2(2ull * (uint64_t)c->max_sessions));
    if (cudaMalloc(&c->sess.slots, ((size_t)1 << lg) * sizeof(SessSlot)) != cudaSuccess) {
      cudaGetLastError();
      return fail(MISAT_ERR_OOM);
    }
    if (cudaMemsetAsync(c->sess.slots, 0, ((size_t)1 << lg) * sizeof(SessSlot), c->stream) != cudaSuccess)
      return fail(MISAT_ERR_CUDA);
    c->sess.log2n = lg;
    c->sess.used = c->d_meta + c->ml.sess_used;
  }
  // per-instance layout: the batch-local index of distinct block-0 keys (2 max_batch slots)
  if (cfg->prefix_index == MISAT_PREFIX_PER_INSTANCE) {
    c->fb.mw = (uint32_t)((W + 63) / 64);
    const size_t fslots = (size_t)4 << std::max(0, bm_log2 - 2);
    if ((rc = dalloc_n(c, &c->fb.keys, fslots)) || (rc = dalloc_n(c, &c->fb.masks, fslots * c->fb.mw)) ||
        (rc = dalloc_n(c, &c->d_fb_list, NB)))
      return fail(rc);
  }
  // global prefix index, sized for full tables (up to 2^26 keys; rebuilds grow it)
  if (cfg->prefix_index == MISAT_PREFIX_GLOBAL) {
    c->use_gix = true;
    c->gix.mw = (uint32_t)((W + 63) / 64);
    c->gix.used = c->d_meta + c->ml.g_used;
    int64_t total_cap = 0;
    for (int w = 0; w < W; ++w) total_cap += c->cap[w];
    total_cap = std::min<int64_t>(total_cap, (int64_t)1 << 26);
    if ((rc = gix_alloc(c, buckets_log2_for(std::max<int64_t>(total_cap, 1024), kGixLoad)))) return fail(rc);
    if ((rc = dalloc_n(c, &c->d_gnew, (size_t)c->keys_cap)) || (rc = dalloc_n(c, &c->d_gnew_n, 1))) return fail(rc);
  }
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return fail(MISAT_ERR_CUDA);
  *out = c;
  return MISAT_OK;
}

int misat_set_mixture(misat_ctx* c, const uint32_t rho_ppm[3]) {
  if (!c || !rho_ppm) return MISAT_ERR_INVALID_ARG;
  if ((uint64_t)rho_ppm[0] + rho_ppm[1] + rho_ppm[2] != 1000000) return MISAT_ERR_INVALID_ARG;
  for (int b = 0; b < 3; ++b) c->rho[b] = rho_ppm[b];
  return MISAT_OK;
}

int misat_set_instance_state(misat_ctx* c, const int64_t* backlog_q, const int64_t* tokcost_q,
                             const int32_t* cap_contraction) {
  if (!c) return MISAT_ERR_INVALID_ARG;
  for (int w = 0; w < c->W; ++w) {
    if (backlog_q && (backlog_q[w] < 0 || backlog_q[w] > kBacklogMax)) return MISAT_ERR_INVALID_ARG;
    if (tokcost_q && (tokcost_q[w] < 0 || tokcost_q[w] > ((int64_t)1 << 32))) return MISAT_ERR_INVALID_ARG;
    if (cap_contraction && cap_contraction[w] < 0) return MISAT_ERR_INVALID_ARG;
  }
  auto below = [&](const int64_t* v) {
    for (int w = 0; w < c->W; ++w)
      if (v[w] >= kEnvSmall) return false;
    return true;
  };
  if (backlog_q) c->bk_small = below(backlog_q);
  if (tokcost_q) c->tc_small = below(tokcost_q);
  if (backlog_q) CK(cudaMemcpyAsync(c->d_backlog, backlog_q, c->W * 8, cudaMemcpyHostToDevice, c->stream));
  if (tokcost_q) CK(cudaMemcpyAsync(c->d_tokcost, tokcost_q, c->W * 8, cudaMemcpyHostToDevice, c->stream));
  if (cap_contraction)
    CK(cudaMemcpyAsync(c->d_contraction, cap_contraction, c->W * 4, cudaMemcpyHostToDevice, c->stream));
  return MISAT_OK;
}

int misat_route(misat_ctx* c, const misat_batch* b, misat_decisions* out) {
  if (!c || !b || !out) return MISAT_ERR_INVALID_ARG;
  const int32_t n = b->n;
  if (n < 0 || b->n_tokens < 0) return MISAT_ERR_INVALID_ARG;
  if (n > c->max_batch || b->n_tokens > c->max_tokens) return MISAT_ERR_BATCH_TOO_LARGE;
  if (n > 0 && (!b->cls || !b->session || !b->tok_off || !out->inst || !out->reason || !out->hit_blocks))
    return MISAT_ERR_INVALID_ARG;
  if (b->n_tokens > 0 && (!b->tokens || ((uintptr_t)b->tokens & 15) != 0)) return MISAT_ERR_INVALID_ARG;
  cudaStream_t st = c->stream;
  c->routed = false;
  estimate_classes(c);
  c->last_n = n;
  c->last_ntok = b->n_tokens;
  c->grp_log2 = (uint32_t)std::max(1, ceil_log2(2 * (uint64_t)std::max(n, 1)));  // as enqueue_route
  RouteParams prm{};
  for (int i = 0; i < 3; ++i) {
    prm.v[i] = c->kbar_b[i];
    prm.v[3 + i] = c->T_b[i];
    prm.v[6 + i] = (int64_t)c->rho[i];
  }
  launch_route_params(prm, c->d_params, st);
  CK(cudaGetLastError());
  if (n == 0) {
    // the caps of an empty batch are still defined (no candidate sessions)
    CK(cudaMemsetAsync(c->d_meta + c->ml.stats, 0, 32 * 8, st));
    CK(cudaMemsetAsync(c->d_meta + c->ml.U, 0, c->W * 8, st));
    CK(cudaMemsetAsync(c->d_meta + c->ml.cand, 0, 5 * 8, st));
    launch_caps(caps_args(c), st);
    CK(cudaGetLastError());
    CK(enqueue_meta(c));
    c->routed = true;
    return MISAT_OK;
  }
  // the device work of a route depends on the batch only through these values: it is
  // replayed as one CUDA graph while they repeat
  const std::vector<uint64_t> key{(uint64_t)n,
                                  (uint64_t)b->n_tokens,
                                  reinterpret_cast<uint64_t>(b->cls),
                                  reinterpret_cast<uint64_t>(b->session),
                                  reinterpret_cast<uint64_t>(b->tok_off),
                                  reinterpret_cast<uint64_t>(b->tokens),
                                  reinterpret_cast<uint64_t>(b->out_H),
                                  reinterpret_cast<uint64_t>(out->inst),
                                  reinterpret_cast<uint64_t>(out->reason),
                                  reinterpret_cast<uint64_t>(out->hit_blocks),
                                  reinterpret_cast<uint64_t>(c->sess.slots),
                                  (uint64_t)c->sess.log2n,
                                  reinterpret_cast<uint64_t>(c->gix.keys),
                                  reinterpret_cast<uint64_t>(c->gix.masks),
                                  (uint64_t)c->gix.log2nb,
                                  (uint64_t)(c->bk_small && c->tc_small)};
  if (c->timing) {
    // phase events bracket the kernels directly (events recorded inside a graph do not time)
    enqueue_route(c, b, out, st);
    CK(cudaGetLastError());
  } else {
    const int rc = run_graph(c, c->g_route, key, [&](cudaStream_t s) { enqueue_route(c, b, out, s); });
    if (rc) return rc;
  }
  CK(enqueue_meta(c));
  c->routed = true;
  return MISAT_OK;
}

int misat_route_host(misat_ctx* c, const misat_batch* hb, misat_decisions* ho) {
  if (!c || !hb || !ho || hb->out_H) return MISAT_ERR_INVALID_ARG;
  const int32_t n = hb->n;
  if (n < 0 || hb->n_tokens < 0) return MISAT_ERR_INVALID_ARG;
  if (n > c->max_batch || hb->n_tokens > c->max_tokens) return MISAT_ERR_BATCH_TOO_LARGE;
  if (n > 0 && (!hb->cls || !hb->session || !hb->tok_off || !ho->inst || !ho->reason || !ho->hit_blocks))
    return MISAT_ERR_INVALID_ARG;
  if (hb->n_tokens > 0 && !hb->tokens) return MISAT_ERR_INVALID_ARG;
  cudaStream_t st = c->stream;
  if (n > 0) {
    CK(cudaMemcpyAsync(c->d_stage_off, hb->tok_off, (size_t)(n + 1) * 8, cudaMemcpyHostToDevice, st));
    CK(cudaMemcpyAsync(c->d_stage_cls, hb->cls, (size_t)n, cudaMemcpyHostToDevice, st));
    CK(cudaMemcpyAsync(c->d_stage_ses, hb->session, (size_t)n * 8, cudaMemcpyHostToDevice, st));
    if (hb->n_tokens > 0)
      CK(cudaMemcpyAsync(c->d_stage_tok, hb->tokens, (size_t)hb->n_tokens * 4, cudaMemcpyHostToDevice, st));
  }
  misat_batch db = *hb;
  db.cls = c->d_stage_cls;
  db.session = c->d_stage_ses;
  db.tok_off = c->d_stage_off;
  db.tokens = c->d_stage_tok;
  db.group = nullptr;
  db.out_H = nullptr;
  misat_decisions dd{c->d_out_inst, c->d_out_reason, c->d_out_hit};
  int rc = misat_route(c, &db, &dd);
  if (rc) return rc;
  if (n > 0) {
    CK(cudaMemcpyAsync(ho->inst, c->d_out_inst, (size_t)n * 4, cudaMemcpyDeviceToHost, st));
    CK(cudaMemcpyAsync(ho->reason, c->d_out_reason, (size_t)n, cudaMemcpyDeviceToHost, st));
    CK(cudaMemcpyAsync(ho->hit_blocks, c->d_out_hit, (size_t)n * 4, cudaMemcpyDeviceToHost, st));
  }
  CK(cudaStreamSynchronize(st));
  return MISAT_OK;
}

namespace {

// The staging slots of the pipelined host path, their events and the copy stream.
int ensure_staging(misat_ctx* c) {
  if (c->copy_stream) return MISAT_OK;
  const size_t NB = (size_t)c->max_batch;
  for (auto& sl : c->slot) {
    int rc;
    if ((!sl.tok && (rc = dalloc_n(c, &sl.tok, (size_t)c->max_tokens + 8))) ||
        (!sl.off && (rc = dalloc_n(c, &sl.off, NB + 1))) || (!sl.cls && (rc = dalloc_n(c, &sl.cls, NB))) ||
        (!sl.ses && (rc = dalloc_n(c, &sl.ses, NB))))
      return rc;
    if (!sl.ev_copied) CK(cudaEventCreateWithFlags(&sl.ev_copied, cudaEventDisableTiming));
    if (!sl.ev_free) CK(cudaEventCreateWithFlags(&sl.ev_free, cudaEventDisableTiming));
  }
  CK(cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking));
  return MISAT_OK;
}

}  // namespace

int misat_stage_host(misat_ctx* c, const misat_batch* hb, int32_t slot) {
  if (!c || !hb || hb->out_H || slot < 0 || slot > 1) return MISAT_ERR_INVALID_ARG;
  const int32_t n = hb->n;
  if (n < 0 || hb->n_tokens < 0) return MISAT_ERR_INVALID_ARG;
  if (n > c->max_batch || hb->n_tokens > c->max_tokens) return MISAT_ERR_BATCH_TOO_LARGE;
  if (n > 0 && (!hb->cls || !hb->session || !hb->tok_off)) return MISAT_ERR_INVALID_ARG;
  if (hb->n_tokens > 0 && !hb->tokens) return MISAT_ERR_INVALID_ARG;
  misat_ctx::StageSlot& sl = c->slot[slot];
  if (sl.staged) return MISAT_ERR_STATE;  // staged and not yet routed
  int rc = ensure_staging(c);
  if (rc) return rc;
  cudaStream_t cs = c->copy_stream;
  // the slot's buffers are overwritten only after the route that last read them
  CK(cudaStreamWaitEvent(cs, sl.ev_free, 0));
  if (n > 0) {
    CK(cudaMemcpyAsync(sl.off, hb->tok_off, (size_t)(n + 1) * 8, cudaMemcpyHostToDevice, cs));
    CK(cudaMemcpyAsync(sl.cls, hb->cls, (size_t)n, cudaMemcpyHostToDevice, cs));
    CK(cudaMemcpyAsync(sl.ses, hb->session, (size_t)n * 8, cudaMemcpyHostToDevice, cs));
    if (hb->n_tokens > 0)
      CK(cudaMemcpyAsync(sl.tok, hb->tokens, (size_t)hb->n_tokens * 4, cudaMemcpyHostToDevice, cs));
  }
  CK(cudaEventRecord(sl.ev_copied, cs));
  sl.n = n;
  sl.n_tokens = hb->n_tokens;
  sl.staged = true;
  return MISAT_OK;
}

namespace {

// Device and pinned host buffers of the delta-encoded staging path (first use).
int ensure_delta_staging(misat_ctx* c) {
  const size_t NB = (size_t)c->max_batch;
  for (auto& sl : c->slot) {
    int rc;
    if ((!sl.dbase && (rc = dalloc_n(c, &sl.dbase, NB))) || (!sl.doff && (rc = dalloc_n(c, &sl.doff, NB + 1))) ||
        (!sl.dtok && (rc = dalloc_n(c, &sl.dtok, (size_t)c->max_tokens + 8))))
      return rc;
    if (!sl.h_off) {
      if (cudaMallocHost(&sl.h_off, (NB + 1) * sizeof(int64_t)) != cudaSuccess) {
        cudaGetLastError();
        sl.h_off = nullptr;
        return MISAT_ERR_OOM;
      }
    }
  }
  return MISAT_OK;
}

}  // namespace

int misat_stage_host_delta(misat_ctx* c, const misat_batch_delta* hb, int32_t slot) {
  if (!c || !hb || slot < 0 || slot > 1) return MISAT_ERR_INVALID_ARG;
  const int32_t n = hb->n;
  if (n < 0) return MISAT_ERR_INVALID_ARG;
  if (n > c->max_batch) return MISAT_ERR_BATCH_TOO_LARGE;
  if (n > 0 && (!hb->cls || !hb->session || !hb->base || !hb->delta_off)) return MISAT_ERR_INVALID_ARG;
  misat_ctx::StageSlot& sl = c->slot[slot];
  if (sl.staged) return MISAT_ERR_STATE;
  const int64_t nd = n > 0 ? hb->delta_off[n] : 0;
  if (n > 0 && hb->delta_off[0] != 0) return MISAT_ERR_INVALID_ARG;
  if (nd < 0 || nd > c->max_tokens) return MISAT_ERR_BATCH_TOO_LARGE;
  if (nd > 0 && !hb->delta_tokens) return MISAT_ERR_INVALID_ARG;
  int rc = ensure_staging(c);
  if (rc) return rc;
  if ((rc = ensure_delta_staging(c))) return rc;
  // full lengths and offsets: prompt(r) = prompt(base[r]) ++ delta(r), written to the slot's
  // pinned buffer once the copy of the slot's previous batch has read it
  CK(cudaEventSynchronize(sl.ev_copied));
  c->delta_len.resize((size_t)n);
  c->delta_depth.resize((size_t)n);
  int64_t* off = sl.h_off;
  off[0] = 0;
  for (int32_t r = 0; r < n; ++r) {
    const int32_t b = hb->base[r];
    const int64_t d = hb->delta_off[r + 1] - hb->delta_off[r];
    if (b < -1 || b >= r || d < 0) return MISAT_ERR_INVALID_ARG;
    const int64_t L = (b >= 0 ? c->delta_len[b] : 0) + d;
    const int depth = (b >= 0 ? c->delta_depth[b] : 0) + 1;
    if (depth > MISAT_DELTA_MAX_DEPTH || L >= ((int64_t)1 << 20)) return MISAT_ERR_INVALID_ARG;
    c->delta_len[r] = L;
    c->delta_depth[r] = (uint8_t)depth;
    off[r + 1] = off[r] + L;
    if (off[r + 1] > c->max_tokens) return MISAT_ERR_BATCH_TOO_LARGE;
  }
  cudaStream_t cs = c->copy_stream;
  CK(cudaStreamWaitEvent(cs, sl.ev_free, 0));
  if (n > 0) {
    CK(cudaMemcpyAsync(sl.off, off, (size_t)(n + 1) * 8, cudaMemcpyHostToDevice, cs));
    CK(cudaMemcpyAsync(sl.cls, hb->cls, (size_t)n, cudaMemcpyHostToDevice, cs));
    CK(cudaMemcpyAsync(sl.ses, hb->session, (size_t)n * 8, cudaMemcpyHostToDevice, cs));
    CK(cudaMemcpyAsync(sl.dbase, hb->base, (size_t)n * 4, cudaMemcpyHostToDevice, cs));
    CK(cudaMemcpyAsync(sl.doff, hb->delta_off, (size_t)(n + 1) * 8, cudaMemcpyHostToDevice, cs));
    if (nd > 0) CK(cudaMemcpyAsync(sl.dtok, hb->delta_tokens, (size_t)nd * 4, cudaMemcpyHostToDevice, cs));
    DeltaArgs da{n, sl.dbase, sl.doff, sl.dtok, sl.off, sl.tok};
    launch_delta_expand(da, c->num_sms, cs);
    CK(cudaGetLastError());
  }
  CK(cudaEventRecord(sl.ev_copied, cs));
  sl.n = n;
  sl.n_tokens = n > 0 ? off[n] : 0;
  sl.staged = true;
  return MISAT_OK;
}

int misat_route_staged(misat_ctx* c, int32_t slot, misat_decisions* ho) {
  if (!c || !ho || slot < 0 || slot > 1) return MISAT_ERR_INVALID_ARG;
  misat_ctx::StageSlot& sl = c->slot[slot];
  if (!sl.staged) return MISAT_ERR_STATE;
  const int32_t n = sl.n;
  if (n > 0 && (!ho->inst || !ho->reason || !ho->hit_blocks)) return MISAT_ERR_INVALID_ARG;
  cudaStream_t st = c->stream;
  CK(cudaStreamWaitEvent(st, sl.ev_copied, 0));
  misat_batch db{};
  db.n = n;
  db.n_tokens = sl.n_tokens;
  db.cls = sl.cls;
  db.session = sl.ses;
  db.group = nullptr;
  db.tok_off = sl.off;
  db.tokens = sl.tok;
  db.out_H = nullptr;
  misat_decisions dd{c->d_out_inst, c->d_out_reason, c->d_out_hit};
  const int rc = misat_route(c, &db, &dd);
  // the slot is free again once the work enqueued so far has run (also after a failed route)
  sl.staged = false;
  CK(cudaEventRecord(sl.ev_free, st));
  if (rc) return rc;
  if (n > 0) {
    CK(cudaMemcpyAsync(ho->inst, c->d_out_inst, (size_t)n * 4, cudaMemcpyDeviceToHost, st));
    CK(cudaMemcpyAsync(ho->reason, c->d_out_reason, (size_t)n, cudaMemcpyDeviceToHost, st));
    CK(cudaMemcpyAsync(ho->hit_blocks, c->d_out_hit, (size_t)n * 4, cudaMemcpyDeviceToHost, st));
  }
  CK(cudaStreamSynchronize(st));
  return MISAT_OK;
}

int misat_commit(misat_ctx* c) {
  if (!c) return MISAT_ERR_INVALID_ARG;
  if (!c->routed) return MISAT_ERR_STATE;
  cudaStream_t st = c->stream;
  CK(cudaEventSynchronize(c->ev_meta));
  if (c->h_err()) return c->h_err();
  c->routed = false;
  const int n = c->last_n;
  if (n > 0) {
    std::vector<int64_t> sizes(c->W), add(c->W);
    for (int w = 0; w < c->W; ++w) {
      sizes[w] = c->h_size(w);
      add[w] = c->h_U(w);
    }
    int rc = ensure_capacity(c, sizes, add);
    if (rc) return rc;
    int64_t add_all = 0;
    for (int64_t x : add) add_all += x;
    if ((rc = gix_ensure(c, sizes, add_all))) return rc;
    rc = maybe_rebuild_sessions(c, n);
    if (rc) return rc;
  }
  CK(cudaMemsetAsync(c->stats_ptr() + 18, 0, 2 * 8, st));
  CK(cudaMemsetAsync(c->stats_ptr() + 24, 0, 8, st));
  c->mark(8);
  if (n > 0) {
    InsertArgs ia{};
    ia.desc = c->d_desc;
    ia.n_inst = c->W;
    ia.n = n;
    ia.units = c->d_units;
    ia.n_units = c->d_units_n;
    ia.units_cap = c->units_cap;
    ia.nb = c->rq.nb;
    ia.kbase = c->rq.kbase;
    ia.inst = c->rq.inst;
    ia.keys = c->d_keys;
    ia.seq = c->seq + 1;
    ia.size = c->size_ptr();
    ia.new_keys = c->stats_ptr() + 18;
    ia.err = c->err_ptr();
    ia.gix = gix_or_null(c);
    ia.gnew = c->d_gnew;
    ia.n_gnew = c->d_gnew_n;
    ia.gnew_cap = c->keys_cap;
    ia.grp = c->d_grp;
    ia.grp_log2 = c->grp_log2;
    ia.skip = c->d_skip;
    ia.ops = c->stats_ptr() + 24;
    launch_insert_tables(ia, c->num_sms, st);
    c->mark(9);
    cudaEvent_t join = nullptr;
    if (ia.gix.keys) {
      if (c->side_stream && !c->timing) {
        CK(cudaEventRecord(c->ev_fork, st));
        CK(cudaStreamWaitEvent(c->side_stream, c->ev_fork, 0));
        launch_insert_gix(ia, c->num_sms * 4, c->side_stream);
        CK(cudaEventRecord(c->ev_join, c->side_stream));
        join = c->ev_join;
      } else {
        launch_insert_gix(ia, c->num_sms * 8, st);
      }
    }
    c->mark(10);
    SessUpdateArgs sa{n, c->rq, c->sess, c->d_prot, c->err_ptr()};
    launch_session_update(sa, st);
    c->mark(11);
    int rc = evict_all(c, c->stats_ptr() + 19, join);
    if (rc) return rc;
  } else {
    for (int i = 9; i <= 16; ++i) c->mark(i);
  }
  CK(cudaGetLastError());
  CK(enqueue_meta(c));
  c->seq += 1;
  return MISAT_OK;
}

int misat_complete(misat_ctx* c, int32_t n, const uint64_t* session, const uint8_t* cls, const int32_t* total_blocks,
                   const int64_t* residency_us, const uint8_t* done) {
  if (!c || n < 0) return MISAT_ERR_INVALID_ARG;
  if (n == 0) return MISAT_OK;
  if (!session || !cls || !total_blocks || !residency_us || !done) return MISAT_ERR_INVALID_ARG;
  {
    // distinct sessions: open addressing in one flat table (session ids are nonzero)
    const int lg = ceil_log2(2 * (uint64_t)n);
    const uint64_t mask = ((uint64_t)1 << lg) - 1;
    std::vector<uint64_t> seen(mask + 1, 0);
    for (int i = 0; i < n; ++i) {
      if (cls[i] > 2 || total_blocks[i] < 0 || residency_us[i] < 0 || session[i] == 0) return MISAT_ERR_INVALID_ARG;
      uint64_t h = session[i] * kGold;
      h = (h ^ (h >> 29)) & mask;
      while (seen[h] != 0) {
        if (seen[h] == session[i]) return MISAT_ERR_INVALID_ARG;
        h = (h + 1) & mask;
      }
      seen[h] = session[i];
    }
  }
  for (int i = 0; i < n; ++i) {
    if (!done[i]) continue;
    const int b = cls[i];
    c->hist_blocks[b].push_back(total_blocks[i]);
    c->hist_res[b].push_back(residency_us[i]);
    while ((int32_t)c->hist_blocks[b].size() > c->hist_window) c->hist_blocks[b].pop_front();
    while ((int32_t)c->hist_res[b].size() > c->hist_window) c->hist_res[b].pop_front();
  }
  // device part: sessions and done flags, in chunks of max_batch, through one of two pinned
  // host copies (reused once the kernel that last read it has run); nothing here waits for
  // the stream
  cudaStream_t st = c->stream;
  for (int off = 0; off < n; off += c->max_batch) {
    const int m = std::min(c->max_batch, n - off);
    misat_ctx::CompBuf& cb = c->comp[c->comp_turn];
    c->comp_turn ^= 1;
    if (!cb.ev) {
      // first use: mapped pinned buffers and their event; on any failure nothing is kept
      const bool ok =
          cudaHostAlloc(&cb.h_ses, (size_t)c->max_batch * 8, cudaHostAllocMapped) == cudaSuccess &&
          cudaHostAlloc(&cb.h_done, (size_t)c->max_batch, cudaHostAllocMapped) == cudaSuccess &&
          cudaHostGetDevicePointer(reinterpret_cast<void**>(&cb.d_ses), cb.h_ses, 0) == cudaSuccess &&
          cudaHostGetDevicePointer(reinterpret_cast<void**>(&cb.d_done), cb.h_done, 0) == cudaSuccess &&
          cudaEventCreateWithFlags(&cb.ev, cudaEventDisableTiming) == cudaSuccess;
      if (!ok) {
        cudaGetLastError();
        if (cb.h_ses) cudaFreeHost(cb.h_ses);
        if (cb.h_done) cudaFreeHost(cb.h_done);
        if (cb.ev) cudaEventDestroy(cb.ev);
        cb = misat_ctx::CompBuf{};
        return MISAT_ERR_OOM;
      }
    } else {
      CK(cudaEventSynchronize(cb.ev));
    }
    std::memcpy(cb.h_ses, session + off, (size_t)m * 8);
    std::memcpy(cb.h_done, done + off, (size_t)m);
    // the kernel reads the pinned copy over the host link: no copy-engine transfer, so the
    // update does not queue behind a staged batch's copy
    CompleteArgs a{m, cb.d_ses, cb.d_done, c->sess, c->d_prot};
    launch_complete(a, st);
    CK(cudaGetLastError());
    CK(cudaEventRecord(cb.ev, st));
  }
  return MISAT_OK;
}

int misat_reset_instance(misat_ctx* c, int32_t w) {
  if (!c || w < 0 || w >= c->W) return MISAT_ERR_INVALID_ARG;
  if (c->use_gix) {
    launch_gix_clear_table(c->h_desc[w], w, c->gix, c->err_ptr(), c->stream);
    CK(cudaGetLastError());
  }
  CK(cudaMemsetAsync(c->h_desc[w].tab, 0, ((size_t)1 << c->h_desc[w].log2nb) * sizeof(Bucket), c->stream));
  CK(cudaMemsetAsync(c->size_ptr() + w, 0, 8, c->stream));
  return MISAT_OK;
}

int misat_evict(misat_ctx* c, int32_t w, const uint64_t* keys, int64_t n) {
  if (!c || w < 0 || w >= c->W || n < 0 || (n > 0 && !keys)) return MISAT_ERR_INVALID_ARG;
  cudaStream_t st = c->stream;
  uint64_t* dk = nullptr;
  if (n > 0) {
    if (cudaMalloc(&dk, (size_t)n * 8) != cudaSuccess) {
      cudaGetLastError();
      return MISAT_ERR_OOM;
    }
    CK(cudaMemcpyAsync(dk, keys, (size_t)n * 8, cudaMemcpyHostToDevice, st));
  }
  CK(cudaMemcpyAsync(c->d_onew, &w, 4, cudaMemcpyHostToDevice, st));
  MarkArgs ma{c->h_desc[w], n, dk, c->size_ptr() + w, c->h_bufs[w].bitmap, c->d_active + w};
  EvictArgs ev = evict_args(c, c->stats_ptr() + 20);
  ev.only_w = c->d_onew;
  launch_mark_evict(ma, w, ev, st);
  CK(cudaGetLastError());
  CK(cudaStreamSynchronize(st));
  cudaFree(dk);
  return MISAT_OK;
}

static int load_common_evict(misat_ctx* c) {
  int rc = evict_all(c, c->stats_ptr() + 20);
  if (rc) return rc;
  CK(cudaStreamSynchronize(c->stream));
  return read_meta(c);
}

int misat_load_entries(misat_ctx* c, int32_t w, const misat_entry* entries, int64_t n) {
  if (!c || w < 0 || w >= c->W || n < 0 || (n > 0 && !entries)) return MISAT_ERR_INVALID_ARG;
  for (int64_t i = 0; i < n; ++i)
    if (entries[i].key < 2 || (entries[i].meta & 0xffff) == 0 || (entries[i].meta >> 36) >= (1ull << 28))
      return MISAT_ERR_INVALID_ARG;
  int rc = read_meta(c);
  if (rc) return rc;
  if (c->h_err()) return c->h_err();
  std::vector<int64_t> sizes(c->W), add(c->W, 0);
  for (int x = 0; x < c->W; ++x) sizes[x] = c->h_size(x);
  add[w] = n;
  if ((rc = ensure_capacity(c, sizes, add))) return rc;
  if ((rc = gix_ensure(c, sizes, n))) return rc;
  misat_entry* de = nullptr;
  if (n > 0) {
    if (cudaMalloc(&de, (size_t)n * sizeof(misat_entry)) != cudaSuccess) {
      cudaGetLastError();
      return MISAT_ERR_OOM;
    }
    CK(cudaMemcpyAsync(de, entries, (size_t)n * sizeof(misat_entry), cudaMemcpyHostToDevice, c->stream));
    EntryInsertArgs a{c->h_desc[w], n, de, c->size_ptr() + w, c->err_ptr(), w, gix_or_null(c)};
    launch_insert_entries(a, c->stream);
    CK(cudaGetLastError());
  }
  rc = load_common_evict(c);
  cudaFree(de);
  if (rc) return rc;
  return c->h_err();
}

int misat_load_chains(misat_ctx* c, int32_t n_chains, const int64_t* tok_off, const int32_t* tokens,
                      const int32_t* inst, const uint64_t* seq, const uint32_t* arr, const int32_t* max_blocks) {
  if (!c || n_chains < 0) return MISAT_ERR_INVALID_ARG;
  if (n_chains == 0) return MISAT_OK;
  if (!tok_off || !inst || !seq || !arr || !max_blocks) return MISAT_ERR_INVALID_ARG;
  if (n_chains > c->max_batch) return MISAT_ERR_BATCH_TOO_LARGE;
  if (tok_off[0] != 0) return MISAT_ERR_INVALID_ARG;
  const int64_t ntok = tok_off[n_chains];
  if (ntok > c->max_tokens) return MISAT_ERR_BATCH_TOO_LARGE;
  if (ntok > 0 && !tokens) return MISAT_ERR_INVALID_ARG;
  std::vector<int64_t> add(c->W, 0);
  for (int i = 0; i < n_chains; ++i) {
    const int64_t L = tok_off[i + 1] - tok_off[i];
    if (L < 0 || L >= (1 << 20) || inst[i] < 0 || inst[i] >= c->W || seq[i] >= (1ull << 28) ||
        arr[i] >= (1u << 20) || max_blocks[i] < 0)
      return MISAT_ERR_INVALID_ARG;
    add[inst[i]] += std::min<int64_t>(L / 16, max_blocks[i]);
  }
  if (c->routed) return MISAT_ERR_STATE;  // the staging and key buffers hold a pending route
  int rc = read_meta(c);
  if (rc) return rc;
  if (c->h_err()) return c->h_err();
  std::vector<int64_t> sizes(c->W);
  for (int x = 0; x < c->W; ++x) sizes[x] = c->h_size(x);
  if ((rc = ensure_capacity(c, sizes, add))) return rc;
  int64_t add_all = 0;
  for (int64_t x : add) add_all += x;
  if ((rc = gix_ensure(c, sizes, add_all))) return rc;
  cudaStream_t st = c->stream;
  // stage: offsets, tokens, per-chain inst / tick / limit (reuse request scratch arrays)
  CK(cudaMemcpyAsync(c->d_stage_off, tok_off, (size_t)(n_chains + 1) * 8, cudaMemcpyHostToDevice, st));
  if (ntok > 0) CK(cudaMemcpyAsync(c->d_stage_tok, tokens, (size_t)ntok * 4, cudaMemcpyHostToDevice, st));
  std::vector<int32_t> nbv(n_chains);
  std::vector<int64_t> kbv(n_chains);
  for (int i = 0; i < n_chains; ++i) {
    nbv[i] = (int32_t)((tok_off[i + 1] - tok_off[i]) >> 4);
    kbv[i] = tok_off[i] >> 4;
  }
  CK(cudaMemcpyAsync(c->rq.nb, nbv.data(), (size_t)n_chains * 4, cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->rq.kbase, kbv.data(), (size_t)n_chains * 8, cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->rq.inst, inst, (size_t)n_chains * 4, cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->rq.session, seq, (size_t)n_chains * 8, cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->d_chain_max, max_blocks, (size_t)n_chains * 4, cudaMemcpyHostToDevice, st));
  CK(cudaMemcpyAsync(c->d_out_hit, arr, (size_t)n_chains * 4, cudaMemcpyHostToDevice, st));
  CK(cudaMemsetAsync(c->work_ptr(), 0, 4, st));
  HashArgs ha{};
  ha.tok_off = c->d_stage_off;
  ha.tokens = c->d_stage_tok;
  ha.n_tokens = ntok;
  ha.n = n_chains;
  ha.seed = c->seed;
  ha.keys = c->d_keys;
  ha.keys_cap = c->keys_cap;
  ha.work = c->work_ptr();
  ha.err = c->err_ptr();
  launch_block_hash(ha, c->num_sms, st);
  InsertArgs ia{};
  ia.desc = c->d_desc;
  ia.n_inst = c->W;
  ia.n = n_chains;
  ia.units = c->d_units;
  ia.n_units = c->d_units_n;
  ia.units_cap = c->units_cap;
  ia.nb = c->rq.nb;
  ia.kbase = c->rq.kbase;
  ia.inst = c->rq.inst;
  ia.keys = c->d_keys;
  ia.meta_seq = c->rq.session;
  ia.meta_arr = reinterpret_cast<const uint32_t*>(c->d_out_hit);
  ia.max_blocks = c->d_chain_max;
  ia.size = c->size_ptr();
  ia.new_keys = c->stats_ptr() + 21;
  ia.err = c->err_ptr();
  ia.gix = gix_or_null(c);
  ia.gnew = c->d_gnew;
  ia.n_gnew = c->d_gnew_n;
  ia.gnew_cap = c->keys_cap;
  launch_insert(ia, c->num_sms, st);
  CK(cudaGetLastError());
  rc = load_common_evict(c);
  if (rc) return rc;
  return c->h_err();
}

int misat_index_size(misat_ctx* c, int32_t w, int64_t* out) {
  if (!c || !out || w < 0 || w >= c->W) return MISAT_ERR_INVALID_ARG;
  int rc = read_meta(c);
  if (rc) return rc;
  *out = c->h_size(w);
  return c->h_err();
}

int misat_index_buckets(misat_ctx* c, int32_t w, int64_t* out) {
  if (!c || !out || w < 0 || w >= c->W) return MISAT_ERR_INVALID_ARG;
  *out = (int64_t)1 << c->h_desc[w].log2nb;
  return MISAT_OK;
}

int misat_dump_index(misat_ctx* c, int32_t w, misat_entry* host_out, int64_t cap, int64_t* n_out) {
  if (!c || !n_out || w < 0 || w >= c->W || cap < 0 || (cap > 0 && !host_out)) return MISAT_ERR_INVALID_ARG;
  const size_t nb = (size_t)1 << c->h_desc[w].log2nb;
  std::vector<Bucket> hb(nb);
  CK(cudaMemcpyAsync(hb.data(), c->h_desc[w].tab, nb * sizeof(Bucket), cudaMemcpyDeviceToHost, c->stream));
  int rc = read_meta(c);
  if (rc) return rc;
  std::vector<misat_entry> v;
  for (auto& B : hb)
    for (int s = 0; s < 4; ++s)
      if (B.key[s] != kEmpty) v.push_back(misat_entry{B.key[s], B.meta[s]});
  std::sort(v.begin(), v.end(), [](const misat_entry& a, const misat_entry& b) { return a.key < b.key; });
  *n_out = (int64_t)v.size();
  if ((int64_t)v.size() > cap) return MISAT_ERR_INVALID_ARG;
  std::copy(v.begin(), v.end(), host_out);
  return c->h_err();
}

int misat_dump_keys(misat_ctx* c, uint64_t* host_out, int64_t cap, int64_t* n_out) {
  if (!c || !n_out || cap < 0 || (cap > 0 && !host_out)) return MISAT_ERR_INVALID_ARG;
  const int n = c->last_n;
  std::vector<int32_t> nb(n);
  std::vector<int64_t> kb(n);
  const int64_t slots = c->last_ntok / 16;
  std::vector<uint64_t> keys(slots);
  if (n > 0) {
    CK(cudaMemcpyAsync(nb.data(), c->rq.nb, (size_t)n * 4, cudaMemcpyDeviceToHost, c->stream));
    CK(cudaMemcpyAsync(kb.data(), c->rq.kbase, (size_t)n * 8, cudaMemcpyDeviceToHost, c->stream));
  }
  if (slots > 0) CK(cudaMemcpyAsync(keys.data(), c->d_keys, (size_t)slots * 8, cudaMemcpyDeviceToHost, c->stream));
  int rc = read_meta(c);
  if (rc) return rc;
  int64_t k = 0;
  for (int r = 0; r < n; ++r)
    for (int j = 0; j < nb[r]; ++j) {
      if (k >= cap) return MISAT_ERR_INVALID_ARG;
      host_out[k++] = keys[kb[r] + j];
    }
  *n_out = k;
  return c->h_err();
}

int misat_dump_caps(misat_ctx* c, int64_t* K_w, int64_t* K_wb, int64_t* N_wb, int64_t* kbar_w, int64_t* kbar_b,
                    int64_t* T_b) {
  if (!c) return MISAT_ERR_INVALID_ARG;
  cudaStream_t st = c->stream;
  if (K_w) CK(cudaMemcpyAsync(K_w, c->ia.K_w, c->W * 8, cudaMemcpyDeviceToHost, st));
  if (K_wb) CK(cudaMemcpyAsync(K_wb, c->ia.K_wb, c->W * 24, cudaMemcpyDeviceToHost, st));
  if (N_wb) CK(cudaMemcpyAsync(N_wb, c->ia.N_wb, c->W * 24, cudaMemcpyDeviceToHost, st));
  if (kbar_w) CK(cudaMemcpyAsync(kbar_w, c->ia.kbar_w, c->W * 8, cudaMemcpyDeviceToHost, st));
  CK(cudaStreamSynchronize(st));
  for (int b = 0; b < 3; ++b) {
    if (kbar_b) kbar_b[b] = c->kbar_b[b];
    if (T_b) T_b[b] = c->T_b[b];
  }
  return MISAT_OK;
}

int misat_dump_counts(misat_ctx* c, int32_t* prot) {
  if (!c || !prot) return MISAT_ERR_INVALID_ARG;
  CK(cudaMemcpyAsync(prot, c->d_prot, c->W * 12, cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  return MISAT_OK;
}

int misat_dump_sessions(misat_ctx* c, uint64_t* ids, int32_t* state, int32_t* inst, int32_t* cls, int64_t cap,
                        int64_t* n_out) {
  if (!c || !n_out || cap < 0) return MISAT_ERR_INVALID_ARG;
  const size_t N = (size_t)1 << c->sess.log2n;
  std::vector<SessSlot> hs(N);
  CK(cudaMemcpyAsync(hs.data(), c->sess.slots, N * sizeof(SessSlot), cudaMemcpyDeviceToHost, c->stream));
  CK(cudaStreamSynchronize(c->stream));
  std::vector<SessSlot> v;
  for (auto& s : hs)
    if (s.key && (sess_state(s.val) == kSessProtected || sess_state(s.val) == kSessReleased)) v.push_back(s);
  std::sort(v.begin(), v.end(), [](const SessSlot& a, const SessSlot& b) { return a.key < b.key; });
  *n_out = (int64_t)v.size();
  if ((int64_t)v.size() > cap) return MISAT_ERR_INVALID_ARG;
  for (size_t i = 0; i < v.size(); ++i) {
    if (ids) ids[i] = v[i].key;
    if (state) state[i] = (int32_t)sess_state(v[i].val);
    if (inst) inst[i] = (int32_t)sess_inst(v[i].val);
    if (cls) cls[i] = (int32_t)sess_cls(v[i].val);
  }
  return MISAT_OK;
}

int misat_stats(misat_ctx* c, misat_batch_stats* o) {
  if (!c || !o) return MISAT_ERR_INVALID_ARG;
  int rc = read_meta(c);
  if (rc) return rc;
  const unsigned long long* s = c->h_meta + c->ml.stats;
  std::memset(o, 0, sizeof(*o));
  o->n_requests = c->last_n;
  for (int i = 0; i < 8; ++i) o->by_reason[i] = (int64_t)s[i];
  for (int b = 0; b < 3; ++b) {
    o->admitted_by_class[b] = (int64_t)s[8 + b];
    o->held_by_class[b] = (int64_t)s[11 + b];
    o->n_admitted += (int64_t)s[8 + b];
    o->n_held += (int64_t)s[11 + b];
  }
  o->hit_tokens = (int64_t)s[14];
  o->query_tokens = (int64_t)s[15];
  o->probes = (int64_t)(s[16] + s[22]);
  o->bucket_reads = (int64_t)(s[17] + s[23]);
  o->probes_first = (int64_t)s[16];
  o->bucket_reads_first = (int64_t)s[17];
  o->new_keys = (int64_t)s[18];
  o->evicted = (int64_t)s[19];
  o->seq = (int64_t)c->seq;
  o->insert_ops = (int64_t)s[24];
  o->joint_selection = (int64_t)s[25];
  o->first_block_keys = (int64_t)s[26];
  o->first_block_lookups = (int64_t)s[27];
  // D_TV (Sec. 3.3) of the admitted class mix against rho, in ppm
  const int64_t A = o->n_admitted;
  if (A > 0) {
    __int128 acc = 0;
    for (int b = 0; b < 3; ++b) {
      const __int128 d = (__int128)1000000 * o->admitted_by_class[b] - (__int128)c->rho[b] * A;
      acc += d < 0 ? -d : d;
    }
    o->dtv_ppm = (int64_t)(acc / (2 * (__int128)A));
  } else {
    o->dtv_ppm = -1;
  }
  return c->h_err();
}

int misat_global_info(misat_ctx* c, int32_t* mask_words, int64_t* slots, int64_t* claimed) {
  if (!c) return MISAT_ERR_INVALID_ARG;
  if (!c->use_gix) return MISAT_ERR_STATE;
  int rc = read_meta(c);
  if (rc) return rc;
  if (mask_words) *mask_words = (int32_t)c->gix.mw;
  if (slots) *slots = (int64_t)gix_slots(c);
  if (claimed) *claimed = (int64_t)c->h_meta[c->ml.g_used];
  return c->h_err();
}

int misat_global_dump(misat_ctx* c, uint64_t* keys, uint64_t* masks, int64_t cap, int64_t* n_out) {
  if (!c || cap < 0 || !n_out || (cap > 0 && (!keys || !masks))) return MISAT_ERR_INVALID_ARG;
  if (!c->use_gix) return MISAT_ERR_STATE;
  const size_t slots = gix_slots(c), mw = c->gix.mw;
  std::vector<unsigned long long> hk(slots), hm(slots * mw);
  CK(cudaMemcpyAsync(hk.data(), c->gix.keys, slots * 8, cudaMemcpyDeviceToHost, c->stream));
  CK(cudaMemcpyAsync(hm.data(), c->gix.masks, slots * mw * 8, cudaMemcpyDeviceToHost, c->stream));
  int rc = read_meta(c);
  if (rc) return rc;
  int64_t n = 0;
  for (size_t i = 0; i < slots; ++i) {
    if (hk[i] == kEmpty) continue;
    bool any = false;
    for (size_t j = 0; j < mw; ++j) any |= hm[i * mw + j] != 0;
    if (!any) continue;
    if (n < cap) {
      keys[n] = hk[i];
      for (size_t j = 0; j < mw; ++j) masks[n * mw + j] = hm[i * mw + j];
    }
    ++n;
  }
  *n_out = n;
  return c->h_err();
}

int misat_global_rebuild(misat_ctx* c) {
  if (!c) return MISAT_ERR_INVALID_ARG;
  if (!c->use_gix) return MISAT_ERR_STATE;
  int rc = read_meta(c);
  if (rc) return rc;
  if (c->h_err()) return c->h_err();
  int64_t live = 0;
  for (int w = 0; w < c->W; ++w) live += c->h_size(w);
  return gix_rebuild(c, live);
}

int misat_set_timing(misat_ctx* c, int enable) {
  if (!c) return MISAT_ERR_INVALID_ARG;
  if (enable && !c->ev[0])
    for (auto& e : c->ev) CK(cudaEventCreate(&e));
  c->timing = enable != 0;
  return MISAT_OK;
}

int misat_phase_times(misat_ctx* c, float* ms) {
  if (!c || !ms) return MISAT_ERR_INVALID_ARG;
  if (!c->timing) return MISAT_ERR_STATE;
  CK(cudaStreamSynchronize(c->stream));
  // route phases: consecutive events 0..7; commit: 8 start, 9 tables inserted, 10 global index,
  // 11 sessions, 12..16 after each eviction kernel
  const int from[MISAT_N_PHASES] = {0, 1, 2, 3, 4, 5, 6, 8, 10, 11, 9, 11, 12, 13, 14, 15};
  const int to[MISAT_N_PHASES] = {1, 2, 3, 4, 5, 6, 7, 9, 11, 16, 10, 12, 13, 14, 15, 16};
  for (int i = 0; i < MISAT_N_PHASES; ++i) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, c->ev[from[i]], c->ev[to[i]]) != cudaSuccess) {
      cudaGetLastError();
      t = 0.f;  // phase not recorded (e.g. empty batch)
    }
    ms[i] = t;
  }
  return MISAT_OK;
}

}  // extern "C"

// ---- checkpoint / resume ----
struct misat_checkpoint {
  int W = 0;
  std::vector<InstDesc> desc;  // saved tables (device copies) with their geometry
  std::vector<int64_t> size;
  SessSlot* sess = nullptr;
  uint32_t sess_log2 = 0;
  uint64_t sess_used = 0;
  int32_t* prot = nullptr;
  int64_t* backlog = nullptr;
  int64_t* tokcost = nullptr;
  int32_t* contraction = nullptr;
  std::deque<int64_t> hist_blocks[3], hist_res[3];
  uint32_t rho[3] = {0, 0, 0};
  uint64_t seq = 0;
  // global prefix index copy (NULL when the context has none)
  unsigned long long* gkeys = nullptr;
  unsigned long long* gmasks = nullptr;
  uint32_t g_log2 = 0;
  uint64_t g_used = 0;
  // device copy of the counters restored with the state: [W] sizes, sessions used, global
  // slots claimed (restored device to device: a host-to-device copy on the context's stream
  // would queue behind a staged batch copy in flight on the copy engine)
  unsigned long long* counters = nullptr;
};

extern "C" {

int misat_checkpoint_free(misat_checkpoint* k) {
  if (!k) return MISAT_ERR_INVALID_ARG;
  for (auto& d : k->desc) cudaFree(d.tab);
  cudaFree(k->sess);
  cudaFree(k->prot);
  cudaFree(k->backlog);
  cudaFree(k->tokcost);
  cudaFree(k->contraction);
  cudaFree(k->gkeys);
  cudaFree(k->gmasks);
  cudaFree(k->counters);
  delete k;
  return MISAT_OK;
}

int misat_checkpoint_save(misat_ctx* c, misat_checkpoint** out) {
  if (!c || !out) return MISAT_ERR_INVALID_ARG;
  *out = nullptr;
  int rc = read_meta(c);
  if (rc) return rc;
  if (c->h_err()) return c->h_err();
  misat_checkpoint* k = new (std::nothrow) misat_checkpoint();
  if (!k) return MISAT_ERR_OOM;
  cudaStream_t st = c->stream;
  k->W = c->W;
  k->desc = c->h_desc;
  for (auto& d : k->desc) d.tab = nullptr;
  bool oom = false;
  for (int w = 0; w < c->W && !oom; ++w) {
    const size_t bytes = ((size_t)1 << c->h_desc[w].log2nb) * sizeof(Bucket);
    if (cudaMalloc(&k->desc[w].tab, bytes) != cudaSuccess) {
      oom = true;
      break;
    }
    if (cudaMemcpyAsync(k->desc[w].tab, c->h_desc[w].tab, bytes, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
      oom = true;
  }
  const size_t sbytes = ((size_t)1 << c->sess.log2n) * sizeof(SessSlot);
  if (!oom && (cudaMalloc(&k->sess, sbytes) != cudaSuccess || cudaMalloc(&k->prot, c->W * 12) != cudaSuccess ||
               cudaMalloc(&k->backlog, c->W * 8) != cudaSuccess || cudaMalloc(&k->tokcost, c->W * 8) != cudaSuccess ||
               cudaMalloc(&k->contraction, c->W * 4) != cudaSuccess ||
               cudaMalloc(&k->counters, (c->W + 2) * 8) != cudaSuccess))
    oom = true;
  if (!oom && c->use_gix &&
      (cudaMalloc(&k->gkeys, gix_slots(c) * 8) != cudaSuccess ||
       cudaMalloc(&k->gmasks, gix_slots(c) * c->gix.mw * 8) != cudaSuccess))
    oom = true;
  if (oom) {
    cudaGetLastError();
    misat_checkpoint_free(k);
    return MISAT_ERR_OOM;
  }
  CK(cudaMemcpyAsync(k->sess, c->sess.slots, sbytes, cudaMemcpyDeviceToDevice, st));
  CK(cudaMemcpyAsync(k->prot, c->d_prot, c->W * 12, cudaMemcpyDeviceToDevice, st));
  CK(cudaMemcpyAsync(k->backlog, c->d_backlog, c->W * 8, cudaMemcpyDeviceToDevice, st));
  CK(cudaMemcpyAsync(k->tokcost, c->d_tokcost, c->W * 8, cudaMemcpyDeviceToDevice, st));
  CK(cudaMemcpyAsync(k->contraction, c->d_contraction, c->W * 4, cudaMemcpyDeviceToDevice, st));
  CK(cudaMemcpyAsync(k->counters, c->d_meta + c->ml.size, (c->W + 1) * 8, cudaMemcpyDeviceToDevice, st));
  CK(cudaMemcpyAsync(k->counters + c->W + 1, c->d_meta + c->ml.g_used, 8, cudaMemcpyDeviceToDevice, st));
  if (c->use_gix) {
    CK(cudaMemcpyAsync(k->gkeys, c->gix.keys, gix_slots(c) * 8, cudaMemcpyDeviceToDevice, st));
    CK(cudaMemcpyAsync(k->gmasks, c->gix.masks, gix_slots(c) * c->gix.mw * 8, cudaMemcpyDeviceToDevice, st));
    k->g_log2 = c->gix.log2nb;
    k->g_used = c->h_meta[c->ml.g_used];
  }
  CK(cudaStreamSynchronize(st));
  k->sess_log2 = c->sess.log2n;
  k->sess_used = c->h_meta[c->ml.sess_used];
  k->size.resize(c->W);
  for (int w = 0; w < c->W; ++w) k->size[w] = c->h_size(w);
  for (int b = 0; b < 3; ++b) {
    k->hist_blocks[b] = c->hist_blocks[b];
    k->hist_res[b] = c->hist_res[b];
    k->rho[b] = c->rho[b];
  }
  k->seq = c->seq;
  *out = k;
  return MISAT_OK;
}

namespace {

// Device-to-device copies of a restore, gathered into copy lists and run by one kernel per
// list (the SMs, not a copy engine, move the bytes).
struct RestoreCopies {
  misat_ctx* c;
  cudaStream_t st;
  CopyList* l;
  int add(void* dst, const void* src, uint64_t bytes) {
    if (bytes == 0) return MISAT_OK;
    if (l->n == kMaxCopies) {
      const int rc = flush();
      if (rc) return rc;
    }
    const uintptr_t a = reinterpret_cast<uintptr_t>(dst) | reinterpret_cast<uintptr_t>(src);
    const uint32_t lg = (a & 15) == 0 ? 4 : (a & 7) == 0 ? 3 : (a & 3) == 0 ? 2 : 0;
    CopyItem& it = l->item[l->n++];
    it.dst = dst;
    it.src = src;
    it.bytes = bytes;
    it.start = l->units;
    it.lg = lg;
    it.pad = 0;
    l->units += (bytes + (1ull << lg) - 1) >> lg;
    return MISAT_OK;
  }
  int flush() {
    launch_copy_list(*l, c->num_sms, st);
    CK(cudaGetLastError());
    l->n = 0;
    l->units = 0;
    return MISAT_OK;
  }
};

}  // namespace

int misat_checkpoint_restore(misat_ctx* c, const misat_checkpoint* k) {
  if (!c || !k || k->W != c->W) return MISAT_ERR_INVALID_ARG;
  cudaStream_t st = c->stream;
  // the counters block is mirrored in pinned host memory: let pending copies land first
  CK(cudaStreamSynchronize(st));
  std::unique_ptr<CopyList> list(new (std::nothrow) CopyList());
  if (!list) return MISAT_ERR_OOM;
  RestoreCopies cp{c, st, list.get()};
  int crc = MISAT_OK;
#define ADD_COPY(dst, src, bytes)                 \
  do {                                            \
    if ((crc = cp.add((dst), (src), (bytes)))) return crc; \
  } while (0)
  for (int w = 0; w < c->W; ++w) {
    if (c->h_desc[w].log2nb > k->desc[w].log2nb) {
      // the table grew after the save: keep the larger table and re-insert the saved
      // entries into it (same entry set, so every later result is the same)
      CK(cudaMemsetAsync(c->h_desc[w].tab, 0, ((size_t)1 << c->h_desc[w].log2nb) * sizeof(Bucket), st));
      RehashArgs ra{k->desc[w], c->h_desc[w], c->err_ptr()};
      launch_rehash(ra, st);
      CK(cudaGetLastError());
      continue;
    }
    if (c->h_desc[w].log2nb != k->desc[w].log2nb) {
      InstDesc nd;
      InstBufs nb;
      int rc = alloc_instance(c, w, k->desc[w].log2nb, &nd, &nb);
      if (rc) return rc;
      if ((rc = swap_instance(c, w, nd, nb))) return rc;
    }
    ADD_COPY(c->h_desc[w].tab, k->desc[w].tab, ((size_t)1 << k->desc[w].log2nb) * sizeof(Bucket));
  }
  if (c->sess.log2n != k->sess_log2) {
    CK(cudaStreamSynchronize(st));
    SessSlot* ns = nullptr;
    if (cudaMalloc(&ns, ((size_t)1 << k->sess_log2) * sizeof(SessSlot)) != cudaSuccess) {
      cudaGetLastError();
      return MISAT_ERR_OOM;
    }
    cudaFree(c->sess.slots);
    c->sess.slots = ns;
    c->sess.log2n = k->sess_log2;
  }
  ADD_COPY(c->sess.slots, k->sess, ((size_t)1 << k->sess_log2) * sizeof(SessSlot));
  ADD_COPY(c->d_prot, k->prot, c->W * 12);
  ADD_COPY(c->d_backlog, k->backlog, c->W * 8);
  ADD_COPY(c->d_tokcost, k->tokcost, c->W * 8);
  ADD_COPY(c->d_contraction, k->contraction, c->W * 4);
  if (c->use_gix) {
    if (!k->gkeys) return MISAT_ERR_INVALID_ARG;
    if (c->gix.log2nb != k->g_log2) {
      int rc = gix_alloc(c, k->g_log2);
      if (rc) return rc;
    }
    ADD_COPY(c->gix.keys, k->gkeys, gix_slots(c) * 8);
    ADD_COPY(c->gix.masks, k->gmasks, gix_slots(c) * c->gix.mw * 8);
    c->h_meta[c->ml.g_used] = k->g_used;
    ADD_COPY(c->d_meta + c->ml.g_used, k->counters + c->W + 1, 8);
  }
  // sizes and the session-slot counter live in the counters block (host mirror and device)
  for (int w = 0; w < c->W; ++w) reinterpret_cast<long long*>(c->h_meta + c->ml.size)[w] = k->size[w];
  c->h_meta[c->ml.sess_used] = k->sess_used;
  ADD_COPY(c->d_meta + c->ml.size, k->counters, (c->W + 1) * 8);
#undef ADD_COPY
  if ((crc = cp.flush())) return crc;
  for (int b = 0; b < 3; ++b) {
    c->hist_blocks[b] = k->hist_blocks[b];
    c->hist_res[b] = k->hist_res[b];
    c->rho[b] = k->rho[b];
  }
  c->seq = k->seq;
  c->routed = false;
  return MISAT_OK;
}

int misat_sync(misat_ctx* c) {
  if (!c) return MISAT_ERR_INVALID_ARG;
  int rc = read_meta(c);
  if (rc) return rc;
  const int32_t e = c->h_err();
  if (e) {
    // reported once: clear the device error word so that the context can be reused
    CK(cudaMemsetAsync(c->err_ptr(), 0, 4, c->stream));
    CK(cudaStreamSynchronize(c->stream));
    c->routed = false;
  }
  return e;
}

}  // extern "C"
