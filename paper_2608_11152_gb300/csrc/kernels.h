// Kernel argument blocks and host-side launchers of the MISA-T routing library.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "gindex.cuh"

namespace misat {

// ---- K1 ----
struct HashArgs {
  const int64_t* tok_off;
  const int32_t* tokens;
  int64_t n_tokens;
  int32_t n;
  uint64_t seed;
  uint64_t* keys;       // key of (r, j) at floor(tok_off[r]/16) + j
  int64_t keys_cap;
  unsigned* work;       // zeroed before the launch
  const int32_t* err;
};
void launch_block_hash(const HashArgs& a, int num_sms, cudaStream_t st);

// ---- per-request derived data shared by the route and commit kernels ----
struct ReqArrays {
  int32_t* nb;          // full blocks
  int64_t* kbase;       // first key index
  int32_t* L;           // prompt tokens
  uint8_t* cls;         // copy of the batch classes
  uint64_t* session;    // copy of the batch sessions
  uint8_t* sst;         // session state at batch start (0 absent, 1 protected, 2 released)
  int32_t* sinst;       // protected / last instance
  int32_t* leader;      // first request of the session in the batch
  uint8_t* status;      // kStUnresolved / kStResolved / kStFollower / kStHeld
  uint8_t* last_reason; // hold reason of a held leader
  int32_t* inst;        // decision (internal copy)
  uint8_t* reason;      // reason (internal copy)
  uint32_t* hbest;      // max over instances of (H_rw << 16 | 65535 - w): the largest H and,
                        // among instances with it, the lowest index (set by the probe kernels)
};

// ---- per-instance caps of the current route ----
struct InstArrays {
  int64_t* K_w;         // [W]
  int64_t* K_wb;        // [W*3]
  int64_t* N_wb;        // [W*3]
  int64_t* kbar_w;      // [W]
  int32_t* tot;         // [W] protected sessions at batch start
  int32_t* gh;          // [W] global headroom at batch start, K_w - tot (>= 0)
  int32_t* ch;          // [W*3] class headroom at batch start, K_wb - prot_wb (>= 0)
  long long* U;         // [W] upper bound of new keys of the pending commit
};

// ---- K2 ----
struct ProbeArgs {
  const InstDesc* desc;
  int32_t W;
  int32_t n;
  const int32_t* nb;
  const int64_t* kbase;
  const uint64_t* keys;
  uint16_t* H;                 // [n*W]
  int2* hits;                  // (r, w) pairs with block 0 resident and nb >= 2
  uint32_t* hbest;             // [n] packed best (H, instance) per request, see ReqArrays
  unsigned* n_hits;
  int64_t hits_cap;
  unsigned long long* stats;         // phase 1: [0] probes, [1] bucket reads
  unsigned long long* stats_search;  // phase 2: [0] probes, [1] bucket reads
  int32_t* err;
  GIndex gix;                        // phase 1 reads the global index when gix.keys != NULL
  // per-instance layout: a batch-local index of the distinct block-0 keys (GIndex layout,
  // keys cleared per batch), the list of its claimed slots, the list's length (also the
  // distinct-key count reported by the statistics) and the counters of its lookups
  GIndex fb;
  int32_t* fb_list;
  unsigned long long* fb_count;
  unsigned long long* stats_fb;      // [0] batch-index lookups, [1] their bucket reads
};
void launch_probe_first(const ProbeArgs& a, int num_sms, cudaStream_t st);
void launch_probe_search(const ProbeArgs& a, int num_sms, cudaStream_t st);

// ---- route ----
struct SessTable {
  SessSlot* slots;
  uint32_t log2n;
  unsigned long long* used;    // slots ever claimed
};

struct PrologueArgs {
  int32_t n;
  int64_t n_tokens;
  const uint8_t* cls;
  const uint64_t* session;
  const int64_t* tok_off;
  ReqArrays rq;
  SessTable st;
  unsigned long long* bm_key;  // batch-local session map
  int32_t* bm_val;
  uint32_t bm_log2;
  long long* cand;             // [3]
  int32_t* err;
};
void launch_prologue(const PrologueArgs& a, cudaStream_t st);

struct CapsArgs {
  int32_t W;
  const InstDesc* desc;
  const int32_t* prot;         // [W*3]
  const long long* cand;       // [3]
  const int64_t* params;       // [9] device: kbar_b[3], T_b[3], rho_ppm[3] of this route
  int32_t pf_q16;
  int32_t mode;
  const int32_t* contraction;  // [W]
  InstArrays ia;
  const int32_t* err;
};
void launch_caps(const CapsArgs& a, cudaStream_t st);
// Writes the host's per-route class parameters (footprints, residencies, mixture) to the
// device (kernel arguments are taken at launch, so the host array may change right after).
struct RouteParams {
  int64_t v[9];
};
void launch_route_params(const RouteParams& p, int64_t* dst, cudaStream_t st);

// ---- serial selection (select.cu) ----
constexpr int kSelectThreads = 512;        // leaders per window of the joint selection CTA
constexpr int kSelectClassThreads = 512;   // leaders per window of a per-class selection CTA

struct SelectPrepArgs {
  int32_t n;
  int32_t W;
  ReqArrays rq;
  const uint16_t* H;
  int4* rec;                   // [2n] per-request records of the selection
  int32_t* adm;                // [W] zeroed here: admissions per instance of the per-class path
  unsigned* ticket;            // zeroed here
  int32_t* coupled;            // zeroed here
  int32_t* seg;                // [3n] out: per class and block of 256 requests, its leaders in order
  int32_t* segcnt;             // [3 * blocks] out: leaders per class and block
  const int32_t* err;
};
void launch_select_prep(const SelectPrepArgs& a, cudaStream_t st);

struct EnvInitArgs {
  int32_t W;
  const int64_t* backlog;      // [W] d_w
  const int64_t* tokcost;      // [W] 1/mu_w
  const int32_t* gh;           // [W] global headroom at batch start
  const int32_t* ch;           // [W*3] class headroom at batch start
  uint8_t* onhull;             // [3*W] out: line w on the lower envelope of class b's instances
  int32_t* rank;               // [W] out: position of line w in slope order
  int32_t* rank_a;             // [W] out: position of line w in (d_w, w) order
  bool small;                  // every d_w and 1/mu_w below 2^25: 64-bit envelope arithmetic
  const int32_t* err;
};
void launch_env_init(const EnvInitArgs& a, cudaStream_t st);

struct SelectArgs {
  int32_t n;
  int32_t W;
  const int4* rec;             // [2n] from launch_select_prep
  ReqArrays rq;                // out: status, inst, reason, last_reason of every leader
  const int32_t* gh;           // [W] global headroom at batch start
  const int32_t* ch;           // [W*3] class headroom at batch start
  const int64_t* backlog;      // [W] d_w
  const int64_t* tokcost;      // [W] 1/mu_w
  const uint8_t* onhull;       // [3*W] initial envelopes (launch_env_init)
  const int32_t* rank;         // [W] slope order (launch_env_init)
  const int32_t* rank_a;       // [W] (d_w, w) order (launch_env_init)
  const uint16_t* H;           // [n*W]
  int64_t hold_delay_q;
  bool small;                  // as EnvInitArgs::small
  const int32_t* coupled;      // the joint selection runs only when the per-class path set this
  int32_t* err;
};
size_t select_smem_bytes(int W);
cudaError_t select_configure();  // per device, before the first launch: shared memory of the selection CTA
void launch_select(const SelectArgs& a, cudaStream_t st);

// Per-class selection (one CTA per class), valid while no instance runs out of global
// headroom; otherwise it sets *coupled and launch_select decides the batch.
struct SelectClassArgs {
  int32_t n;
  int32_t W;
  const int4* rec;             // [2n] from launch_select_prep
  ReqArrays rq;                // out: status, inst, reason, last_reason of every leader
  const int32_t* gh;           // [W] global headroom at batch start
  const int32_t* ch;           // [W*3] class headroom at batch start
  const int64_t* backlog;      // [W] d_w
  const int64_t* tokcost;      // [W] 1/mu_w
  const uint8_t* onhull;       // [3*W] initial envelopes (launch_env_init)
  const int32_t* rank;         // [W] slope order (launch_env_init)
  const int32_t* rank_a;       // [W] (d_w, w) order (launch_env_init)
  const uint16_t* H;           // [n*W]
  int64_t hold_delay_q;
  bool small;                  // as EnvInitArgs::small
  const int32_t* seg;          // [3n] per class and block of 256 requests, its leaders (prep)
  const int32_t* segcnt;       // [3 * blocks] leaders per class and block (prep)
  int32_t* adm;                // [W] zeroed by launch_select_prep
  unsigned* ticket;            // zeroed by launch_select_prep
  int32_t* coupled;            // zeroed by launch_select_prep; set when the joint kernel must run
  unsigned long long* stats;   // route stats block: [25] = 1 when the joint kernel runs
  int32_t* err;
};
size_t select_class_smem_bytes(int W, int n);
cudaError_t select_class_configure();
void launch_select_class(const SelectClassArgs& a, cudaStream_t st);

struct FinalizeArgs {
  int32_t n;
  int32_t W;
  ReqArrays rq;
  const uint16_t* H;
  int32_t* out_inst;
  uint8_t* out_reason;
  int32_t* out_hit;
  long long* U;
  unsigned long long* stats;   // route stats block (see api)
  ulonglong2* grp;             // zeroed before the launch: (first key, instance) groups of the
  uint32_t grp_log2;           //   admitted requests (grp_note), read back at commit
  const uint64_t* keys;
  const int32_t* err;
};
void launch_finalize(const FinalizeArgs& a, cudaStream_t st);

// ---- commit ----
struct InsertArgs {
  const InstDesc* desc;
  int32_t n;
  int4* units;                 // work list: 32-byte unit records (2 int4), up to 128 blocks each
  unsigned* n_units;           // units listed (zeroed by the launcher)
  int64_t units_cap;
  const int32_t* nb;
  const int64_t* kbase;
  const int32_t* inst;         // instance per request (-1: skip)
  const uint64_t* keys;
  const uint64_t* meta_seq;    // per request tick source: NULL -> (seq, r)
  const uint32_t* meta_arr;    // per request arrival when meta_seq != NULL
  const int32_t* max_blocks;   // per request insert limit (NULL: all)
  uint64_t seq;
  int32_t n_inst;              // W
  long long* size;             // [W] live entries
  unsigned long long* new_keys;
  int32_t* err;
  GIndex gix;                  // mirrored when gix.keys != NULL
  ulonglong2* gnew;            // keys new to an instance table, (key, instance), for the
  unsigned* n_gnew;            //   global index pass (zeroed by the launcher)
  int64_t gnew_cap;
  const ulonglong2* grp;       // groups of the admitted requests (NULL: insert every block)
  uint32_t grp_log2;
  int32_t* skip;               // [n] leading blocks a later request of the group inserts
  unsigned long long* ops;     // blocks in the work list (NULL: not counted)
};
void launch_insert(const InsertArgs& a, int num_sms, cudaStream_t st);  // tables, then global index
void launch_insert_tables(const InsertArgs& a, int num_sms, cudaStream_t st);
void launch_insert_gix(const InsertArgs& a, int ctas, cudaStream_t st);

struct EntryInsertArgs {
  InstDesc desc;
  int64_t n;
  const misat_entry* entries;
  long long* size;             // &size[w]
  int32_t* err;
  int32_t w;
  GIndex gix;
};
void launch_insert_entries(const EntryInsertArgs& a, cudaStream_t st);

struct SessUpdateArgs {
  int32_t n;
  ReqArrays rq;
  SessTable st;
  int32_t* prot;               // [W*3]
  int32_t* err;
};
void launch_session_update(const SessUpdateArgs& a, cudaStream_t st);

struct CompleteArgs {
  int32_t n;
  const uint64_t* session;
  const uint8_t* done;
  SessTable st;
  int32_t* prot;
};
void launch_complete(const CompleteArgs& a, cudaStream_t st);

struct EvictArgs {
  const InstDesc* desc;
  int32_t W;
  const int32_t* only_w;       // if not NULL: evict only instance *only_w
  long long* size;             // [W]
  uint32_t* const* bitmaps;    // [W] per instance fullness bitmap (NB/32 words)
  uint4* const* cand_a;        // [W] candidate lists (meta, key) as uint4: the collected list
  uint4* const* cand_b;        //     and two work lists of the radix narrowing
  uint4* const* cand_c;
  uint32_t* const* slots;      // [W] slot (bucket*4+s) of each entry of cand_a
  uint32_t* const* dslots;     // [W] slots certainly evicted (meta below the bracket)
  uint32_t* const* dmask;      // [W] deleted-slot mask, 4 bits per bucket (NB/8 words)
  unsigned* n_cand;            // [W] entries in cand_a
  unsigned* n_d;               // [W] entries in dslots
  unsigned long long* thr_lo;  // [W] meta bracket of the E-th smallest
  unsigned long long* thr_hi;  // [W]
  unsigned long long* theta;   // [W*2] (meta, key)
  int32_t* active;             // [W] 1: delete entries <= theta, 2: marked entries only
  unsigned long long* evicted;
  int32_t* err;
  GIndex gix;                  // deletions clear the instance's bit when gix.keys != NULL
  int32_t* act;                // [W] instances over capacity (listed by the estimate pass)
  unsigned* n_act;             // entries in act (zeroed by the launcher)
};
void launch_evict(const EvictArgs& a, int chunks_per_inst, int num_sms, cudaStream_t st);
// the two halves: select (estimate, collect, select; reads the tables only) and apply
// (delete, shift; also clears global-index bits)
// marks (may be NULL): events recorded after each kernel (select: 3, apply: 2), for phase timing
void launch_evict_select(const EvictArgs& a, int chunks_per_inst, int num_sms, cudaStream_t st,
                         const cudaEvent_t* marks);
void launch_evict_apply(const EvictArgs& a, int num_sms, cudaStream_t st,
                        const cudaEvent_t* marks);
void launch_compact_marked(const EvictArgs& a, cudaStream_t st);

struct MarkArgs {
  InstDesc desc;
  int64_t n;
  const uint64_t* keys;
  long long* size;             // &size[w]
  uint32_t* bitmap;
  int32_t* active;             // &active[w], set to 0
};
void launch_mark_evict(const MarkArgs& a, int32_t w, const EvictArgs& ev, cudaStream_t st);

struct RehashArgs {
  InstDesc from;
  InstDesc to;
  int32_t* err;
};
void launch_rehash(const RehashArgs& a, cudaStream_t st);

// Device-to-device copies of a checkpoint restore, done by one kernel on the SMs (a
// cudaMemcpyAsync between device buffers may be given to a copy engine, where it waits
// behind a host-to-device copy in flight).  The list travels as the kernel's parameter block,
// so the launch itself copies nothing from the host.
constexpr int kMaxCopies = 768;  // the list fits the 32 KB kernel parameter space
struct CopyItem {
  void* dst;
  const void* src;
  uint64_t bytes;
  uint64_t start;  // first unit of this item in the flattened list
  uint32_t lg;     // log2 of the unit size in bytes (4, 3, 2 or 0: both pointers aligned to it)
  uint32_t pad;
};
struct CopyList {
  int32_t n;
  int32_t pad;
  uint64_t units;  // total units
  CopyItem item[kMaxCopies];
};
void launch_copy_list(const CopyList& l, int num_sms, cudaStream_t st);

// ---- delta-encoded host batches (misat_stage_host_delta) ----
constexpr int kDeltaMaxDepth = MISAT_DELTA_MAX_DEPTH;
struct DeltaArgs {
  int32_t n;
  const int32_t* base;     // [n] base request or -1
  const int64_t* doff;     // [n+1] offsets of the deltas
  const int32_t* dtok;     // delta tokens
  const int64_t* tok_off;  // [n+1] full offsets (computed on the host)
  int32_t* tokens;         // full tokens (output)
};
void launch_delta_expand(const DeltaArgs& a, int num_sms, cudaStream_t st);

struct SessRehashArgs {
  SessTable from;
  SessTable to;
  int32_t* err;
};
void launch_sess_rehash(const SessRehashArgs& a, cudaStream_t st);

// ---- global prefix index maintenance ----
// Rebuild: set bit w for every key of every instance table (index zeroed beforehand).
void launch_gix_build(const InstDesc* desc, int32_t W, uint32_t max_log2nb, const GIndex& g, int32_t* err,
                      cudaStream_t st);
// Clear bit w of every key of instance w's table (before the table is reset).
void launch_gix_clear_table(const InstDesc& d, int32_t w, const GIndex& g, int32_t* err, cudaStream_t st);

}  // namespace misat
