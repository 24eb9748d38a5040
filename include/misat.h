/*
 * misat.h -- C ABI of the GB300 (sm_103a) MISA-T batched routing decision.
 *
 * MISA-T ("Scheduling Mixed RL Rollouts Beyond Prefix Locality") is a routing-layer
 * admission policy for mixed RLVR / RLHF / agentic rollout serving.  For each
 * request r the router outputs pi(r) in W u {HOLD} (Sec. 3.1): it admits and
 * places the request on an inference instance, or holds it for re-evaluation.
 * This library computes that decision for a whole batch on one GPU:
 *
 *   1. chained 16-token block hashes of every prompt (Sec. 4.4),
 *   2. the longest cached prefix H_rw of every request on every instance's
 *      resident-block index, held as GPU open-addressing hash tables (Sec. 4.4),
 *   3. caps K_w and K_wb (Sec. 4.1, Eqs. 9-13), eligibility (Eq. 6), prefill
 *      cost (Eq. 1) and the hold-vs-cold rule (Eq. 7), argmin placement,
 *   4. admission in arrival order under the global and class caps (Eq. 6, Sec. 4.2):
 *      the leaders of a batch (first request of each session) are decided one at a
 *      time, each against the batch-start snapshot plus the sessions admitted before
 *      it, which are pending on their instances; then a deterministic commit: index
 *      insert, session table update and eviction down to each instance's KV block
 *      capacity.
 *
 * Conventions
 *   - Return value: MISAT_OK (0) or a negative MISAT_ERR_* code.  Calls validate
 *     their host-visible arguments before enqueueing anything; an invalid call
 *     changes no state.
 *   - Streams: every call is stream-ordered on the stream given to misat_create.
 *     Calls marked [async] return after enqueueing; calls marked [sync] wait.
 *   - Device errors (a malformed batch found on the device, a full table) are
 *     sticky: they are recorded on the device and returned by the next
 *     misat_sync, misat_stats or misat_dump_* call.  Kernels skip their work once
 *     an error is recorded, and no device loop is unbounded.
 *   - Ownership: the caller owns every buffer it passes (batch inputs, decision
 *     outputs, host arrays); the library owns its tables, counters and scratch
 *     and frees them in misat_destroy.  Device pointers are raw CUDA device
 *     addresses on the context's device (e.g. torch tensor data_ptr()).
 *   - Block size is 16 tokens.  Limits: W <= 1024 instances, capacity <= 2^26
 *     blocks per instance, <= 2^20 requests per batch, prompts < 2^20 tokens,
 *     < 2^28 commits per context.
 */
#ifndef MISAT_H
#define MISAT_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- return codes ---- */
#define MISAT_OK 0
#define MISAT_ERR_INVALID_ARG (-1)     /* argument outside its documented range */
#define MISAT_ERR_OOM (-2)             /* device or pinned host allocation failed */
#define MISAT_ERR_CUDA (-3)            /* a CUDA runtime call failed */
#define MISAT_ERR_STATE (-4)           /* commit without a pending route */
#define MISAT_ERR_TABLE_FULL (-5)      /* a bounded probe found no free slot */
#define MISAT_ERR_BATCH_TOO_LARGE (-6) /* batch exceeds max_batch / max_tokens */
#define MISAT_ERR_INTERNAL (-7)        /* the global index no longer mirrors the instance tables */

/* ---- prefix index used by the block-0 probe (misat_config.prefix_index) ---- */
#define MISAT_PREFIX_GLOBAL 0       /* key -> instance bitmask, one lookup per request (default) */
#define MISAT_PREFIX_PER_INSTANCE 1 /* one lookup per (request, instance) pair */

/* ---- policy modes (Sec. 5.1: the policies the evaluation compares) ---- */
#define MISAT_MODE_MISA_T 0            /* block-time quota, Eqs. (11),(13) (default) */
#define MISAT_MODE_MISA 1              /* spatial quota, Eqs. (9)-(10) */
#define MISAT_MODE_SESSION_ADMISSION 2 /* global cap only (class-agnostic) */
#define MISAT_MODE_PLACEMENT_ONLY 3    /* no admission control (cache-aware placement) */

/* ---- decision reasons ---- */
#define MISAT_ADMIT_CONT 1         /* session already protected on the instance (Eq. 6, case 1) */
#define MISAT_ADMIT_NEW 2          /* new, released or rebound session admitted with headroom */
#define MISAT_ADMIT_FOLLOW 3       /* later request of a session whose leader was admitted */
#define MISAT_HOLD_GLOBAL_CAP 16   /* at its turn no instance had global headroom (K_w reached) */
#define MISAT_HOLD_CLASS_CAP 17    /* at its turn every instance with global headroom had reached
                                      the session's class cap K_wb */
#define MISAT_HOLD_NO_ELIGIBLE 18  /* not produced (the two reasons above cover every hold for
                                      headroom); the value stays reserved */
#define MISAT_HOLD_PREFER_CACHE 19 /* Eq. (7): waiting for the cached instance is cheaper */
#define MISAT_HOLD_LEADER_HELD 20  /* later request of a session whose leader was held */

typedef struct misat_ctx misat_ctx;

/* Router configuration (misat_create).  All sizes in KV blocks of 16 tokens. */
typedef struct misat_config {
  int32_t n_instances;          /* W, 1..1024 */
  const int64_t* cap_blocks;    /* host [W]: resident-block capacity Cap_w, 1..2^26 */
  int32_t protected_frac_q16;   /* C_w = floor(Cap_w * q / 65536), 1..65536 (0.9 -> 58982) */
  int32_t mode;                 /* MISAT_MODE_* */
  int32_t max_batch;            /* largest n passed to misat_route, 1..2^20 */
  int64_t max_tokens;           /* largest total prompt tokens of one batch, >= 16 */
  int32_t max_sessions;         /* expected live sessions (table is sized 2x and grows) */
  int32_t hist_window;          /* completed sessions kept per class, 1..4096 (256) */
  int32_t min_obs;              /* observations before T_b leaves the prior, >= 1 (8) */
  int64_t hold_delay_q;         /* Delta_r of Eq. (7), cost units, 0..2^61 */
  int64_t prior_kbar_blocks[3]; /* conservative class footprint priors, 1..2^30 */
  int64_t prior_T_us;           /* shared neutral residency prior (Sec. 4.3), 0..2^40 */
  uint64_t hash_seed;           /* a_{-1} of the block-hash chain (0x9e3779b97f4a7c15) */
  double table_load;            /* max load of an instance table before it grows, 0.25..0.9 (0.75) */
  int32_t prefix_index;         /* MISAT_PREFIX_* (0 = global) */
} misat_config;

/* One routing batch.  Device pointers, except n and n_tokens. */
typedef struct misat_batch {
  int32_t n;                /* requests, 0..max_batch */
  int64_t n_tokens;         /* tok_off[n] */
  const uint8_t* cls;       /* [n] workload class b_r: 0 RLVR, 1 RLHF, 2 agentic */
  const uint64_t* session;  /* [n] session id s_r, nonzero; a session keeps one class */
  const uint64_t* group;    /* [n] prompt group g_r, may be NULL (carried, not used) */
  const int64_t* tok_off;   /* [n+1] CSR offsets into tokens, tok_off[0] = 0, non-decreasing,
                               each prompt < 2^20 tokens */
  const int32_t* tokens;    /* [n_tokens] token ids; 16-byte aligned and readable up to the
                               next 16-byte boundary past n_tokens */
  uint16_t* out_H;          /* optional [n*W] device output: H_rw in blocks, row-major */
} misat_batch;

/* Decisions of one batch.  Device pointers (misat_route) or host pointers
 * (misat_route_host). */
typedef struct misat_decisions {
  int32_t* inst;        /* [n] instance, -1 = HOLD */
  uint8_t* reason;      /* [n] MISAT_ADMIT_* / MISAT_HOLD_* */
  int32_t* hit_blocks;  /* [n] H on the chosen instance; for HOLD the max over instances */
} misat_decisions;

/* Index entry (dump / load).  meta = seq<<36 | arrival<<16 | (65535 - depth):
 * ascending (meta, key) is the eviction order (oldest commit first, deeper block
 * first).  key >= 2. */
typedef struct misat_entry {
  uint64_t key;
  uint64_t meta;
} misat_entry;

/* Statistics of the last route and commit (misat_stats). */
typedef struct misat_batch_stats {
  int64_t n_requests, n_admitted, n_held;
  int64_t by_reason[8];          /* CONT NEW FOLLOW GLOBAL CLASS NO_ELIGIBLE PREFER_CACHE LEADER_HELD */
  int64_t admitted_by_class[3];
  int64_t held_by_class[3];
  int64_t hit_tokens;            /* 16 * hit blocks over admitted requests */
  int64_t query_tokens;          /* prompt tokens of admitted requests */
  int64_t dtv_ppm;               /* D_TV(admitted class mix, rho) in ppm, -1 if none admitted */
  int64_t probes;                /* key lookups executed by the probe kernels */
  int64_t bucket_reads;          /* 32-byte key groups read by the probe kernels */
  int64_t probes_first;          /* of which: block-0 probes (phase 1) */
  int64_t bucket_reads_first;    /* of which: key groups read by phase 1 */
  int64_t new_keys;              /* keys inserted by the last commit */
  int64_t evicted;               /* keys evicted by the last commit */
  int64_t seq;                   /* commits applied so far */
  int64_t insert_ops;            /* key operations of the last commit's insert: full blocks of the
                                    admitted requests, less the leading blocks that a later request
                                    of the same instance inserts with the same keys */
  int64_t joint_selection;       /* 1 if some instance ran out of global headroom during the last
                                    route, so its leaders were decided by the joint chain over all
                                    classes; 0 if the per-class chains decided them */
  int64_t first_block_keys;      /* per-instance layout: distinct block-0 keys of the last route
                                    (each probed once per instance); 0 with the global index */
  int64_t first_block_lookups;   /* per-instance layout: lookups of the requests' block-0 keys in
                                    the route's index of distinct keys; 0 with the global index */
} misat_batch_stats;

/* Create a router on the current CUDA device.  cuda_stream: a cudaStream_t (NULL =
 * legacy default stream).  [sync] Errors: INVALID_ARG, OOM, CUDA. */
int misat_create(const misat_config* cfg, void* cuda_stream, misat_ctx** out);

/* Free all device and host memory of ctx (waits for the stream). */
int misat_destroy(misat_ctx* ctx);

/* Trainer target mixture rho (Sec. 3.1), ppm per class, sum = 10^6.  Used only for
 * D_TV (Sec. 3.3) and for splitting C_w when no class has demand.  [host] */
int misat_set_mixture(misat_ctx* ctx, const uint32_t rho_ppm[3]);

/* Per-instance runtime state from the serving layer, host arrays [W], each may be NULL
 * to keep the previous values:
 *   backlog_q       d_w of Eq. (1), fixed-point cost units, 0..2^61
 *   tokcost_q       1/mu_w of Eq. (1), cost units per prompt token, 0..2^32
 *   cap_contraction overload contraction of K_w (Sec. 4.1), >= 0
 * [async] */
int misat_set_instance_state(misat_ctx* ctx, const int64_t* backlog_q, const int64_t* tokcost_q,
                             const int32_t* cap_contraction);

/* Route one batch (Sec. 3.1, Sec. 4).  The leaders -- the first request of each session in
 * the batch -- are decided in arrival order, as the router decides requests online: each
 * sees the state at batch start (caches, sessions, d_w, mu_w) and the sessions admitted
 * before it in the batch, pending on their instances.  A leader takes the cheapest instance
 * of Eq. (1) where Admit (Eq. 6, with the class cap of Sec. 4.2) holds, ties to the lower
 * index, or is held when none has headroom for it (or by Eq. 7); later requests of its
 * session follow it.  Inputs and outputs are device pointers; outputs are written before
 * the call's work ends on the stream.  A second route without a commit replaces the
 * pending one.  [async]
 * The second time a set of batch and output buffers (and sizes) comes among the last four
 * sets seen, the route's kernels are captured into a CUDA graph (on a private stream) and
 * replayed from then on; the graphs of the four most recently used sets are kept.  While
 * the caller captures the context's stream itself, or phase timing is on, they are launched
 * directly.  Errors: INVALID_ARG, BATCH_TOO_LARGE; malformed contents are
 * reported by misat_sync. */
int misat_route(misat_ctx* ctx, const misat_batch* batch, misat_decisions* out);

/* misat_route with HOST batch arrays (pinned memory recommended) and host outputs:
 * copies the batch to library staging buffers, routes, and copies the decisions
 * back.  out_H must be NULL.  [sync] */
int misat_route_host(misat_ctx* ctx, const misat_batch* host_batch, misat_decisions* host_out);

/* Pipelined host path: the copy of the next batch overlaps the routing of the current one.
 * Not in the paper, which routes requests one at a time; this is the batch ingestion of a
 * router whose requests arrive in host memory, where the host link (not the GPU) bounds the
 * end-to-end rate.
 *
 * misat_stage_host copies a HOST batch (pinned memory, or the copies are not asynchronous)
 * into staging slot 0 or 1 on a library copy stream and returns at once.  The copies start
 * after the last route from that slot has finished reading it.  The host arrays must stay
 * unchanged until misat_route_staged of that slot has returned.  out_H must be NULL.  The
 * first call allocates both slots (2 x (4 max_tokens + 17 max_batch) bytes of device memory)
 * and the copy stream.  [async]  Errors: INVALID_ARG, BATCH_TOO_LARGE, STATE (the slot holds
 * a batch not yet routed), OOM, CUDA.
 *
 * misat_route_staged routes the batch of `slot` on the context's stream once its copies are
 * done, exactly as misat_route would route it, and copies the decisions to the HOST arrays
 * of host_out ([n] each).  Returns when they are there.  A staged batch is routed once; the
 * slot is then free for the next misat_stage_host.  Not for use while the caller captures
 * the context's stream.  [sync]  Errors: as misat_route, STATE (nothing staged in the slot).
 *
 * Typical loop: stage(0, batch 0); for k: stage((k+1)%2, batch k+1); route_staged(k%2);
 * commit.  The GPU's copy engine takes host-to-device copies in order, so a host copy that
 * another call enqueues on the context's stream (misat_set_instance_state, misat_load_*)
 * while a staged batch is being copied starts after that batch's copy; misat_route_staged,
 * misat_commit and misat_complete make no host-to-device copy. */
int misat_stage_host(misat_ctx* ctx, const misat_batch* host_batch, int32_t slot);
int misat_route_staged(misat_ctx* ctx, int32_t slot, misat_decisions* host_out);

/* A batch whose prompts are sent as extensions of earlier prompts of the same batch (HOST
 * pointers).  An agentic turn re-sends its session's whole history, and the samples of an
 * RL prompt group share one prompt; with this layout each request carries only the tokens
 * that follow the prompt of an earlier request it extends, so far fewer bytes cross the
 * host link.  No counterpart in the paper: it is an input encoding; the routing decision is
 * the one of the full batch.
 *   base[r]    -1, or an earlier request (0 <= base[r] < r) whose whole prompt is the start
 *              of r's prompt; chains of bases at most MISAT_DELTA_MAX_DEPTH long
 *   delta_off  [n+1] CSR offsets into delta_tokens, delta_off[0] = 0, non-decreasing
 *   delta_tokens  request r's prompt = prompt(base[r]) followed by
 *              delta_tokens[delta_off[r] .. delta_off[r+1]) */
#define MISAT_DELTA_MAX_DEPTH 64
typedef struct misat_batch_delta {
  int32_t n;
  const uint8_t* cls;
  const uint64_t* session;
  const int32_t* base;
  const int64_t* delta_off;
  const int32_t* delta_tokens;
} misat_batch_delta;

/* misat_stage_host for a delta-encoded batch: copies cls, session, bases and delta tokens
 * into staging slot 0 or 1 on the copy stream, then rebuilds the slot's full token array on
 * the GPU (on the same stream), so that misat_route_staged routes exactly the batch the
 * bases and deltas describe.  The full offsets are computed on the host; full prompts must
 * stay below 2^20 tokens and their total within max_tokens.  The first delta call also
 * allocates the slots' delta buffers (4 max_tokens + 12 max_batch bytes of device memory
 * each, and 8 max_batch bytes of pinned host memory).  Host arrays as for misat_stage_host.
 * [async]  Errors: INVALID_ARG (a base out of range, a chain deeper than
 * MISAT_DELTA_MAX_DEPTH, offsets out of order), BATCH_TOO_LARGE, STATE, OOM, CUDA. */
int misat_stage_host_delta(misat_ctx* ctx, const misat_batch_delta* host_batch, int32_t slot);

/* Apply the pending route: insert every admitted request's blocks into its instance's
 * index (tick = commit number and arrival index, depth = block index, max-merge), make
 * newly admitted sessions protected on their instance (a rebound session leaves its old
 * instance), then evict each instance down to Cap_w (Sec. 4.1, Sec. 4.4).  Waits for the
 * route's small summary, then enqueues.  Errors: STATE (no pending route). */
int misat_commit(misat_ctx* ctx);

/* Completion events, host arrays [n] with distinct sessions:
 *   done != 0: the session finished: (total_blocks, residency_us) join class cls's
 *              bounded histories (Sec. 4.1, Sec. 4.3) and the session leaves the
 *              protected set and is forgotten;
 *   done == 0: protection is released but the session is remembered; its next
 *              request is a continuation that must be admitted again (Eq. 7).
 * Unknown sessions only update the histories.  The arrays are copied into one of two
 * library buffers of mapped pinned host memory before the call returns, so the caller may
 * reuse them at once; the first call allocates them (2 x 9 max_batch bytes).  The device
 * update is a kernel on the context's stream that reads that buffer over the host link (no
 * copy-engine transfer, so it does not queue behind a staged batch's copy), and the call
 * does not wait for it.
 * [async]  Errors: INVALID_ARG (a class above 2, a negative count, session 0 or a session
 * listed twice), OOM, CUDA. */
int misat_complete(misat_ctx* ctx, int32_t n, const uint64_t* session, const uint8_t* cls,
                   const int32_t* total_blocks, const int64_t* residency_us, const uint8_t* done);

/* Engine removal events (Sec. 4.4): remove the listed keys (host array) from instance
 * w's index.  The removed set must be suffix-closed (no remaining block may lose its
 * parent).  [sync] */
int misat_evict(misat_ctx* ctx, int32_t w, const uint64_t* keys, int64_t n);

/* Cache reset of instance w (e.g. after a weight sync): its index becomes empty. [async] */
int misat_reset_instance(misat_ctx* ctx, int32_t w);

/* Warm-up of prompt chains, host arrays: chain c (tokens tok_off[c]..tok_off[c+1]) is
 * hashed and its first min(full blocks, max_blocks[c]) blocks are inserted on inst[c]
 * with tick (seq[c] < 2^28, arr[c] < 2^20), then every instance is evicted to Cap.
 * [sync] */
int misat_load_chains(misat_ctx* ctx, int32_t n_chains, const int64_t* tok_off,
                      const int32_t* tokens, const int32_t* inst, const uint64_t* seq,
                      const uint32_t* arr, const int32_t* max_blocks);

/* Load index entries (host array) into instance w with max-merge of meta, then evict w
 * to Cap.  Loaded state must be prefix-closed.  [sync] */
int misat_load_entries(misat_ctx* ctx, int32_t w, const misat_entry* entries, int64_t n);

/* Number of resident blocks of instance w.  [sync] */
int misat_index_size(misat_ctx* ctx, int32_t w, int64_t* out);

/* Buckets (4 slots each) of instance w's table: 2^k, at least 2 Cap_w slots at creation,
 * doubled when a commit would fill it past table_load.  [host] */
int misat_index_buckets(misat_ctx* ctx, int32_t w, int64_t* out);

/* Copy instance w's index to host_out sorted by key (cap entries available; *n_out =
 * count).  [sync] */
int misat_dump_index(misat_ctx* ctx, int32_t w, misat_entry* host_out, int64_t cap,
                     int64_t* n_out);

/* Block keys of the last routed batch, request order (host, cap entries). [sync] */
int misat_dump_keys(misat_ctx* ctx, uint64_t* host_out, int64_t cap, int64_t* n_out);

/* Caps of the last route (host arrays): K_w [W], K_wb [W*3], N_wb [W*3], kbar_w [W],
 * kbar_b [3], T_b [3].  Any pointer may be NULL.  [sync] */
int misat_dump_caps(misat_ctx* ctx, int64_t* K_w, int64_t* K_wb, int64_t* N_wb, int64_t* kbar_w,
                    int64_t* kbar_b, int64_t* T_b);

/* Protected session counts per (w, b), host [W*3].  [sync] */
int misat_dump_counts(misat_ctx* ctx, int32_t* prot);

/* Live sessions sorted by id (host arrays, cap entries): state 1 = protected,
 * 2 = released; inst; class.  [sync] */
int misat_dump_sessions(misat_ctx* ctx, uint64_t* ids, int32_t* state, int32_t* inst,
                        int32_t* cls, int64_t cap, int64_t* n_out);

/* Statistics of the last route / commit.  [sync] */
int misat_stats(misat_ctx* ctx, misat_batch_stats* host_out);

/* Global prefix index (Sec. 4.4: the router maps every prefix block hash to the set of
 * instances that currently cache it).  With MISAT_PREFIX_GLOBAL the library keeps, next to
 * the per-instance tables, one table key -> W-bit instance mask that mirrors them exactly;
 * the block-0 probe of a request reads one mask instead of W tables.
 *
 * misat_global_info [sync]: mask words per entry (ceil(W/64)), slots of the index and
 *   slots claimed (live keys plus keys whose mask became empty; the index is rebuilt from
 *   the instance tables when claimed slots pass 70% of the slots).  Any output may be NULL.
 * misat_global_dump [sync]: the keys with a non-empty mask (unordered) and their masks,
 *   host arrays keys[cap] and masks[cap * mask_words]; *n_out = number of such keys (may
 *   exceed cap: only cap are written).
 * misat_global_rebuild [async]: rebuild the index from the instance tables now.
 * All three return MISAT_ERR_STATE when the context uses MISAT_PREFIX_PER_INSTANCE. */
int misat_global_info(misat_ctx* ctx, int32_t* mask_words, int64_t* slots, int64_t* claimed);
int misat_global_dump(misat_ctx* ctx, uint64_t* keys, uint64_t* masks, int64_t cap, int64_t* n_out);
int misat_global_rebuild(misat_ctx* ctx);

/* ---- checkpoint / resume (the paper has no counterpart: state snapshots of the router) ----
 * A checkpoint is a device-resident copy of the whole router state: every instance index
 * (with its table geometry), the session table, protected counts, per-instance inputs,
 * class histories and the commit counter.  save [sync]; restore [async, stream-ordered]:
 * the context returns to exactly the saved state (a table that grew since keeps its
 * larger size and receives the saved entries); a pending route is dropped.  free
 * releases the copy. */
typedef struct misat_checkpoint misat_checkpoint;
int misat_checkpoint_save(misat_ctx* ctx, misat_checkpoint** out);
int misat_checkpoint_restore(misat_ctx* ctx, const misat_checkpoint* ckpt);
int misat_checkpoint_free(misat_checkpoint* ckpt);

/* ---- per-phase device time (measurement; the paper has no counterpart) ----
 * With timing enabled, the route and commit kernels are launched directly (no graph
 * replay, the global-index pass on the context's stream instead of beside the session
 * update) with CUDA events on the context's stream between them.  misat_phase_times waits
 * and writes the durations (ms) of the last route / commit, indexed by MISAT_PHASE_*
 * (MISAT_N_PHASES values). */
#define MISAT_PHASE_PROLOGUE 0      /* validation, session snapshot, leaders */
#define MISAT_PHASE_HASH 1          /* K1 chained block hash */
#define MISAT_PHASE_CAPS 2          /* K3a caps */
#define MISAT_PHASE_PROBE_FIRST 3   /* K2 block-0 probe of every (request, instance) pair */
#define MISAT_PHASE_PROBE_SEARCH 4  /* K2 binary search of the hit pairs */
#define MISAT_PHASE_SELECT 5        /* K3b placement + K4a admission: the serial selection */
#define MISAT_PHASE_FINALIZE 6      /* holds, followers, outputs */
#define MISAT_PHASE_INSERT 7        /* K4b index insert (work list + table inserts) */
#define MISAT_PHASE_SESSIONS 8      /* session table update */
#define MISAT_PHASE_EVICT 9         /* K4c eviction, all five kernels */
#define MISAT_PHASE_GIX_INSERT 10   /* global prefix index bits of the new keys (inline while timing) */
#define MISAT_PHASE_EVICT_ESTIMATE 11
#define MISAT_PHASE_EVICT_COLLECT 12
#define MISAT_PHASE_EVICT_SELECT 13
#define MISAT_PHASE_EVICT_DELETE 14
#define MISAT_PHASE_EVICT_SHIFT 15
#define MISAT_N_PHASES 16
int misat_set_timing(misat_ctx* ctx, int enable);
int misat_phase_times(misat_ctx* ctx, float* ms_out);

/* ---- allocation-free block hashing (the paper has no counterpart) ----
 * For callers that cannot allocate device memory: an inference engine that has already
 * given all free HBM to its KV-cache pool (a new cudaMalloc would fail, or fragment and
 * shrink that pool), or a hook that runs inside another framework's allocator or
 * memory-accounting scope where device allocations are not allowed.  It writes the same
 * chained 16-token block keys as misat_route, in request order (request 0's full blocks,
 * then request 1's, ... -- the layout of misat_dump_keys), and allocates nothing: its
 * scratch (per-request key offsets, a work counter, an error word) is a fixed array of
 * about 513 KiB inside this library, held by every GPU that loads it until exit.
 *   tok_off   device [n+1], as in misat_batch
 *   tokens    device [n_tokens], 16-byte aligned, readable to the next 16-byte boundary
 *   keys_out  device [keys_cap] u64
 * n above MISAT_NOALLOC_MAX_REQUESTS returns MISAT_ERR_BATCH_TOO_LARGE; malformed offsets
 * or keys_cap below the number of full blocks return MISAT_ERR_INVALID_ARG (nothing is
 * written then).  The first call on a device looks the scratch array up
 * (cudaGetSymbolAddress, with that device current) and should come before any stream
 * capture.  Every call shares the one array: calls that overlap on the GPU (e.g. from
 * two streams at once) race.  [sync: waits for its stream to report errors] */
#define MISAT_NOALLOC_MAX_REQUESTS 65536
int misat_block_hash_noalloc(const int64_t* tok_off, const int32_t* tokens, int32_t n, int64_t n_tokens,
                             uint64_t hash_seed, uint64_t* keys_out, int64_t keys_cap, void* cuda_stream);

/* ---- overload pressure controller (host only; Sec. 4.1) ----
 * The operational cap K_w stays at or below its base floor(C_w / kbar_w).  A confirmed
 * decline of instance w's prefix-cache hit rate relative to its recent healthy windows, or
 * a persistent waiting queue, contracts the cap; it recovers gradually afterwards.  Per
 * observation window and instance:
 *   h_w   = floor(10^6 * hit_tokens / query_tokens) (none when query_tokens = 0)
 *   h*_w  = the largest h of the last ref_windows healthy windows (once min_ref exist)
 *   G_w   = max(0, h*_w - h_w)                         (the paper's hit-rate gap)
 *   hit signal   G_w > gap_ppm and h_w <= the previous window's h (slope check)
 *   queue signal waiting > queue_thresh
 *   after `confirm` consecutive signalling windows, each further signalling window adds
 *   max(1, floor(k_base * G_w / 10^6)) (hit) or max(1, floor(k_base / 8)) (queue),
 *   whichever is larger; each run of recover_after windows without a signal removes 1;
 *   the contraction stays within [0, floor(k_base * max_contraction_pct / 100)].
 *   A window is healthy (joins the reference) when observed, G_w <= gap_ppm and no queue
 *   signal.
 * The paper gives the signals, not their thresholds: every number in the configuration is
 * this library's choice (misat_overload_default_config).  The output is the
 * cap_contraction argument of misat_set_instance_state.  No CUDA call is made. */
typedef struct misat_overload misat_overload;
typedef struct misat_overload_config {
  int32_t ref_windows;         /* healthy windows kept for h*, 1..64 (8) */
  int32_t min_ref;             /* healthy windows before G_w is evaluated, 1..ref_windows (3) */
  int32_t gap_ppm;             /* hit-rate gap that signals degradation, 0..10^6 (100000) */
  int32_t confirm;             /* consecutive signalling windows before a contraction, 1..1000 (2) */
  int64_t queue_thresh;        /* waiting requests above which the queue signals, >= 0 (64) */
  int32_t recover_after;       /* windows without a signal per recovery step, 1..1000 (2) */
  int32_t max_contraction_pct; /* largest contraction in percent of the base cap, 0..100 (50) */
} misat_overload_config;

void misat_overload_default_config(misat_overload_config* cfg);
/* W instances, 1..1024.  Errors: INVALID_ARG (a field out of range), OOM. */
int misat_overload_create(int32_t n_instances, const misat_overload_config* cfg, misat_overload** out);
int misat_overload_destroy(misat_overload* ov);
/* One observation window, host arrays [W]: hit_tokens and query_tokens of the window's
 * admitted requests (0 <= hit <= query <= 2^40), waiting requests, the base cap
 * floor(C_w / kbar_w) (0..2^31); writes the new contraction per instance to
 * contraction_out (may be NULL).  Errors: INVALID_ARG (state unchanged). */
int misat_overload_observe(misat_overload* ov, const int64_t* hit_tokens, const int64_t* query_tokens,
                           const int64_t* waiting, const int64_t* k_base, int32_t* contraction_out);

/* ---- grouped-rollout recheck delays (host only; Sec. 4.1: the recheck delay of a held
 * request decreases as more siblings of its prompt group become visible) ----
 * Host arrays [n]: prompt group (0 = none) and held flag of each request the scheduler
 * currently sees.  delay_out = 0 for a request not held, base_delay_us without a group, and
 * max(min_delay_us, floor(base_delay_us / v)) with v = requests of its group in the list.
 * The 1/v law is this library's choice (the paper gives none).  Errors: INVALID_ARG. */
int misat_recheck_delays(int32_t n, const uint64_t* group, const uint8_t* held, int64_t base_delay_us,
                         int64_t min_delay_us, int64_t* delay_out);

/* Wait for the stream and return the sticky device error (0 if none), then clear it and
 * drop any pending route.  A batch rejected on the device changes no persistent state;
 * after TABLE_FULL during a commit the index of the affected instance may hold part of
 * that commit's blocks.  [sync] */
int misat_sync(misat_ctx* ctx);

/* Static description of an error code. */
const char* misat_strerror(int code);

#ifdef __cplusplus
}
#endif
#endif /* MISAT_H */
