// Commit kernels (K4b, K4c): index insert, session table update, completions,
// eviction down to capacity, table growth.
//
// Index tables are bucketed linear-probing hash sets (4 keys per 32-byte sector).
// Insert claims only empty slots with a CAS, so two threads inserting the same new
// key always meet in the same slot (no duplicates) and an existing key is found by
// every later inserter; the tick is merged with atomicMax (Sec. 4.4 reading: LRU).
// Eviction never leaves tombstones: the exact eviction threshold theta (the E-th
// smallest (meta, key)) is found by a per-instance radix select, then every run of
// full buckets is compacted by one thread with backward shifts, so lookups keep
// stopping at the first bucket with a free slot.
#include "common.cuh"
#include "kernels.h"

namespace misat {

namespace {
constexpr unsigned kFull = 0xffffffffu;

// Find-or-claim `key` in an instance table and merge `meta`, starting at bucket `b` whose
// four keys the caller has already read into k[] (possibly stale: keys are only ever
// added while inserts run, so a stale read can only miss a claim, which the CAS catches).
// Returns 1 if the key was new, 0 if it existed, -1 if no free slot was found.
__device__ __forceinline__ int table_insert_at(const InstDesc& d, uint64_t key, uint64_t meta, uint32_t b,
                                               unsigned long long k[4]) {
  const uint32_t mask = (1u << d.log2nb) - 1;
  for (uint32_t it = 0; it <= mask; ++it) {
    Bucket* B = d.tab + b;
    for (int tries = 0; tries < 2 * kSlots; ++tries) {
      if (it | tries) ld_bucket_keys_cg(B, k);
      int s = -1;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (k[i] == key) s = i;
      if (s >= 0) {
        atomicMax(&B->meta[s], (unsigned long long)meta);
        return 0;
      }
      int e = -1;
#pragma unroll
      for (int i = 3; i >= 0; --i)
        if (k[i] == kEmpty) e = i;
      if (e < 0) break;  // bucket full without the key: next bucket
      const unsigned long long old = atomicCAS(&B->key[e], kEmpty, (unsigned long long)key);
      if (old == kEmpty || old == key) {
        atomicMax(&B->meta[e], (unsigned long long)meta);
        return old == kEmpty ? 1 : 0;
      }
      // the slot went to another key: re-read this bucket
    }
    b = (b + 1) & mask;
  }
  return -1;
}

__device__ __forceinline__ int table_insert(const InstDesc& d, uint64_t key, uint64_t meta) {
  const uint32_t b = home_bucket(key, d.log2nb);
  unsigned long long k[4];
  ld_bucket_keys_cg(d.tab + b, k);
  return table_insert_at(d, key, meta, b, k);
}

}  // namespace

// ---------------------------------------------------------------------------
// Insert.  Work is listed first: every request with an instance contributes one unit per
// kUnitBlocks of its blocks, so that the insert kernel touches only admitted keys and a
// long prompt is spread over many warps.  A unit is a self-contained 32-byte record
// (pointer to its first key, the instance table, the tick of its request, first depth,
// instance, table size, block count), so a warp reaches its keys in one dependent load
// instead of walking request -> instance -> table descriptor.  A warp then inserts one unit:
// lane l takes blocks l, l+32, l+64, l+96 of it and issues all four home-bucket reads
// before the first atomic; a key already present costs one fire-and-forget atomicMax on
// its meta, a new one a CAS.  While those are in flight the warp already loads its next
// unit's record and keys (software pipelining over the warp's units).  The order of the
// units is free: the final key set and metas do not depend on it.
constexpr int kIns = 4;
constexpr int kUnitBlocks = 32 * kIns;
constexpr int kInsThreads = 256;

struct UnitRec {
  const unsigned long long* keys;  // key of block j0 (lane l, k: keys[l + 32k])
  Bucket* tab;
  uint64_t mhi;                    // seq << 36 | arrival << 16 of the request's tick
  int32_t j0;                      // depth of the first block
  int32_t w;
  uint32_t log2nb;
  int32_t cnt;                     // blocks in the unit, 1..kUnitBlocks
};

__device__ __forceinline__ UnitRec load_unit(const int4* units, int64_t u) {
  const int4 x = __ldg(units + 2 * u), y = __ldg(units + 2 * u + 1);
  UnitRec r;
  r.keys = reinterpret_cast<const unsigned long long*>(((uint64_t)(uint32_t)x.y << 32) | (uint32_t)x.x);
  r.tab = reinterpret_cast<Bucket*>(((uint64_t)(uint32_t)x.w << 32) | (uint32_t)x.z);
  r.mhi = ((uint64_t)(uint32_t)y.y << 32) | (uint32_t)y.x;
  r.j0 = y.z;
  r.w = y.w & 0xffff;
  r.log2nb = ((uint32_t)y.w >> 16) & 0xff;
  r.cnt = (int32_t)((uint32_t)y.w >> 24) + 1;
  return r;
}

__device__ __forceinline__ void load_unit_keys(const UnitRec& u, int lane, uint64_t key[kIns]) {
#pragma unroll
  for (int k = 0; k < kIns; ++k) key[k] = lane + 32 * k < u.cnt ? __ldg(u.keys + lane + 32 * k) : 0;
}

__global__ void __launch_bounds__(256) k4_units(InsertArgs a) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  const int lane = threadIdx.x & 31;
  int u = 0, c = 0, w = 0, s0 = 0;
  if (r < a.n && *a.err == 0 && a.inst[r] >= 0) {
    w = a.inst[r];
    c = a.nb[r];
    if (a.max_blocks && a.max_blocks[r] < c) c = a.max_blocks[r];
    if (a.skip) s0 = min(a.skip[r], c);
    u = (c - s0 + kUnitBlocks - 1) / kUnitBlocks;
  }
  int incl = u;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += t;
  }
  const int tot = __shfl_sync(kFull, incl, 31);
  if (a.ops) {
    const int blocks = __reduce_add_sync(kFull, (unsigned)(c - s0));
    if (lane == 0 && blocks) atomicAdd(a.ops, (unsigned long long)blocks);
  }
  if (tot == 0) return;
  unsigned base = 0;
  if (lane == 31) base = atomicAdd(a.n_units, (unsigned)tot);
  base = __shfl_sync(kFull, base, 31) + (unsigned)(incl - u);
  if (u == 0) return;
  const InstDesc d = a.desc[w];
  const uint64_t seq = a.meta_seq ? a.meta_seq[r] : a.seq;
  const uint64_t arr = a.meta_seq ? (uint64_t)a.meta_arr[r] : (uint64_t)r;
  const uint64_t mhi = pack_meta(seq, arr, 0);  // meta of depth j = mhi - j
  const uint64_t kp = reinterpret_cast<uint64_t>(a.keys + a.kbase[r]);
  const uint64_t tp = reinterpret_cast<uint64_t>(d.tab);
  int4* units = reinterpret_cast<int4*>(a.units);
  for (int i = 0; i < u; ++i) {
    if ((int64_t)base + i >= a.units_cap) {
      set_error(a.err, MISAT_ERR_TABLE_FULL);
      break;
    }
    const int j0 = s0 + i * kUnitBlocks;
    const int cnt = min(kUnitBlocks, c - j0);
    const uint64_t k0 = kp + 8ull * (uint64_t)j0;
    units[2 * ((int64_t)base + i)] = make_int4((int)(uint32_t)k0, (int)(uint32_t)(k0 >> 32), (int)(uint32_t)tp,
                                               (int)(uint32_t)(tp >> 32));
    units[2 * ((int64_t)base + i) + 1] =
        make_int4((int)(uint32_t)mhi, (int)(uint32_t)(mhi >> 32), j0,
                  (int)((uint32_t)w | (d.log2nb << 16) | ((uint32_t)(cnt - 1) << 24)));
  }
}

// Insert work that a later request does anyway.  Keys chain the whole prefix, so request r
// and a later request r' of the same instance whose keys agree on blocks 0 .. p-1 insert the
// same p keys at the same depths, and r' with the larger tick (same commit, later arrival):
// after r' the index holds exactly what it holds after both, for every order of the atomics
// (max-merged ticks, a key claimed once).  Per request, r' is the latest admitted request of
// its (first key, instance) group (grp_note at route time), and skip[r] = p is the length of
// the common prefix, compared key by key (one warp per request, 32 keys per step).  An agentic
// turn and the next turn of its session, or two samples of one prompt, share their prefix.
__global__ void __launch_bounds__(256) k4_dedup(InsertArgs a) {
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= a.n) return;
  int p = 0;
  const int w = a.inst[r];
  const int c = a.nb[r];
  if (w >= 0 && c > 0 && *a.err == 0) {
    const uint64_t* kr = a.keys + a.kbase[r];
    const int last = grp_last(a.grp, a.grp_log2, __ldg(kr), w);
    if (last > r) {
      const uint64_t* kl = a.keys + a.kbase[last];
      const int m = min(c, a.nb[last]);
      p = m;
      // 128 keys per step: four loads per lane in flight
      for (int j0 = 0; j0 < m; j0 += 128) {
        bool ne[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int j = j0 + 32 * k + lane;
          ne[k] = j < m && __ldg(kr + j) != __ldg(kl + j);
        }
        unsigned first = 0;
        int at = -1;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const unsigned b = __ballot_sync(kFull, ne[k]);
          if (at < 0 && b) {
            first = b;
            at = k;
          }
        }
        if (at >= 0) {
          p = j0 + 32 * at + __ffs(first) - 1;
          break;
        }
      }
    }
  }
  if (lane == 0) a.skip[r] = p;
}

__global__ void __launch_bounds__(kInsThreads, 3) k4_insert(InsertArgs a) {
  __shared__ unsigned s_new[kMaxW];  // new keys per instance, flushed once per CTA
  if (block_error(a.err)) return;
  for (int i = threadIdx.x; i < a.n_inst; i += blockDim.x) s_new[i] = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  unsigned long long nnew = 0;
  const int4* units = reinterpret_cast<const int4*>(a.units);
  const int64_t n_units = min((int64_t)__ldcg(a.n_units), a.units_cap);
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  int64_t u = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  UnitRec cur{};
  uint64_t key[kIns];
  if (u < n_units) {
    cur = load_unit(units, u);
    load_unit_keys(cur, lane, key);
  }
  for (; u < n_units; u += warps) {
    // home-bucket reads of this unit's keys
    uint32_t hb[kIns];
    unsigned long long kk[kIns][4];
#pragma unroll
    for (int k = 0; k < kIns; ++k) {
      hb[k] = home_bucket(key[k], cur.log2nb);
      if (lane + 32 * k < cur.cnt) ld_bucket_keys_cg(cur.tab + hb[k], kk[k]);
    }
    // the next unit's record and keys, while the buckets are in flight
    UnitRec nxt{};
    uint64_t nkey[kIns] = {0, 0, 0, 0};
    if (u + warps < n_units) {
      nxt = load_unit(units, u + warps);
      load_unit_keys(nxt, lane, nkey);
    }
    const InstDesc d{cur.tab, cur.log2nb, 0, 0};
    unsigned cnt = 0;
    int isnew[kIns];
#pragma unroll
    for (int k = 0; k < kIns; ++k) {
      const int j = lane + 32 * k;
      isnew[k] = 0;
      if (j < cur.cnt) {
        const int res = table_insert_at(d, key[k], cur.mhi - (uint64_t)(cur.j0 + j), hb[k], kk[k]);
        if (res < 0)
          set_error(a.err, MISAT_ERR_TABLE_FULL);
        else
          isnew[k] = res;
      }
      cnt += __popc(__ballot_sync(kFull, isnew[k]));
    }
    if (a.gix.keys && cnt) {
      // keys new to instance w are listed for the global-index pass (one slot range per warp)
      unsigned base = 0;
      if (lane == 0) base = atomicAdd(a.n_gnew, cnt);
      base = __shfl_sync(kFull, base, 0);
#pragma unroll
      for (int k = 0; k < kIns; ++k) {
        const unsigned bal = __ballot_sync(kFull, isnew[k]);
        if (isnew[k]) {
          const unsigned pos = base + __popc(bal & lanemask_lt());
          if ((int64_t)pos < a.gnew_cap)
            a.gnew[pos] = make_ulonglong2((unsigned long long)key[k], (unsigned long long)cur.w);
          else
            set_error(a.err, MISAT_ERR_TABLE_FULL);
        }
        base += __popc(bal);
      }
    }
    if (lane == 0 && cnt) {
      atomicAdd(&s_new[cur.w], cnt);
      nnew += cnt;
    }
    cur = nxt;
#pragma unroll
    for (int k = 0; k < kIns; ++k) key[k] = nkey[k];
  }
  const long long tot = block_sum((long long)nnew);
  if (threadIdx.x == 0 && tot) atomicAdd(a.new_keys, (unsigned long long)tot);
  __syncthreads();
  for (int i = threadIdx.x; i < a.n_inst; i += blockDim.x)
    if (s_new[i]) atomic_add_i64(&a.size[i], (long long)s_new[i]);
}

// Global index pass: bit w for every key new to instance w, one thread per listed key.
__global__ void __launch_bounds__(256) k4_gix_insert(InsertArgs a) {
  if (block_error(a.err)) return;
  const int64_t n = min((int64_t)__ldcg(a.n_gnew), a.gnew_cap);
  long long claimed = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const ulonglong2 e = a.gnew[i];
    const int g = gix_set(a.gix, e.x, (int)e.y);
    if (g < 0)
      set_error(a.err, MISAT_ERR_TABLE_FULL);
    else
      claimed += g;
  }
  const long long tot = block_sum(claimed);
  if (threadIdx.x == 0 && tot) atomicAdd(a.gix.used, (unsigned long long)tot);
}

void launch_insert_tables(const InsertArgs& a, int num_sms, cudaStream_t st) {
  if (a.n <= 0) return;
  cudaMemsetAsync(a.n_units, 0, sizeof(unsigned), st);
  if (a.gix.keys) cudaMemsetAsync(a.n_gnew, 0, sizeof(unsigned), st);
  if (a.grp && a.skip) k4_dedup<<<(a.n + 7) / 8, 256, 0, st>>>(a);
  k4_units<<<(a.n + 255) / 256, 256, 0, st>>>(a);
  k4_insert<<<num_sms * 3, kInsThreads, 0, st>>>(a);  // resident CTAs: 3 per SM
}

void launch_insert_gix(const InsertArgs& a, int ctas, cudaStream_t st) {
  if (a.n <= 0 || !a.gix.keys) return;
  k4_gix_insert<<<ctas, 256, 0, st>>>(a);
}

void launch_insert(const InsertArgs& a, int num_sms, cudaStream_t st) {
  launch_insert_tables(a, num_sms, st);
  launch_insert_gix(a, num_sms * 8, st);
}

__global__ void __launch_bounds__(256) k4_insert_entries(EntryInsertArgs a) {
  if (block_error(a.err)) return;
  long long nnew = 0, gclaim = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < a.n; i += (int64_t)gridDim.x * blockDim.x) {
    const misat_entry e = a.entries[i];
    const int res = table_insert(a.desc, e.key, e.meta);
    if (res < 0) {
      set_error(a.err, MISAT_ERR_TABLE_FULL);
    } else {
      nnew += res;
      if (res && a.gix.keys) {
        const int g = gix_set(a.gix, e.key, a.w);
        if (g < 0)
          set_error(a.err, MISAT_ERR_TABLE_FULL);
        else
          gclaim += g;
      }
    }
  }
  if (a.gix.keys) {
    const long long gt = block_sum(gclaim);
    if (threadIdx.x == 0 && gt) atomicAdd(a.gix.used, (unsigned long long)gt);
  }
  const long long tot = block_sum(nnew);
  if (threadIdx.x == 0 && tot) atomic_add_i64(a.size, tot);
}

void launch_insert_entries(const EntryInsertArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  int64_t blocks = (a.n + 255) / 256;
  k4_insert_entries<<<(int)(blocks < 4096 ? blocks : 4096), 256, 0, st>>>(a);
}

// ---------------------------------------------------------------------------
// Session table update at commit (Sec. 4.1: an admitted new session becomes pending /
// protected on its instance; a rebound one leaves its previous instance's count).
// Only leaders with ADMIT_NEW change anything; each session has one leader per batch.
__global__ void __launch_bounds__(256) k4_sessions(SessUpdateArgs a) {
  if (block_error(a.err)) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= a.n || a.rq.leader[r] != r || a.rq.reason[r] != MISAT_ADMIT_NEW) return;
  const uint64_t s = a.rq.session[r];
  const int w = a.rq.inst[r];
  const int b = a.rq.cls[r];
  const uint64_t nv = sess_val(kSessProtected, (uint32_t)b, (uint32_t)w);
  const uint32_t mask = (1u << a.st.log2n) - 1;
  uint32_t h = sess_home(s, a.st.log2n);
  for (uint32_t it = 0; it <= mask; ++it) {
    SessSlot* sl = a.st.slots + h;
    unsigned long long k = __ldcg(&sl->key);
    if (k == 0) {
      k = atomicCAS(&sl->key, 0ull, (unsigned long long)s);
      if (k == 0) {
        sl->val = nv;
        atomicAdd(a.st.used, 1ull);
        atomicAdd(&a.prot[w * 3 + b], 1);
        return;
      }
    }
    if (k == s) {
      const uint64_t ov = sl->val;
      if (sess_state(ov) == kSessProtected) atomicSub(&a.prot[sess_inst(ov) * 3 + sess_cls(ov)], 1);
      sl->val = nv;
      atomicAdd(&a.prot[w * 3 + b], 1);
      return;
    }
    h = (h + 1) & mask;
  }
  set_error(a.err, MISAT_ERR_TABLE_FULL);
}

void launch_session_update(const SessUpdateArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  k4_sessions<<<(a.n + 255) / 256, 256, 0, st>>>(a);
}

// Completion events (distinct sessions): leave the protected set; done -> dead slot,
// otherwise released (a later request must be admitted again, Eq. 7).
__global__ void __launch_bounds__(256) k_complete(CompleteArgs a) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= a.n) return;
  const uint64_t s = a.session[i];
  const uint32_t mask = (1u << a.st.log2n) - 1;
  uint32_t h = sess_home(s, a.st.log2n);
  for (uint32_t it = 0; it <= mask; ++it) {
    SessSlot* sl = a.st.slots + h;
    const unsigned long long k = sl->key;
    if (k == 0) return;
    if (k == s) {
      const uint64_t v = sl->val;
      const uint32_t stv = sess_state(v);
      if (stv == kSessDead) return;
      if (stv == kSessProtected) atomicSub(&a.prot[sess_inst(v) * 3 + sess_cls(v)], 1);
      sl->val = sess_val(a.done[i] ? kSessDead : kSessReleased, sess_cls(v), sess_inst(v));
      return;
    }
    h = (h + 1) & mask;
  }
}

void launch_complete(const CompleteArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  k_complete<<<(a.n + 255) / 256, 256, 0, st>>>(a);
}

// External removal (Sec. 4.4 engine events): mark listed keys (meta = 0), rebuild the
// fullness bitmap from the keys, then compact with theta inactive.
__global__ void __launch_bounds__(256) k_mark(MarkArgs a) {
  long long cnt = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < a.n; i += (int64_t)gridDim.x * blockDim.x) {
    const uint64_t key = a.keys[i];
    const uint32_t mask = (1u << a.desc.log2nb) - 1;
    uint32_t b = home_bucket(key, a.desc.log2nb);
    for (uint32_t it = 0; it <= mask; ++it) {
      Bucket* B = a.desc.tab + b;
      bool open = false, found = false;
      for (int s = 0; s < 4; ++s) {
        const unsigned long long k = B->key[s];
        if (k == key) {
          if (atomicExch(&B->meta[s], 0ull) != 0ull) ++cnt;
          found = true;
        }
        open |= k == kEmpty;
      }
      if (found || open) break;
      b = (b + 1) & mask;
    }
  }
  (void)cnt;
}

__global__ void __launch_bounds__(256) k_bitmap_keys(MarkArgs a) {
  const uint32_t NB = 1u << a.desc.log2nb;
  // compaction of this instance deletes marked entries only
  if (threadIdx.x == 0 && blockIdx.x == 0) *a.active = 2;
  for (uint32_t b0 = blockIdx.x * blockDim.x; b0 < NB; b0 += gridDim.x * blockDim.x) {
    const uint32_t b = b0 + threadIdx.x;
    bool full = false;
    if (b < NB) {
      const Bucket* B = a.desc.tab + b;
      full = B->key[0] && B->key[1] && B->key[2] && B->key[3];
    }
    const unsigned bits = __ballot_sync(kFull, full);
    if ((threadIdx.x & 31) == 0 && b < NB) a.bitmap[b >> 5] = bits;
  }
}

void launch_mark_evict(const MarkArgs& a, int32_t w, const EvictArgs& ev, cudaStream_t st) {
  (void)w;
  if (a.n > 0) {
    int64_t blocks = (a.n + 255) / 256;
    k_mark<<<(int)(blocks < 4096 ? blocks : 4096), 256, 0, st>>>(a);
  }
  const uint32_t NB = 1u << a.desc.log2nb;
  k_bitmap_keys<<<(NB + 255) / 256 < 4096 ? (NB + 255) / 256 : 4096, 256, 0, st>>>(a);
  launch_compact_marked(ev, st);
}

// Growth: re-insert every entry of `from` into the empty, larger table `to`.
// Copy list: CTAs take spans of kSpan units of the flattened list; the item holding a span's
// first unit is found by a (uniform) binary search, later items by stepping forward.
__global__ void __launch_bounds__(256) k_copy_list(const __grid_constant__ CopyList L) {
  constexpr uint64_t kSpan = 256 * 16;
  for (uint64_t s0 = (uint64_t)blockIdx.x * kSpan; s0 < L.units; s0 += (uint64_t)gridDim.x * kSpan) {
    int lo = 0, hi = L.n - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (L.item[mid].start <= s0)
        lo = mid;
      else
        hi = mid - 1;
    }
    int i = lo;
    const uint64_t s1 = min(s0 + kSpan, L.units);
    for (uint64_t u = s0 + threadIdx.x; u < s1; u += blockDim.x) {
      while (i < L.n - 1 && u >= L.item[i].start + ((L.item[i].bytes + (1ull << L.item[i].lg) - 1) >> L.item[i].lg)) ++i;
      const CopyItem& it = L.item[i];
      const uint64_t off = (u - it.start) << it.lg;
      char* d = static_cast<char*>(it.dst) + off;
      const char* sp = static_cast<const char*>(it.src) + off;
      if (off + (1ull << it.lg) <= it.bytes) {
        switch (it.lg) {
          case 4: *reinterpret_cast<int4*>(d) = *reinterpret_cast<const int4*>(sp); break;
          case 3: *reinterpret_cast<unsigned long long*>(d) = *reinterpret_cast<const unsigned long long*>(sp); break;
          case 2: *reinterpret_cast<unsigned*>(d) = *reinterpret_cast<const unsigned*>(sp); break;
          default: *d = *sp; break;
        }
      } else {
        for (uint64_t b = off; b < it.bytes; ++b) static_cast<char*>(it.dst)[b] = static_cast<const char*>(it.src)[b];
      }
    }
  }
}

void launch_copy_list(const CopyList& l, int num_sms, cudaStream_t st) {
  if (l.n <= 0 || l.units == 0) return;
  const uint64_t spans = (l.units + 256 * 16 - 1) / (256 * 16);
  const int grid = (int)(spans < (uint64_t)num_sms * 8 ? spans : (uint64_t)num_sms * 8);
  k_copy_list<<<grid, 256, 0, st>>>(l);
}

__global__ void __launch_bounds__(256) k_rehash(RehashArgs a) {
  const uint32_t NB = 1u << a.from.log2nb;
  for (uint32_t b = blockIdx.x * blockDim.x + threadIdx.x; b < NB; b += gridDim.x * blockDim.x) {
    const Bucket B = a.from.tab[b];
    for (int s = 0; s < 4; ++s)
      if (B.key[s] != kEmpty && table_insert(a.to, B.key[s], B.meta[s]) < 0) set_error(a.err, MISAT_ERR_TABLE_FULL);
  }
}

void launch_rehash(const RehashArgs& a, cudaStream_t st) {
  const uint32_t NB = 1u << a.from.log2nb;
  k_rehash<<<(NB + 255) / 256 < 8192 ? (NB + 255) / 256 : 8192, 256, 0, st>>>(a);
}

__global__ void __launch_bounds__(256) k_sess_rehash(SessRehashArgs a) {
  const uint32_t N = 1u << a.from.log2n;
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < N; i += gridDim.x * blockDim.x) {
    const SessSlot sl = a.from.slots[i];
    if (sl.key == 0) continue;
    const uint32_t stv = sess_state(sl.val);
    if (stv != kSessProtected && stv != kSessReleased) continue;
    const uint32_t mask = (1u << a.to.log2n) - 1;
    uint32_t h = sess_home(sl.key, a.to.log2n);
    bool placed = false;
    for (uint32_t it = 0; it <= mask && !placed; ++it) {
      if (atomicCAS(&a.to.slots[h].key, 0ull, sl.key) == 0ull) {
        a.to.slots[h].val = sl.val;
        atomicAdd(a.to.used, 1ull);
        placed = true;
      }
      h = (h + 1) & mask;
    }
    if (!placed) set_error(a.err, MISAT_ERR_TABLE_FULL);
  }
}

void launch_sess_rehash(const SessRehashArgs& a, cudaStream_t st) {
  const uint32_t N = 1u << a.from.log2n;
  k_sess_rehash<<<(N + 255) / 256 < 8192 ? (N + 255) / 256 : 8192, 256, 0, st>>>(a);
}

}  // namespace misat
