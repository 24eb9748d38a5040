// Commit kernels (K4b, K4c): index insert, session table update, completions,
// eviction down to capacity, table growth.
//
// Index tables are bucketed linear-probing hash sets (4 keys per 32-byte sector).
// Insert claims only empty slots with a CAS, so two threads inserting the same new
// key always meet in the same slot (no duplicates) and an existing key is found by
// every later inserter; the tick is merged with atomicMax (Sec. 4.5 reading: LRU).
// Eviction never leaves tombstones: the exact eviction threshold theta (the E-th
// smallest (meta, key)) is found by a per-instance radix select, then every run of
// full buckets is compacted by one thread with backward shifts, so lookups keep
// stopping at the first bucket with a free slot.
#include "common.cuh"
#include "kernels.h"

namespace misat {

namespace {
constexpr unsigned kFull = 0xffffffffu;

// Find-or-claim `key` in an instance table and merge `meta`.  Returns 1 if the key was
// new, 0 if it existed, -1 if no free slot was found within the table.
__device__ int table_insert(const InstDesc& d, uint64_t key, uint64_t meta) {
  const uint32_t mask = (1u << d.log2nb) - 1;
  uint32_t b = home_bucket(key, d.log2nb);
  for (uint32_t it = 0; it <= mask; ++it) {
    Bucket* B = d.tab + b;
    for (int tries = 0; tries < 2 * kSlots; ++tries) {
      unsigned long long k[4];
      ld_bucket_keys_cg(B, k);
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
      if (old == kEmpty) {
        atomicMax(&B->meta[e], (unsigned long long)meta);
        return 1;
      }
      if (old == key) {
        atomicMax(&B->meta[e], (unsigned long long)meta);
        return 0;
      }
      // the slot went to another key: re-read this bucket
    }
    b = (b + 1) & mask;
  }
  return -1;
}

}  // namespace

// ---------------------------------------------------------------------------
// Insert: one thread per key slot of the batch; the owning request comes from the owner
// map the hash kernel wrote next to the keys.
__global__ void __launch_bounds__(256) k4_insert(InsertArgs a) {
  __shared__ unsigned s_new[kMaxW];  // new keys per instance, flushed once per CTA
  if (block_error(a.err)) return;
  for (int i = threadIdx.x; i < a.n_inst; i += blockDim.x) s_new[i] = 0;
  __syncthreads();
  constexpr int kPer = 4;  // independent key slots per thread per iteration
  const int lane = threadIdx.x & 31;
  unsigned long long nnew = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x * kPer;
  // a warp covers 32*kPer consecutive slots per iteration; lane handles base + lane + 32 k
  const int64_t start = ((int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31)) * kPer;
  for (int64_t base = start; base < a.n_slots; base += stride) {
    int r[kPer], w[kPer];
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int64_t q = base + lane + 32 * k;
      r[k] = q < a.n_slots ? a.owner[q] : -1;
    }
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      w[k] = -1;
      if (r[k] >= 0) {
        w[k] = a.inst[r[k]];
        const int64_t j = base + lane + 32 * k - a.kbase[r[k]];
        if (w[k] >= 0 && a.max_blocks && j >= a.max_blocks[r[k]]) w[k] = -1;
      }
    }
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int64_t q = base + lane + 32 * k;
      int isnew = 0;
      if (w[k] >= 0) {
        const int64_t j = q - a.kbase[r[k]];
        const uint64_t meta = a.meta_seq ? pack_meta(a.meta_seq[r[k]], a.meta_arr[r[k]], (uint64_t)j)
                                         : pack_meta(a.seq, (uint64_t)r[k], (uint64_t)j);
        const int res = table_insert(a.desc[w[k]], a.keys[q], meta);
        if (res < 0)
          set_error(a.err, MISAT_ERR_TABLE_FULL);
        else
          isnew = res;
      }
      // per-instance size increments, aggregated over the warp's lanes with the same instance
      const unsigned peers = __match_any_sync(kFull, isnew ? w[k] : -1 - lane);
      const unsigned newmask = __ballot_sync(kFull, isnew);
      if (isnew && lane == __ffs(peers) - 1) {
        const int c = __popc(peers & newmask);
        atomicAdd(&s_new[w[k]], (unsigned)c);
        nnew += c;
      }
    }
  }
  const long long tot = block_sum((long long)nnew);
  if (threadIdx.x == 0 && tot) atomicAdd(a.new_keys, (unsigned long long)tot);
  __syncthreads();
  for (int i = threadIdx.x; i < a.n_inst; i += blockDim.x)
    if (s_new[i]) atomic_add_i64(&a.size[i], (long long)s_new[i]);
}

void launch_insert(const InsertArgs& a, int num_sms, cudaStream_t st) {
  if (a.n_slots <= 0 || a.n <= 0) return;
  int64_t blocks = (a.n_slots + 1023) / 1024;
  int grid = (int)(blocks < (int64_t)num_sms * 8 ? blocks : (int64_t)num_sms * 8);
  k4_insert<<<grid, 256, 0, st>>>(a);
}

__global__ void __launch_bounds__(256) k4_insert_entries(EntryInsertArgs a) {
  if (block_error(a.err)) return;
  long long nnew = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < a.n; i += (int64_t)gridDim.x * blockDim.x) {
    const misat_entry e = a.entries[i];
    const int res = table_insert(a.desc, e.key, e.meta);
    if (res < 0)
      set_error(a.err, MISAT_ERR_TABLE_FULL);
    else
      nnew += res;
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
// otherwise released (a later request must reacquire admission, Eq. 7).
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

// External removal (Sec. 4.5 engine events): mark listed keys (meta = 0), rebuild the
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
