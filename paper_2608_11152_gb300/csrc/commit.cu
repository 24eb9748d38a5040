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

// Owner request of key slot q (keys of request r live at kbase[r] .. kbase[r]+nb[r]-1,
// kbase non-decreasing): the last r with kbase[r] <= q, or -1 if q is a gap.
__device__ __forceinline__ int owner_of(int64_t q, const int64_t* kbase, const int32_t* nb, int n) {
  int lo = 0, hi = n - 1, r = -1;
  while (lo <= hi) {
    const int mid = (lo + hi) >> 1;
    if (kbase[mid] <= q) {
      r = mid;
      lo = mid + 1;
    } else {
      hi = mid - 1;
    }
  }
  // several requests can share kbase when earlier ones have no full block; the owner is
  // the last of them, which is the one found.
  if (r < 0 || q >= kbase[r] + nb[r]) return -1;
  return r;
}

__device__ __forceinline__ bool le128(uint64_t ma, uint64_t ka, uint64_t mb, uint64_t kb) {
  return ma < mb || (ma == mb && ka <= kb);
}
}  // namespace

// ---------------------------------------------------------------------------
// Insert: one thread per key slot of the batch; owner request found by binary search.
__global__ void __launch_bounds__(256) k4_insert(InsertArgs a) {
  if (block_error(a.err)) return;
  const int lane = threadIdx.x & 31;
  unsigned long long nnew = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t start = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31);
  for (int64_t base = start; base < a.n_slots; base += stride) {
    const int64_t q = base + lane;
    int w = -1, isnew = 0;
    if (q < a.n_slots) {
      const int r = owner_of(q, a.kbase, a.nb, a.n);
      if (r >= 0) {
        w = a.inst[r];
        const int64_t j = q - a.kbase[r];
        if (w >= 0 && a.max_blocks && j >= a.max_blocks[r]) w = -1;
        if (w >= 0) {
          const uint64_t meta = a.meta_seq ? pack_meta(a.meta_seq[r], a.meta_arr[r], (uint64_t)j)
                                           : pack_meta(a.seq, (uint64_t)r, (uint64_t)j);
          const int res = table_insert(a.desc[w], a.keys[q], meta);
          if (res < 0) {
            set_error(a.err, MISAT_ERR_TABLE_FULL);
          } else {
            isnew = res;
          }
        }
      }
    }
    // per-instance size increments, aggregated over the warp's lanes with the same instance
    const unsigned peers = __match_any_sync(kFull, isnew ? w : -1 - lane);
    const unsigned newmask = __ballot_sync(kFull, isnew);
    if (isnew && lane == __ffs(peers) - 1) {
      const int c = __popc(peers & newmask);
      atomic_add_i64(&a.size[w], (long long)c);
      nnew += c;
    }
  }
  if (nnew) atomicAdd(a.new_keys, nnew);
}

void launch_insert(const InsertArgs& a, int num_sms, cudaStream_t st) {
  if (a.n_slots <= 0 || a.n <= 0) return;
  int64_t blocks = (a.n_slots + 255) / 256;
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
  if (nnew) atomic_add_i64(a.size, nnew);
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

// ---------------------------------------------------------------------------
// Eviction select: one CTA per instance with E = size - Cap > 0 finds theta, the E-th
// smallest (meta, key) (ascending = oldest commit first, deeper block first, key last).
// Pass A: histogram of the commit age of every entry (12-bit digit) and the fullness
// bitmap of the buckets.  Pass B: entries of the threshold age bin become candidates
// (copied with their values).  Then radix passes over the candidates, each on the 12
// bits below the highest bit in which candidates still differ, until one is left.
constexpr int kSelThreads = 1024;
constexpr int kBins = 4096;

__device__ __forceinline__ uint32_t age_digit(uint64_t meta, uint64_t cur_seq) {
  const uint64_t seq = meta >> 36;
  const uint64_t age = cur_seq > seq ? cur_seq - seq : 0;
  return (uint32_t)(kBins - 1 - (age < (uint64_t)(kBins - 1) ? age : (uint64_t)(kBins - 1)));
}

// Block-wide: find bin t with cum(<t) < E <= cum(<=t); returns t, writes cum(<t).
__device__ int find_threshold_bin(uint32_t* hist, long long E, long long* below, long long* s_tmp) {
  // each thread owns 4 consecutive bins
  const int t = threadIdx.x;
  long long local = (long long)hist[4 * t] + hist[4 * t + 1] + hist[4 * t + 2] + hist[4 * t + 3];
  // block exclusive scan of `local` (1024 threads) via warp scans
  const int lane = t & 31, wid = t >> 5;
  long long incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long v = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) s_tmp[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    long long v = s_tmp[lane];
    long long sc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long u = __shfl_up_sync(kFull, sc, o);
      if (lane >= o) sc += u;
    }
    s_tmp[lane] = sc - v;  // exclusive warp offsets
  }
  __syncthreads();
  const long long excl = s_tmp[wid] + incl - local;
  __shared__ int s_bin;
  __shared__ long long s_below;
  if (t == 0) s_bin = -1;
  __syncthreads();
  long long c = excl;
  for (int i = 0; i < 4; ++i) {
    const long long h = hist[4 * t + i];
    if (c < E && E <= c + h) {
      s_bin = 4 * t + i;
      s_below = c;
    }
    c += h;
  }
  __syncthreads();
  *below = s_below;
  const int bin = s_bin;
  __syncthreads();
  return bin;
}

__device__ __forceinline__ uint32_t digit128(uint64_t hi, uint64_t lo, int shift) {
  // 12 bits of the 128-bit value (hi:lo) starting at bit `shift`
  if (shift >= 64) return (uint32_t)(hi >> (shift - 64)) & (kBins - 1);
  uint64_t v = lo >> shift;
  if (shift > 0 && shift + 12 > 64) v |= hi << (64 - shift);
  return (uint32_t)v & (kBins - 1);
}

__global__ void __launch_bounds__(kSelThreads) k4_evict_select(EvictArgs a) {
  __shared__ uint32_t hist[kBins];
  __shared__ long long s_tmp[32];
  __shared__ unsigned s_cnt;
  __shared__ unsigned long long s_or_hi, s_or_lo, s_v0_hi, s_v0_lo;
  const int w = a.only_w ? *a.only_w : blockIdx.x;
  if (block_error(a.err)) return;
  const long long E = a.size[w] - a.desc[w].cap;
  if (threadIdx.x == 0) a.active[w] = E > 0 ? 1 : 0;
  if (E <= 0) return;
  const InstDesc d = a.desc[w];
  const uint32_t NB = 1u << d.log2nb;
  uint32_t* bitmap = a.bitmaps[w];
  for (int i = threadIdx.x; i < kBins; i += blockDim.x) hist[i] = 0;
  __syncthreads();
  // pass A: age histogram + fullness bitmap
  for (uint32_t b0 = 0; b0 < NB; b0 += blockDim.x) {
    const uint32_t b = b0 + threadIdx.x;
    bool full = false;
    if (b < NB) {
      const ulonglong2* mp = reinterpret_cast<const ulonglong2*>(d.tab[b].meta);
      const ulonglong2 m01 = __ldcg(mp), m23 = __ldcg(mp + 1);
      const unsigned long long m[4] = {m01.x, m01.y, m23.x, m23.y};
      full = true;
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        if (m[s]) atomicAdd(&hist[age_digit(m[s], a.cur_seq)], 1u);
        else full = false;
      }
    }
    const unsigned bits = __ballot_sync(kFull, full);
    if ((threadIdx.x & 31) == 0 && b < NB) bitmap[b >> 5] = bits;
  }
  __syncthreads();
  long long below;
  int t1 = find_threshold_bin(hist, E, &below, s_tmp);
  long long Erem = E - below;
  // pass B: candidates of the threshold bin
  if (threadIdx.x == 0) s_cnt = 0;
  __syncthreads();
  uint4* cur = a.cand_a[w];
  uint4* nxt = a.cand_b[w];
  for (uint32_t b = threadIdx.x; b < NB; b += blockDim.x) {
    const Bucket* B = d.tab + b;
#pragma unroll
    for (int s = 0; s < 4; ++s) {
      const unsigned long long m = __ldcg(&B->meta[s]);
      if (m && age_digit(m, a.cur_seq) == (uint32_t)t1) {
        const unsigned long long k = __ldcg(&B->key[s]);
        const unsigned pos = atomicAdd(&s_cnt, 1u);
        cur[pos] = make_uint4((uint32_t)m, (uint32_t)(m >> 32), (uint32_t)k, (uint32_t)(k >> 32));
      }
    }
  }
  __syncthreads();
  unsigned cnt = s_cnt;
  // radix narrowing over the candidates
  for (int iter = 0; iter < 16 && cnt > 1; ++iter) {
    if (threadIdx.x == 0) {
      const uint4 v0 = cur[0];
      s_v0_hi = ((unsigned long long)v0.y << 32) | v0.x;
      s_v0_lo = ((unsigned long long)v0.w << 32) | v0.z;
      s_or_hi = 0;
      s_or_lo = 0;
    }
    for (int i = threadIdx.x; i < kBins; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    unsigned long long oh = 0, ol = 0;
    for (unsigned i = threadIdx.x; i < cnt; i += blockDim.x) {
      const uint4 v = cur[i];
      oh |= (((unsigned long long)v.y << 32) | v.x) ^ s_v0_hi;
      ol |= (((unsigned long long)v.w << 32) | v.z) ^ s_v0_lo;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      oh |= __shfl_xor_sync(kFull, oh, o);
      ol |= __shfl_xor_sync(kFull, ol, o);
    }
    if ((threadIdx.x & 31) == 0) {
      if (oh) atomicOr(&s_or_hi, oh);
      if (ol) atomicOr(&s_or_lo, ol);
    }
    __syncthreads();
    const unsigned long long dh = s_or_hi, dl = s_or_lo;
    if (dh == 0 && dl == 0) break;  // all equal (cannot happen for distinct keys)
    const int top = dh ? 64 + 63 - __clzll((long long)dh) : 63 - __clzll((long long)dl);
    const int shift = top >= 11 ? top - 11 : 0;
    for (unsigned i = threadIdx.x; i < cnt; i += blockDim.x) {
      const uint4 v = cur[i];
      atomicAdd(&hist[digit128(((unsigned long long)v.y << 32) | v.x, ((unsigned long long)v.w << 32) | v.z, shift)], 1u);
    }
    __syncthreads();
    long long bl;
    const int t = find_threshold_bin(hist, Erem, &bl, s_tmp);
    Erem -= bl;
    if (threadIdx.x == 0) s_cnt = 0;
    __syncthreads();
    for (unsigned i = threadIdx.x; i < cnt; i += blockDim.x) {
      const uint4 v = cur[i];
      if (digit128(((unsigned long long)v.y << 32) | v.x, ((unsigned long long)v.w << 32) | v.z, shift) == (uint32_t)t) {
        const unsigned pos = atomicAdd(&s_cnt, 1u);
        nxt[pos] = v;
      }
    }
    __syncthreads();
    cnt = s_cnt;
    uint4* tmp = cur;
    cur = nxt;
    nxt = tmp;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    if (cnt < 1) set_error(a.err, MISAT_ERR_TABLE_FULL);
    // the E-th smallest: with cnt == 1 the only candidate; if all remaining candidates
    // are equal (impossible for distinct keys) theta is their common value
    const uint4 v = cur[0];
    a.theta[2 * w] = ((unsigned long long)v.y << 32) | v.x;
    a.theta[2 * w + 1] = ((unsigned long long)v.w << 32) | v.z;
  }
}

// Compaction of one instance table: delete entries with meta == 0 (marked) or
// (meta, key) <= theta, then restore the probing invariant inside each run of full
// buckets.  A run starts after a bucket that was not full before the pass and ends at
// the next such bucket; runs are disjoint, so each is owned by one thread.
__global__ void __launch_bounds__(256) k4_evict_compact(EvictArgs a) {
  const int w = a.only_w ? *a.only_w : blockIdx.y;
  if (block_error(a.err)) return;
  // active: 0 nothing to do (bitmap not built), 1 theta eviction, 2 marked entries only
  const int act = a.active[w];
  if (act == 0) return;
  const InstDesc d = a.desc[w];
  const uint32_t NB = 1u << d.log2nb;
  const uint32_t mask = NB - 1;
  const uint32_t* bitmap = a.bitmaps[w];
  const unsigned long long tm = a.theta[2 * w], tk = a.theta[2 * w + 1];
  const uint32_t nthreads = gridDim.x * blockDim.x;
  const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x;
  const uint32_t per = (NB + nthreads - 1) / nthreads;
  const uint32_t lo = tid * per;
  const uint32_t hi = lo + per < NB ? lo + per : NB;
  long long deleted = 0;
  auto is_full = [&](uint32_t b) { return (bitmap[b >> 5] >> (b & 31)) & 1u; };
  for (uint32_t x0 = lo; x0 < hi; ++x0) {
    if (is_full((x0 - 1) & mask)) continue;  // not a run start
    // run [x0, e]: e = first bucket at or after x0 that was not full
    uint32_t e = x0, len = 0;
    while (is_full(e) && len < NB) {
      e = (e + 1) & mask;
      ++len;
    }
    // delete
    for (uint32_t i = 0; i <= len; ++i) {
      Bucket* B = d.tab + ((x0 + i) & mask);
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        const unsigned long long k = B->key[s];
        if (k == kEmpty) continue;
        const unsigned long long m = B->meta[s];
        if (m == 0 || (act == 1 && le128(m, k, tm, tk))) {
          B->key[s] = kEmpty;
          B->meta[s] = 0;
          ++deleted;
        }
      }
    }
    if (len == 0) continue;
    // backward shift: fill free slots of bucket x from the first later entry of the run
    // whose home lies in [x0, x]
    for (uint32_t i = 0; i < len; ++i) {
      Bucket* X = d.tab + ((x0 + i) & mask);
      for (int s = 0; s < 4; ++s) {
        if (X->key[s] != kEmpty) continue;
        bool moved = false;
        for (uint32_t j = i + 1; j <= len && !moved; ++j) {
          Bucket* Y = d.tab + ((x0 + j) & mask);
          for (int t = 0; t < 4; ++t) {
            const unsigned long long k = Y->key[t];
            if (k == kEmpty) continue;
            const uint32_t rel = (home_bucket(k, d.log2nb) - x0) & mask;
            if (rel <= i) {
              X->key[s] = k;
              X->meta[s] = Y->meta[t];
              Y->key[t] = kEmpty;
              Y->meta[t] = 0;
              moved = true;
              break;
            }
          }
        }
        if (!moved) break;  // no later entry can move into x
      }
    }
  }
  if (deleted) {
    atomic_add_i64(&a.size[w], -deleted);
    atomicAdd(a.evicted, (unsigned long long)deleted);
  }
}

void launch_evict(const EvictArgs& a, int chunks_per_inst, cudaStream_t st) {
  if (a.only_w) {
    k4_evict_select<<<1, kSelThreads, 0, st>>>(a);
    k4_evict_compact<<<dim3(chunks_per_inst, 1), 256, 0, st>>>(a);
  } else {
    k4_evict_select<<<a.W, kSelThreads, 0, st>>>(a);
    k4_evict_compact<<<dim3(chunks_per_inst, a.W), 256, 0, st>>>(a);
  }
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
  k4_evict_compact<<<dim3(8, 1), 256, 0, st>>>(ev);
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
