// Eviction down to capacity (K4c): after a commit's inserts, each instance whose index
// holds E = size - Cap_w > 0 entries too many loses its E smallest (meta, key): the
// least recently committed blocks, deepest first among equal ticks (Sec. 4.4 reading:
// LRU; the commit-tick order keeps every index prefix-closed).
//
// Admissions concentrate on few instances (every cold request of a round prefers the
// same cheapest instance), so E ranges from 0 to a large part of an instance; the work
// is spread over many CTAs per instance and the one serial step is kept small:
//   k4_evict_estimate  (1 CTA / instance)  sorted sample of up to 4096 metas -> a meta
//                      bracket [lo, hi] that contains the E-th smallest w.h.p.
//   k4_evict_collect   (many CTAs / instance, streaming)  fullness bitmap; entries with
//                      meta < lo are certainly evicted (slot list D), entries with
//                      lo <= meta <= hi go to a short list U with their values and slots
//   k4_evict_select    (1 CTA / instance)  theta = the (E - |D|)-th smallest of U by
//                      radix narrowing; if the bracket missed, the CTA re-collects the
//                      whole instance and selects exactly anyway
//   k4_evict_delete    deletes D and the entries of U at or below theta
//   k4_evict_shift     refills the holes of every run of full buckets that lost an entry
//                      with backward shifts (no tombstones), one thread per run
#include "common.cuh"
#include "kernels.h"

namespace misat {

namespace {
constexpr unsigned kFull = 0xffffffffu;
constexpr int kSelThreads = 1024;
constexpr int kBins = 4096;

__device__ __forceinline__ bool le128(uint64_t ma, uint64_t ka, uint64_t mb, uint64_t kb) {
  return ma < mb || (ma == mb && ka <= kb);
}

__device__ __forceinline__ uint64_t v_hi(const uint4& v) { return ((unsigned long long)v.y << 32) | v.x; }
__device__ __forceinline__ uint64_t v_lo(const uint4& v) { return ((unsigned long long)v.w << 32) | v.z; }

// Block-wide (1024 threads, 4096 bins): bin t with cum(<t) < E <= cum(<=t); cum(<t) in *below.
__device__ int find_threshold_bin(uint32_t* hist, long long E, long long* below, long long* s_tmp) {
  const int t = threadIdx.x;
  long long local = (long long)hist[4 * t] + hist[4 * t + 1] + hist[4 * t + 2] + hist[4 * t + 3];
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
    s_tmp[lane] = sc - v;
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

// 12 bits of the 128-bit value (hi:lo) starting at bit `shift`.
__device__ __forceinline__ uint32_t digit128(uint64_t hi, uint64_t lo, int shift) {
  if (shift >= 64) return (uint32_t)(hi >> (shift - 64)) & (kBins - 1);
  uint64_t v = lo >> shift;
  if (shift > 0 && shift + 12 > 64) v |= hi << (64 - shift);
  return (uint32_t)v & (kBins - 1);
}

}  // namespace


__global__ void __launch_bounds__(kSelThreads) k4_evict_estimate(EvictArgs a) {
  constexpr int kEst = 2048;  // 4 slots of up to 512 evenly spaced buckets
  __shared__ unsigned long long s_smp[kEst];
  __shared__ uint32_t hist[kBins];
  __shared__ long long s_tmp[32];
  __shared__ unsigned long long s_min, s_max;
  __shared__ unsigned s_m;
  const int w = a.only_w ? *a.only_w : blockIdx.x;
  if (block_error(a.err)) return;
  const long long size = a.size[w];
  const long long E = size - a.desc[w].cap;
  const int tid = threadIdx.x;
  if (tid == 0) {
    a.active[w] = E > 0 ? 1 : 0;
    a.n_d[w] = 0;
    a.n_cand[w] = 0;
    if (E > 0) a.act[atomicAdd(a.n_act, 1u)] = w;  // the streaming passes visit only these
  }
  if (E <= 0) return;
  const InstDesc d = a.desc[w];
  const uint32_t NB = 1u << d.log2nb;
  if (tid == 0) {
    s_m = 0;
    s_min = ~0ull;
    s_max = 0;
  }
  for (int i = tid; i < kBins; i += kSelThreads) hist[i] = 0;
  __syncthreads();
  // samples: the metas of up to 512 evenly spaced buckets
  unsigned long long mn = ~0ull, mx = 0;
  {
    const uint32_t nsb = NB < 512u ? NB : 512u;
    unsigned occ = 0;
    if ((uint32_t)tid < nsb) {
      const uint32_t b = (uint32_t)(((uint64_t)tid * NB) / nsb);
      const ulonglong2* mp = reinterpret_cast<const ulonglong2*>(d.tab[b].meta);
      const ulonglong2 m01 = __ldcg(mp), m23 = __ldcg(mp + 1);
      const unsigned long long m[4] = {m01.x, m01.y, m23.x, m23.y};
      for (int s = 0; s < 4; ++s) {
        s_smp[4 * tid + s] = m[s];
        if (m[s]) {
          ++occ;
          mn = m[s] < mn ? m[s] : mn;
          mx = m[s] > mx ? m[s] : mx;
        }
      }
    } else if (tid < kEst / 4) {
      for (int s = 0; s < 4; ++s) s_smp[4 * tid + s] = 0;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long a1 = __shfl_xor_sync(kFull, mn, o), a2 = __shfl_xor_sync(kFull, mx, o);
      mn = a1 < mn ? a1 : mn;
      mx = a2 > mx ? a2 : mx;
      occ += __shfl_xor_sync(kFull, occ, o);
    }
    if ((tid & 31) == 0 && occ) {
      atomicAdd(&s_m, occ);
      atomicMin(&s_min, mn);
      atomicMax(&s_max, mx);
    }
  }
  __syncthreads();
  const unsigned m = s_m;
  unsigned long long lo = 0, hi = ~0ull;
  if (m > 0 && size > 0) {
    // histogram of the samples over [min, max], 4096 equal bins
    const unsigned long long smin = s_min;
    const unsigned __int128 range = (unsigned __int128)(s_max - s_min) + 1;
    auto bin_of = [&](unsigned long long x) {
      return (uint32_t)((((unsigned __int128)(x - smin)) << 12) / range);
    };
    for (int i = tid; i < kEst; i += kSelThreads) {
      const unsigned long long x = s_smp[i];
      if (x) atomicAdd(&hist[bin_of(x)], 1u);
    }
    __syncthreads();
    // the E-th smallest sits near sample rank p = E m / size; bracket it by ~3 standard
    // deviations of the sample count plus a constant on both sides
    const double p = (double)E * (double)m / (double)size;
    const double margin = 3.0 * sqrt(p + 1.0) + 16.0;
    const long long rl = (long long)(p - margin), rh = (long long)(p + margin) + 1;
    long long below;
    const int bl = rl >= 1 ? find_threshold_bin(hist, rl, &below, s_tmp) : -1;
    const int bh = rh <= (long long)m ? find_threshold_bin(hist, rh, &below, s_tmp) : -1;
    // bin edges: every sample of bin b lies in [edge(b), edge(b + 1) - 1]
    auto edge = [&](int b) {
      return smin + (unsigned long long)((range * (unsigned)b + 4095) >> 12);
    };
    if (bl >= 0) lo = edge(bl);
    if (bh >= 0) hi = edge(bh + 1) - 1;
  }
  if (tid == 0) {
    a.thr_lo[w] = lo;
    a.thr_hi[w] = hi;
  }
}

// Streaming pass over the instance's metas: chunk `cidx` of `chunks` of instance w, a range
// of whole 32-bucket bitmap words.  A CTA takes 4 x blockDim buckets at a time: each thread
// loads the metas of four buckets (all loads in flight together), keeps only which slots
// are certainly evicted (meta < lo) or candidates (lo <= meta <= hi) as bit masks, writes
// the fullness bitmap words and clears the deleted-slot masks; the list entries are
// reserved with one CTA-wide scan per step, and only candidates re-read their meta and key.
__device__ __forceinline__ void collect_chunk(const EvictArgs& a, int w, uint32_t cidx, uint32_t chunks) {
  __shared__ unsigned s_wd[32], s_wu[32], s_bd, s_bu;
  const InstDesc d = a.desc[w];
  const uint32_t NB = 1u << d.log2nb;
  const unsigned long long lo = a.thr_lo[w], hi = a.thr_hi[w];
  uint32_t* bitmap = a.bitmaps[w];
  uint32_t* dmask = a.dmask[w];
  uint32_t* dsl = a.dslots[w];
  uint4* u = a.cand_a[w];
  uint32_t* usl = a.slots[w];
  const int lane = threadIdx.x & 31;
  const int wid = threadIdx.x >> 5;
  const uint32_t words = (NB + 31) >> 5;
  const uint32_t b_beg = (uint32_t)(((uint64_t)words * cidx / chunks) << 5);
  const uint32_t b_end = min(NB, (uint32_t)(((uint64_t)words * (cidx + 1) / chunks) << 5));
  for (uint32_t base = b_beg; base < b_end; base += 4 * blockDim.x) {
    ulonglong2 m01[4], m23[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint32_t b = base + k * blockDim.x + threadIdx.x;
      if (b < b_end) {
        const ulonglong2* mp = reinterpret_cast<const ulonglong2*>(d.tab[b].meta);
        m01[k] = __ldcg(mp);
        m23[k] = __ldcg(mp + 1);
      } else {
        m01[k] = make_ulonglong2(0, 0);
        m23[k] = make_ulonglong2(0, 0);
      }
    }
    unsigned dm = 0, um = 0;  // bit 4k + s: slot s of this thread's k-th bucket
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint32_t b = base + k * blockDim.x + threadIdx.x;
      const unsigned long long m[4] = {m01[k].x, m01[k].y, m23[k].x, m23[k].y};
      const bool full = m[0] && m[1] && m[2] && m[3];
      const unsigned bits = __ballot_sync(kFull, full);
      if (lane == 0 && b < b_end) bitmap[b >> 5] = bits;
      if ((lane & 7) == 0 && b < b_end) dmask[b >> 3] = 0;
#pragma unroll
      for (int sl = 0; sl < 4; ++sl) {
        if (!m[sl]) continue;
        if (m[sl] < lo) dm |= 1u << (4 * k + sl);
        else if (m[sl] <= hi) um |= 1u << (4 * k + sl);
      }
    }
    const int nd = __popc(dm), nu = __popc(um);
    // CTA-wide reservation in both lists: warp scans, then one atomic pair per CTA
    int id = nd, iu = nu;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int vd = __shfl_up_sync(kFull, id, o), vu = __shfl_up_sync(kFull, iu, o);
      if (lane >= o) {
        id += vd;
        iu += vu;
      }
    }
    if (lane == 31) {
      s_wd[wid] = id;
      s_wu[wid] = iu;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      unsigned td = 0, tu = 0;
      for (int k = 0; k < (int)(blockDim.x >> 5); ++k) {
        const unsigned xd = s_wd[k], xu = s_wu[k];
        s_wd[k] = td;
        s_wu[k] = tu;
        td += xd;
        tu += xu;
      }
      s_bd = td ? atomicAdd(&a.n_d[w], td) : 0;
      s_bu = tu ? atomicAdd(&a.n_cand[w], tu) : 0;
    }
    __syncthreads();
    unsigned bd = s_bd + s_wd[wid] + (unsigned)(id - nd);
    unsigned bu = s_bu + s_wu[wid] + (unsigned)(iu - nu);
    __syncthreads();  // the shared offsets are rewritten by the next step
    while (dm) {
      const int bit = __ffs(dm) - 1;
      dm &= dm - 1;
      const uint32_t b = base + (bit >> 2) * blockDim.x + threadIdx.x;
      dsl[bd++] = b * 4 + (bit & 3);
    }
    while (um) {
      const int bit = __ffs(um) - 1;
      um &= um - 1;
      const uint32_t b = base + (bit >> 2) * blockDim.x + threadIdx.x;
      const int sl = bit & 3;
      const unsigned long long x = __ldcg(&d.tab[b].meta[sl]);
      const unsigned long long key = __ldcg(&d.tab[b].key[sl]);
      u[bu] = make_uint4((uint32_t)x, (uint32_t)(x >> 32), (uint32_t)key, (uint32_t)(key >> 32));
      usl[bu] = b * 4 + sl;
      ++bu;
    }
  }
}

// Work items (active instance, chunk), taken by a grid of resident CTAs: instances within
// capacity cost nothing (their list entries are never made).
__global__ void __launch_bounds__(256) k4_evict_collect(EvictArgs a, uint32_t chunks) {
  if (block_error(a.err)) return;
  const uint32_t items = *(volatile const unsigned*)a.n_act * chunks;
  for (uint32_t it = blockIdx.x; it < items; it += gridDim.x) collect_chunk(a, a.act[it / chunks], it % chunks, chunks);
}

__global__ void __launch_bounds__(kSelThreads) k4_evict_select(EvictArgs a) {
  __shared__ uint32_t hist[kBins];
  __shared__ long long s_tmp[32];
  __shared__ unsigned s_cnt;
  __shared__ unsigned long long s_or_hi, s_or_lo, s_v0_hi, s_v0_lo;
  const int w = a.only_w ? *a.only_w : blockIdx.x;
  if (block_error(a.err)) return;
  if (a.active[w] != 1) return;
  const long long E = a.size[w] - a.desc[w].cap;
  const int tid = threadIdx.x;
  const InstDesc d = a.desc[w];
  const uint32_t NB = 1u << d.log2nb;
  uint4* c0 = a.cand_a[w];
  unsigned cnt = a.n_cand[w];
  const unsigned nd = a.n_d[w];
  long long Erem = E - (long long)nd;
  if (Erem <= 0 || Erem > (long long)cnt) {
    // the bracket missed the E-th smallest: collect every entry of the instance here
    if (tid == 0) s_cnt = 0;
    __syncthreads();
    uint32_t* usl = a.slots[w];
    for (uint32_t b = tid; b < NB; b += kSelThreads) {
      for (int s = 0; s < 4; ++s) {
        const unsigned long long m = __ldcg(&d.tab[b].meta[s]);
        if (!m) continue;
        const unsigned long long key = __ldcg(&d.tab[b].key[s]);
        const unsigned pos = atomicAdd(&s_cnt, 1u);
        c0[pos] = make_uint4((uint32_t)m, (uint32_t)(m >> 32), (uint32_t)key, (uint32_t)(key >> 32));
        usl[pos] = b * 4 + s;
      }
    }
    __syncthreads();
    cnt = s_cnt;
    Erem = E;
    if (tid == 0) {
      a.n_cand[w] = cnt;
      a.n_d[w] = 0;
    }
  }
  // radix narrowing over the candidates: each pass takes the 12 bits below the highest
  // bit in which the remaining candidates differ and keeps the bin holding the target
  uint4* cur = c0;
  uint4* nxt = a.cand_b[w];
  uint4* spare = a.cand_c[w];
  for (int iter = 0; iter < 16 && cnt > 1; ++iter) {
    if (tid == 0) {
      s_v0_hi = v_hi(cur[0]);
      s_v0_lo = v_lo(cur[0]);
      s_or_hi = 0;
      s_or_lo = 0;
    }
    for (int i = tid; i < kBins; i += kSelThreads) hist[i] = 0;
    __syncthreads();
    unsigned long long oh = 0, ol = 0;
    for (unsigned i = tid; i < cnt; i += kSelThreads) {
      const uint4 v = cur[i];
      oh |= v_hi(v) ^ s_v0_hi;
      ol |= v_lo(v) ^ s_v0_lo;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      oh |= __shfl_xor_sync(kFull, oh, o);
      ol |= __shfl_xor_sync(kFull, ol, o);
    }
    if ((tid & 31) == 0) {
      if (oh) atomicOr(&s_or_hi, oh);
      if (ol) atomicOr(&s_or_lo, ol);
    }
    __syncthreads();
    const unsigned long long dh = s_or_hi, dl = s_or_lo;
    if (dh == 0 && dl == 0) break;  // all equal (cannot happen for distinct keys)
    const int top = dh ? 64 + 63 - __clzll((long long)dh) : 63 - __clzll((long long)dl);
    const int shift = top >= 11 ? top - 11 : 0;
    for (unsigned i = tid; i < cnt; i += kSelThreads) {
      const uint4 v = cur[i];
      atomicAdd(&hist[digit128(v_hi(v), v_lo(v), shift)], 1u);
    }
    __syncthreads();
    long long bl;
    const int t = find_threshold_bin(hist, Erem, &bl, s_tmp);
    Erem -= bl;
    if (tid == 0) s_cnt = 0;
    __syncthreads();
    for (unsigned i0 = 0; i0 < cnt; i0 += kSelThreads) {
      // keep the target bin: one shared add per warp, positions by ballot rank
      const unsigned i = i0 + tid;
      uint4 v = make_uint4(0, 0, 0, 0);
      bool keep = false;
      if (i < cnt) {
        v = cur[i];
        keep = digit128(v_hi(v), v_lo(v), shift) == (uint32_t)t;
      }
      const unsigned bal = __ballot_sync(kFull, keep);
      unsigned base = 0;
      if ((tid & 31) == 0 && bal) base = atomicAdd(&s_cnt, (unsigned)__popc(bal));
      base = __shfl_sync(kFull, base, 0);
      if (keep) nxt[base + __popc(bal & lanemask_lt())] = v;
    }
    __syncthreads();
    cnt = s_cnt;
    uint4* done = cur;  // the collected list (with its slots) is kept for the delete pass
    cur = nxt;
    nxt = (done == c0) ? spare : done;
    __syncthreads();
  }
  if (tid == 0) {
    if (cnt < 1) set_error(a.err, MISAT_ERR_TABLE_FULL);
    const uint4 v = cur[0];
    a.theta[2 * w] = v_hi(v);
    a.theta[2 * w + 1] = v_lo(v);
  }
}

namespace {
// The apply passes take the entries of all instances over capacity as one index space, so
// that every thread gets about the same number whatever the instances' shares: entry g
// belongs to the k-th active instance with s_pre[k] <= g < s_pre[k + 1] (its D list first,
// then its candidates).  Built by each CTA in shared memory; returns the total.
__device__ unsigned long long list_prefix(const EvictArgs& a, unsigned long long* s_pre, int nact) {
  // the lengths are loaded in parallel, then warp 0 scans them 32 at a time
  for (int k = threadIdx.x; k < nact; k += blockDim.x) {
    const int w = a.act[k];
    s_pre[k + 1] = (unsigned long long)a.n_d[w] + a.n_cand[w];
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    unsigned long long carry = 0;
    for (int k0 = 0; k0 < nact; k0 += 32) {
      const int k = k0 + lane;
      const unsigned long long v = k < nact ? s_pre[k + 1] : 0;
      unsigned long long incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long t = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += t;
      }
      if (k < nact) s_pre[k + 1] = carry + incl;
      carry += __shfl_sync(kFull, incl, 31);
    }
    if (lane == 0) s_pre[0] = 0;
  }
  __syncthreads();
  return s_pre[nact];
}

// The k with s_pre[k] <= g < s_pre[k + 1] (binary search over nact entries).
__device__ __forceinline__ int list_owner(const unsigned long long* s_pre, int nact, unsigned long long g) {
  int lo = 0, hi = nact - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_pre[mid] <= g) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// Delete slot sl of instance w's table; the global index (if any) loses bit w of its key.
__device__ __forceinline__ void delete_slot(const GIndex& g, int w, Bucket* tab, uint32_t* dmask, uint32_t sl,
                                            int32_t* err) {
  const uint32_t b = sl >> 2, s = sl & 3;
  if (g.keys && gix_clear(g, tab[b].key[s], w) < 0) set_error(err, MISAT_ERR_INTERNAL);
  tab[b].key[s] = kEmpty;
  tab[b].meta[s] = 0;
  atomicOr(&dmask[b >> 3], 1u << ((b & 7) * 4 + s));
}
}  // namespace

// Delete D and the candidates at or below theta; record them in the deleted-slot masks.
// Deletions are counted per instance in shared memory and added to the sizes once per CTA.
__global__ void __launch_bounds__(256) k4_evict_delete(EvictArgs a) {
  __shared__ unsigned long long s_pre[kMaxW + 1];
  __shared__ unsigned s_del[kMaxW];
  if (block_error(a.err)) return;
  const int nact = (int)*(volatile const unsigned*)a.n_act;
  for (int k = threadIdx.x; k < nact; k += blockDim.x) s_del[k] = 0;
  const unsigned long long total = list_prefix(a, s_pre, nact);
  const unsigned long long stride = (unsigned long long)gridDim.x * blockDim.x;
  for (unsigned long long g = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; g < total; g += stride) {
    const int k = list_owner(s_pre, nact, g);
    const int w = a.act[k];
    const unsigned i = (unsigned)(g - s_pre[k]), nd = a.n_d[w];
    uint32_t sl;
    if (i < nd) {
      sl = a.dslots[w][i];
    } else {
      const uint4 v = a.cand_a[w][i - nd];
      if (!le128(v_hi(v), v_lo(v), a.theta[2 * w], a.theta[2 * w + 1])) continue;
      sl = a.slots[w][i - nd];
    }
    delete_slot(a.gix, w, a.desc[w].tab, a.dmask[w], sl, a.err);
    atomicAdd(&s_del[k], 1u);
  }
  __syncthreads();
  unsigned long long mine = 0;
  for (int k = threadIdx.x; k < nact; k += blockDim.x) {
    const unsigned d = s_del[k];
    if (d) {
      atomic_add_i64(&a.size[a.act[k]], -(long long)d);
      mine += d;
    }
  }
  const long long tot = block_sum((long long)mine);
  if (threadIdx.x == 0 && tot) atomicAdd(a.evicted, (unsigned long long)tot);
}

// Refill the holes of every run of full buckets that lost an entry.  The thread of the
// run's first deleted slot (lowest bucket, then lowest slot) owns the run.
__global__ void __launch_bounds__(256) k4_evict_shift(EvictArgs a) {
  __shared__ unsigned long long s_pre[kMaxW + 1];
  if (block_error(a.err)) return;
  const int nact = (int)*(volatile const unsigned*)a.n_act;
  const unsigned long long total = list_prefix(a, s_pre, nact);
  const unsigned long long stride = (unsigned long long)gridDim.x * blockDim.x;
  for (unsigned long long g = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x; g < total; g += stride) {
    const int k = list_owner(s_pre, nact, g);
    const int w = a.act[k];
    const unsigned i = (unsigned)(g - s_pre[k]), nd = a.n_d[w];
    const uint32_t* full = a.bitmaps[w];
    const uint32_t* dmask = a.dmask[w];
    const InstDesc d = a.desc[w];
    const uint32_t NB = 1u << d.log2nb, mask = NB - 1;
    uint32_t sl;
    if (i < nd) {
      sl = a.dslots[w][i];
    } else {
      const uint4 v = a.cand_a[w][i - nd];
      if (!le128(v_hi(v), v_lo(v), a.theta[2 * w], a.theta[2 * w + 1])) continue;
      sl = a.slots[w][i - nd];
    }
    // the bitmap and deleted-mask words last read (runs are short: mostly one word each)
    uint32_t fw_i = 0xffffffffu, fw = 0, dw_i = 0xffffffffu, dw = 0;
    auto is_full = [&](uint32_t b) {
      if ((b >> 5) != fw_i) {
        fw_i = b >> 5;
        fw = full[fw_i];
      }
      return (fw >> (b & 31)) & 1u;
    };
    auto dmask_at = [&](uint32_t b) {
      if ((b >> 3) != dw_i) {
        dw_i = b >> 3;
        dw = dmask[dw_i];
      }
      return (dw >> ((b & 7) * 4)) & 0xFu;
    };
    const uint32_t x = sl >> 2, sx = sl & 3;
    // a hole in the last (not full) bucket of a run needs no refill
    if (!is_full(x)) continue;
    // my deletion must be the lowest deleted slot of bucket x (the masks are not modified
    // by this kernel, unlike the buckets)
    if ((uint32_t)(__ffs(dmask_at(x)) - 1) != sx) continue;
    // run start: walk back over full buckets; no earlier bucket of the run may hold a deletion
    uint32_t s0 = x, len = 0;
    bool lead = true;
    while (is_full((s0 - 1) & mask) && len < NB) {
      s0 = (s0 - 1) & mask;
      ++len;
      if (dmask_at(s0)) {
        lead = false;
        break;
      }
    }
    if (!lead) continue;
    // run end: the first bucket after x that was not full
    uint32_t e = x, rl = 0;
    while (is_full(e) && rl < NB) {
      e = (e + 1) & mask;
      ++rl;
    }
    const uint32_t runlen = ((e - s0) & mask);  // buckets s0 .. e-1 are full, e ends the run
    for (uint32_t ii = 0; ii < runlen; ++ii) {
      Bucket* X = d.tab + ((s0 + ii) & mask);
      unsigned long long xk[4];
      {
        const ulonglong2* p = reinterpret_cast<const ulonglong2*>(X->key);
        const ulonglong2 u0 = p[0], u1 = p[1];
        xk[0] = u0.x;
        xk[1] = u0.y;
        xk[2] = u1.x;
        xk[3] = u1.y;
      }
      bool stop = false;
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        if (stop || xk[s] != kEmpty) continue;
        bool moved = false;
        for (uint32_t j = ii + 1; j <= runlen && !moved; ++j) {
          Bucket* Y = d.tab + ((s0 + j) & mask);
          const ulonglong2* p = reinterpret_cast<const ulonglong2*>(Y->key);
          const ulonglong2 u0 = p[0], u1 = p[1];
          const unsigned long long yk[4] = {u0.x, u0.y, u1.x, u1.y};
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const unsigned long long k = yk[t];
            if (moved || k == kEmpty) continue;
            const uint32_t rel = (home_bucket(k, d.log2nb) - s0) & mask;
            if (rel <= ii) {
              X->key[s] = k;
              X->meta[s] = Y->meta[t];
              Y->key[t] = kEmpty;
              Y->meta[t] = 0;
              xk[s] = k;
              moved = true;
            }
          }
        }
        if (!moved) stop = true;  // no later entry of the run can move into this bucket
      }
    }
  }
}


namespace {
int stream_grid(const EvictArgs& a, int chunks_per_inst, int resident) {
  // streaming passes: resident CTAs over (active instance, chunk) items
  const int64_t items = (int64_t)(a.only_w ? 1 : a.W) * chunks_per_inst;
  return (int)(items < (int64_t)resident ? items : (int64_t)resident);
}
}  // namespace

void launch_evict_select(const EvictArgs& a, int chunks_per_inst, int num_sms, cudaStream_t st,
                         const cudaEvent_t* marks) {
  const int W = a.only_w ? 1 : a.W;
  cudaMemsetAsync(a.n_act, 0, sizeof(unsigned), st);
  k4_evict_estimate<<<W, kSelThreads, 0, st>>>(a);
  if (marks) cudaEventRecord(marks[0], st);
  k4_evict_collect<<<stream_grid(a, chunks_per_inst, resident_grid<k4_evict_collect>(256, 0, num_sms)), 256, 0, st>>>(
      a, (uint32_t)chunks_per_inst);
  if (marks) cudaEventRecord(marks[1], st);
  k4_evict_select<<<W, kSelThreads, 0, st>>>(a);
  if (marks) cudaEventRecord(marks[2], st);
}

void launch_evict_apply(const EvictArgs& a, int num_sms, cudaStream_t st, const cudaEvent_t* marks) {
  // one grid-stride pass over the list entries of every instance over capacity, one wave each
  k4_evict_delete<<<resident_grid<k4_evict_delete>(256, 0, num_sms), 256, 0, st>>>(a);
  if (marks) cudaEventRecord(marks[0], st);
  k4_evict_shift<<<resident_grid<k4_evict_shift>(256, 0, num_sms), 256, 0, st>>>(a);
  if (marks) cudaEventRecord(marks[1], st);
}

void launch_evict(const EvictArgs& a, int chunks_per_inst, int num_sms, cudaStream_t st) {
  launch_evict_select(a, chunks_per_inst, num_sms, st, nullptr);
  launch_evict_apply(a, num_sms, st, nullptr);
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
          if (a.gix.keys && gix_clear(a.gix, k, w) < 0) set_error(a.err, MISAT_ERR_INTERNAL);
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
  const long long tot = block_sum(deleted);
  if (threadIdx.x == 0 && tot) {
    atomic_add_i64(&a.size[w], -tot);
    atomicAdd(a.evicted, (unsigned long long)tot);
  }
}

void launch_compact_marked(const EvictArgs& a, cudaStream_t st) {
  k4_evict_compact<<<dim3(8, 1), 256, 0, st>>>(a);
}

}  // namespace misat
