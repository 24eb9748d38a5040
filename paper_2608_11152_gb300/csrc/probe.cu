// K2: longest cached prefix H_rw of every request on every instance (Sec. 3.2, Eq. 1;
// Sec. 4.4: the reusable prefix on an instance is the longest run of the prompt's block
// hashes that the instance caches).
//
// Every instance index is prefix-closed (a commit writes whole prefixes with one
// tick and eviction takes the deepest block of a tick first), so "block h-1 is
// resident" is monotone in h and H is found by binary search.
//
// Phase 1: block 0 of every request on every instance.  With the global index one lookup
// per request answers all instances (k2_probe_first_gix).  With per-instance tables every
// distinct block-0 key of the batch is probed once per instance (k2_first_claim,
// k2_probe_distinct) and the requests' rows are expanded from the keys' instance masks by
// the same kernel.  A table probe reads one 32-byte sector (the four keys of the home
// bucket) and continues to the next bucket only when the bucket is full without a match.
// Pairs with block 0 resident and at least two blocks are appended to a compact hit list.
// Phase 2 (k2_probe_search): a group of 16 lanes per hit pair searches [1, nb] with 16
// parallel lookups per step (monotone predicate under prefix closure).
#include "common.cuh"
#include "kernels.h"

namespace misat {

namespace {

__device__ __forceinline__ void block_add_stats(unsigned long long* stats, unsigned long long probes,
                                                unsigned long long reads) {
  __shared__ unsigned long long s_p, s_r;
  if (threadIdx.x == 0) {
    s_p = 0;
    s_r = 0;
  }
  __syncthreads();
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    probes += __shfl_xor_sync(0xffffffffu, probes, o);
    reads += __shfl_xor_sync(0xffffffffu, reads, o);
  }
  if ((threadIdx.x & 31) == 0) {
    atomicAdd(&s_p, probes);
    atomicAdd(&s_r, reads);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    atomicAdd(&stats[0], s_p);
    atomicAdd(&stats[1], s_r);
  }
}

}  // namespace

// Phase 1, per-instance layout with the block-0 lookups of a batch shared by key: requests
// that start with the same block (the members of a rollout group, the turns of a session)
// have the same block-0 residency on every instance, so each distinct key is probed once.
// (a) k2_first_claim: every request finds or claims its block-0 key in the batch-local index;
//     a claimer zeroes the key's instance mask and lists its slot (one atomic per warp).
// (b) k2_probe_distinct: a warp per listed key looks it up in the W instance tables (lane j
//     takes the instances congruent to j mod 32) and writes the key's instance mask, one
//     64-bit word per two ballots.
// (c) k2_probe_first_gix on the batch-local index writes every request's H row, hbest and
//     hit-list entries from its key's mask, as with the global index.
__global__ void __launch_bounds__(256) k2_first_claim(ProbeArgs a) {
  if (block_error(a.err)) return;
  const int lane = threadIdx.x & 31;
  const int stride = gridDim.x * blockDim.x;
  const uint32_t mw = a.fb.mw;
  for (int r0 = blockIdx.x * blockDim.x + (threadIdx.x & ~31); r0 < a.n; r0 += stride) {
    const int r = r0 + lane;
    bool claimed = false;
    int64_t slot = -1;
    if (r < a.n && a.nb[r] > 0) {
      slot = gix_claim(a.fb, a.keys[a.kbase[r]], &claimed);
      if (slot < 0) set_error(a.err, MISAT_ERR_TABLE_FULL);
    }
    if (claimed)
      for (uint32_t i = 0; i < mw; ++i) a.fb.masks[(size_t)slot * mw + i] = 0ull;
    const unsigned m = __ballot_sync(0xffffffffu, claimed);
    if (m) {
      const int leader = __ffs(m) - 1;
      unsigned long long base = 0;
      if (lane == leader) base = atomicAdd(a.fb_count, (unsigned long long)__popc(m));
      base = __shfl_sync(0xffffffffu, base, leader);
      if (claimed) a.fb_list[base + __popc(m & lanemask_lt())] = (int32_t)slot;
    }
  }
}

constexpr int kDistIlp = 4;  // tables per lane with their home sectors in flight together

__global__ void __launch_bounds__(256) k2_probe_distinct(ProbeArgs a) {
  __shared__ Bucket* s_tab[kMaxW];
  __shared__ uint32_t s_lg[kMaxW];
  if (block_error(a.err)) return;
  for (int w = threadIdx.x; w < a.W; w += blockDim.x) {
    s_tab[w] = a.desc[w].tab;
    s_lg[w] = a.desc[w].log2nb;
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int nd = (int)*a.fb_count;
  const uint32_t mw = a.fb.mw;
  unsigned long long probes = 0, reads = 0;
  for (int d = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; d < nd; d += (gridDim.x * blockDim.x) >> 5) {
    const int64_t slot = a.fb_list[d];
    const uint64_t key = a.fb.keys[slot];
    for (int w0 = 0; w0 < a.W; w0 += 32 * kDistIlp) {
      // the home-bucket sectors of the lane's kDistIlp tables are requested before any is
      // examined; a full home bucket without the key continues its probe sequence after
      ulonglong2 k01[kDistIlp], k23[kDistIlp];
#pragma unroll
      for (int i = 0; i < kDistIlp; ++i) {
        const int w = w0 + 32 * i + lane;
        k01[i] = make_ulonglong2(kEmpty, kEmpty);
        k23[i] = k01[i];
        if (w < a.W) {
          const ulonglong2* p = reinterpret_cast<const ulonglong2*>(s_tab[w][home_bucket(key, s_lg[w])].key);
          k01[i] = __ldg(p);
          k23[i] = __ldg(p + 1);
        }
      }
#pragma unroll
      for (int i = 0; i < kDistIlp; ++i) {
        const int w = w0 + 32 * i + lane;
        int h = 0;
        if (w < a.W) {
          h = (k01[i].x == key) | (k01[i].y == key) | (k23[i].x == key) | (k23[i].y == key);
          const bool open =
              (k01[i].x == kEmpty) | (k01[i].y == kEmpty) | (k23[i].x == kEmpty) | (k23[i].y == kEmpty);
          uint32_t rd = 1;
          if (!h && !open) {
            InstDesc dd;
            dd.tab = s_tab[w];
            dd.log2nb = s_lg[w];
            h = table_contains_from(dd, key, (home_bucket(key, dd.log2nb) + 1) & ((1u << dd.log2nb) - 1), &rd);
          }
          probes += 1;
          reads += rd;
        }
        const unsigned m = __ballot_sync(0xffffffffu, h);
        if (lane == 0) {
          const int wb = w0 + 32 * i;
          if (wb < a.W) {
            unsigned* mw32 = reinterpret_cast<unsigned*>(a.fb.masks + (size_t)slot * mw);
            mw32[wb >> 5] = m;  // 32-bit halves of the little-endian 64-bit mask words
          }
        }
      }
    }
  }
  block_add_stats(a.stats, probes, reads);
}

// Phase 2: a group of kSG lanes per hit pair.  H is the largest h in [1, nb] with block h-1
// resident, and residency is prefix-closed, so "block h-1 resident" holds exactly for
// h <= H.  Each step the lanes test kSG points spread over the current interval [lo, hi]
// (the last one at hi) with one table lookup each; the points that hold form a prefix, so
// one ballot leaves an interval kSG times shorter: about log_kSG(nb) dependent lookups per
// pair instead of log_2(nb).  Points that repeat (short intervals) are tested once.
constexpr int kSG = 16;

__global__ void __launch_bounds__(256) k2_probe_search(ProbeArgs a) {
  if (block_error(a.err)) return;
  const unsigned nh = *a.n_hits;
  const unsigned lim = (int64_t)nh < a.hits_cap ? nh : (unsigned)a.hits_cap;
  const int lane = threadIdx.x & 31;
  const int gl = lane & (kSG - 1);
  const int g0 = lane & ~(kSG - 1);
  const unsigned gmask = ((1u << kSG) - 1) << g0;
  unsigned long long probes = 0, reads = 0;
  const unsigned groups = (gridDim.x * blockDim.x) / kSG;
  for (unsigned i = (blockIdx.x * blockDim.x + threadIdx.x) / kSG; i < lim; i += groups) {
    const int2 pr = a.hits[i];
    const int r = pr.x, w = pr.y;
    const int32_t nb = a.nb[r];
    const uint64_t* k = a.keys + a.kbase[r];
    const InstDesc d = a.desc[w];
    int32_t lo = 1, hi = nb;  // H in [lo, hi]; block 0 is resident
    uint32_t rd = 0;
    while (lo < hi) {
      const int64_t span = hi - lo;
      // point of lane gl: lo + ceil((gl + 1) * span / kSG), increasing, the last one = hi
      const int32_t h = lo + (int32_t)(((int64_t)(gl + 1) * span + kSG - 1) / kSG);
      const int32_t hprev = gl == 0 ? lo : lo + (int32_t)(((int64_t)gl * span + kSG - 1) / kSG);
      bool res = false;
      if (h != hprev) {
        probes += 1;
        res = table_contains(d, k[h - 1], &rd) != 0;
      }
      // repeated points take the answer of the lane that tested them
      const unsigned tested = __ballot_sync(gmask, h != hprev) >> g0;
      const unsigned yes = __ballot_sync(gmask, res) >> g0;
      // lanes in increasing point order: the largest tested point that holds, and the
      // smallest tested point that does not
      const int last_yes = yes ? 31 - __clz(yes) : -1;
      const unsigned no = tested & ~yes;
      const int first_no = no ? __ffs(no) - 1 : kSG;
      const int32_t nlo = last_yes >= 0 ? __shfl_sync(gmask, h, g0 + last_yes) : lo;
      const int32_t nhi = first_no < kSG ? __shfl_sync(gmask, h, g0 + first_no) - 1 : hi;
      lo = nlo;
      hi = nhi;
    }
    if (gl == 0) {
      a.H[(int64_t)r * a.W + w] = (uint16_t)lo;
      atomicMax(a.hbest + r, ((uint32_t)lo << 16) | (65535u - (uint32_t)w));
    }
    reads += rd;
  }
  block_add_stats(a.stats_search, probes, reads);
}

// Phase 1 through the global index: a warp takes 32 requests, each lane looks up the
// block-0 key of one of them (one lookup answers every instance) and the masks go to shared
// memory.  The warp's 32 H rows are one contiguous run of 32W u16 (64W bytes, 16-byte
// aligned), written as 16-byte stores of eight entries (H = 1 where the bit is set) spread
// over the lanes; each set bit of a request with at least two blocks also becomes a hit
// pair, at its request's base (one atomic per warp) plus the rank of the bit in the mask.
__global__ void __launch_bounds__(256) k2_probe_first_gix(ProbeArgs a) {
  extern __shared__ unsigned long long s_gm[];  // [warps][32][mw] masks, then [warps][32] (nb, base)
  if (block_error(a.err)) return;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int wpb = blockDim.x >> 5;
  const uint32_t mw = a.gix.mw;
  unsigned long long* sm = s_gm + (size_t)wid * 32 * mw;
  int2* s_nbb = reinterpret_cast<int2*>(s_gm + (size_t)wpb * 32 * mw) + wid * 32;
  unsigned long long probes = 0, reads = 0;
  const int groups = (a.n + 31) >> 5;
  const int W = a.W;
  for (int grp = blockIdx.x * wpb + wid; grp < groups; grp += gridDim.x * wpb) {
    const int r = grp * 32 + lane;
    int nb = 0;
    int64_t slot = -1;
    if (r < a.n) {
      nb = a.nb[r];
      if (nb > 0) {
        uint32_t rd = 0;
        slot = gix_find(a.gix, a.keys[a.kbase[r]], &rd);
        probes += 1;
        reads += rd;
      }
    }
    int bits = 0, wmin = INT32_MAX;
    for (uint32_t i = 0; i < mw; ++i) {
      const unsigned long long m = slot >= 0 ? __ldg(a.gix.masks + (size_t)slot * mw + i) : 0ull;
      sm[lane * mw + i] = m;
      bits += __popcll(m);
      if (m && wmin == INT32_MAX) wmin = 64 * (int)i + __ffsll((long long)m) - 1;
    }
    if (r < a.n) a.hbest[r] = wmin < W ? (1u << 16) | (65535u - (uint32_t)wmin) : 65535u;
    // hit-list positions: one atomic per warp
    const int nh = nb > 1 ? bits : 0;
    int incl = nh;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    const int tot = __shfl_sync(0xffffffffu, incl, 31);
    unsigned base = 0;
    if (lane == 31 && tot) base = atomicAdd(a.n_hits, (unsigned)tot);
    base = __shfl_sync(0xffffffffu, base, 31) + (unsigned)(incl - nh);
    s_nbb[lane] = make_int2(nb, (int)base);
    __syncwarp();
    // the group's rows: elements e = i*W + w of a run of cnt*W entries
    const int cnt = min(32, a.n - grp * 32);
    const int64_t run = (int64_t)cnt * W;
    uint16_t* rows = a.H + (int64_t)grp * 32 * W;
    const int64_t n8 = (run + 7) >> 3;
    if ((W & 7) == 0) {
      // eight entries of one row per chunk: one mask byte gives them all
      const int cpr = W >> 3;  // chunks per row
      for (int c8 = lane; c8 < (int)n8; c8 += 32) {
        const int i = c8 / cpr;
        const int w0 = (c8 - i * cpr) << 3;
        const unsigned long long* mi = sm + i * mw;
        const uint32_t b8 = (uint32_t)(mi[w0 >> 6] >> (w0 & 63)) & 0xffu;
        uint4 v;
        v.x = (b8 & 1u) | (((b8 >> 1) & 1u) << 16);
        v.y = ((b8 >> 2) & 1u) | (((b8 >> 3) & 1u) << 16);
        v.z = ((b8 >> 4) & 1u) | (((b8 >> 5) & 1u) << 16);
        v.w = ((b8 >> 6) & 1u) | (((b8 >> 7) & 1u) << 16);
        *reinterpret_cast<uint4*>(rows + ((int64_t)c8 << 3)) = v;
        if (b8) {
          const int2 q = s_nbb[i];
          if (q.x > 1) {
            // rank of the chunk's first entry among the row's set bits
            unsigned rank = (unsigned)__popcll(mi[w0 >> 6] & ((1ull << (w0 & 63)) - 1ull));
            for (int j = 0; j < (w0 >> 6); ++j) rank += (unsigned)__popcll(mi[j]);
            uint32_t rest = b8;
            while (rest) {
              const int bit = __ffs(rest) - 1;
              rest &= rest - 1;
              const unsigned p = (unsigned)q.y + rank++;
              if ((int64_t)p < a.hits_cap)
                a.hits[p] = make_int2(grp * 32 + i, w0 + bit);
              else
                set_error(a.err, MISAT_ERR_TABLE_FULL);
            }
          }
        }
      }
      __syncwarp();
      continue;
    }
    for (int64_t c8 = lane; c8 < n8; c8 += 32) {
      const int64_t e0 = c8 << 3;
      int i = (int)(e0 / W);
      int w = (int)(e0 - (int64_t)i * W);
      uint32_t packed[4] = {0u, 0u, 0u, 0u};
      const int ne = run - e0 < 8 ? (int)(run - e0) : 8;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (k >= ne) break;
        const unsigned long long* mi = sm + i * mw;
        const uint32_t wd = (uint32_t)w >> 6;
        const unsigned long long m = mi[wd];
        const unsigned long long below = m & ((1ull << (w & 63)) - 1ull);
        if ((m >> (w & 63)) & 1ull) {
          packed[k >> 1] |= 1u << (16 * (k & 1));
          const int2 q = s_nbb[i];
          if (q.x > 1) {
            unsigned rank = (unsigned)__popcll(below);
            for (uint32_t j = 0; j < wd; ++j) rank += (unsigned)__popcll(mi[j]);
            const unsigned p = (unsigned)q.y + rank;
            if ((int64_t)p < a.hits_cap)
              a.hits[p] = make_int2(grp * 32 + i, w);
            else
              set_error(a.err, MISAT_ERR_TABLE_FULL);
          }
        }
        if (++w == W) {
          w = 0;
          ++i;
        }
      }
      if (ne == 8) {
        *reinterpret_cast<uint4*>(rows + e0) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
      } else {
#pragma unroll
        for (int k = 0; k < 8; ++k)
          if (k < ne) rows[e0 + k] = (uint16_t)((packed[k >> 1] >> (16 * (k & 1))) & 0xffffu);
      }
    }
    __syncwarp();
  }
  block_add_stats(a.stats, probes, reads);
}

void launch_probe_first(const ProbeArgs& a, int num_sms, cudaStream_t st) {
  const int64_t total = (int64_t)a.n * a.W;
  if (total <= 0) return;
  const int groups = (a.n + 31) / 32;
  const int gblocks = (groups + 7) / 8;
  const size_t gsmem = 8 * 32 * ((a.gix.keys ? a.gix.mw : a.fb.mw) * sizeof(unsigned long long) + sizeof(int2));
  const int gres = resident_grid<k2_probe_first_gix>(256, gsmem, num_sms);
  const int ggrid = gblocks < gres ? gblocks : gres;
  if (a.gix.keys) {
    k2_probe_first_gix<<<ggrid, 256, 8 * 32 * (a.gix.mw * sizeof(unsigned long long) + sizeof(int2)), st>>>(a);
    return;
  }
  // per-instance tables: the context allocates the batch-local index with the tables
  k2_first_claim<<<ggrid, 256, 0, st>>>(a);
  k2_probe_distinct<<<num_sms * 8, 256, 0, st>>>(a);  // two waves: measured faster than one for this pass
  ProbeArgs e = a;
  e.gix = a.fb;
  e.stats = a.stats_fb;
  k2_probe_first_gix<<<ggrid, 256, 8 * 32 * (a.fb.mw * sizeof(unsigned long long) + sizeof(int2)), st>>>(e);
}

void launch_probe_search(const ProbeArgs& a, int num_sms, cudaStream_t st) {
  if ((int64_t)a.n * a.W <= 0) return;
  k2_probe_search<<<resident_grid<k2_probe_search>(256, 0, num_sms), 256, 0, st>>>(a);
}

}  // namespace misat
