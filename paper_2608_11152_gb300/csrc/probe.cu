// K2: longest cached prefix H_rw of every request on every instance (Sec. 3.2, Eq. 1;
// Sec. 4.5: "the longest matching prompt-block hash determines the reusable prefix").
//
// Every instance index is prefix-closed (a commit writes whole prefixes with one
// tick and eviction takes the deepest block of a tick first), so "block h-1 is
// resident" is monotone in h and H is found by binary search.
//
// Phase 1 (k2_probe_first): one thread per (r, w) pair probes block 0.  A probe
// reads one 32-byte sector (the four keys of the home bucket) and continues to
// the next bucket only when the bucket is full without a match.  Most pairs miss
// and finish after one sector.  Pairs with block 0 resident and at least two
// blocks are appended to a compact hit list (warp-aggregated).
// Phase 2 (k2_probe_search): one thread per hit pair probes the last block
// (fully cached prefixes finish there), then binary-searches [1, nb-1].
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

__global__ void __launch_bounds__(256) k2_probe_first(ProbeArgs a) {
  __shared__ Bucket* s_tab[kMaxW];
  __shared__ uint32_t s_lg[kMaxW];
  if (block_error(a.err)) return;
  for (int w = threadIdx.x; w < a.W; w += blockDim.x) {
    s_tab[w] = a.desc[w].tab;
    s_lg[w] = a.desc[w].log2nb;
  }
  __syncthreads();
  const int64_t total = (int64_t)a.n * a.W;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  unsigned long long probes = 0, reads = 0;
  const int lane = threadIdx.x & 31;
  // the loop trip count is uniform per warp so that ballots see every lane
  const int64_t start = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31);
  for (int64_t base = start; base < total; base += stride) {
    const int64_t p = base + lane;
    bool hit_list = false;
    int r = 0, w = 0;
    if (p < total) {
      r = (int)(p / a.W);
      w = (int)(p - (int64_t)r * a.W);
      const int32_t nb = a.nb[r];
      uint16_t h = 0;
      if (nb > 0) {
        const uint64_t key = a.keys[a.kbase[r]];
        InstDesc d;
        d.tab = s_tab[w];
        d.log2nb = s_lg[w];
        uint32_t rd = 0;
        const int res = table_contains(d, key, &rd);
        probes += 1;
        reads += rd;
        if (res) {
          h = 1;
          hit_list = nb > 1;
        }
      }
      a.H[p] = h;
    }
    const unsigned m = __ballot_sync(0xffffffffu, hit_list);
    if (m) {
      unsigned pos = 0;
      const int leader = __ffs(m) - 1;
      if (lane == leader) pos = atomicAdd(a.n_hits, (unsigned)__popc(m));
      pos = __shfl_sync(0xffffffffu, pos, leader) + __popc(m & lanemask_lt());
      if (hit_list) {
        if ((int64_t)pos < a.hits_cap)
          a.hits[pos] = make_int2(r, w);
        else
          set_error(a.err, MISAT_ERR_TABLE_FULL);
      }
    }
  }
  block_add_stats(a.stats, probes, reads);
}

// Phase 1, sub-warp layout: a group of S lanes (S = min(32, pow2 >= W)) owns one request;
// its block-0 key is read once and broadcast, each lane probes instances w = lane, lane+S,
// ... with up to kIlp independent sector loads in flight before any of them is consumed.
template <int S>
__global__ void __launch_bounds__(256) k2_probe_first_group(ProbeArgs a) {
  constexpr int kIlp = 4;
  __shared__ Bucket* s_tab[kMaxW];
  __shared__ uint32_t s_lg[kMaxW];
  if (block_error(a.err)) return;
  for (int w = threadIdx.x; w < a.W; w += blockDim.x) {
    s_tab[w] = a.desc[w].tab;
    s_lg[w] = a.desc[w].log2nb;
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int sub = lane & (S - 1);
  const int gid = (blockIdx.x * blockDim.x + threadIdx.x) / S;  // group index
  const int ngroups = (gridDim.x * blockDim.x) / S;
  unsigned long long probes = 0, reads = 0;
  // groups per warp iterate in lockstep so that the warp-wide ballots see every lane
  const int warp_first_group = ((blockIdx.x * blockDim.x + (threadIdx.x & ~31)) / S);
  for (int rb = warp_first_group; rb < a.n; rb += ngroups) {
    const int r = rb + (gid - warp_first_group);
    const bool live = r < a.n;
    int32_t nb = 0;
    uint64_t key = 0;
    if (live) {
      nb = a.nb[r];
      if (nb > 0) key = a.keys[a.kbase[r]];
    }
    for (int w0 = 0; w0 < a.W; w0 += S * kIlp) {
      int res[kIlp];
      uint32_t rd[kIlp];
#pragma unroll
      for (int i = 0; i < kIlp; ++i) {
        const int w = w0 + i * S + sub;
        res[i] = 0;
        rd[i] = 0;
        if (live && nb > 0 && w < a.W) {
          InstDesc d;
          d.tab = s_tab[w];
          d.log2nb = s_lg[w];
          res[i] = table_contains(d, key, &rd[i]);
        }
      }
#pragma unroll
      for (int i = 0; i < kIlp; ++i) {
        const int w = w0 + i * S + sub;
        const bool valid = live && w < a.W;
        if (valid) {
          a.H[(int64_t)r * a.W + w] = (uint16_t)res[i];
          if (nb > 0) {
            probes += 1;
            reads += rd[i];
          }
        }
        const bool hl = valid && res[i] && nb > 1;
        const unsigned m = __ballot_sync(0xffffffffu, hl);
        if (m) {
          unsigned pos = 0;
          const int leader = __ffs(m) - 1;
          if (lane == leader) pos = atomicAdd(a.n_hits, (unsigned)__popc(m));
          pos = __shfl_sync(0xffffffffu, pos, leader) + __popc(m & lanemask_lt());
          if (hl) {
            if ((int64_t)pos < a.hits_cap)
              a.hits[pos] = make_int2(r, w);
            else
              set_error(a.err, MISAT_ERR_TABLE_FULL);
          }
        }
      }
    }
  }
  block_add_stats(a.stats, probes, reads);
}

__global__ void __launch_bounds__(256) k2_probe_search(ProbeArgs a) {
  if (block_error(a.err)) return;
  const unsigned nh = *a.n_hits;
  const unsigned lim = (int64_t)nh < a.hits_cap ? nh : (unsigned)a.hits_cap;
  unsigned long long probes = 0, reads = 0;
  for (unsigned i = blockIdx.x * blockDim.x + threadIdx.x; i < lim; i += gridDim.x * blockDim.x) {
    const int2 pr = a.hits[i];
    const int r = pr.x, w = pr.y;
    const int32_t nb = a.nb[r];
    const uint64_t* k = a.keys + a.kbase[r];
    const InstDesc d = a.desc[w];
    uint32_t rd = 0;
    int32_t h;
    probes += 1;
    if (table_contains(d, k[nb - 1], &rd)) {
      h = nb;
    } else {
      int32_t lo = 1, hi = nb - 1;  // H in [lo, hi]: block 0 resident, block nb-1 not
      while (lo < hi) {
        const int32_t mid = (lo + hi + 1) >> 1;
        probes += 1;
        if (table_contains(d, k[mid - 1], &rd))
          lo = mid;
        else
          hi = mid - 1;
      }
      h = lo;
    }
    reads += rd;
    a.H[(int64_t)r * a.W + w] = (uint16_t)h;
  }
  block_add_stats(a.stats_search, probes, reads);
}

void launch_probe_first(const ProbeArgs& a, int num_sms, cudaStream_t st) {
  const int64_t total = (int64_t)a.n * a.W;
  if (total <= 0) return;
  if (a.flat) {
    int64_t blocks = (total + 255) / 256;
    int grid = (int)(blocks < (int64_t)num_sms * 8 ? blocks : (int64_t)num_sms * 8);
    k2_probe_first<<<grid, 256, 0, st>>>(a);
    return;
  }
  int S = 1;
  while (S < a.W && S < 32) S <<= 1;
  const int64_t threads = (int64_t)a.n * S;
  int64_t blocks = (threads + 255) / 256;
  const int grid = (int)(blocks < (int64_t)num_sms * 8 ? blocks : (int64_t)num_sms * 8);
  switch (S) {
    case 1: k2_probe_first_group<1><<<grid, 256, 0, st>>>(a); break;
    case 2: k2_probe_first_group<2><<<grid, 256, 0, st>>>(a); break;
    case 4: k2_probe_first_group<4><<<grid, 256, 0, st>>>(a); break;
    case 8: k2_probe_first_group<8><<<grid, 256, 0, st>>>(a); break;
    case 16: k2_probe_first_group<16><<<grid, 256, 0, st>>>(a); break;
    default: k2_probe_first_group<32><<<grid, 256, 0, st>>>(a); break;
  }
}

void launch_probe_search(const ProbeArgs& a, int num_sms, cudaStream_t st) {
  if ((int64_t)a.n * a.W <= 0) return;
  k2_probe_search<<<num_sms * 4, 256, 0, st>>>(a);
}

}  // namespace misat
