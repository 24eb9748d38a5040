// K1: chained 16-token block hash (Sec. 4.5: the router's prefix index is keyed by
// block hashes of the engine's prefix cache).
//
// Key of block j of a prompt:  c_j = mix64(XOR_i mix64(x_i + (i+1)G)) over the
// block's eight 64-bit token pairs, a_j = a_{j-1} G + c_j (a_{-1} = seed),
// k_j = mix64(a_j ^ (j+1)) (+2 if < 2).  The chain step is affine mod 2^64, so a
// warp evaluates 32 consecutive blocks as an inclusive scan of affine maps:
// in-chunk sums s_j = sum_{i<=j} c_i G^{j-i} (Hillis-Steele, multiplier G^d at
// distance d), then a_j = carry G^{j+1} + s_j.
//
// Layout: one warp per request (dynamic work counter).  A chunk of 32 blocks is
// 512 tokens = 2 KiB, read as four fully coalesced 512-byte warp loads of int4;
// a prompt that does not start on a 16-byte boundary is realigned in registers
// (funnel of the lane's int4 and its right neighbour's).  Lanes 4m..4m+3 hold the
// four quarters of one block and combine their partial hashes with two xor
// shuffles.  Keys are written coalesced at keys[floor(tok_off[r]/16) + j].
#include <mutex>

#include "common.cuh"
#include "kernels.h"

namespace misat {

namespace {

__host__ __device__ constexpr uint64_t gold_pow(int k) {
  uint64_t r = 1;
  for (int i = 0; i < k; ++i) r *= kGold;
  return r;
}

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ int4 shfl_int4(int4 v, int src) {
  int4 o;
  o.x = __shfl_sync(kFull, v.x, src);
  o.y = __shfl_sync(kFull, v.y, src);
  o.z = __shfl_sync(kFull, v.z, src);
  o.w = __shfl_sync(kFull, v.w, src);
  return o;
}

__device__ __forceinline__ int4 shfl_down_int4(int4 v) {
  int4 o;
  o.x = __shfl_down_sync(kFull, v.x, 1);
  o.y = __shfl_down_sync(kFull, v.y, 1);
  o.z = __shfl_down_sync(kFull, v.z, 1);
  o.w = __shfl_down_sync(kFull, v.w, 1);
  return o;
}

// The four tokens at word offset `off` (0..3) of the 8-word window (cur, nxt).
__device__ __forceinline__ int4 funnel(int4 cur, int4 nxt, int off) {
  int4 t;
  if (off == 1) {
    t.x = cur.y; t.y = cur.z; t.z = cur.w; t.w = nxt.x;
  } else if (off == 2) {
    t.x = cur.z; t.y = cur.w; t.z = nxt.x; t.w = nxt.y;
  } else {
    t.x = cur.w; t.y = nxt.x; t.z = nxt.y; t.w = nxt.z;
  }
  return t;
}

__device__ __forceinline__ int4 load_tok4(const int4* base, int64_t idx, int64_t n_int4) {
  if (idx < n_int4) return ld_stream_v4(base + idx);
  return make_int4(0, 0, 0, 0);
}

}  // namespace

__global__ void __launch_bounds__(256) k1_block_hash(HashArgs a) {
  if (*a.err) return;
  const int lane = threadIdx.x & 31;
  const int q = lane & 3;
  const int64_t n_int4 = (a.n_tokens + 3) >> 2;
  const int4* tok4 = reinterpret_cast<const int4*>(a.tokens);
  // G^(lane+1): multiplier of the incoming carry for block `lane` of a chunk
  uint64_t pw = kGold;
  for (int i = 0; i < lane; ++i) pw *= kGold;
  const uint64_t addA = (uint64_t)(2 * q + 1) * kGold;
  const uint64_t addB = (uint64_t)(2 * q + 2) * kGold;

  while (true) {
    int r = 0;
    if (lane == 0) r = (int)atomicAdd(a.work, 1u);
    r = __shfl_sync(kFull, r, 0);
    if (r >= a.n) break;
    const int64_t t0 = a.tok_off[r];
    const int64_t t1 = a.tok_off[r + 1];
    const int32_t nb = (int32_t)((t1 - t0) >> 4);
    const int64_t kb = t0 >> 4;
    if (nb <= 0) continue;
    const int64_t q0 = t0 >> 2;
    const int off = (int)(t0 & 3);
    uint64_t carry = a.seed;
    const int n_chunks = (nb + 31) >> 5;

    int4 v[4], ex;
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = load_tok4(tok4, q0 + 32 * i + lane, n_int4);
    ex = (off != 0 && lane == 0) ? load_tok4(tok4, q0 + 128, n_int4) : make_int4(0, 0, 0, 0);

    for (int c = 0; c < n_chunks; ++c) {
      // prefetch the next chunk while this one is hashed
      int4 vn[4], exn = make_int4(0, 0, 0, 0);
      const bool more = (c + 1) < n_chunks;
      const int64_t nbase = q0 + 128ll * (c + 1);
#pragma unroll
      for (int i = 0; i < 4; ++i) vn[i] = more ? load_tok4(tok4, nbase + 32 * i + lane, n_int4) : make_int4(0, 0, 0, 0);
      if (more && off != 0 && lane == 0) exn = load_tok4(tok4, nbase + 128, n_int4);

      // pre-mix XOR of block 8i + lane/4 after sub-iteration i (same in its 4 lanes); lane
      // 4m + i' keeps the one of sub-iteration i' = lane % 4, i.e. block 8(lane%4) + lane/4
      uint64_t pkeep = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        int4 t = v[i];
        if (off != 0) {
          int4 nxt = shfl_down_int4(v[i]);
          int4 wrap = shfl_int4(i < 3 ? v[i + 1] : ex, 0);
          if (lane == 31) nxt = wrap;
          t = funnel(v[i], nxt, off);
        }
        // this lane holds tokens 4q..4q+3 of block 8i + lane/4 of the chunk
        const uint64_t xa = (uint64_t)(uint32_t)t.x | ((uint64_t)(uint32_t)t.y << 32);
        const uint64_t xb = (uint64_t)(uint32_t)t.z | ((uint64_t)(uint32_t)t.w << 32);
        uint64_t p = mix64(xa + addA) ^ mix64(xb + addB);
        p ^= __shfl_xor_sync(kFull, p, 1);
        p ^= __shfl_xor_sync(kFull, p, 2);
        if (q == i) pkeep = p;
      }
      // one finishing mix per lane, then block j moves to lane j (it sits on lane 4(j%8) + j/8)
      const uint64_t cown = mix64(pkeep);
      const uint64_t cmine = __shfl_sync(kFull, cown, 4 * (lane & 7) + (lane >> 3));
      const int cnt = min(32, nb - 32 * c);
      uint64_t s = lane < cnt ? cmine : 0;
      {
        uint64_t t = __shfl_up_sync(kFull, s, 1);
        if (lane >= 1) s += t * gold_pow(1);
        t = __shfl_up_sync(kFull, s, 2);
        if (lane >= 2) s += t * gold_pow(2);
        t = __shfl_up_sync(kFull, s, 4);
        if (lane >= 4) s += t * gold_pow(4);
        t = __shfl_up_sync(kFull, s, 8);
        if (lane >= 8) s += t * gold_pow(8);
        t = __shfl_up_sync(kFull, s, 16);
        if (lane >= 16) s += t * gold_pow(16);
      }
      const uint64_t av = carry * pw + s;
      uint64_t key = mix64(av ^ (uint64_t)(32 * c + lane + 1));
      key += key < 2 ? 2 : 0;
      const int64_t dst = kb + 32ll * c + lane;
      if (lane < cnt && dst < a.keys_cap) a.keys[dst] = key;
      carry = __shfl_sync(kFull, av, 31);
#pragma unroll
      for (int i = 0; i < 4; ++i) v[i] = vn[i];
      ex = exn;
    }
  }
}

void launch_block_hash(const HashArgs& a, int num_sms, cudaStream_t st) {
  int grid = num_sms * 8;  // 8 CTAs x 8 warps per SM; warps pull requests dynamically
  k1_block_hash<<<grid, 256, 0, st>>>(a);
}

// ---------------------------------------------------------------------------
// Allocation-free block hashing.
//
// Some callers of this library cannot allocate device memory: an inference engine
// that has already handed all free HBM to its KV-cache pool (a new cudaMalloc would
// fail, or fragment and shrink that pool), or a hook that runs inside another
// framework's allocator or memory-accounting scope, where new device allocations are
// not allowed.  misat_block_hash_noalloc serves them: it computes the same chained
// block keys as the routing path and allocates nothing.  Its only scratch -- the
// per-request key offsets, a work counter and an error word -- lives in the
// file-scope array below, which every GPU that loads this library holds
// (about 513 KiB) until the process exits.

// scratch layout in 8-byte words: [0] work counter (low 32 bits) | [1] error word |
// [2] total blocks | [3..7] unused | [8 .. 8 + max requests] exclusive key offsets
constexpr int kNoAllocMaxRequests = MISAT_NOALLOC_MAX_REQUESTS;
constexpr int kNoAllocWords = 8 + kNoAllocMaxRequests + 1;
static __device__ __align__(256) unsigned long long g_noalloc_scratch[kNoAllocWords];

namespace {

// One CTA: clear the counters, validate the offsets and write the exclusive prefix of
// floor(L_r / 16) (compact key positions) into the scratch array.
__global__ void __launch_bounds__(1024) k1na_offsets(const int64_t* tok_off, int32_t n, int64_t n_tokens,
                                                     int64_t keys_cap, unsigned long long* scratch) {
  __shared__ long long s_warp[32];
  __shared__ int s_bad;
  const int t = threadIdx.x, lane = t & 31, wid = t >> 5;
  if (t == 0) {
    scratch[0] = 0;
    scratch[1] = 0;
    s_bad = 0;
  }
  __syncthreads();
  const int per = (n + blockDim.x - 1) / blockDim.x;
  const int lo = t * per, hi = min(n, lo + per);
  long long local = 0;
  bool bad = false;
  for (int r = lo; r < hi; ++r) {
    const int64_t t0 = tok_off[r], t1 = tok_off[r + 1];
    if (t0 < 0 || t1 < t0 || t1 > n_tokens || (t1 - t0) >= (1 << 20)) bad = true;
    local += (t1 - t0) >> 4;
  }
  if (t == 0 && tok_off[0] != 0) bad = true;
  if (t == 0 && tok_off[n] != n_tokens) bad = true;
  if (bad) atomicOr(&s_bad, 1);
  long long incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long v = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) s_warp[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    const long long v = s_warp[lane];
    long long sc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long u = __shfl_up_sync(kFull, sc, o);
      if (lane >= o) sc += u;
    }
    s_warp[lane] = sc - v;
  }
  __syncthreads();
  long long run = s_warp[wid] + incl - local;
  for (int r = lo; r < hi; ++r) {
    scratch[8 + r] = (unsigned long long)run;
    run += (tok_off[r + 1] - tok_off[r]) >> 4;
  }
  if (t == blockDim.x - 1) {
    scratch[8 + n] = (unsigned long long)run;
    scratch[2] = (unsigned long long)run;
  }
  __syncthreads();
  if (t == 0) {
    const long long total = (long long)scratch[2];
    if (s_bad || total > keys_cap) scratch[1] = (unsigned long long)(long long)MISAT_ERR_INVALID_ARG;
  }
}

// The block hash of k1_block_hash with compact output positions: block j of request r
// goes to keys[off[r] + j] (off = the exclusive prefix above).
__global__ void __launch_bounds__(256) k1na_hash(const int64_t* tok_off, const int32_t* tokens, int64_t n_tokens,
                                                 int32_t n, uint64_t seed, uint64_t* keys,
                                                 unsigned long long* scratch) {
  if (scratch[1]) return;
  unsigned* work = reinterpret_cast<unsigned*>(scratch);
  const unsigned long long* off_r = scratch + 8;
  const int lane = threadIdx.x & 31;
  const int q = lane & 3;
  const int64_t n_int4 = (n_tokens + 3) >> 2;
  const int4* tok4 = reinterpret_cast<const int4*>(tokens);
  uint64_t pw = kGold;
  for (int i = 0; i < lane; ++i) pw *= kGold;
  const uint64_t addA = (uint64_t)(2 * q + 1) * kGold;
  const uint64_t addB = (uint64_t)(2 * q + 2) * kGold;
  while (true) {
    int r = 0;
    if (lane == 0) r = (int)atomicAdd(work, 1u);
    r = __shfl_sync(kFull, r, 0);
    if (r >= n) break;
    const int64_t t0 = tok_off[r];
    const int32_t nb = (int32_t)((tok_off[r + 1] - t0) >> 4);
    if (nb <= 0) continue;
    const int64_t kb = (int64_t)off_r[r];
    const int64_t q0 = t0 >> 2;
    const int off = (int)(t0 & 3);
    uint64_t carry = seed;
    const int n_chunks = (nb + 31) >> 5;
    for (int c = 0; c < n_chunks; ++c) {
      const int64_t base = q0 + 128ll * c;
      int4 v[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) v[i] = load_tok4(tok4, base + 32 * i + lane, n_int4);
      const int4 ex = (off != 0 && lane == 0) ? load_tok4(tok4, base + 128, n_int4) : make_int4(0, 0, 0, 0);
      uint64_t cmine = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        int4 t = v[i];
        if (off != 0) {
          int4 nxt = shfl_down_int4(v[i]);
          const int4 wrap = shfl_int4(i < 3 ? v[i + 1] : ex, 0);
          if (lane == 31) nxt = wrap;
          t = funnel(v[i], nxt, off);
        }
        const uint64_t xa = (uint64_t)(uint32_t)t.x | ((uint64_t)(uint32_t)t.y << 32);
        const uint64_t xb = (uint64_t)(uint32_t)t.z | ((uint64_t)(uint32_t)t.w << 32);
        uint64_t p = mix64(xa + addA) ^ mix64(xb + addB);
        p ^= __shfl_xor_sync(kFull, p, 1);
        p ^= __shfl_xor_sync(kFull, p, 2);
        const uint64_t cb = mix64(p);
        const uint64_t got = __shfl_sync(kFull, cb, 4 * (lane & 7));
        if ((lane >> 3) == i) cmine = got;
      }
      const int cnt = min(32, nb - 32 * c);
      uint64_t s = lane < cnt ? cmine : 0;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const uint64_t u = __shfl_up_sync(kFull, s, d);
        if (lane >= d) s += u * gold_pow(d);
      }
      const uint64_t av = carry * pw + s;
      uint64_t key = mix64(av ^ (uint64_t)(32 * c + lane + 1));
      key += key < 2 ? 2 : 0;
      if (lane < cnt) keys[kb + 32ll * c + lane] = key;
      carry = __shfl_sync(kFull, av, 31);
    }
  }
}

std::mutex g_noalloc_mu;
unsigned long long* g_noalloc_ptr[256];  // device address of the scratch array, per device
int g_noalloc_sms[256];

// Per device, once, with that device current: the device address of the scratch array.
int noalloc_setup(unsigned long long** scratch, int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) return MISAT_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) {
      cudaGetLastError();
      return MISAT_ERR_CUDA;
    }
    int s = 0;
    if (cudaDeviceGetAttribute(&s, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return MISAT_ERR_CUDA;
    g_noalloc_sms[dev] = s;
    g_noalloc_ptr[dev] = reinterpret_cast<unsigned long long*>(p);
  }
  *scratch = g_noalloc_ptr[dev];
  *sms = g_noalloc_sms[dev];
  return MISAT_OK;
}

}  // namespace
}  // namespace misat

extern "C" int misat_block_hash_noalloc(const int64_t* tok_off, const int32_t* tokens, int32_t n, int64_t n_tokens,
                                        uint64_t seed, uint64_t* keys_out, int64_t keys_cap, void* cuda_stream) {
  using namespace misat;
  if (n < 0 || n_tokens < 0 || keys_cap < 0) return MISAT_ERR_INVALID_ARG;
  if (n > kNoAllocMaxRequests) return MISAT_ERR_BATCH_TOO_LARGE;
  if (n == 0) return MISAT_OK;
  if (!tok_off || (keys_cap > 0 && !keys_out)) return MISAT_ERR_INVALID_ARG;
  if (n_tokens > 0 && (!tokens || ((uintptr_t)tokens & 15) != 0)) return MISAT_ERR_INVALID_ARG;
  unsigned long long* scratch = nullptr;
  int sms = 1;
  int rc = noalloc_setup(&scratch, &sms);
  if (rc) return rc;
  cudaStream_t st = (cudaStream_t)cuda_stream;
  k1na_offsets<<<1, 1024, 0, st>>>(tok_off, n, n_tokens, keys_cap, scratch);
  k1na_hash<<<sms * 8, 256, 0, st>>>(tok_off, tokens, n_tokens, n, seed, keys_out, scratch);
  if (cudaGetLastError() != cudaSuccess) return MISAT_ERR_CUDA;
  unsigned long long err = 0;
  if (cudaMemcpyAsync(&err, scratch + 1, sizeof(err), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return MISAT_ERR_CUDA;
  return (int)(long long)err;
}
