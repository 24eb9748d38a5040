// K1: chained 16-token block hash (Sec. 4.4: the router's prefix index is keyed by
// block hashes of the engine's prefix cache).
//
// Key of block j of a prompt:  c_j = mix64(XOR_i (x_i + (i+1)G) M) over the block's
// eight 64-bit token pairs x_i (M odd: a bijection of each word), a_j = a_{j-1} G + c_j
// (a_{-1} = seed),
// k_j = mix64(a_j ^ (j+1)) (+2 if < 2).  The chain step is affine mod 2^64, so a
// warp evaluates 32 consecutive blocks as an inclusive scan of affine maps:
// in-chunk sums s_j = sum_{i<=j} c_i G^{j-i} (Hillis-Steele, multiplier G^d at
// distance d), then a_j = carry G^{j+1} + s_j.
//
// Layout: one warp per request (dynamic work counter).  A chunk of 32 blocks is
// 512 tokens = 2 KiB, read as four fully coalesced 512-byte warp loads of int4
// (the next chunk's loads are issued before the current one is hashed).  In
// sub-row i of a chunk, lane 4m+q holds tokens 4q..4q+3 of block 8i+m.  A prompt
// that does not start on a 16-byte boundary is realigned in registers: the
// misalignment (0..3 words) is the same for the whole warp, so the chunk loop is
// specialised on it and only the 1..3 words a lane needs from its right neighbour
// are shuffled.  The four lanes of a block combine their partial XORs once per
// chunk with a two-step reduce-scatter (lane 4m+q ends with block 8q+m), then one
// shuffle moves block j to lane j for the scan.  Keys are written coalesced.
//
// Per block: eight 64-bit multiplies and two 64-bit mixes (the content hash's and the
// key's), so the kernel streams tokens near the memory roof; the structure above keeps
// the instructions around them few.
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
constexpr uint64_t kWordMul = 0x94d049bb133111ebull;  // the content hash's odd word multiplier

__device__ __forceinline__ int4 load_tok4(const int4* base, int64_t idx, int64_t n_int4) {
  if (idx < n_int4) return ld_stream_v4(base + idx);
  return make_int4(0, 0, 0, 0);
}

// Per-lane constants of the chunk loop.
struct LaneConst {
  int lane;
  int src;          // lane that holds block `lane` after the reduce-scatter
  bool b0, b1;      // bits of the quarter index q = lane & 3
  uint64_t pw;      // G^(lane+1): multiplier of the incoming carry for block `lane`
  uint64_t addA;    // (2q+1) G: increment of the lane's first token pair
  uint64_t addB;    // (2q+2) G: increment of its second pair
};

__device__ __forceinline__ LaneConst lane_const() {
  LaneConst c;
  c.lane = threadIdx.x & 31;
  const int q = c.lane & 3;
  c.src = 4 * (c.lane & 7) + (c.lane >> 3);
  c.b0 = (q & 1) != 0;
  c.b1 = (q & 2) != 0;
  uint64_t pw = kGold;
  for (int i = 0; i < c.lane; ++i) pw *= kGold;
  c.pw = pw;
  c.addA = (uint64_t)(2 * q + 1) * kGold;
  c.addB = (uint64_t)(2 * q + 2) * kGold;
  return c;
}

// The four tokens that start OFF words into `cur`, continued by `nxt`.
template <int OFF>
__device__ __forceinline__ int4 align_words(int4 cur, int4 nxt) {
  if (OFF == 1) return make_int4(cur.y, cur.z, cur.w, nxt.x);
  if (OFF == 2) return make_int4(cur.z, cur.w, nxt.x, nxt.y);
  if (OFF == 3) return make_int4(cur.w, nxt.x, nxt.y, nxt.z);
  return cur;
}

// The first OFF words of the int4 that follows this lane's `cur` in memory: lane l+1's
// `cur`, or for lane 31 lane 0's `after` (the first int4 of the next sub-row).
template <int OFF>
__device__ __forceinline__ int4 next_words(int4 cur, int4 after, int lane) {
  int4 nx = make_int4(0, 0, 0, 0);
  const int src = (lane + 1) & 31;
  const bool first = lane == 0;
  if (OFF >= 1) nx.x = __shfl_sync(kFull, first ? after.x : cur.x, src);
  if (OFF >= 2) nx.y = __shfl_sync(kFull, first ? after.y : cur.y, src);
  if (OFF >= 3) nx.z = __shfl_sync(kFull, first ? after.z : cur.z, src);
  return nx;
}

// Keys of one prompt of nb >= 1 full blocks whose first token is word OFF of int4 q0:
// key j goes to out[j] for j < out_lim.
template <int OFF>
__device__ __forceinline__ void hash_chain(const int4* tok4, int64_t n_int4, int64_t q0, int32_t nb, uint64_t seed,
                                           uint64_t* out, int64_t out_lim, const LaneConst& lc) {
  const int lane = lc.lane;
  uint64_t carry = seed;
  const int n_chunks = (nb + 31) >> 5;
  int4 v[4], ex = make_int4(0, 0, 0, 0);
#pragma unroll
  for (int i = 0; i < 4; ++i) v[i] = load_tok4(tok4, q0 + 32 * i + lane, n_int4);
  if (OFF != 0 && lane == 0) ex = load_tok4(tok4, q0 + 128, n_int4);

  for (int c = 0; c < n_chunks; ++c) {
    // issue the next chunk's loads before this chunk is hashed
    const bool more = (c + 1) < n_chunks;
    const int64_t nbase = q0 + 128ll * (c + 1);
    int4 vn[4], exn = make_int4(0, 0, 0, 0);
#pragma unroll
    for (int i = 0; i < 4; ++i) vn[i] = more ? load_tok4(tok4, nbase + 32 * i + lane, n_int4) : make_int4(0, 0, 0, 0);
    if (OFF != 0 && more && lane == 0) exn = load_tok4(tok4, nbase + 128, n_int4);

    // partial XOR of the lane's two multiplied token pairs, per sub-row
    uint64_t p[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      int4 t = v[i];
      if (OFF != 0) t = align_words<OFF>(v[i], next_words<OFF>(v[i], i < 3 ? v[i + 1] : ex, lane));
      const uint64_t xa = (uint64_t)(uint32_t)t.x | ((uint64_t)(uint32_t)t.y << 32);
      const uint64_t xb = (uint64_t)(uint32_t)t.z | ((uint64_t)(uint32_t)t.w << 32);
      p[i] = ((xa + lc.addA) * kWordMul) ^ ((xb + lc.addB) * kWordMul);
    }
    // reduce-scatter over the quad: after the exchange with lane^1 a lane keeps the
    // sub-rows with bit 0 = its q's bit 0, after lane^2 the sub-row i = q: block 8q + m
    uint64_t k0 = lc.b0 ? p[1] : p[0], k1 = lc.b0 ? p[3] : p[2];
    const uint64_t s0 = lc.b0 ? p[0] : p[1], s1 = lc.b0 ? p[2] : p[3];
    k0 ^= __shfl_xor_sync(kFull, s0, 1);
    k1 ^= __shfl_xor_sync(kFull, s1, 1);
    uint64_t kq = lc.b1 ? k1 : k0;
    const uint64_t sq = lc.b1 ? k0 : k1;
    kq ^= __shfl_xor_sync(kFull, sq, 2);
    // finishing mix, then block j moves to lane j
    const uint64_t cmine = __shfl_sync(kFull, mix64(kq), lc.src);
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
    const uint64_t av = carry * lc.pw + s;
    uint64_t key = mix64(av ^ (uint64_t)(32 * c + lane + 1));
    key += key < 2 ? 2 : 0;
    const int64_t j = 32ll * c + lane;
    if (lane < cnt && j < out_lim) out[j] = key;
    carry = __shfl_sync(kFull, av, 31);
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = vn[i];
    ex = exn;
  }
}

// One prompt: dispatch on its (warp-uniform) misalignment.
__device__ __forceinline__ void hash_prompt(const int4* tok4, int64_t n_int4, int64_t t0, int32_t nb, uint64_t seed,
                                            uint64_t* out, int64_t out_lim, const LaneConst& lc) {
  const int64_t q0 = t0 >> 2;
  switch ((int)(t0 & 3)) {
    case 0: hash_chain<0>(tok4, n_int4, q0, nb, seed, out, out_lim, lc); break;
    case 1: hash_chain<1>(tok4, n_int4, q0, nb, seed, out, out_lim, lc); break;
    case 2: hash_chain<2>(tok4, n_int4, q0, nb, seed, out, out_lim, lc); break;
    default: hash_chain<3>(tok4, n_int4, q0, nb, seed, out, out_lim, lc); break;
  }
}

}  // namespace

__global__ void __launch_bounds__(256) k1_block_hash(HashArgs a) {
  if (*a.err) return;
  const LaneConst lc = lane_const();
  const int64_t n_int4 = (a.n_tokens + 3) >> 2;
  const int4* tok4 = reinterpret_cast<const int4*>(a.tokens);
  while (true) {
    int r = 0;
    if (lc.lane == 0) r = (int)atomicAdd(a.work, 1u);
    r = __shfl_sync(kFull, r, 0);
    if (r >= a.n) break;
    const int64_t t0 = a.tok_off[r];
    const int32_t nb = (int32_t)((a.tok_off[r + 1] - t0) >> 4);
    if (nb <= 0) continue;
    const int64_t kb = t0 >> 4;
    hash_prompt(tok4, n_int4, t0, nb, a.seed, a.keys + kb, a.keys_cap - kb, lc);
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
// floor(L_r / 16) (compact key positions) into the scratch array.  The offsets are read in
// coalesced tiles of blockDim.x requests (thread t takes request tile + t); each tile is
// scanned across the block and carried into the next.
__global__ void __launch_bounds__(1024) k1na_offsets(const int64_t* tok_off, int32_t n, int64_t n_tokens,
                                                     int64_t keys_cap, unsigned long long* scratch) {
  __shared__ long long s_wsum[32], s_wex[32], s_tot;
  __shared__ int s_bad;
  const int t = threadIdx.x, lane = t & 31, wid = t >> 5;
  const int nw = (blockDim.x + 31) >> 5;
  if (t == 0) {
    scratch[0] = 0;
    scratch[1] = 0;
    s_bad = 0;
  }
  bool bad = t == 0 && (tok_off[0] != 0 || tok_off[n] != n_tokens);
  long long carry = 0;  // key positions of the tiles before this one (block-uniform)
  for (int base = 0; base < n; base += blockDim.x) {
    const int r = base + t;
    long long v = 0;
    if (r < n) {
      const int64_t t0 = tok_off[r], t1 = tok_off[r + 1];
      if (t0 < 0 || t1 < t0 || t1 > n_tokens || (t1 - t0) >= (1 << 20)) bad = true;
      v = (t1 - t0) >> 4;
    }
    long long incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long u = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += u;
    }
    if (lane == 31) s_wsum[wid] = incl;
    __syncthreads();
    if (wid == 0) {
      const long long w = lane < nw ? s_wsum[lane] : 0;
      long long sc = w;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const long long u = __shfl_up_sync(kFull, sc, o);
        if (lane >= o) sc += u;
      }
      s_wex[lane] = sc - w;
      if (lane == 31) s_tot = sc;
    }
    __syncthreads();
    if (r < n) scratch[8 + r] = (unsigned long long)(carry + s_wex[wid] + incl - v);
    carry += s_tot;
  }
  if (bad) atomicOr(&s_bad, 1);
  __syncthreads();
  if (t == 0) {
    scratch[8 + n] = (unsigned long long)carry;
    scratch[2] = (unsigned long long)carry;
    if (s_bad || carry > keys_cap) scratch[1] = (unsigned long long)(long long)MISAT_ERR_INVALID_ARG;
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
  const int64_t total = (int64_t)scratch[2];
  const LaneConst lc = lane_const();
  const int64_t n_int4 = (n_tokens + 3) >> 2;
  const int4* tok4 = reinterpret_cast<const int4*>(tokens);
  while (true) {
    int r = 0;
    if (lc.lane == 0) r = (int)atomicAdd(work, 1u);
    r = __shfl_sync(kFull, r, 0);
    if (r >= n) break;
    const int64_t t0 = tok_off[r];
    const int32_t nb = (int32_t)((tok_off[r + 1] - t0) >> 4);
    if (nb <= 0) continue;
    const int64_t kb = (int64_t)off_r[r];
    hash_prompt(tok4, n_int4, t0, nb, seed, keys + kb, total - kb, lc);
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
