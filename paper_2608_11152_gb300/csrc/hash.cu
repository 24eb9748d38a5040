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
    if (nb <= 0) continue;
    const int64_t kb = t0 >> 4;
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

      uint64_t cmine = 0;
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
        const uint64_t cb = mix64(p);
        const uint64_t got = __shfl_sync(kFull, cb, 4 * (lane & 7));
        if ((lane >> 3) == i) cmine = got;
      }
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

}  // namespace misat
