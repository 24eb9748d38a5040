// Shared device-side definitions of the MISA-T routing library (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/misat.h"

namespace misat {

// Blocks of `kernel` that fit on the GPU at once at this block size and dynamic shared memory
// (resident blocks per SM x SMs; queried once per kernel).  A grid-stride loop with a static
// split over this many blocks runs in one wave: with more blocks than fit, the blocks of the
// second wave start only as the first finish, and a latency-bound pass takes about twice its
// one-wave time.
template <auto Kernel>
inline int resident_grid(int block, size_t smem, int num_sms) {
  static int per_sm = 0, last_block = -1;
  static size_t last_smem = 0;
  if (per_sm == 0 || block != last_block || smem != last_smem) {
    int v = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, Kernel, block, smem) != cudaSuccess || v < 1) {
      cudaGetLastError();
      v = 1;
    }
    per_sm = v;
    last_block = block;
    last_smem = smem;
  }
  return per_sm * num_sms;
}

constexpr int kBlockTokens = 16;
constexpr uint64_t kGold = 0x9e3779b97f4a7c15ull;  // SplitMix64 increment, chain multiplier
constexpr uint64_t kEmpty = 0;                     // empty slot key (block keys are >= 2)
constexpr int kSlots = 4;                          // keys per bucket: one 32-byte sector
constexpr int64_t kCapInf = 2147483647;            // "no cap"
constexpr int64_t kBacklogMax = (int64_t)1 << 61;  // saturation of the in-batch backlog
constexpr int kMaxW = 1024;

// Session states in the device session table.
constexpr uint32_t kSessProtected = 1;  // in O_w u P_w of `inst`
constexpr uint32_t kSessReleased = 2;   // admitted before, protected nowhere
constexpr uint32_t kSessDead = 3;       // finished; slot reusable

// Request status during the selection rounds.
constexpr uint8_t kStUnresolved = 0;
constexpr uint8_t kStResolved = 1;
constexpr uint8_t kStFollower = 2;
constexpr uint8_t kStHeld = 3;  // leader with no eligible instance: held for the rest of the batch

// One bucket of an instance's resident-block table: four keys in one 32-byte
// sector (what a probe reads) followed by their four metas (what a commit
// updates), 64 bytes aligned.  meta = seq<<36 | arrival<<16 | (65535 - depth);
// an empty slot has key 0 and meta 0.
struct alignas(64) Bucket {
  unsigned long long key[kSlots];
  unsigned long long meta[kSlots];
};
static_assert(sizeof(Bucket) == 64, "bucket must be 64 bytes");

// Per-instance table descriptor (device copy kept in sync by the host).
struct InstDesc {
  Bucket* tab;
  uint32_t log2nb;  // number of buckets = 2^log2nb, log2nb >= 1
  uint32_t pad;
  int64_t cap;      // Cap_w
};

// Session table slot: key = session id (0 = never used), val = state<<40 | cls<<32 | inst.
struct alignas(16) SessSlot {
  unsigned long long key;
  unsigned long long val;
};

__host__ __device__ __forceinline__ uint64_t sess_val(uint32_t state, uint32_t cls, uint32_t inst) {
  return ((uint64_t)state << 40) | ((uint64_t)cls << 32) | (uint64_t)inst;
}
__host__ __device__ __forceinline__ uint32_t sess_state(uint64_t v) { return (uint32_t)(v >> 40); }
__host__ __device__ __forceinline__ uint32_t sess_cls(uint64_t v) { return (uint32_t)(v >> 32) & 0xff; }
__host__ __device__ __forceinline__ uint32_t sess_inst(uint64_t v) { return (uint32_t)v; }

__host__ __device__ __forceinline__ uint64_t pack_meta(uint64_t seq, uint64_t arrival, uint64_t depth) {
  return (seq << 36) | (arrival << 16) | (65535ull - depth);
}

// SplitMix64 finaliser (Steele, Lea & Flood 2014).
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
  z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
  return z ^ (z >> 31);
}

// Home bucket of a key: top log2nb bits of key * G (multiplicative hashing), so that
// loaded entries with skewed keys (e.g. 63-bit values) still spread over the table.
__device__ __forceinline__ uint32_t home_bucket(uint64_t key, uint32_t log2nb) {
  return (uint32_t)((key * kGold) >> (64 - log2nb));
}

// Home slot of a session id in the session table.
__device__ __forceinline__ uint32_t sess_home(uint64_t s, uint32_t log2n) {
  return (uint32_t)(mix64(s) >> (64 - log2n));
}

// Block-uniform early exit once a device error is recorded (safe before __syncthreads).
__device__ __forceinline__ bool block_error(const int32_t* err) {
  __shared__ int32_t s_err;
  if (threadIdx.x == 0) s_err = *(volatile const int32_t*)err;
  __syncthreads();
  return s_err != 0;
}

// Signed 64-bit atomic add (two's complement through the unsigned overload).
__device__ __forceinline__ void atomic_add_i64(long long* p, long long v) {
  atomicAdd(reinterpret_cast<unsigned long long*>(p), (unsigned long long)v);
}

// Sum of v over the block (every thread must call it); the total is valid in thread 0.
// Used so that per-kernel counters cost one global atomic per CTA, not per thread.
__device__ __forceinline__ long long block_sum(long long v) {
  __shared__ long long s_part[32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  __syncthreads();  // s_part may still be read by a previous call
  if (lane == 0) s_part[wid] = v;
  __syncthreads();
  long long t = 0;
  if (threadIdx.x == 0)
    for (int i = 0; i < (int)((blockDim.x + 31) >> 5); ++i) t += s_part[i];
  return t;
}

// Record the first device error (sticky).
__device__ __forceinline__ void set_error(int32_t* err, int32_t code) { atomicCAS(err, 0, code); }

__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Streaming 16-byte read-only load (read once: no L1 allocation, 256-byte L2 prefetch).
__device__ __forceinline__ int4 ld_stream_v4(const int4* p) {
  int4 v;
  asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.s32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Read the four keys of a bucket (one 32-byte sector) through the read-only path.
__device__ __forceinline__ void ld_bucket_keys(const Bucket* b, unsigned long long k[4]) {
  const ulonglong2* p = reinterpret_cast<const ulonglong2*>(b->key);
  ulonglong2 a = __ldg(p);
  ulonglong2 c = __ldg(p + 1);
  k[0] = a.x;
  k[1] = a.y;
  k[2] = c.x;
  k[3] = c.y;
}

// Coherent (L2) read of the four keys, for kernels that modify tables concurrently.
__device__ __forceinline__ void ld_bucket_keys_cg(const Bucket* b, unsigned long long k[4]) {
  const ulonglong2* p = reinterpret_cast<const ulonglong2*>(b->key);
  ulonglong2 a = __ldcg(p);
  ulonglong2 c = __ldcg(p + 1);
  k[0] = a.x;
  k[1] = a.y;
  k[2] = c.x;
  k[3] = c.y;
}

// Look a key up in one instance table (no concurrent writers).  Returns 1 if
// resident.  Adds the number of buckets read to *reads.  Bounded by the table size.
// Look a key up from bucket b0 on (the later buckets of its probe sequence, after a full
// home bucket without it).  Adds the buckets read to *reads.
__device__ __forceinline__ int table_contains_from(const InstDesc& d, uint64_t key, uint32_t b0, uint32_t* reads) {
  const uint32_t mask = (1u << d.log2nb) - 1;
  uint32_t b = b0;
  for (uint32_t it = 0; it < mask; ++it) {
    unsigned long long k[4];
    ld_bucket_keys(d.tab + b, k);
    *reads += 1;
    if ((k[0] == key) | (k[1] == key) | (k[2] == key) | (k[3] == key)) return 1;
    if ((k[0] == kEmpty) | (k[1] == kEmpty) | (k[2] == kEmpty) | (k[3] == kEmpty)) return 0;
    b = (b + 1) & mask;
  }
  return 0;
}

__device__ __forceinline__ int table_contains(const InstDesc& d, uint64_t key, uint32_t* reads) {
  const uint32_t mask = (1u << d.log2nb) - 1;
  uint32_t b = home_bucket(key, d.log2nb);
  for (uint32_t it = 0; it <= mask; ++it) {
    unsigned long long k[4];
    ld_bucket_keys(d.tab + b, k);
    *reads += 1;
    bool hit = (k[0] == key) | (k[1] == key) | (k[2] == key) | (k[3] == key);
    if (hit) return 1;
    bool open = (k[0] == kEmpty) | (k[1] == kEmpty) | (k[2] == kEmpty) | (k[3] == kEmpty);
    if (open) return 0;
    b = (b + 1) & mask;
  }
  return 0;
}

// ---- groups of the admitted requests of a batch (commit work dedup) ----
// Open-addressing table over (first block key, instance): per group the latest admitted
// request.  Slot {key0, tag}: tag = (instance + 1) << 32 | (arrival + 1), 0 = empty.  A slot's
// key is claimed first, then its instance; a slot whose instance differs is passed over, so
// every (key0, instance) pair owns exactly one slot of its probe sequence.
__device__ __forceinline__ uint32_t grp_home(uint64_t key0, int w, uint32_t log2n) {
  return (uint32_t)(mix64(key0 ^ ((uint64_t)(w + 1) * kGold)) >> (64 - log2n));
}

__device__ __forceinline__ void grp_note(ulonglong2* tab, uint32_t log2n, uint64_t key0, int w, int r) {
  const uint32_t mask = (1u << log2n) - 1;
  uint32_t h = grp_home(key0, w, log2n);
  for (uint32_t it = 0; it <= mask; ++it) {
    unsigned long long* kp = &tab[h].x;
    unsigned long long k = __ldcg(kp);
    if (k == 0) {
      k = atomicCAS(kp, 0ull, (unsigned long long)key0);
      if (k == 0) k = key0;
    }
    if (k == key0) {
      unsigned* tag = reinterpret_cast<unsigned*>(&tab[h].y);  // [0] arrival + 1, [1] instance + 1
      const unsigned wv = atomicCAS(tag + 1, 0u, (unsigned)(w + 1));
      if (wv == 0 || wv == (unsigned)(w + 1)) {
        atomicMax(tag, (unsigned)(r + 1));
        return;
      }
    }
    h = (h + 1) & mask;
  }
}

// The latest admitted request of group (key0, w), -1 if the group is not in the table.
__device__ __forceinline__ int grp_last(const ulonglong2* tab, uint32_t log2n, uint64_t key0, int w) {
  const uint32_t mask = (1u << log2n) - 1;
  uint32_t h = grp_home(key0, w, log2n);
  for (uint32_t it = 0; it <= mask; ++it) {
    const ulonglong2 e = __ldcg(&tab[h]);
    if (e.x == 0) return -1;
    if (e.x == key0 && (uint32_t)(e.y >> 32) == (uint32_t)(w + 1)) return (int)(uint32_t)e.y - 1;
    h = (h + 1) & mask;
  }
  return -1;
}

}  // namespace misat
