// Global prefix index: block key -> bitmask of the instances whose table holds the key
// (Sec. 4.4: the router keeps, for every prefix hash, the set of instances caching it).
//
// The per-instance tables stay the source of truth (they carry the eviction order); the
// global index mirrors their key sets exactly: a key enters instance w's table <=> bit w
// is set, and every deletion from a table clears the bit.  One lookup then answers the
// block-0 probe of a request for all W instances at once.
//
// Layout: bucketed linear probing over 32-byte buckets of four keys (one sector per probe)
// with the masks in a separate array, mw = ceil(W/64) words per slot.  Slots are claimed
// by CAS and never released while the index is in use: a key whose mask drops to zero
// keeps its slot (a later insert of the same key reuses it), and the host rebuilds the
// whole index from the instance tables once claimed slots pass a load threshold.
#pragma once

#include "common.cuh"

namespace misat {

struct GIndex {
  unsigned long long* keys;   // [4 << log2nb]; 0 = empty
  unsigned long long* masks;  // [(4 << log2nb) * mw]
  uint32_t log2nb;            // buckets = 2^log2nb; 0 with keys == NULL: index disabled
  uint32_t mw;                // mask words per slot
  unsigned long long* used;   // claimed slots
};

// Slot of `key`, or -1.  Only for phases without concurrent claims.  Adds buckets read.
__device__ __forceinline__ int64_t gix_find(const GIndex& g, uint64_t key, uint32_t* reads) {
  const uint32_t mask = (1u << g.log2nb) - 1;
  uint32_t b = home_bucket(key, g.log2nb);
  for (uint32_t it = 0; it <= mask; ++it) {
    const ulonglong2* p = reinterpret_cast<const ulonglong2*>(g.keys + 4 * (size_t)b);
    const ulonglong2 x = __ldg(p), y = __ldg(p + 1);
    *reads += 1;
    if (x.x == key) return 4 * (int64_t)b;
    if (x.y == key) return 4 * (int64_t)b + 1;
    if (y.x == key) return 4 * (int64_t)b + 2;
    if (y.y == key) return 4 * (int64_t)b + 3;
    if (x.x == kEmpty || x.y == kEmpty || y.x == kEmpty || y.y == kEmpty) return -1;
    b = (b + 1) & mask;
  }
  return -1;
}

// Slot of `key` while other threads may claim slots (their claims are only additions).
__device__ __forceinline__ int64_t gix_find_cg(const GIndex& g, uint64_t key) {
  const uint32_t mask = (1u << g.log2nb) - 1;
  uint32_t b = home_bucket(key, g.log2nb);
  for (uint32_t it = 0; it <= mask; ++it) {
    const ulonglong2* p = reinterpret_cast<const ulonglong2*>(g.keys + 4 * (size_t)b);
    const ulonglong2 x = __ldcg(p), y = __ldcg(p + 1);
    if (x.x == key) return 4 * (int64_t)b;
    if (x.y == key) return 4 * (int64_t)b + 1;
    if (y.x == key) return 4 * (int64_t)b + 2;
    if (y.y == key) return 4 * (int64_t)b + 3;
    if (x.x == kEmpty || x.y == kEmpty || y.x == kEmpty || y.y == kEmpty) return -1;
    b = (b + 1) & mask;
  }
  return -1;
}

// Find-or-claim `key` and set bit w.  Returns 1 if a slot was claimed, 0 if the key had
// one, -1 if the index has no free slot.
__device__ __forceinline__ int gix_set(const GIndex& g, uint64_t key, int w) {
  const uint32_t mask = (1u << g.log2nb) - 1;
  uint32_t b = home_bucket(key, g.log2nb);
  const unsigned long long bit = 1ull << (w & 63);
  for (uint32_t it = 0; it <= mask; ++it) {
    unsigned long long* kb = g.keys + 4 * (size_t)b;
    for (int tries = 0; tries < 2 * kSlots; ++tries) {
      const ulonglong2* p = reinterpret_cast<const ulonglong2*>(kb);
      const ulonglong2 x = __ldcg(p), y = __ldcg(p + 1);
      const unsigned long long k[4] = {x.x, x.y, y.x, y.y};
      int s = -1, e = -1;
#pragma unroll
      for (int i = 3; i >= 0; --i) {
        if (k[i] == key) s = i;
        if (k[i] == kEmpty) e = i;
      }
      if (s >= 0) {
        atomicOr(g.masks + (4 * (size_t)b + s) * g.mw + (w >> 6), bit);
        return 0;
      }
      if (e < 0) break;  // full without the key: next bucket
      const unsigned long long old = atomicCAS(kb + e, kEmpty, (unsigned long long)key);
      if (old == kEmpty || old == key) {
        atomicOr(g.masks + (4 * (size_t)b + e) * g.mw + (w >> 6), bit);
        return old == kEmpty ? 1 : 0;
      }
    }
    b = (b + 1) & mask;
  }
  return -1;
}

// Find-or-claim `key` without touching its mask.  Returns its slot (and sets *claimed when
// this call took it), or -1 if the index has no free slot.
__device__ __forceinline__ int64_t gix_claim(const GIndex& g, uint64_t key, bool* claimed) {
  const uint32_t mask = (1u << g.log2nb) - 1;
  uint32_t b = home_bucket(key, g.log2nb);
  *claimed = false;
  for (uint32_t it = 0; it <= mask; ++it) {
    unsigned long long* kb = g.keys + 4 * (size_t)b;
    for (int tries = 0; tries < 2 * kSlots; ++tries) {
      const ulonglong2* p = reinterpret_cast<const ulonglong2*>(kb);
      const ulonglong2 x = __ldcg(p), y = __ldcg(p + 1);
      const unsigned long long k[4] = {x.x, x.y, y.x, y.y};
      int s = -1, e = -1;
#pragma unroll
      for (int i = 3; i >= 0; --i) {
        if (k[i] == key) s = i;
        if (k[i] == kEmpty) e = i;
      }
      if (s >= 0) return 4 * (int64_t)b + s;
      if (e < 0) break;  // full without the key: next bucket
      const unsigned long long old = atomicCAS(kb + e, kEmpty, (unsigned long long)key);
      if (old == kEmpty || old == key) {
        *claimed = old == kEmpty;
        return 4 * (int64_t)b + e;
      }
    }
    b = (b + 1) & mask;
  }
  return -1;
}

// Clear bit w of `key`.  Returns 0, or -1 if the key is not in the index (an index that
// no longer mirrors the tables).
__device__ __forceinline__ int gix_clear(const GIndex& g, uint64_t key, int w) {
  const int64_t s = gix_find_cg(g, key);
  if (s < 0) return -1;
  atomicAnd(g.masks + (size_t)s * g.mw + (w >> 6), ~(1ull << (w & 63)));
  return 0;
}

}  // namespace misat
