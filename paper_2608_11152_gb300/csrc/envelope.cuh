// Lower envelope of the cold placement costs of Eq. (1), used by the serial selection.
//
// A request of prompt length x with no cached prefix on instance w costs
//   cost_w(x) = d_w + x / mu_w  =  bk_w + x * tc_w        (fixed point, Eq. 1)
// and the router takes the argmin over the instances with headroom, ties to the lower
// index.  Ordering the pairs (cost, w) lexicographically is ordering the integers
//   key_w(x) = 1024 * cost_w(x) + w = A_w + x * B_w,  A_w = 1024 bk_w + w,  B_w = 1024 tc_w
// (w < 1024), and for w != v the keys differ at every integer x.  So the cheapest available
// instance at x is the line of the lower envelope of {A_w + x B_w} over x >= 0, and two
// lines never tie at an integer x: a line that wins only at a crossing point wins no request.
//
// Lines are kept in "slope order": B descending, then A ascending (a line with the same slope
// and a larger A never wins).  Along the envelope (x increasing) lines appear in slope order.
// A line i is on the envelope of a set S iff the interval of x >= 0 where it beats every other
// line of S is non-empty:
//   lo_i = max(0, max over steeper j of (A_i - A_j) / (B_j - B_i))
//   hi_i = min over shallower j of (A_j - A_i) / (B_i - B_j)
// and lo_i < hi_i.  The fractions are compared by cross-multiplication in 128-bit integers
// (|A_i - A_j| < 2^72, |B_i - B_j| < 2^43), without division.
//
// For a query at integer x >= 0 along an envelope h_0 .. h_{m-1} (slope order), "h_{k+1} beats
// h_k at x" is true exactly for k below the answer's index, so a binary search on it finds the
// answer; it compares 64-bit costs (bk + x tc < 2^62) with the index as the tie-break.
#pragma once

#include <stdint.h>

#ifdef __CUDACC__
#define MISAT_HD __host__ __device__ __forceinline__
#else
#define MISAT_HD inline
#endif

namespace misat {

// (A_i - A_j) for A = 1024 bk + w
MISAT_HD __int128 env_adiff(int64_t bk_i, int i, int64_t bk_j, int j) {
  return (__int128)(bk_i - bk_j) * 1024 + (__int128)(i - j);
}

// a/b < c/d for b, d > 0
MISAT_HD bool env_frac_lt(__int128 a, int64_t b, __int128 c, int64_t d) {
  return a * (__int128)d < c * (__int128)b;
}

// Running state of the on-envelope test of one line against a set of others (the set may be
// split among several threads and the partial states combined).
struct EnvTest {
  __int128 lo_num;  // lo = lo_num / lo_den (starts at 0 / 1: the domain x >= 0)
  int64_t lo_den;
  __int128 hi_num;  // hi = hi_num / hi_den, valid when has_hi
  int64_t hi_den;
  int has_hi;
  int dominated;    // a line with the same slope and a smaller A exists
};

MISAT_HD void env_test_init(EnvTest& t) {
  t.lo_num = 0;
  t.lo_den = 1;
  t.hi_num = 0;
  t.hi_den = 1;
  t.has_hi = 0;
  t.dominated = 0;
}

// Account for line j (bk_j, tc_j) against line i (bk_i, tc_i); j != i.
MISAT_HD void env_test_add(EnvTest& t, int64_t bk_i, int64_t tc_i, int i, int64_t bk_j, int64_t tc_j, int j) {
  if (tc_j == tc_i) {
    if (bk_j < bk_i || (bk_j == bk_i && j < i)) t.dominated = 1;
    return;
  }
  if (tc_j > tc_i) {  // steeper: i beats j for x > (A_i - A_j) / (B_j - B_i)
    const __int128 num = env_adiff(bk_i, i, bk_j, j);
    const int64_t den = (tc_j - tc_i) * 1024;
    if (env_frac_lt(t.lo_num, t.lo_den, num, den)) {
      t.lo_num = num;
      t.lo_den = den;
    }
  } else {  // shallower: i beats j for x < (A_j - A_i) / (B_i - B_j)
    const __int128 num = env_adiff(bk_j, j, bk_i, i);
    const int64_t den = (tc_i - tc_j) * 1024;
    if (!t.has_hi || env_frac_lt(num, den, t.hi_num, t.hi_den)) {
      t.hi_num = num;
      t.hi_den = den;
      t.has_hi = 1;
    }
  }
}

// Merge a partial state computed over another part of the set.
MISAT_HD void env_test_merge(EnvTest& t, const EnvTest& o) {
  t.dominated |= o.dominated;
  if (env_frac_lt(t.lo_num, t.lo_den, o.lo_num, o.lo_den)) {
    t.lo_num = o.lo_num;
    t.lo_den = o.lo_den;
  }
  if (o.has_hi && (!t.has_hi || env_frac_lt(o.hi_num, o.hi_den, t.hi_num, t.hi_den))) {
    t.hi_num = o.hi_num;
    t.hi_den = o.hi_den;
    t.has_hi = 1;
  }
}

MISAT_HD bool env_test_on(const EnvTest& t) {
  if (t.dominated) return false;
  return !t.has_hi || env_frac_lt(t.lo_num, t.lo_den, t.hi_num, t.hi_den);
}

// Does line v come before line u in slope order (B descending, then A ascending)?
MISAT_HD bool env_slope_before(int64_t bk_v, int64_t tc_v, int v, int64_t bk_u, int64_t tc_u, int u) {
  if (tc_v != tc_u) return tc_v > tc_u;
  if (bk_v != bk_u) return bk_v < bk_u;
  return v < u;
}

// Is (cost_v(x), v) below (cost_u(x), u)?
MISAT_HD bool env_beats(int64_t bk_v, int64_t tc_v, int v, int64_t bk_u, int64_t tc_u, int u, int64_t x) {
  const int64_t cv = bk_v + x * tc_v;
  const int64_t cu = bk_u + x * tc_u;
  return cv < cu || (cv == cu && v < u);
}

}  // namespace misat
