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
// and lo_i < hi_i.  The fractions are compared by cross-multiplication, without division
// (EnvFrac below).
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

// A crossing abscissa as a fraction of differences of the line parameters:
//   x = (1024 dbk + dw) / (1024 dtc) = (1024 dbk + dw) / dtc / 1024,   dtc > 0,
// where dbk and dtc are differences of d_w and 1/mu_w and dw a difference of indices.  Two
// such fractions compare as the sign of
//   (1024 dbk1 + dw1) dtc2 - (1024 dbk2 + dw2) dtc1
//     = 1024 (dbk1 dtc2 - dbk2 dtc1) + (dw1 dtc2 - dw2 dtc1),
// exact in 64-bit integers when |dbk| and |dtc| are below 2^25 (every product below 2^50,
// the sum below 2^62), and in 128-bit integers otherwise.
struct EnvFrac {
  int64_t dbk;
  int64_t dw;
  int64_t dtc;  // > 0
};

constexpr int64_t kEnvSmall = (int64_t)1 << 25;

// a < b as fractions; small: every |dbk| and |dtc| of the instance set is below 2^25
MISAT_HD bool env_frac_lt(const EnvFrac& a, const EnvFrac& b, bool small) {
  if (small) {  // every factor fits in 32 bits: one widening multiply per product
    const int64_t d1 = (int64_t)(int32_t)a.dbk * (int32_t)b.dtc - (int64_t)(int32_t)b.dbk * (int32_t)a.dtc;
    const int64_t d2 = (int64_t)(int32_t)a.dw * (int32_t)b.dtc - (int64_t)(int32_t)b.dw * (int32_t)a.dtc;
    return 1024 * d1 + d2 < 0;
  }
  const __int128 na = (__int128)a.dbk * 1024 + a.dw, nb = (__int128)b.dbk * 1024 + b.dw;
  return na * (__int128)b.dtc < nb * (__int128)a.dtc;
}

// Running state of the on-envelope test of one line against a set of others (the set may be
// split among several threads and the partial states combined).
struct EnvTest {
  EnvFrac lo;   // lo starts at 0: the domain x >= 0
  EnvFrac hi;   // valid when has_hi
  int has_hi;
  int dominated;  // a line with the same slope and a smaller A exists
};

MISAT_HD void env_test_init(EnvTest& t) {
  t.lo = EnvFrac{0, 0, 1};
  t.hi = EnvFrac{0, 0, 1};
  t.has_hi = 0;
  t.dominated = 0;
}

// Account for line j (bk_j, tc_j) against line i (bk_i, tc_i); j != i.
MISAT_HD void env_test_add(EnvTest& t, int64_t bk_i, int64_t tc_i, int i, int64_t bk_j, int64_t tc_j, int j,
                           bool small) {
  if (tc_j == tc_i) {
    if (bk_j < bk_i || (bk_j == bk_i && j < i)) t.dominated = 1;
    return;
  }
  if (tc_j > tc_i) {  // steeper: i beats j for x > (A_i - A_j) / (B_j - B_i)
    const EnvFrac f{bk_i - bk_j, (int64_t)(i - j), tc_j - tc_i};
    if (env_frac_lt(t.lo, f, small)) t.lo = f;
  } else {  // shallower: i beats j for x < (A_j - A_i) / (B_i - B_j)
    const EnvFrac f{bk_j - bk_i, (int64_t)(j - i), tc_i - tc_j};
    if (!t.has_hi || env_frac_lt(f, t.hi, small)) {
      t.hi = f;
      t.has_hi = 1;
    }
  }
}

// Merge a partial state computed over another part of the set.
MISAT_HD void env_test_merge(EnvTest& t, const EnvTest& o, bool small) {
  t.dominated |= o.dominated;
  if (env_frac_lt(t.lo, o.lo, small)) t.lo = o.lo;
  if (o.has_hi && (!t.has_hi || env_frac_lt(o.hi, t.hi, small))) {
    t.hi = o.hi;
    t.has_hi = 1;
  }
}

MISAT_HD bool env_test_on(const EnvTest& t, bool small) {
  if (t.dominated) return false;
  return !t.has_hi || env_frac_lt(t.lo, t.hi, small);
}

// Dual point i strictly below the segment p-q (slopes p > i > q), i.e. line i is below the
// crossing of p and q: (A_i - A_p)(B_p - B_q) < (A_q - A_p)(B_p - B_i).
MISAT_HD bool env_below_chord(int64_t bki, int64_t tci, int i, int64_t bkp, int64_t tcp, int p, int64_t bkq,
                              int64_t tcq, int q, bool small) {
  const EnvFrac a{bki - bkp, (int64_t)(i - p), tcp - tci};  // (A_i - A_p) / (B_p - B_i)
  const EnvFrac c{bkq - bkp, (int64_t)(q - p), tcp - tcq};  // (A_q - A_p) / (B_p - B_q)
  return env_frac_lt(a, c, small);
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
