// Selection of one batch: the leaders (first request of each session in the batch) are
// decided one at a time in arrival order, as the online router of Sec. 4 decides requests.
// Each sees the snapshot taken at batch start (caches, sessions, backlog d_w, throughput
// mu_w) and the sessions admitted before it, which are pending on their instances
// (P_w, Sec. 4.1-4.2).  A leader takes the cheapest instance of Eq. (1) where Admit holds
// (Eq. 6 with the class cap of Sec. 4.2; Sec. 4.4: placement among instances with
// headroom), or is held when no instance has headroom for it; a released continuation may
// prefer to wait for its cached instance (Eq. 7).
//
// The decisions form a serial chain, but the state that a leader's choice depends on
// changes only when an instance runs out of headroom (at most 4 W times per batch).
// Between such events every leader's choice is independent of the others', so one CTA
// takes the batch in windows of kSelectThreads leaders (one per thread):
//   1. every undecided leader of the window chooses against the state at the window's
//      current start: for a cold prompt (nothing cached) the cheapest instance with
//      headroom for its class is a query of the lower envelope of the lines
//      d_w + L / mu_w (envelope.cuh), plus its few cached or protected instances;
//   2. the admissions are counted per (instance, class); where an instance would be
//      over-subscribed, arrival-order ranks (warp counts, one scan over the warps) find the
//      first leader whose instance has no headroom left at its turn;
//   3. the leaders before that one are final (their instance still had headroom, and every
//      other instance only lost headroom, so the argmin stands); instances that ran out leave
//      the envelopes of the classes they no longer admit, and the window continues from
//      that leader.
// Released continuations with a cached prefix (Eq. 7 compares two instances) are decided
// only at the head of the window, where the state is exactly that of their turn.
#include "common.cuh"
#include "envelope.cuh"
#include "kernels.h"

namespace misat {

namespace {
constexpr unsigned kFull = 0xffffffffu;
constexpr int kNT = kSelectThreads;
constexpr int kNW = kNT / 32;
constexpr int kMaxGaps = 32;   // envelope gaps handled incrementally per update
constexpr int kSlotInst = kNT / (4 * kNW);  // over-subscribed instances given exact ranks per pass
static_assert(kNW == 16 && kSlotInst == 8, "one thread per (counter, warp) in the rank scan");
}  // namespace

// ---------------------------------------------------------------------------
// Per-request records for the selection (32 bytes, one coalesced pair of loads):
//   rec[2r]   = {L, cls | sst << 8 | leader << 16, protected / last instance, hbest}
//   rec[2r+1] = {instances with H > 0, first two of them as (w << 16 | H), 0}
__global__ void __launch_bounds__(256) k3_select_prep(SelectPrepArgs a) {
  __shared__ int s_wc[3][8];
  if (blockIdx.x == 0) {
    for (int w = threadIdx.x; w < a.W; w += blockDim.x) a.adm[w] = 0;
    if (threadIdx.x == 0) {
      *a.ticket = 0;
      *a.coupled = 0;
    }
  }
  if (block_error(a.err)) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  // this block's leaders of each class, in arrival order, for the per-class selection
  {
    const int c = r < a.n && a.rq.status[r] == kStUnresolved ? a.rq.cls[r] : 3;
    unsigned mine = 0;
#pragma unroll
    for (int b = 0; b < 3; ++b) {
      const unsigned m = __ballot_sync(kFull, c == b);
      if (lane == 0) s_wc[b][wid] = __popc(m);
      if (c == b) mine = m;
    }
    __syncthreads();
    if (c < 3) {
      int off = __popc(mine & lanemask_lt());
      for (int k = 0; k < wid; ++k) off += s_wc[c][k];
      a.seg[(int64_t)c * a.n + blockIdx.x * 256 + off] = r;
    }
    if (threadIdx.x < 3) {
      int t = 0;
      for (int k = 0; k < 8; ++k) t += s_wc[threadIdx.x][k];
      a.segcnt[threadIdx.x * gridDim.x + blockIdx.x] = t;
    }
  }
  if (r >= a.n) return;
  const int lead = a.rq.status[r] == kStUnresolved;
  const uint32_t hb = a.rq.hbest[r];
  int nh = 0;
  uint32_t h0 = 0, h1 = 0;
  if (lead && (hb >> 16) > 0) {
    const uint16_t* row = a.H + (int64_t)r * a.W;
    for (int w = 0; w < a.W; ++w) {
      const uint32_t h = row[w];
      if (h) {
        if (nh == 0) h0 = ((uint32_t)w << 16) | h;
        else if (nh == 1) h1 = ((uint32_t)w << 16) | h;
        ++nh;
      }
    }
  }
  a.rec[2 * r] = make_int4(a.rq.L[r], a.rq.cls[r] | (a.rq.sst[r] << 8) | (lead << 16), a.rq.sinst[r], (int)hb);
  a.rec[2 * r + 1] = make_int4(nh, (int)h0, (int)h1, 0);
}

// ---------------------------------------------------------------------------
// Initial envelopes and orders.  blockIdx.y = class b (0..2): is line i on the lower envelope
// of the instances with headroom for class b?  blockIdx.y = 3: position of line i in slope
// order; 4: its position in (d_w, w) order.  Eight lanes share line i, each taking every
// eighth other line.
__global__ void __launch_bounds__(1024) k3_env_init(EnvInitArgs a) {
  if (block_error(a.err)) return;
  const int i = blockIdx.x * 128 + (threadIdx.x >> 3);
  const int sub = threadIdx.x & 7;
  const int b = blockIdx.y;
  const bool line = i < a.W;
  const int64_t bki = line ? a.backlog[i] : 0, tci = line ? a.tokcost[i] : 0;
  if (b >= 3) {  // 3: position in slope order; 4: position in (d_w, w) order
    int cnt = 0;
    if (line)
      for (int j = sub; j < a.W; j += 8) {
        const int64_t bkj = a.backlog[j];
        if (j != i && (b == 3 ? env_slope_before(bkj, a.tokcost[j], j, bki, tci, i) : (bkj < bki || (bkj == bki && j < i))))
          ++cnt;
      }
#pragma unroll
    for (int o = 4; o > 0; o >>= 1) cnt += __shfl_xor_sync(kFull, cnt, o);
    if (line && sub == 0) (b == 3 ? a.rank : a.rank_a)[i] = cnt;
    return;
  }
  auto avail = [&](int w) { return a.gh[w] > 0 && a.ch[w * 3 + b] > 0; };
  const bool ai = line && avail(i);
  EnvTest t;
  env_test_init(t);
  if (ai)
    for (int j = sub; j < a.W; j += 8)
      if (j != i && avail(j)) env_test_add(t, bki, tci, i, a.backlog[j], a.tokcost[j], j, a.small);
#pragma unroll
  for (int o = 4; o > 0; o >>= 1) {
    EnvTest u;
    u.lo = EnvFrac{__shfl_xor_sync(kFull, t.lo.dbk, o), __shfl_xor_sync(kFull, t.lo.dw, o),
                   __shfl_xor_sync(kFull, t.lo.dtc, o)};
    u.hi = EnvFrac{__shfl_xor_sync(kFull, t.hi.dbk, o), __shfl_xor_sync(kFull, t.hi.dw, o),
                   __shfl_xor_sync(kFull, t.hi.dtc, o)};
    u.has_hi = __shfl_xor_sync(kFull, t.has_hi, o);
    u.dominated = __shfl_xor_sync(kFull, t.dominated, o);
    env_test_merge(t, u, a.small);
  }
  if (line && sub == 0) a.onhull[b * a.W + i] = ai && env_test_on(t, a.small) ? 1 : 0;
}

void launch_select_prep(const SelectPrepArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  k3_select_prep<<<(a.n + 255) / 256, 256, 0, st>>>(a);
}

void launch_env_init(const EnvInitArgs& a, cudaStream_t st) {
  dim3 grid((a.W + 127) / 128, 5);
  k3_env_init<<<grid, 1024, 0, st>>>(a);
}

// ---------------------------------------------------------------------------
// Shared state of the selection CTA.  Per class, the headroom flags are kept both by instance
// (queries) and in slope order (envelope updates read them as contiguous bytes); the envelope
// keeps its lines' d_w and 1/mu_w beside their indices, so a query step is one load level.
struct SelSmem {
  int64_t* bk;     // [W] d_w
  int64_t* tc;     // [W] 1/mu_w
  int64_t* hbk;    // [3][W] d_w of the envelope lines
  int64_t* htc;    // [3][W] 1/mu_w of the envelope lines
  int32_t* gh;     // [W] global headroom
  int32_t* ch;     // [3][W] class headroom
  int32_t* T;      // [W] admissions of the window's current choices
  int32_t* Tb;     // [3][W]
  int32_t* slot;   // [W] exact-rank slot of an over-subscribed instance, -1
  int32_t* wc;     // [4 * kSlotInst counters][kNW warps]
  int32_t* surv;   // [3][W] envelope candidates of each class's update
  int16_t* ord;    // [W] instances in slope order
  int16_t* pos;    // [W] position in slope order
  int16_t* aord;   // [W] instances in (d_w, w) order
  int16_t* hull;   // [3][W] envelope lines per class, slope order
  uint8_t* av;     // [3][W] headroom for the class (gh > 0 and ch > 0), by instance
  uint8_t* avp;    // [3][W] the same by slope position
  uint8_t* onp;    // [3][W] on the envelope of the class, by slope position
};

// Per-class scratch of an envelope update (one warp per class).  headroom only shrinks, so
// the first line with headroom in (d_w, w) order (the one that wins at x = 0) and the last in
// slope order (the least 1/mu_w) are found by pointers that only move forward.
struct EnvScratch {
  int gp[kMaxGaps];
  int gq[kMaxGaps];
  int first_a;     // position in (d_w, w) order of the first line that may have headroom
  int last_s;      // position in slope order of the last line that may have headroom
};

// Rebuild hull[b] from the on-envelope flags (compaction in slope order).  One warp.
__device__ void env_compact_warp(const SelSmem& s, int W, int b, int* hm) {
  const int lane = threadIdx.x & 31;
  int base = 0;
  for (int x0 = 0; x0 < W; x0 += 128) {
    bool f[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int x = x0 + 32 * u + lane;
      f[u] = x < W && s.onp[b * W + x];
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int x = x0 + 32 * u + lane;
      const unsigned m = __ballot_sync(kFull, f[u]);
      if (f[u]) {
        const int k = base + __popc(m & lanemask_lt());
        const int w = s.ord[x];
        s.hull[b * W + k] = (int16_t)w;
        s.hbk[b * W + k] = s.bk[w];
        s.htc[b * W + k] = s.tc[w];
      }
      base += __popc(m);
    }
  }
  if (lane == 0) *hm = base;
  __syncwarp();
}

// The line of class b with headroom that wins at x = 0 (least (d_w, w)), -1 if none.  One warp
// (warp-uniform result).
__device__ __forceinline__ int env_first_line(const SelSmem& s, int W, int b, EnvScratch& sc) {
  int k = sc.first_a;
  while (k < W && !s.av[b * W + s.aord[k]]) ++k;
  __syncwarp();
  if ((threadIdx.x & 31) == 0) sc.first_a = k;
  __syncwarp();
  return k < W ? s.aord[k] : -1;
}

// The line of class b with headroom that wins for large x: least 1/mu_w, then least d_w (the
// first of the last run of equal slopes in slope order), -1 if none.  One warp.
__device__ __forceinline__ int env_last_line(const SelSmem& s, int W, int b, EnvScratch& sc) {
  int x = sc.last_s;
  while (x >= 0 && !s.avp[b * W + x]) --x;
  __syncwarp();
  if ((threadIdx.x & 31) == 0) sc.last_s = x;
  __syncwarp();
  if (x < 0) return -1;
  const int64_t t = s.tc[s.ord[x]];
  int y = x;
  for (int z = x - 1; z >= 0 && s.tc[s.ord[z]] == t; --z)
    if (s.avp[b * W + z]) y = z;
  return s.ord[y];
}

// Remove the lines of class b that lost their headroom from its envelope.  One warp.
// Each maximal run of removed envelope lines leaves a gap between its surviving neighbours p
// and q (slope order).  A gap at the start of the envelope is closed by the line that now
// wins at x = 0 (least d_w: it is on the envelope), one at the end by the line that now wins
// for large x (least 1/mu_w).  Between p and q the envelope is that of p, q and the lines of
// slope strictly between them that lie below the chord p-q: a line above it cannot be on the
// envelope there, and does not change the envelope of the ones below it.
__device__ void env_update_warp(const SelSmem& s, int W, int b, int* hm, EnvScratch& sc, bool small) {
  const int lane = threadIdx.x & 31;
  const int m = *hm;
  const int16_t* hull = s.hull + b * W;
  int ng = 0;
  // gaps, in hull order
  for (int k0 = 0; k0 < m; k0 += 32) {
    const int k = k0 + lane;
    const int w = k < m ? hull[k] : 0;
    const bool del = k < m && !s.av[b * W + w];
    const unsigned md = __ballot_sync(kFull, del);
    const bool prev_del = lane > 0 ? (md >> (lane - 1)) & 1 : (k > 0 && !s.av[b * W + hull[k - 1]]);
    const bool start = del && !prev_del;
    if (del) s.onp[b * W + s.pos[w]] = 0;
    const unsigned ms = __ballot_sync(kFull, start);
    if (start) {
      int c = k + 1;
      while (c < m && !s.av[b * W + hull[c]]) ++c;
      const int g = ng + __popc(ms & lanemask_lt());
      if (g < kMaxGaps) {
        sc.gp[g] = k > 0 ? hull[k - 1] : -1;
        sc.gq[g] = c < m ? hull[c] : -1;
      }
    }
    ng += __popc(ms);
  }
  __syncwarp();
  if (ng > kMaxGaps) {
    // full rebuild: every line with headroom tested against all the others
    for (int x = lane; x < W; x += 32) {
      bool on = false;
      if (s.avp[b * W + x]) {
        const int i = s.ord[x];
        EnvTest t;
        env_test_init(t);
        for (int j = 0; j < W; ++j)
          if (j != i && s.av[b * W + j]) env_test_add(t, s.bk[i], s.tc[i], i, s.bk[j], s.tc[j], j, small);
        on = env_test_on(t, small);
      }
      s.onp[b * W + x] = on;
    }
    __syncwarp();
  } else {
    int ns = 0;
    int* surv = s.surv + b * W;
    for (int g = 0; g < ng; ++g) {
      int p = sc.gp[g], q = sc.gq[g];
      if (p < 0) {  // the envelope's start was removed: the line that now wins at x = 0
        p = env_first_line(s, W, b, sc);
        if (p >= 0 && lane == 0) s.onp[b * W + s.pos[p]] = 1;
      }
      if (p >= 0 && q < 0) {  // the end was removed: the line that now wins for large x
        q = env_last_line(s, W, b, sc);
        if (lane == 0) s.onp[b * W + s.pos[q]] = 1;
      }
      if (p < 0 || q < 0 || p == q) continue;
      const int g0 = ns;
      const int xp = s.pos[p], xq = s.pos[q];
      const int64_t bkp = s.bk[p], tcp = s.tc[p], bkq = s.bk[q], tcq = s.tc[q];
      for (int x0 = xp + 1; x0 < xq; x0 += 128) {
        bool c[4];
        int iv[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int x = x0 + 32 * u + lane;
          c[u] = false;
          iv[u] = 0;
          if (x < xq && s.avp[b * W + x]) {
            const int i = s.ord[x];
            const int64_t tci = s.tc[i];
            iv[u] = i;
            c[u] = tci != tcp && env_below_chord(s.bk[i], tci, i, bkp, tcp, p, bkq, tcq, q, small);
          }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const unsigned mc = __ballot_sync(kFull, c[u]);
          if (c[u]) surv[ns + __popc(mc & lanemask_lt())] = iv[u];
          ns += __popc(mc);
        }
      }
      __syncwarp();
      // each candidate against p, q and the other candidates of this gap
      for (int e = g0 + lane; e < ns; e += 32) {
        const int i = surv[e];
        const int64_t bki = s.bk[i], tci = s.tc[i];
        EnvTest t;
        env_test_init(t);
        env_test_add(t, bki, tci, i, bkp, tcp, p, small);
        env_test_add(t, bki, tci, i, bkq, tcq, q, small);
        for (int f = g0; f < ns; ++f) {
          const int j = surv[f];
          if (j != i) env_test_add(t, bki, tci, i, s.bk[j], s.tc[j], j, small);
        }
        if (env_test_on(t, small)) s.onp[b * W + s.pos[i]] = 1;
      }
      __syncwarp();
    }
  }
  env_compact_warp(s, W, b, hm);
}

// Decision of one leader against the current state (see the file comment).  Returns the
// instance (or -1) and sets *dec to MISAT_ADMIT_NEW, MISAT_ADMIT_CONT, MISAT_HOLD_PREFER_CACHE,
// MISAT_HOLD_CLASS_CAP or MISAT_HOLD_GLOBAL_CAP.
__device__ __forceinline__ int sel_choose(const SelSmem& s, const int* s_hm, int W, int nglobal, int L, int b,
                                          int sst, int pw, uint32_t hb, int nh, uint32_t h0, uint32_t h1,
                                          const uint16_t* Hrow, int64_t hold, uint8_t* dec) {
  int64_t best_c = INT64_MAX;
  int best_w = INT32_MAX;
  const int m = s_hm[b];
  const int16_t* hull = s.hull + b * W;
  const int64_t* hbk = s.hbk + b * W;
  const int64_t* htc = s.htc + b * W;
  const int64_t x = L;
  if (m > 0) {
    int lo = 0, hi = m - 1;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      const int64_t cu = hbk[mid] + x * htc[mid], cv = hbk[mid + 1] + x * htc[mid + 1];
      // line mid + 1 beats line mid at x (ties to the lower index)
      if (cv < cu || (cv == cu && hull[mid + 1] < hull[mid])) lo = mid + 1;
      else hi = mid;
    }
    best_w = hull[lo];
    best_c = hbk[lo] + x * htc[lo];
  }
  auto consider = [&](int w, int64_t h) {
    const int64_t c = s.bk[w] + (x - 16 * h) * s.tc[w];
    if (c < best_c || (c == best_c && w < best_w)) {
      best_c = c;
      best_w = w;
    }
  };
  // cached instances with headroom (or the protected one): below their line of the envelope
  if (nh > 0 && nh <= 2) {
    const int w0 = (int)(h0 >> 16);
    if (s.av[b * W + w0] || w0 == pw) consider(w0, h0 & 0xffff);
    if (nh == 2) {
      const int w1 = (int)(h1 >> 16);
      if (s.av[b * W + w1] || w1 == pw) consider(w1, h1 & 0xffff);
    }
  } else if (nh > 2) {
    for (int w = 0; w < W; ++w) {
      const int h = Hrow[w];
      if (h && (s.av[b * W + w] || w == pw)) consider(w, h);
    }
  }
  // the protected instance is eligible without headroom (its cached cost was considered above)
  if (pw >= 0) consider(pw, 0);
  if (best_w == INT32_MAX) {
    *dec = nglobal > 0 ? MISAT_HOLD_CLASS_CAP : MISAT_HOLD_GLOBAL_CAP;
    return -1;
  }
  const int hmax = (int)(hb >> 16), whit = 65535 - (int)(hb & 0xffffu);
  if (sst == kSessReleased && hmax > 0 && !s.av[b * W + whit]) {
    const int64_t lhs = hold + s.bk[whit] - s.bk[best_w];
    const int64_t rhs = 16 * (int64_t)hmax * s.tc[whit];
    if (lhs < rhs) {
      *dec = MISAT_HOLD_PREFER_CACHE;
      return -1;
    }
  }
  *dec = best_w == pw ? MISAT_ADMIT_CONT : MISAT_ADMIT_NEW;
  return best_w;
}

// First set position >= from in the window's kNW-word bitmask held by lanes 0 .. kNW-1 of
// every warp (kNT if none).  Warp-uniform.
__device__ __forceinline__ int first_set_from(unsigned word, int lane, int from) {
  const int fw = from >> 5;
  unsigned m = lane < fw ? 0u : word;
  if (lane == fw) m &= ~0u << (from & 31);
  const unsigned nz = __ballot_sync(kFull, m != 0);
  if (!nz) return kNT;
  const int w = __ffs(nz) - 1;
  return w * 32 + __ffs(__shfl_sync(kFull, m, w)) - 1;
}

// An instance's headroom dropped to `g` (global) or its class b headroom to `c`: clear its
// flags for the classes it no longer admits.
__device__ __forceinline__ void sel_flags(const SelSmem& s, int W, int w, int b, bool gone_g, bool gone_c,
                                          int* s_dirty) {
  const int x = s.pos[w];
#pragma unroll
  for (int c = 0; c < 3; ++c)
    if ((gone_g || (gone_c && c == b)) && s.av[c * W + w]) {
      s.av[c * W + w] = 0;
      s.avp[c * W + x] = 0;
      if (s.onp[c * W + x]) s_dirty[c] = 1;
    }
}

__global__ void __launch_bounds__(kNT, 1) k4_select(SelectArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int s_hm[3], s_q, s_nslot, s_nglobal, s_f, s_dirty[3];
  __shared__ unsigned s_lead[kNW], s_sens[kNW];
  __shared__ EnvScratch s_env[3];
  if (block_error(a.err)) return;
  // the per-class path decided the batch unless it raised the flag (no flag: always run)
  if (a.coupled != nullptr && *(volatile const int32_t*)a.coupled == 0) return;
  const int W = a.W;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  SelSmem s;
  {
    unsigned char* p = smem;
    s.bk = reinterpret_cast<int64_t*>(p);
    p += (size_t)W * 8;
    s.tc = reinterpret_cast<int64_t*>(p);
    p += (size_t)W * 8;
    s.hbk = reinterpret_cast<int64_t*>(p);
    p += (size_t)W * 24;
    s.htc = reinterpret_cast<int64_t*>(p);
    p += (size_t)W * 24;
    s.gh = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.ch = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 12;
    s.T = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.Tb = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 12;
    s.slot = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.wc = reinterpret_cast<int32_t*>(p);
    p += (size_t)kNT * 4;
    s.surv = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 12;
    s.ord = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.pos = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.aord = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.hull = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 6;
    s.av = p;
    p += (size_t)W * 3;
    s.avp = p;
    p += (size_t)W * 3;
    s.onp = p;
  }
  if (tid == 0) {
    s_nglobal = 0;
    s_q = kNT;
    s_nslot = 0;
    s_f = -1;
    s_dirty[0] = s_dirty[1] = s_dirty[2] = 0;
  }
  __syncthreads();
  for (int w = tid; w < W; w += kNT) {
    const int r = a.rank[w];
    s.ord[r] = (int16_t)w;
    s.pos[w] = (int16_t)r;
    s.aord[a.rank_a[w]] = (int16_t)w;
    s.bk[w] = a.backlog[w];
    s.tc[w] = a.tokcost[w];
    const int32_t g = a.gh[w];
    s.gh[w] = g;
    if (g > 0) atomicAdd(&s_nglobal, 1);
    s.T[w] = 0;
    s.slot[w] = -1;
#pragma unroll
    for (int b = 0; b < 3; ++b) {
      const int32_t c = a.ch[w * 3 + b];
      const uint8_t v = g > 0 && c > 0;
      s.ch[b * W + w] = c;
      s.Tb[b * W + w] = 0;
      s.av[b * W + w] = v;
      s.avp[b * W + r] = v;
      s.onp[b * W + r] = a.onhull[b * W + w];
    }
  }
  s.wc[tid] = 0;
  if (tid < 3) {
    s_env[tid].first_a = 0;
    s_env[tid].last_s = W - 1;
  }
  __syncthreads();
  if (wid < 3) env_compact_warp(s, W, wid, &s_hm[wid]);
  __syncthreads();

  // records of the first window
  int4 n0 = make_int4(0, 0, 0, 0), n1 = make_int4(0, 0, 0, 0);
  if (tid < a.n) {
    n0 = a.rec[2 * tid];
    n1 = a.rec[2 * tid + 1];
  }
#pragma unroll 1
  for (int base = 0; base < a.n; base += kNT) {
    const int i = base + tid;
    const int4 r0 = n0, r1 = n1;
    if (i + kNT < a.n) {  // next window's records, in flight during this one
      n0 = a.rec[2 * (i + kNT)];
      n1 = a.rec[2 * (i + kNT) + 1];
    }
    const int L = r0.x;
    const int b = r0.y & 0xff;
    const int sst = (r0.y >> 8) & 0xff;
    const int pw = sst == (int)kSessProtected ? r0.z : -1;
    const uint32_t hb = (uint32_t)r0.w;
    const int nh = r1.x;
    const uint32_t h0 = (uint32_t)r1.y, h1 = (uint32_t)r1.z;
    const bool lead = i < a.n && ((r0.y >> 16) & 1);
    const bool sens = sst == (int)kSessReleased && (hb >> 16) > 0;
    {
      const unsigned ml = __ballot_sync(kFull, lead), ms = __ballot_sync(kFull, lead && sens);
      if (lane == 0) {
        s_lead[wid] = ml;
        s_sens[wid] = ms;
      }
    }
    __syncthreads();
    const unsigned lead_word = lane < kNW ? s_lead[lane] : 0u;
    const unsigned sens_word = lane < kNW ? s_sens[lane] : 0u;
    // the window's leaders before `done` are decided; a leader's tentative decision is kept
    // over the iterations while it stays right: an admission stays the argmin as long as its
    // instance keeps headroom for the class (the other instances only lose headroom), and a
    // hold stays a hold
    int done = 0;
    bool have = false;
    uint8_t dec = 0;
    int dw = -1;
    // every iteration finalises at least the window's first undecided leader (its choice is
    // taken against the exact state of its turn), so a window needs at most kNT iterations
    int guard = 0;
#pragma unroll 1
    while (true) {
      const int head = first_set_from(lead_word, lane, done);
      if (head == kNT) break;
      if (++guard > kNT) {
        if (tid == 0) set_error(a.err, MISAT_ERR_INTERNAL);
        return;
      }
      // the first undecided Eq. (7) leader: the leaders before it are decided now, and an
      // Eq. (7) leader at the head is decided alone
      const int qcut = max(first_set_from(sens_word, lane, head), head + 1);
      const int ng0 = s_nglobal;
      const bool act = lead && tid >= head && tid < qcut;
      // 1. choices against the state at the window's current start
      if (act && !have) {
        dw = sel_choose(s, s_hm, W, ng0, L, b, sst, pw, hb, nh, h0, h1, a.H + (int64_t)i * W, a.hold_delay_q, &dec);
        have = true;
      }
      const bool cons = act && dec == MISAT_ADMIT_NEW;
      // 2. admissions per (instance, class)
      const unsigned pm = __match_any_sync(kFull, cons ? dw : -1 - lane);
      const unsigned pc = __match_any_sync(kFull, cons ? dw * 3 + b : -1 - lane);
      const bool gl = cons && lane == __ffs(pm) - 1;  // first lane of its instance in the warp
      const bool cl = cons && lane == __ffs(pc) - 1;
      if (gl) atomicAdd(&s.T[dw], __popc(pm));
      if (cl) atomicAdd(&s.Tb[b * W + dw], __popc(pc));
      __syncthreads();
      bool any;
      {
        const bool over = gl && s.T[dw] > s.gh[dw];
        const bool overc = cl && s.Tb[b * W + dw] > s.ch[b * W + dw];
        if ((over || overc) && atomicCAS(&s.slot[dw], -1, -2) == -1) s.slot[dw] = atomicAdd(&s_nslot, 1);
        any = __syncthreads_or(over || overc);
      }
      int qv = kNT;
      if (any) {
        // exact arrival-order ranks at the over-subscribed instances, kSlotInst at a time: a
        // consumer is invalid when the consumers before it fill its instance or its class
        const int nslot = s_nslot;
        for (int p0 = 0; p0 < nslot; p0 += kSlotInst) {
          const int sl = cons ? s.slot[dw] - p0 : -1;
          const bool mine = sl >= 0 && sl < kSlotInst;
          if (mine && gl) s.wc[(sl * 4) * kNW + wid] = __popc(pm);
          if (mine && cl) s.wc[(sl * 4 + 1 + b) * kNW + wid] = __popc(pc);
          __syncthreads();
          {  // exclusive scan over the warps of each counter: thread = (counter, warp)
            const int v = s.wc[tid];
            int incl = v;
#pragma unroll
            for (int o = 1; o < kNW; o <<= 1) {
              const int t = __shfl_up_sync(kFull, incl, o, kNW);
              if ((lane & (kNW - 1)) >= o) incl += t;
            }
            s.wc[tid] = incl - v;
          }
          __syncthreads();
          bool bad = false;
          if (mine) {
            const unsigned lt = lanemask_lt();
            const int ag = __popc(pm & lt) + s.wc[(sl * 4) * kNW + wid];
            const int ac = __popc(pc & lt) + s.wc[(sl * 4 + 1 + b) * kNW + wid];
            bad = ag >= s.gh[dw] || ac >= s.ch[b * W + dw];
          }
          const unsigned mb = __ballot_sync(kFull, bad);
          if (lane == 0 && mb) atomicMin(&s_q, wid * 32 + __ffs(mb) - 1);
          __syncthreads();
          s.wc[tid] = 0;
          __syncthreads();
        }
        qv = s_q;
      }
      const int q = min(qv, qcut);
      // 3. the leaders before q are final: take their admissions out of the headroom (per
      //    warp, atomically; the one that empties an instance or class clears its flags)
      {
        const bool cc = cons && tid < q;
        const int qw = q - wid * 32;  // lanes of this warp before q
        const unsigned below = qw >= 32 ? kFull : (qw <= 0 ? 0u : ((1u << qw) - 1));
        const unsigned qm = pm & below, qc = pc & below;
        if (cc && lane == __ffs(qm) - 1) {
          const int k = __popc(qm);
          const int g = atomicSub(&s.gh[dw], k);
          if (g > 0 && g - k <= 0) {
            atomicSub(&s_nglobal, 1);
            sel_flags(s, W, dw, b, true, false, s_dirty);
          }
        }
        if (cc && lane == __ffs(qc) - 1) {
          const int k = __popc(qc);
          const int c = atomicSub(&s.ch[b * W + dw], k);
          if (c > 0 && c - k <= 0) sel_flags(s, W, dw, b, false, true, s_dirty);
        }
      }
      __syncthreads();
      if (gl) {
        s.T[dw] = 0;
        s.slot[dw] = -1;
      }
      if (cl) s.Tb[b * W + dw] = 0;
      // the last instance with global headroom filled in this prefix: the holds after the
      // admission that filled it found no global headroom at their turn
      const bool exhausted = ng0 > 0 && s_nglobal == 0;
      if (exhausted) {  // uniform
        const unsigned mf = __ballot_sync(kFull, cons && tid < q);
        if (lane == 0 && mf) atomicMax(&s_f, wid * 32 + 31 - __clz(mf));
        __syncthreads();
      }
      if (act && tid < q) {
        if (dec == MISAT_HOLD_CLASS_CAP && (ng0 == 0 || (exhausted && tid > s_f))) dec = MISAT_HOLD_GLOBAL_CAP;
        if (dec == MISAT_ADMIT_NEW || dec == MISAT_ADMIT_CONT) {
          a.rq.status[i] = kStResolved;
          a.rq.inst[i] = dw;
          a.rq.reason[i] = dec;
        } else {  // (inst may hold an admission of the per-class path, which this replaces)
          a.rq.status[i] = kStHeld;
          a.rq.inst[i] = -1;
          a.rq.last_reason[i] = dec;
        }
      } else if (have && dec == MISAT_ADMIT_NEW && !s.av[b * W + dw]) {
        have = false;  // its instance has no headroom for the class any more: choose again
      }
      done = q;
      // envelopes of the classes that lost an envelope line: one warp per class
      if (wid < 3 && s_dirty[wid]) env_update_warp(s, W, wid, &s_hm[wid], s_env[wid], a.small);
      __syncthreads();
      // nobody reads these again before the next iteration's first barrier
      if (tid == 0) {
        s_q = kNT;
        s_nslot = 0;
        s_f = -1;
        s_dirty[0] = s_dirty[1] = s_dirty[2] = 0;
      }
    }
    __syncthreads();  // the window's bitmasks are read until here
  }
}

size_t select_smem_bytes(int W) {
  return (size_t)W * 8 * 2 + (size_t)W * 48 + (size_t)W * 4 * 4 + (size_t)W * 4 * 4 + (size_t)W * 4 +
         (size_t)kNT * 4 + (size_t)W * 12 + (size_t)W * 2 * 6 + (size_t)W * 9 + 16;
}

cudaError_t select_configure() {
  // sized for the largest instance count, so that contexts of any size share the setting
  return cudaFuncSetAttribute(k4_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)select_smem_bytes(kMaxW));
}

void launch_select(const SelectArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  k4_select<<<1, kNT, select_smem_bytes(a.W), st>>>(a);
}

// ---------------------------------------------------------------------------
// Per-class selection: the path taken when no instance runs out of global headroom.
//
// A leader of class b is eligible on w when w has global headroom and class-b headroom
// (Eq. 6 with the class cap of Sec. 4.2).  As long as every instance keeps global headroom,
// eligibility depends only on the admissions of the leader's own class, so the leaders of the
// three classes form three independent chains.  One CTA per class decides its class's leaders
// in arrival order with the window scheme of k4_select, on one envelope and per-instance
// counters.  At the end the CTAs add up their admissions per instance: if every instance that
// had global headroom at batch start keeps some, no decision could have depended on the global
// cap, and the result is exactly that of the joint arrival order (by induction over the arrival
// order: each instance's global headroom stays positive at every leader's turn, so the joint
// eligibility equals the per-class one, and a hold's reason -- class cap while some instance
// has global headroom -- is the class cap exactly when some instance had it at batch start).
// Otherwise the last CTA sets `coupled` and k4_select decides the whole batch again.
//
// Within a window a tentative admission is final once the registered choosers of its
// instance before it leave it headroom; the first leader that finds none cuts the window.
// Registrations stay in place for the whole window (decided ones included), so the slot where
// an instance runs out (the ch-th registered chooser, ch its headroom at the window's start)
// and the slot of its first chooser that finds none only move earlier as leaders register,
// and are recomputed (one warp per instance) only for the instances that received
// registrations since their last scan.  An instance that runs out leaves the envelope by a
// local repair (the lines between its neighbours that lie below their chord, envelope.cuh),
// and only the undecided leaders that had chosen it choose again.
namespace {
constexpr int kCT = kSelectClassThreads;
constexpr int kMaxBatchBlocks = 4096;  // blocks of 256 requests: batches of up to 2^20 requests
constexpr int kCW = kCT / 32;
static_assert(kCW <= 32 && (kCW & (kCW - 1)) == 0, "the window bitmask is at most one word per lane of a warp");
}  // namespace

struct ClsSmem {
  unsigned* regm;  // [W][kCW] registered choosers of each instance in the window: one bit per slot
  longlong2* ln;   // [W] {d_w, 1/mu_w}
  longlong2* hl;   // [W] {d_w, 1/mu_w} of the envelope lines, slope order
  longlong2* tl;   // [W] scratch of the envelope repair
  int32_t* ch;     // [W] class headroom at the window's start (0 without global headroom)
  int32_t* T;      // [W] registered choosers in the window
  int32_t* fpos;   // [W] window slot of the chooser that takes an instance's last headroom, kCT
  int32_t* pp;     // [W] window slot of its first chooser that finds no headroom, kCT
  int32_t* cand;   // [W] envelope repair candidates
  int32_t* rem;    // [W] instances that ran out in this iteration
  int16_t* hull;   // [W] envelope lines, slope order
  int16_t* th;     // [W] scratch of the envelope repair
  int16_t* hp;     // [W] position of an instance on the envelope, -1 if it is not on it
  int16_t* ord;    // [W] instances in slope order
  int16_t* pos;    // [W] position in slope order
  int16_t* aord;   // [W] instances in (d_w, w) order
  uint8_t* av;     // [W] class headroom left
  unsigned* tm;    // [32] "tight" instances: registered choosers >= class headroom > 0
  unsigned* dm;    // [32] tight instances with registrations since their last scan
};

size_t select_class_smem_bytes(int W, int n) {
  const size_t nblk = ((size_t)n + 255) >> 8;
  return (size_t)256 + (size_t)W * (4 * kCW + 16 * 3 + 4 * 6 + 2 * 6) + (((size_t)W + 15) & ~(size_t)15) +
         nblk * 4 + 64;
}

// First set position >= from in a kCT-bit mask held one word per lane (kCT if none).  Warp-uniform.
__device__ __forceinline__ int cls_first_set(unsigned word, int lane, int from) {
  if (from >= kCT) return kCT;
  const int fw = from >> 5;
  unsigned m = lane < fw ? 0u : word;
  if (lane == fw) m &= ~0u << (from & 31);
  const unsigned nz = __ballot_sync(kFull, m != 0);
  if (!nz) return kCT;
  const int w = __ffs(nz) - 1;
  return w * 32 + __ffs(__shfl_sync(kFull, m, w)) - 1;
}

// Position of the (k+1)-th set bit of x (0 <= k < popc(x)): a binary search on bit counts.
__device__ __forceinline__ int nth_set(unsigned x, int k) {
  int pos = 0;
  int c = __popc(x & 0xffffu);
  if (k >= c) { k -= c; x >>= 16; pos += 16; }
  c = __popc(x & 0xffu);
  if (k >= c) { k -= c; x >>= 8; pos += 8; }
  c = __popc(x & 0xfu);
  if (k >= c) { k -= c; x >>= 4; pos += 4; }
  c = __popc(x & 0x3u);
  if (k >= c) { k -= c; x >>= 2; pos += 2; }
  if (k >= (int)(x & 1u)) pos += 1;
  return pos;
}

// Decision of one leader of the CTA's class against the current state; see sel_choose.
__device__ __forceinline__ int cls_choose(const ClsSmem& s, int m, int nglobal, int64_t x, int sst, int pw,
                                          uint32_t hb, int nh, uint32_t h0, uint32_t h1, const uint16_t* Hrow,
                                          int W, int64_t hold, uint8_t* dec) {
  int64_t best_c = INT64_MAX;
  int best_w = INT32_MAX;
  if (m > 0) {
    int lo = 0, hi = m - 1;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      const longlong2 u = s.hl[mid], v = s.hl[mid + 1];
      const int64_t cu = u.x + x * u.y, cv = v.x + x * v.y;
      // line mid + 1 beats line mid at x (ties to the lower index)
      if (cv < cu || (cv == cu && s.hull[mid + 1] < s.hull[mid])) lo = mid + 1;
      else hi = mid;
    }
    const longlong2 t = s.hl[lo];
    best_w = s.hull[lo];
    best_c = t.x + x * t.y;
  }
  auto consider = [&](int w, int64_t h) {
    const longlong2 t = s.ln[w];
    const int64_t c = t.x + (x - 16 * h) * t.y;
    if (c < best_c || (c == best_c && w < best_w)) {
      best_c = c;
      best_w = w;
    }
  };
  if (nh > 0 && nh <= 2) {
    const int w0 = (int)(h0 >> 16);
    if (s.av[w0] || w0 == pw) consider(w0, h0 & 0xffff);
    if (nh == 2) {
      const int w1 = (int)(h1 >> 16);
      if (s.av[w1] || w1 == pw) consider(w1, h1 & 0xffff);
    }
  } else if (nh > 2) {
    for (int w = 0; w < W; ++w) {
      const int h = Hrow[w];
      if (h && (s.av[w] || w == pw)) consider(w, h);
    }
  }
  if (pw >= 0) consider(pw, 0);
  if (best_w == INT32_MAX) {
    *dec = nglobal > 0 ? MISAT_HOLD_CLASS_CAP : MISAT_HOLD_GLOBAL_CAP;
    return -1;
  }
  const int hmax = (int)(hb >> 16), whit = 65535 - (int)(hb & 0xffffu);
  if (sst == kSessReleased && hmax > 0 && !s.av[whit]) {
    const int64_t lhs = hold + s.ln[whit].x - s.ln[best_w].x;
    const int64_t rhs = 16 * (int64_t)hmax * s.ln[whit].y;
    if (lhs < rhs) {
      *dec = MISAT_HOLD_PREFER_CACHE;
      return -1;
    }
  }
  *dec = best_w == pw ? MISAT_ADMIT_CONT : MISAT_ADMIT_NEW;
  return best_w;
}

__device__ __forceinline__ bool cls_present(const ClsSmem& s, int i) { return s.av[i] || s.hp[i] >= 0; }

// Envelope repair after instance w ran out of headroom (one warp).  The lines p and q that bound
// the repaired stretch are w's neighbours on the envelope, or, where w was the first (last)
// line, the line that now wins at x = 0 (for large x).  The lines strictly between p and q in
// slope order that lie below the chord p-q are the candidates; each is tested against p, q and
// the other candidates (EnvTest over the domain x >= 0), and the ones on the envelope replace
// w.  A line that ran out in the same iteration but is still on the envelope counts as present
// until its own repair, so that every repair computes the envelope of a well-defined set; the
// order of the repairs does not change the final envelope.  first_a / last_s: forward-only
// pointers to the lines that may win at x = 0 ((d_w, w) order) and for large x (slope order).
__device__ __forceinline__ void cls_repair(const ClsSmem& s, int W, int w, int* hm, int* first_a, int* last_s,
                                           bool small) {
  const int lane = threadIdx.x & 31;
  const int k = s.hp[w];
  __syncwarp();
  if (k < 0) return;
  if (lane == 0) s.hp[w] = -1;
  __syncwarp();
  const int m = *hm;
  const int P = k > 0 ? s.hull[k - 1] : -1, Q = k + 1 < m ? s.hull[k + 1] : -1;
  int p = P, q = Q;
  if (p < 0) {  // the line that now wins at x = 0
    int a = *first_a;
    while (a < W && !cls_present(s, s.aord[a])) ++a;
    p = a < W ? s.aord[a] : -1;
    __syncwarp();
    if (lane == 0) *first_a = a;
  }
  if (q < 0 && p >= 0) {  // the line that now wins for large x: least 1/mu_w, then least d_w
    int x = *last_s;
    while (x >= 0 && !cls_present(s, s.ord[x])) --x;
    __syncwarp();
    if (lane == 0) *last_s = x;
    const int64_t t = s.ln[s.ord[x]].y;
    int y = x;
    for (int z = x - 1; z >= 0 && s.ln[s.ord[z]].y == t; --z)
      if (cls_present(s, s.ord[z])) y = z;
    q = s.ord[y];
  }
  int nnew = 0;
  if (P < 0 && p >= 0 && p != Q) {
    if (lane == 0) s.th[0] = (int16_t)p;
    nnew = 1;
  }
  if (p >= 0 && q != p) {
    const int xp = s.pos[p], xq = s.pos[q];
    const longlong2 lp = s.ln[p], lq = s.ln[q];
    int nc = 0;
    for (int x0 = xp + 1; x0 < xq; x0 += 32) {
      const int x = x0 + lane;
      bool c = false;
      int i = 0;
      if (x < xq) {
        i = s.ord[x];
        if (s.av[i]) {
          const longlong2 li = s.ln[i];
          c = li.y != lp.y && env_below_chord(li.x, li.y, i, lp.x, lp.y, p, lq.x, lq.y, q, small);
        }
      }
      const unsigned mc = __ballot_sync(kFull, c);
      if (c) s.cand[nc + __popc(mc & lanemask_lt())] = i;
      nc += __popc(mc);
    }
    __syncwarp();
    if (nc == 1) {
      // a single line below the chord beats p and q around their crossing (x >= 0): it is on
      // the envelope, and nothing else enters between p and q
      if (lane == 0) s.th[nnew] = (int16_t)s.cand[0];
      nnew += 1;
    }
    for (int e0 = 0; nc > 1 && e0 < nc; e0 += 32) {
      const int e = e0 + lane;
      bool on = false;
      int i = 0;
      if (e < nc) {
        i = s.cand[e];
        const longlong2 li = s.ln[i];
        EnvTest t;
        env_test_init(t);
        env_test_add(t, li.x, li.y, i, lp.x, lp.y, p, small);
        env_test_add(t, li.x, li.y, i, lq.x, lq.y, q, small);
        for (int f = 0; f < nc; ++f) {
          const int j = s.cand[f];
          if (j != i) {
            const longlong2 lj = s.ln[j];
            env_test_add(t, li.x, li.y, i, lj.x, lj.y, j, small);
          }
        }
        on = env_test_on(t, small);
      }
      const unsigned mo = __ballot_sync(kFull, on);
      if (on) s.th[nnew + __popc(mo & lanemask_lt())] = (int16_t)i;
      nnew += __popc(mo);
    }
    if (Q < 0 && q != P) {
      if (lane == 0) s.th[nnew] = (int16_t)q;
      nnew += 1;
    }
  }
  __syncwarp();
  // splice: hull[0..k-1] ++ th[0..nnew-1] ++ hull[k+1..m-1]
  const int tail = m - k - 1;
  for (int t = lane; t < tail; t += 32) {
    s.th[nnew + t] = s.hull[k + 1 + t];
    s.tl[nnew + t] = s.hl[k + 1 + t];
  }
  for (int t = lane; t < nnew; t += 32) s.tl[t] = s.ln[s.th[t]];
  __syncwarp();
  const int total = nnew + tail;
  for (int t = lane; t < total; t += 32) {
    const int v = s.th[t];
    s.hull[k + t] = (int16_t)v;
    s.hl[k + t] = s.tl[t];
    s.hp[v] = (int16_t)(k + t);
  }
  if (lane == 0) *hm = k + total;
  __syncwarp();
}

__global__ void __launch_bounds__(kCT, 1) k4_select_class(SelectClassArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int s_nc, s_hm, s_first_a, s_last_s, s_nglobal, s_last, s_navail;
  __shared__ int s_qb[2];  // cut bound of the current and the next iteration
  __shared__ int s_ws[kCW];
  __shared__ unsigned s_lead[kCW], s_sens[kCW];
  if (block_error(a.err)) return;
  const int W = a.W, b = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  ClsSmem s;
  {
    unsigned char* p = smem;
    s.tm = reinterpret_cast<unsigned*>(p);
    s.dm = s.tm + 32;
    p += 256;
    s.regm = reinterpret_cast<unsigned*>(p);
    p += (size_t)W * kCW * 4;
    s.ln = reinterpret_cast<longlong2*>(p);
    p += (size_t)W * 16;
    s.hl = reinterpret_cast<longlong2*>(p);
    p += (size_t)W * 16;
    s.tl = reinterpret_cast<longlong2*>(p);
    p += (size_t)W * 16;
    s.ch = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.T = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.fpos = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.pp = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.cand = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.rem = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.hull = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.th = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.hp = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.ord = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.pos = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.aord = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.av = p;
  }
  if (tid == 0) {
    s_nglobal = 0;
    s_qb[0] = kCT;
    s_first_a = 0;
    s_last_s = W - 1;
    s_navail = 0;
  }
  __syncthreads();
  for (int w = tid; w < W; w += kCT) {
    const int r = a.rank[w];
    s.ord[r] = (int16_t)w;
    s.pos[w] = (int16_t)r;
    s.aord[a.rank_a[w]] = (int16_t)w;
    s.ln[w] = make_longlong2(a.backlog[w], a.tokcost[w]);
    const int g = a.gh[w];
    if (g > 0) atomicAdd(&s_nglobal, 1);
    const int c = g > 0 ? a.ch[w * 3 + b] : 0;
    s.ch[w] = c;
    s.av[w] = c > 0;
    if (c > 0) atomicAdd(&s_navail, 1);
    s.T[w] = 0;
    s.fpos[w] = kCT;
    s.pp[w] = kCT;
    s.hp[w] = -1;
  }
  for (int i = tid; i < W * kCW; i += kCT) s.regm[i] = 0;
  if (tid < 64) s.tm[tid] = 0;  // tm and dm
  __syncthreads();
  // initial envelope of the class (launch_env_init), compacted in slope order
  if (wid == 0) {
    int base = 0;
    for (int x0 = 0; x0 < W; x0 += 32) {
      const int x = x0 + lane;
      const int w = x < W ? s.ord[x] : 0;
      const bool f = x < W && a.onhull[b * W + w];
      const unsigned mf = __ballot_sync(kFull, f);
      if (f) {
        const int k = base + __popc(mf & lanemask_lt());
        s.hull[k] = (int16_t)w;
        s.hl[k] = s.ln[w];
        s.hp[w] = (int16_t)k;
      }
      base += __popc(mf);
    }
    if (lane == 0) s_hm = base;
  }
  // The class's leaders in arrival order: the prep kernel listed them per block of 256
  // requests; the block offsets are an exclusive scan of its counts (s_pre), and the class
  // index g of a leader maps to its block by binary search.
  const int nblk = (a.n + 255) >> 8;
  const int32_t* seg = a.seg + (int64_t)b * a.n;
  int* s_pre = reinterpret_cast<int*>(s.av + ((W + 15) & ~15));
  {
    constexpr int kPer = (kMaxBatchBlocks + kCT - 1) / kCT;
    int v[kPer], t = 0;
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int j = tid * kPer + u;
      v[u] = j < nblk ? a.segcnt[b * nblk + j] : 0;
      t += v[u];
    }
    int incl = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int x = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += x;
    }
    if (lane == 31) s_ws[wid] = incl;
    __syncthreads();
    if (wid == 0) {
      const int x = lane < kCW ? s_ws[lane] : 0;
      int wi = x;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFull, wi, o);
        if (lane >= o) wi += y;
      }
      if (lane < kCW) s_ws[lane] = wi - x;
      if (lane == 31) s_nc = wi;
    }
    __syncthreads();
    int off = s_ws[wid] + incl - t;
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int j = tid * kPer + u;
      if (j < nblk) s_pre[j] = off;
      off += v[u];
    }
    __syncthreads();
  }
  const int nc = s_nc;
  // request of class index g (< nc): the last block whose offset is <= g
  auto leader_at = [&](int g) -> int {
    int lo = 0, hi = nblk - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_pre[mid] <= g) lo = mid;
      else hi = mid - 1;
    }
    return seg[(int64_t)lo * 256 + (g - s_pre[lo])];
  };
  const int nglobal = s_nglobal;

  // records of the first window
  int rn = tid < nc ? leader_at(tid) : 0;
  int4 n0 = make_int4(0, 0, 0, 0), n1 = make_int4(0, 0, 0, 0);
  if (tid < nc) {
    n0 = a.rec[2 * rn];
    n1 = a.rec[2 * rn + 1];
  }
#pragma unroll 1
  for (int base = 0; base < nc; base += kCT) {
    if (s_navail == 0) {
      // no instance has headroom for the class any more: every remaining leader is decided
      // on its own (a protected session continues on its instance, anyone else is held)
      for (int i = base + tid; i < nc; i += kCT) {
        const int r = leader_at(i);
        const int4 r0 = a.rec[2 * r];
        if (((r0.y >> 8) & 0xff) == (int)kSessProtected) {
          a.rq.status[r] = kStResolved;
          a.rq.inst[r] = r0.z;
          a.rq.reason[r] = MISAT_ADMIT_CONT;
        } else {
          a.rq.status[r] = kStHeld;
          a.rq.inst[r] = -1;
          a.rq.last_reason[r] = nglobal > 0 ? MISAT_HOLD_CLASS_CAP : MISAT_HOLD_GLOBAL_CAP;
        }
      }
      break;
    }
    const int i = base + tid;
    const bool valid = i < nc;
    const int r = rn;
    const int4 r0 = n0, r1 = n1;
    if (i + kCT < nc) {  // the next window's records, in flight during this one
      rn = leader_at(i + kCT);
      n0 = a.rec[2 * rn];
      n1 = a.rec[2 * rn + 1];
    }
    const int64_t L = r0.x;
    const int sst = (r0.y >> 8) & 0xff;
    const int pw = sst == (int)kSessProtected ? r0.z : -1;
    const uint32_t hb = (uint32_t)r0.w;
    const int nh = r1.x;
    const uint32_t h0 = (uint32_t)r1.y, h1 = (uint32_t)r1.z;
    const bool sens = valid && sst == (int)kSessReleased && (hb >> 16) > 0;
    {
      const unsigned ml = __ballot_sync(kFull, valid), ms = __ballot_sync(kFull, sens);
      if (lane == 0) {
        s_lead[wid] = ml;
        s_sens[wid] = ms;
      }
    }
    __syncthreads();
    const unsigned lead_word = lane < kCW ? s_lead[lane] : 0u;
    const unsigned sens_word = lane < kCW ? s_sens[lane] : 0u;
    int done = 0, par = 0;
    bool have = false, reg = false;
    uint8_t dec = 0;
    int dw = -1;
    int guard = 0;
#pragma unroll 1
    while (true) {
      const int head = cls_first_set(lead_word, lane, done);
      if (head == kCT) break;
      if (++guard > 2 * kCT) {  // every iteration decides at least the leader at `head`
        if (tid == 0) set_error(a.err, MISAT_ERR_INTERNAL);
        return;
      }
      // an Eq. (7) leader is decided alone, at the head, against the exact state of its turn
      const int qcut = max(cls_first_set(sens_word, lane, head), head + 1);
      const bool act = valid && tid >= head && tid < qcut;
      // 1. an undecided leader whose instance ran out chooses again (its stale registration
      //    stays with that instance, which is never scanned again); choices and registration,
      //    one shared-memory update per (warp, instance)
      if (tid >= done && reg && !s.av[dw]) {
        reg = false;
        have = false;
      }
      bool nreg = false;
      if (act && !have) {
        dw = cls_choose(s, s_hm, nglobal, L, sst, pw, hb, nh, h0, h1, a.H + (int64_t)r * W, W, a.hold_delay_q, &dec);
        have = true;
        nreg = dec == MISAT_ADMIT_NEW;
        reg = nreg;
      }
      if (__any_sync(kFull, nreg)) {
        const unsigned grp = __match_any_sync(kFull, nreg ? dw : -1 - lane);
        if (nreg && lane == __ffs(grp) - 1) {
          s.regm[dw * kCW + wid] |= grp;  // word (dw, wid) is written by this warp only
          const int t1 = atomicAdd(&s.T[dw], __popc(grp)) + __popc(grp);
          if (t1 >= s.ch[dw]) {
            const unsigned bit = 1u << (dw & 31);
            if (!(s.tm[dw >> 5] & bit)) atomicOr(&s.tm[dw >> 5], bit);
            if (!(s.dm[dw >> 5] & bit)) atomicOr(&s.dm[dw >> 5], bit);
          }
        }
      }
      __syncthreads();
      // 2. tight instances with new registrations: the slot of the chooser that takes the last
      //    headroom (fpos) and of the first one that finds none (pp); the k-th such instance
      //    goes to warp k mod kCW.  Both slots only move earlier while the instance is tight,
      //    so the cut bound starts from the others' pp (set by step 3 of the last iteration).
      {
        const unsigned word = s.tm[lane] & s.dm[lane];
        const unsigned nzw = __ballot_sync(kFull, word != 0);
        int seen = 0;
        for (unsigned zz = nzw; zz; zz &= zz - 1) {
          const int wi = __ffs(zz) - 1;
          const unsigned bits = __shfl_sync(kFull, word, wi);
          unsigned mine = 0;
          for (unsigned t = bits; t; t &= t - 1) {
            if ((seen & (kCW - 1)) == wid) mine |= t & (0u - t);
            ++seen;
          }
          while (mine) {
            const int w = 32 * wi + __ffs(mine) - 1;
            mine &= mine - 1;
            const int need = s.ch[w];
            // lane j holds the registered choosers of w among slots [32 j, 32 j + 32)
            const unsigned word = lane < kCW ? s.regm[w * kCW + lane] : 0u;
            const int c = __popc(word);
            int incl = c;
#pragma unroll
            for (int o = 1; o < kCW; o <<= 1) {
              const int t = __shfl_up_sync(kFull, incl, o);
              if (lane >= o) incl += t;
            }
            // slots of the need-th and (need + 1)-th registered choosers of w (kCT if fewer)
            const unsigned mx1 = __ballot_sync(kFull, lane < kCW && incl >= need);
            const unsigned mx2 = __ballot_sync(kFull, lane < kCW && incl > need);
            const int l1 = mx1 ? __ffs(mx1) - 1 : 0, l2 = mx2 ? __ffs(mx2) - 1 : 0;
            const unsigned w1 = __shfl_sync(kFull, word, l1), w2 = __shfl_sync(kFull, word, l2);
            const int before1 = __shfl_sync(kFull, incl - c, l1), before2 = __shfl_sync(kFull, incl - c, l2);
            const int f = mx1 ? 32 * l1 + nth_set(w1, need - 1 - before1) : kCT;
            const int p = mx2 ? 32 * l2 + nth_set(w2, need - before2) : kCT;
            if (lane == 0) {
              s.fpos[w] = f;
              s.pp[w] = p;
              if (p < kCT) atomicMin(&s_qb[par], p);
            }
          }
        }
      }
      __syncthreads();
      const int q = min(s_qb[par], qcut);
      // 3. the leaders before q are decided; warp 0 takes the instances whose last headroom
      //    went to one of them out of the envelope, and sets the next iteration's cut bound
      if (act && tid < q) {
        if (dec == MISAT_ADMIT_NEW || dec == MISAT_ADMIT_CONT) {
          a.rq.status[r] = kStResolved;
          a.rq.inst[r] = dw;
          a.rq.reason[r] = dec;
        } else {
          a.rq.status[r] = kStHeld;
          a.rq.inst[r] = -1;
          a.rq.last_reason[r] = dec;
        }
      }
      if (wid == 0) {
        const unsigned word = s.tm[lane];
        unsigned out = 0;
        int mn = kCT;
        for (unsigned t = word; t; t &= t - 1) {  // lane-local: the tight instances of word `lane`
          const int w = 32 * lane + __ffs(t) - 1;
          if (s.fpos[w] < q) {
            out |= t & (0u - t);
            s.fpos[w] = kCT;
            s.pp[w] = kCT;
          } else {
            mn = min(mn, s.pp[w]);
          }
        }
        s.tm[lane] = word & ~out;
        s.dm[lane] = 0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mn = min(mn, __shfl_xor_sync(kFull, mn, o));
        if (lane == 0) s_qb[par ^ 1] = mn;  // last read before the barrier above
        // instances that ran out, in index order
        int cnt = __popc(out), excl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int v = __shfl_up_sync(kFull, excl, o);
          if (lane >= o) excl += v;
        }
        const int nrem = __shfl_sync(kFull, excl, 31);
        excl -= cnt;
        if (lane == 0) s_navail -= nrem;
        for (unsigned t = out; t; t &= t - 1) {
          const int w = 32 * lane + __ffs(t) - 1;
          s.av[w] = 0;
          s.rem[excl++] = w;
        }
        __syncwarp();
        for (int e = 0; e < nrem; ++e) cls_repair(s, W, s.rem[e], &s_hm, &s_first_a, &s_last_s, a.small);
      }
      __syncthreads();
      done = q;
      par ^= 1;
    }
    // end of the window: every tight instance ran out (its last headroom went to a decided
    // leader); the others lose the window's admissions
    for (int w = tid; w < W; w += kCT) {
      s.ch[w] = s.av[w] ? s.ch[w] - s.T[w] : 0;
      s.T[w] = 0;
    }
    for (int i = tid; i < W * kCW; i += kCT) s.regm[i] = 0;
    if (tid == 0) s_qb[0] = kCT;
    __syncthreads();  // s_lead / s_sens are rewritten by the next window
  }
  // admissions per instance, and the check that no instance ran out of global headroom
  for (int w = tid; w < W; w += kCT) {
    const int c0 = a.gh[w] > 0 ? a.ch[w * 3 + b] : 0;
    const int used = c0 - s.ch[w];
    if (used) atomicAdd(&a.adm[w], used);
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(a.ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (s_last) {
    __threadfence();
    bool bad = false;
    for (int w = tid; w < W; w += kCT) {
      const int g = a.gh[w];
      if (g > 0 && __ldcg(&a.adm[w]) >= g) bad = true;
    }
    if (__syncthreads_or(bad) && tid == 0) {
      *a.coupled = 1;
      a.stats[25] = 1;
    }
  }
}

cudaError_t select_class_configure() {
  return cudaFuncSetAttribute(k4_select_class, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)select_class_smem_bytes(kMaxW, 256 * kMaxBatchBlocks));
}

void launch_select_class(const SelectClassArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  k4_select_class<<<3, kCT, select_class_smem_bytes(a.W, a.n), st>>>(a);
}

}  // namespace misat
