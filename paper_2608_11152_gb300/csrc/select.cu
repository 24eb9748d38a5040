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
//   2. the warps then take turns in arrival order (a chain of named barriers): each checks
//      its 32 leaders against the headroom left by the leaders before them and takes their
//      admissions out of it, up to the first leader whose instance has no headroom left at
//      its turn;
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
static_assert(kNW >= 2 && kNW <= 16, "the admission chain uses named barriers 1 .. kNW - 1");
}  // namespace

// ---------------------------------------------------------------------------
// Per-request records for the selection (32 bytes, one coalesced pair of loads):
//   rec[2r]   = {L, cls | sst << 8 | leader << 16, protected / last instance, hbest}
//   rec[2r+1] = {instances with H > 0, first two of them as (w << 16 | H), 0}
__global__ void __launch_bounds__(256) k3_select_prep(SelectPrepArgs a) {
  if (block_error(a.err)) return;
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
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
// Initial envelopes and slope order.  blockIdx.y = class b (0..2): is line i on the lower
// envelope of the instances with headroom for class b?  blockIdx.y = 3: position of line i
// in slope order.  Eight lanes share line i, each taking every eighth other line.
__device__ __forceinline__ __int128 shfl_xor_i128(__int128 v, int o) {
  uint64_t lo = (uint64_t)v, hi = (uint64_t)((unsigned __int128)v >> 64);
  lo = __shfl_xor_sync(kFull, lo, o);
  hi = __shfl_xor_sync(kFull, hi, o);
  return (__int128)(((unsigned __int128)hi << 64) | lo);
}

__global__ void __launch_bounds__(1024) k3_env_init(EnvInitArgs a) {
  if (block_error(a.err)) return;
  const int i = blockIdx.x * 128 + (threadIdx.x >> 3);
  const int sub = threadIdx.x & 7;
  const int b = blockIdx.y;
  const bool line = i < a.W;
  const int64_t bki = line ? a.backlog[i] : 0, tci = line ? a.tokcost[i] : 0;
  if (b == 3) {
    int cnt = 0;
    if (line)
      for (int j = sub; j < a.W; j += 8)
        if (j != i && env_slope_before(a.backlog[j], a.tokcost[j], j, bki, tci, i)) ++cnt;
#pragma unroll
    for (int o = 4; o > 0; o >>= 1) cnt += __shfl_xor_sync(kFull, cnt, o);
    if (line && sub == 0) a.rank[i] = cnt;
    return;
  }
  auto avail = [&](int w) { return a.gh[w] > 0 && a.ch[w * 3 + b] > 0; };
  const bool ai = line && avail(i);
  EnvTest t;
  env_test_init(t);
  if (ai)
    for (int j = sub; j < a.W; j += 8)
      if (j != i && avail(j)) env_test_add(t, bki, tci, i, a.backlog[j], a.tokcost[j], j);
#pragma unroll
  for (int o = 4; o > 0; o >>= 1) {
    EnvTest u;
    u.lo_num = shfl_xor_i128(t.lo_num, o);
    u.lo_den = __shfl_xor_sync(kFull, t.lo_den, o);
    u.hi_num = shfl_xor_i128(t.hi_num, o);
    u.hi_den = __shfl_xor_sync(kFull, t.hi_den, o);
    u.has_hi = __shfl_xor_sync(kFull, t.has_hi, o);
    u.dominated = __shfl_xor_sync(kFull, t.dominated, o);
    env_test_merge(t, u);
  }
  if (line && sub == 0) a.onhull[b * a.W + i] = ai && env_test_on(t) ? 1 : 0;
}

void launch_select_prep(const SelectPrepArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  k3_select_prep<<<(a.n + 255) / 256, 256, 0, st>>>(a);
}

void launch_env_init(const EnvInitArgs& a, cudaStream_t st) {
  dim3 grid((a.W + 127) / 128, 4);
  k3_env_init<<<grid, 1024, 0, st>>>(a);
}

// ---------------------------------------------------------------------------
// Shared state of the selection CTA.  Per class, the headroom flags are kept both by instance
// (queries) and in slope order (envelope updates read them as contiguous bytes).
struct SelSmem {
  int64_t* bk;     // [W] d_w
  int64_t* tc;     // [W] 1/mu_w
  int32_t* gh;     // [W] global headroom
  int32_t* ch;     // [3][W] class headroom
  int32_t* surv;   // [3][W] envelope candidates of each class's update
  int16_t* ord;    // [W] instances in slope order
  int16_t* pos;    // [W] position in slope order
  int16_t* hull;   // [3][W] envelope lines per class, slope order
  uint8_t* av;     // [3][W] headroom for the class (gh > 0 and ch > 0), by instance
  uint8_t* avp;    // [3][W] the same by slope position
  uint8_t* onp;    // [3][W] on the envelope of the class, by slope position
};

// Per-class scratch of an envelope update (one warp per class).
struct EnvScratch {
  int gp[kMaxGaps];
  int gq[kMaxGaps];
};

// Rebuild hull[b] from the on-envelope flags (compaction in slope order).  One warp.
__device__ void env_compact_warp(const SelSmem& s, int W, int b, int* hm) {
  const int lane = threadIdx.x & 31;
  int base = 0;
#pragma unroll 4
  for (int x0 = 0; x0 < W; x0 += 32) {
    const int x = x0 + lane;
    const bool f = x < W && s.onp[b * W + x];
    const unsigned m = __ballot_sync(kFull, f);
    if (f) s.hull[b * W + base + __popc(m & lanemask_lt())] = s.ord[x];
    base += __popc(m);
  }
  if (lane == 0) *hm = base;
  __syncwarp();
}

// Dual point i strictly below the segment p-q (slopes p > i > q): below every chord, a line
// may join the envelope between p and q; above it, it cannot.
__device__ __forceinline__ bool env_below_chord(const SelSmem& s, int i, int p, int q) {
  const __int128 lhs = env_adiff(s.bk[i], i, s.bk[p], p) * (__int128)((s.tc[p] - s.tc[q]) * 1024);
  const __int128 rhs = env_adiff(s.bk[q], q, s.bk[p], p) * (__int128)((s.tc[p] - s.tc[i]) * 1024);
  return lhs < rhs;
}

// The line of class b's available ones at slope positions [x0, x1] with the least key:
// by_slope = 0: (d_w, w) -- the line that wins at x = 0; by_slope = 1: (1/mu_w, d_w, w) -- the
// line that wins as x grows.  -1 if none.  One warp.
__device__ int env_end_line_warp(const SelSmem& s, int W, int b, int x0, int x1, int by_slope) {
  const int lane = threadIdx.x & 31;
  int64_t k1 = INT64_MAX, k2 = INT64_MAX;
  int bw = INT32_MAX;
  auto better = [](int64_t a1, int64_t a2, int aw, int64_t c1, int64_t c2, int cw) {
    return a1 < c1 || (a1 == c1 && (a2 < c2 || (a2 == c2 && aw < cw)));
  };
  for (int x = x0 + lane; x <= x1; x += 32) {
    if (!s.avp[b * W + x]) continue;
    const int i = s.ord[x];
    const int64_t c1 = by_slope ? s.tc[i] : s.bk[i];
    const int64_t c2 = by_slope ? s.bk[i] : 0;
    if (better(c1, c2, i, k1, k2, bw)) {
      k1 = c1;
      k2 = c2;
      bw = i;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const int64_t o1 = __shfl_xor_sync(kFull, k1, o), o2 = __shfl_xor_sync(kFull, k2, o);
    const int ow = __shfl_xor_sync(kFull, bw, o);
    if (better(o1, o2, ow, k1, k2, bw)) {
      k1 = o1;
      k2 = o2;
      bw = ow;
    }
  }
  return bw == INT32_MAX ? -1 : bw;
}

// Remove the lines of class b that lost their headroom from its envelope.  One warp.
// Each maximal run of removed envelope lines leaves a gap between its surviving neighbours p
// and q (slope order).  A gap at the start of the envelope is closed by the line that now
// wins at x = 0 (least d_w: it is on the envelope), one at the end by the line that now wins
// for large x (least 1/mu_w).  Between p and q the envelope is that of p, q and the lines of
// slope strictly between them that lie below the chord p-q: a line above it cannot be on the
// envelope there, and does not change the envelope of the ones below it.
__device__ void env_update_warp(const SelSmem& s, int W, int b, int* hm, EnvScratch& sc) {
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
          if (j != i && s.av[b * W + j]) env_test_add(t, s.bk[i], s.tc[i], i, s.bk[j], s.tc[j], j);
        on = env_test_on(t);
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
        p = env_end_line_warp(s, W, b, 0, q >= 0 ? s.pos[q] : W - 1, 0);
        if (p >= 0 && lane == 0) s.onp[b * W + s.pos[p]] = 1;
      }
      if (p >= 0 && q < 0) {  // the end was removed: the line that now wins for large x
        q = env_end_line_warp(s, W, b, s.pos[p], W - 1, 1);
        if (lane == 0) s.onp[b * W + s.pos[q]] = 1;
      }
      if (p < 0 || q < 0 || p == q) continue;
      const int g0 = ns;
      const int xp = s.pos[p], xq = s.pos[q];
      const int64_t tcp = s.tc[p];
      for (int x0 = xp + 1; x0 < xq; x0 += 32) {
        const int x = x0 + lane;
        bool c = false;
        int i = 0;
        if (x < xq && s.avp[b * W + x]) {
          i = s.ord[x];
          c = s.tc[i] != tcp && env_below_chord(s, i, p, q);
        }
        const unsigned mc = __ballot_sync(kFull, c);
        if (c) surv[ns + __popc(mc & lanemask_lt())] = i;
        ns += __popc(mc);
      }
      __syncwarp();
      // each candidate against p, q and the other candidates of this gap
      for (int e = g0 + lane; e < ns; e += 32) {
        const int i = surv[e];
        EnvTest t;
        env_test_init(t);
        env_test_add(t, s.bk[i], s.tc[i], i, s.bk[p], s.tc[p], p);
        env_test_add(t, s.bk[i], s.tc[i], i, s.bk[q], s.tc[q], q);
        for (int f = g0; f < ns; ++f) {
          const int j = surv[f];
          if (j != i) env_test_add(t, s.bk[i], s.tc[i], i, s.bk[j], s.tc[j], j);
        }
        if (env_test_on(t)) s.onp[b * W + s.pos[i]] = 1;
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
  const int64_t x = L;
  if (m > 0) {
    int lo = 0, hi = m - 1;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      const int u = hull[mid], v = hull[mid + 1];
      if (env_beats(s.bk[v], s.tc[v], v, s.bk[u], s.tc[u], u, x)) lo = mid + 1;
      else hi = mid;
    }
    best_w = hull[lo];
    best_c = s.bk[best_w] + x * s.tc[best_w];
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

// Named barrier k of the admission chain: warp k - 1 arrives, warp k waits (64 threads).
__device__ __forceinline__ void chain_wait(int k) { asm volatile("bar.sync %0, 64;" ::"r"(k) : "memory"); }
__device__ __forceinline__ void chain_pass(int k) { asm volatile("bar.arrive %0, 64;" ::"r"(k) : "memory"); }

// An instance's headroom drops: clear its flags for the classes it no longer admits.
__device__ __forceinline__ void sel_take(const SelSmem& s, int W, int w, int b, int kg, int kc, int* s_nglobal,
                                         int* s_dirty) {
  if (kg) {
    const int g = s.gh[w] - kg;
    s.gh[w] = g;
    if (g <= 0) {
      atomicSub(s_nglobal, 1);
#pragma unroll
      for (int c = 0; c < 3; ++c)
        if (s.av[c * W + w]) {
          s.av[c * W + w] = 0;
          const int x = s.pos[w];
          s.avp[c * W + x] = 0;
          if (s.onp[c * W + x]) s_dirty[c] = 1;
        }
    }
  }
  if (kc) {
    const int c = s.ch[b * W + w] - kc;
    s.ch[b * W + w] = c;
    if (c <= 0 && s.av[b * W + w]) {
      s.av[b * W + w] = 0;
      const int x = s.pos[w];
      s.avp[b * W + x] = 0;
      if (s.onp[b * W + x]) s_dirty[b] = 1;
    }
  }
}

__global__ void __launch_bounds__(kNT, 1) k4_select(SelectArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ int s_hm[3], s_q, s_nglobal, s_dirty[3];
  __shared__ unsigned s_lead[kNW], s_sens[kNW];
  __shared__ EnvScratch s_env[3];
  if (block_error(a.err)) return;
  const int W = a.W;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  SelSmem s;
  {
    unsigned char* p = smem;
    s.bk = reinterpret_cast<int64_t*>(p);
    p += (size_t)W * 8;
    s.tc = reinterpret_cast<int64_t*>(p);
    p += (size_t)W * 8;
    s.gh = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 4;
    s.ch = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 12;
    s.surv = reinterpret_cast<int32_t*>(p);
    p += (size_t)W * 12;
    s.ord = reinterpret_cast<int16_t*>(p);
    p += (size_t)W * 2;
    s.pos = reinterpret_cast<int16_t*>(p);
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
    s_dirty[0] = s_dirty[1] = s_dirty[2] = 0;
  }
  __syncthreads();
  for (int w = tid; w < W; w += kNT) {
    const int r = a.rank[w];
    s.ord[r] = (int16_t)w;
    s.pos[w] = (int16_t)r;
    s.bk[w] = a.backlog[w];
    s.tc[w] = a.tokcost[w];
    const int32_t g = a.gh[w];
    s.gh[w] = g;
    if (g > 0) atomicAdd(&s_nglobal, 1);
#pragma unroll
    for (int b = 0; b < 3; ++b) {
      const int32_t c = a.ch[w * 3 + b];
      const uint8_t v = g > 0 && c > 0;
      s.ch[b * W + w] = c;
      s.av[b * W + w] = v;
      s.avp[b * W + r] = v;
      s.onp[b * W + r] = a.onhull[b * W + w];
    }
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
      const bool act = lead && tid >= head && tid < qcut;
      if (act && !have) {
        dw = sel_choose(s, s_hm, W, s_nglobal, L, b, sst, pw, hb, nh, h0, h1, a.H + (int64_t)i * W, a.hold_delay_q,
                        &dec);
        have = true;
      }
      const bool cons = act && dec == MISAT_ADMIT_NEW;
      const unsigned pm = __match_any_sync(kFull, cons ? dw : -1 - lane);
      const unsigned pc = __match_any_sync(kFull, cons ? dw * 3 + b : -1 - lane);
      // 2. the admission chain: warps in arrival order
      bool fin = false;  // this lane's decision is final in this iteration
      if (wid > 0) chain_wait(wid);
      if (s_q == kNT) {
        const int ng_before = s_nglobal;
        const unsigned lt = lanemask_lt();
        const bool ok = !cons || ((int)__popc(pm & lt) < s.gh[dw] && (int)__popc(pc & lt) < s.ch[b * W + dw]);
        const unsigned bad = __ballot_sync(kFull, !ok);
        const int f = bad ? __ffs(bad) - 1 : 32;  // first lane without headroom at its turn
        const unsigned below = f == 32 ? kFull : ((1u << f) - 1);
        const bool cc = cons && lane < f;
        const unsigned pmc = pm & below, pcc = pc & below;
        const bool gl = cc && lane == __ffs(pmc) - 1, cl = cc && lane == __ffs(pcc) - 1;
        if (gl || cl) sel_take(s, W, dw, b, gl ? __popc(pmc) : 0, cl ? __popc(pcc) : 0, &s_nglobal, s_dirty);
        __syncwarp();
        fin = act && lane < f;
        const unsigned adm = __ballot_sync(kFull, cc);
        if (fin && (dec == MISAT_HOLD_CLASS_CAP || dec == MISAT_HOLD_GLOBAL_CAP)) {
          // at its turn, is there global headroom left?  None before this warp, or the last
          // one filled by an earlier admission of this warp
          const bool gone = ng_before == 0 ||
                            (s_nglobal == 0 && adm != 0 && lane > 31 - (int)__clz(adm));
          dec = gone ? MISAT_HOLD_GLOBAL_CAP : MISAT_HOLD_CLASS_CAP;
        }
        if (f < 32 && lane == 0) s_q = wid * 32 + f;
      }
      if (wid < kNW - 1) chain_pass(wid + 1);
      __syncthreads();
      const int q = min(s_q, qcut);
      // 3. final decisions; a tentative admission whose instance lost headroom chooses again
      if (fin && tid < q) {
        if (dec == MISAT_ADMIT_NEW || dec == MISAT_ADMIT_CONT) {
          a.rq.status[i] = kStResolved;
          a.rq.inst[i] = dw;
          a.rq.reason[i] = dec;
        } else {
          a.rq.status[i] = kStHeld;
          a.rq.last_reason[i] = dec;
        }
      } else if (have && dec == MISAT_ADMIT_NEW && !s.av[b * W + dw]) {
        have = false;
      }
      done = q;
      // envelopes of the classes that lost an envelope line: one warp per class
      if (wid < 3 && s_dirty[wid]) env_update_warp(s, W, wid, &s_hm[wid], s_env[wid]);
      __syncthreads();
      if (tid == 0) {
        s_q = kNT;
        s_dirty[0] = s_dirty[1] = s_dirty[2] = 0;
      }
      __syncwarp();  // warp 0 reads them next; the other warps after warp 0 passes the chain
    }
    __syncthreads();  // the window's bitmasks are read until here
  }
}

size_t select_smem_bytes(int W) {
  return (size_t)W * 8 * 2 + (size_t)W * 4 * 4 + (size_t)W * 12 + (size_t)W * 2 * 5 + (size_t)W * 9 + 16;
}

cudaError_t select_configure() {
  // sized for the largest instance count, so that contexts of any size share the setting
  return cudaFuncSetAttribute(k4_select, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)select_smem_bytes(kMaxW));
}

void launch_select(const SelectArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  k4_select<<<1, kNT, select_smem_bytes(a.W), st>>>(a);
}

}  // namespace misat
