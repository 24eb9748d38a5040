// Route kernels: batch validation and session snapshot, caps (K3a), scoring and
// placement (K3b), arrival-order admission under the caps (K4a) and finalisation.
#include "common.cuh"
#include "kernels.h"

namespace misat {

namespace {
constexpr unsigned kFull = 0xffffffffu;
constexpr int kTile = kAdmitTile;  // requests per admission tile
}  // namespace

// ---------------------------------------------------------------------------
// Prologue: validate the batch, derive per-request sizes, look sessions up in the
// device session table (state at batch start, Sec. 4.1: O_w u P_w merged) and
// insert them into a batch-local map that keeps each session's first arrival.
__global__ void __launch_bounds__(256) k0_prologue(PrologueArgs a) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= a.n) return;
  const uint8_t c = a.cls[r];
  const uint64_t s = a.session[r];
  const int64_t t0 = a.tok_off[r], t1 = a.tok_off[r + 1];
  bool ok = c < 3 && s != 0 && t0 >= 0 && t1 >= t0 && t1 <= a.n_tokens && (t1 - t0) < (1 << 20);
  if (r == 0 && t0 != 0) ok = false;
  if (r == a.n - 1 && t1 != a.n_tokens) ok = false;
  if (!ok) {
    set_error(a.err, MISAT_ERR_INVALID_ARG);
    return;
  }
  const int32_t L = (int32_t)(t1 - t0);
  a.rq.nb[r] = L >> 4;
  a.rq.kbase[r] = t0 >> 4;
  a.rq.L[r] = L;
  a.rq.cls[r] = c;
  a.rq.session[r] = s;
  a.rq.choice[r] = -1;
  a.rq.inst[r] = -1;
  a.rq.reason[r] = 0;
  a.rq.last_reason[r] = MISAT_HOLD_NO_ELIGIBLE;
  // session table lookup
  uint8_t state = 0;
  int32_t inst = -1;
  {
    const uint32_t mask = (1u << a.st.log2n) - 1;
    uint32_t h = sess_home(s, a.st.log2n);
    for (uint32_t it = 0; it <= mask; ++it) {
      const SessSlot sl = a.st.slots[h];
      if (sl.key == 0) break;
      if (sl.key == s) {
        const uint32_t stv = sess_state(sl.val);
        if (stv == kSessProtected || stv == kSessReleased) {
          state = (uint8_t)stv;
          inst = (int32_t)sess_inst(sl.val);
        }
        break;
      }
      h = (h + 1) & mask;
    }
  }
  a.rq.sst[r] = state;
  a.rq.sinst[r] = inst;
  // batch-local first arrival of the session
  {
    const uint32_t mask = (1u << a.bm_log2) - 1;
    uint32_t h = sess_home(s, a.bm_log2);
    for (uint32_t it = 0; it <= mask; ++it) {
      const unsigned long long k = atomicCAS(&a.bm_key[h], 0ull, (unsigned long long)s);
      if (k == 0 || k == s) {
        atomicMin(&a.bm_val[h], r);
        break;
      }
      h = (h + 1) & mask;
    }
  }
}

// Leaders and candidate-session demand: cand_b = distinct sessions of class b in the
// batch that are protected nowhere (Sec. 4.2: held and candidate sessions each count).
__global__ void __launch_bounds__(256) k0_leaders(PrologueArgs a) {
  __shared__ unsigned long long s_cand[3];
  if (block_error(a.err)) return;
  if (threadIdx.x < 3) s_cand[threadIdx.x] = 0;
  __syncthreads();
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r < a.n) {
    const uint64_t s = a.rq.session[r];
    const uint32_t mask = (1u << a.bm_log2) - 1;
    uint32_t h = sess_home(s, a.bm_log2);
    int32_t ld = r;
    for (uint32_t it = 0; it <= mask; ++it) {
      if (a.bm_key[h] == s) {
        ld = a.bm_val[h];
        break;
      }
      h = (h + 1) & mask;
    }
    a.rq.leader[r] = ld;
    a.rq.status[r] = ld == r ? kStUnresolved : kStFollower;
  }
  {
    // candidate sessions by class: warp ballots, one shared add per warp and class
    const bool cand = r < a.n && a.rq.leader[r] == r && a.rq.sst[r] != kSessProtected;
    const int b = cand ? a.rq.cls[r] : -1;
    const unsigned c0 = __popc(__ballot_sync(0xffffffffu, b == 0));
    const unsigned c1 = __popc(__ballot_sync(0xffffffffu, b == 1));
    const unsigned c2 = __popc(__ballot_sync(0xffffffffu, b == 2));
    if ((threadIdx.x & 31) == 0) {
      if (c0) atomicAdd(&s_cand[0], (unsigned long long)c0);
      if (c1) atomicAdd(&s_cand[1], (unsigned long long)c1);
      if (c2) atomicAdd(&s_cand[2], (unsigned long long)c2);
    }
  }
  __syncthreads();
  if (threadIdx.x < 3 && s_cand[threadIdx.x]) atomicAdd((unsigned long long*)&a.cand[threadIdx.x], s_cand[threadIdx.x]);
}

void launch_prologue(const PrologueArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  const int grid = (a.n + 255) / 256;
  k0_prologue<<<grid, 256, 0, st>>>(a);
  k0_leaders<<<grid, 256, 0, st>>>(a);
}

// ---------------------------------------------------------------------------
// K3a caps, one thread per instance (Sec. 4.1; Eqs. 9-10 MISA; Eqs. 11, 13 MISA-T).
__global__ void __launch_bounds__(1024) k3_caps(CapsArgs a) {
  if (block_error(a.err)) return;
  int64_t kbar_b[3], T_b[3];
  uint32_t rho[3];
#pragma unroll
  for (int b = 0; b < 3; ++b) {
    kbar_b[b] = a.params[b];
    T_b[b] = a.params[3 + b];
    rho[b] = (uint32_t)a.params[6 + b];
  }
  if (threadIdx.x == 0) {
    a.ia.live[0] = 1;  // the first selection round always runs
    a.ia.live[1] = 0;
    a.ia.live[2] = 0;
  }
  for (int w = threadIdx.x; w < a.W; w += blockDim.x) {
    int64_t N[3];
    int64_t sumN = 0, tot = 0;
    for (int b = 0; b < 3; ++b) {
      const int64_t p = a.prot[w * 3 + b];
      N[b] = p + a.cand[b];
      sumN += N[b];
      tot += p;
      a.ia.N_wb[w * 3 + b] = N[b];
    }
    // reference footprint kbar_w: demand-weighted class footprint, rounded up
    int64_t kw;
    if (sumN > 0) {
      __int128 num = 0;
      for (int b = 0; b < 3; ++b) num += (__int128)N[b] * kbar_b[b];
      kw = (int64_t)((num + sumN - 1) / sumN);
    } else {
      kw = kbar_b[0] < kbar_b[1] ? kbar_b[0] : kbar_b[1];
      kw = kw < kbar_b[2] ? kw : kbar_b[2];
    }
    const int64_t Cw = (int64_t)(((__int128)a.desc[w].cap * a.pf_q16) >> 16);
    int64_t Kw = Cw / kw - a.contraction[w];
    Kw = Kw < 1 ? 1 : Kw;
    if (a.mode == MISAT_MODE_PLACEMENT_ONLY) Kw = kCapInf;
    int64_t Kwb[3];
    if (a.mode == MISAT_MODE_SESSION_ADMISSION || a.mode == MISAT_MODE_PLACEMENT_ONLY) {
      Kwb[0] = Kwb[1] = Kwb[2] = kCapInf;
    } else {
      unsigned __int128 R[3], sumR = 0;
      for (int b = 0; b < 3; ++b) {
        R[b] = (unsigned __int128)N[b] * (unsigned __int128)kbar_b[b];
        if (a.mode == MISAT_MODE_MISA_T) R[b] *= (unsigned __int128)T_b[b];
        sumR += R[b];
      }
      for (int b = 0; b < 3; ++b) {
        int64_t M;
        if (sumR > 0)
          M = (int64_t)(((unsigned __int128)Cw * R[b]) / sumR);
        else
          M = (int64_t)(((__int128)Cw * rho[b]) / 1000000);
        const int64_t k = M / kbar_b[b];
        Kwb[b] = k < 1 ? 1 : k;
      }
    }
    a.ia.K_w[w] = Kw;
    a.ia.kbar_w[w] = kw;
    a.ia.tot[w] = (int32_t)tot;
    const int64_t g = Kw - tot;
    a.ia.gh[w] = (int32_t)(g < 0 ? 0 : (g > kCapInf ? kCapInf : g));
    for (int b = 0; b < 3; ++b) {
      a.ia.K_wb[w * 3 + b] = Kwb[b];
      const int64_t hdr = Kwb[b] - a.prot[w * 3 + b];
      a.ia.ch[w * 3 + b] = (int32_t)(hdr < 0 ? 0 : (hdr > kCapInf ? kCapInf : hdr));
      a.ia.delta[w * 3 + b] = 0;
    }
    a.ia.backlog_k[w] = a.backlog[w];
    a.ia.prefill[w] = 0;
    a.ia.U[w] = 0;
  }
}

void launch_caps(const CapsArgs& a, cudaStream_t st) { k3_caps<<<1, 1024, 0, st>>>(a); }

__global__ void k_route_params(RouteParams p, int64_t* dst) {
  if (threadIdx.x < 9) dst[threadIdx.x] = p.v[threadIdx.x];
}

void launch_route_params(const RouteParams& p, int64_t* dst, cudaStream_t st) { k_route_params<<<1, 32, 0, st>>>(p, dst); }

// Whether the current selection round runs (block-uniform read of the round flag).
__device__ __forceinline__ bool round_live(const RoundArgs& a) {
  return *(volatile const int32_t*)a.ia.live != 0;
}

// ---------------------------------------------------------------------------
// K3b score: a group of G lanes per unresolved leader (G = 4..32 with W: each lane takes
// 8-instance chunks of the H row, so a group reads its row as one coalesced segment).
// Cost of Eq. (1) in fixed point, cost = backlog_k[w] + (L_r - 16 H_rw) * tokcost[w];
// eligibility of Eq. (6) with the class cap of Sec. 4.2 (headroom at round start) is folded
// into a per-class backlog: an instance without headroom for class b carries a sentinel
// backlog above every eligible cost, so the scan over instances has no branch.  Bounds:
// backlog_k <= 2^61 and (L_r - 16 H_rw) * tokcost < 2^20 * 2^32 + 1, so eligible costs stay
// below 2^62 = sentinel, and sentinel costs below 2^63.  argmin (cost, w) (ties to the lower
// instance) by log2(G) shuffle steps inside the group; the instance a session is protected
// on is eligible without headroom and is compared after the scan.  A session protected on
// its choice is admitted here (ADMIT_CONT); a released session may prefer to wait for its
// cached instance (Eq. 7).
constexpr int64_t kCostSentinel = (int64_t)1 << 62;

template <int G, int CPL>
__global__ void __launch_bounds__(256, 4) k3_score(RoundArgs a) {
  extern __shared__ unsigned char smem[];
  // per-class backlog (sentinel without headroom) and token cost per instance, stored at
  // w + w/8: the lanes of a group read instances 8 apart, which this padding puts in
  // distinct bank pairs
  const int wpad = a.W + (a.W >> 3) + 1;
  int64_t* s_bkc = reinterpret_cast<int64_t*>(smem);  // [3][wpad]
  int64_t* s_tc = s_bkc + 3 * wpad;
  if (block_error(a.err) || !round_live(a)) return;
  for (int w = threadIdx.x; w < a.W; w += blockDim.x) {
    const int wp = w + (w >> 3);
    const int64_t bk = a.ia.backlog_k[w];
    s_tc[wp] = a.tokcost[w];
    const int32_t gh = a.ia.gh[w];
#pragma unroll
    for (int b = 0; b < 3; ++b) s_bkc[b * wpad + wp] = (gh > 0 && a.ia.ch[w * 3 + b] > 0) ? bk : kCostSentinel;
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int gl = lane & (G - 1);                 // lane within the group
  const int g0 = lane & ~(G - 1);                // first lane of the group in the warp
  const unsigned gmask = G == 32 ? kFull : (((1u << G) - 1) << g0);
  const int64_t gid = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) / G;
  const int64_t ngroups = ((int64_t)gridDim.x * blockDim.x) / G;
  const int chunks = (a.W + 7) >> 3;
  const bool row_vec = (a.W & 7) == 0;           // H rows 16-byte aligned
  // a group owns requests gid + k * ngroups; they are taken G at a time: lane k of the
  // group loads request k's status and fields, so the group learns which of its requests
  // are unresolved in one round trip, and each request's H chunks are loaded while the
  // previous request is reduced
  auto load_h = [&](int r, uint4 (&hv)[CPL]) {
    const uint16_t* Hr = a.H + (int64_t)r * a.W;
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      const int ck = gl + G * c;
      hv[c] = make_uint4(0, 0, 0, 0);
      if (ck < chunks) {
        if (row_vec) {
          hv[c] = *reinterpret_cast<const uint4*>(Hr + ck * 8);
        } else {
          uint32_t t[4] = {0, 0, 0, 0};
          for (int i = 0; i < 8; ++i)
            if (ck * 8 + i < a.W) t[i >> 1] |= (uint32_t)Hr[ck * 8 + i] << (16 * (i & 1));
          hv[c] = make_uint4(t[0], t[1], t[2], t[3]);
        }
      }
    }
  };
  for (int64_t base = gid; base < a.n; base += ngroups * G) {
    const int64_t rk = base + (int64_t)gl * ngroups;
    uint8_t st = kStResolved, kb = 0, ksst = 0;
    int ksinst = -1, kL = 0;
    uint32_t khb = 0;
    if (rk < a.n) {
      st = a.rq.status[rk];
      if (st == kStUnresolved) {
        kb = a.rq.cls[rk];
        ksst = a.rq.sst[rk];
        ksinst = a.rq.sinst[rk];
        kL = a.rq.L[rk];
        khb = a.rq.hbest[rk];
      }
    }
    unsigned todo = (__ballot_sync(gmask, st == kStUnresolved) >> g0) & (G == 32 ? kFull : ((1u << G) - 1));
    if (!todo) continue;
    int k = __ffs(todo) - 1;
    uint4 hv[CPL];
    load_h((int)(base + (int64_t)k * ngroups), hv);
    while (true) {
      todo &= todo - 1;
      const int knext = todo ? __ffs(todo) - 1 : -1;
      uint4 hn[CPL];
      if (knext >= 0) load_h((int)(base + (int64_t)knext * ngroups), hn);
      const int r = (int)(base + (int64_t)k * ngroups);
      const int b = __shfl_sync(gmask, (int)kb, g0 + k);
      const uint8_t sst = (uint8_t)__shfl_sync(gmask, (int)ksst, g0 + k);
      const int sinst = __shfl_sync(gmask, ksinst, g0 + k);
      const int64_t Lr = __shfl_sync(gmask, kL, g0 + k);
      const uint32_t hb = __shfl_sync(gmask, khb, g0 + k);
      const int hmax = (int)(hb >> 16), whit = 65535 - (int)(hb & 0xffffu);  // max H, lowest such w
      const int pw = sst == kSessProtected ? sinst : -1;
      const int64_t* bkc = s_bkc + b * wpad;
      int64_t best_c = INT64_MAX;
      int best_w = INT32_MAX;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int ck = gl + G * c;
        if (ck >= chunks) break;
        const uint32_t hw[4] = {hv[c].x, hv[c].y, hv[c].z, hv[c].w};
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int w = ck * 8 + i;
          if (w >= a.W) break;
          const uint32_t h = (hw[i >> 1] >> (16 * (i & 1))) & 0xffffu;
          const uint32_t cold = (uint32_t)Lr - 16u * h;  // L_r - 16 H_rw >= 0, < 2^20
          const int wp = w + (w >> 3);
          const int64_t cost = bkc[wp] + (int64_t)((uint64_t)cold * (uint64_t)s_tc[wp]);
          if (cost < best_c) {
            best_c = cost;
            best_w = w;
          }
        }
      }
#pragma unroll
      for (int o = G / 2; o > 0; o >>= 1) {
        const int64_t oc = __shfl_xor_sync(gmask, best_c, o, G);
        const int ow = __shfl_xor_sync(gmask, best_w, o, G);
        if (oc < best_c || (oc == best_c && ow < best_w)) {
          best_c = oc;
          best_w = ow;
        }
      }
      if (gl == 0) {
        if (best_c >= kCostSentinel) best_w = INT32_MAX;  // no instance with headroom
        if (pw >= 0 && bkc[pw + (pw >> 3)] >= kCostSentinel) {
          // protected on pw: eligible there without headroom, at its real cost
          const int64_t hp = a.H[(int64_t)r * a.W + pw];
          const int64_t cpw = a.ia.backlog_k[pw] + (Lr - 16 * hp) * s_tc[pw + (pw >> 3)];
          if (best_w == INT32_MAX || cpw < best_c || (cpw == best_c && pw < best_w)) {
            best_c = cpw;
            best_w = pw;
          }
        }
        int choice = -1;
        uint8_t reason = 0;
        if (best_w == INT32_MAX) {
          // no instance has headroom: headroom only shrinks over the rounds and protection
          // is fixed by the snapshot, so no later round can admit it
          reason = MISAT_HOLD_NO_ELIGIBLE;
          a.rq.status[r] = kStHeld;
        } else {
          choice = best_w;
          if (sst == kSessReleased && hmax > 0) {
            const bool elig_hit = bkc[whit + (whit >> 3)] < kCostSentinel;
            if (!elig_hit) {
              const int64_t lhs = a.hold_delay_q + a.ia.backlog_k[whit] - a.ia.backlog_k[best_w];
              const int64_t rhs = 16 * (int64_t)hmax * s_tc[whit + (whit >> 3)];
              if (lhs < rhs) {
                choice = -1;
                reason = MISAT_HOLD_PREFER_CACHE;
              }
            }
          }
        }
        if (choice >= 0 && choice == pw) {
          a.rq.status[r] = kStResolved;
          a.rq.inst[r] = choice;
          a.rq.reason[r] = MISAT_ADMIT_CONT;
          a.rq.choice[r] = -1;
          atomicAdd(&a.ia.prefill[choice], (unsigned long long)(Lr - 16 * (int64_t)a.H[(int64_t)r * a.W + choice]));
          atomicAdd(&a.ia.live[1], 1);
        } else {
          a.rq.choice[r] = choice;
          if (choice < 0) a.rq.last_reason[r] = reason;
        }
      }
      if (knext < 0) break;
      k = knext;
#pragma unroll
      for (int c = 0; c < CPL; ++c) hv[c] = hn[c];
    }
  }
}

// Arrival-order admission, three passes over tiles of kTile requests.
// A chooser needs headroom (it is not protected on its choice).  For chooser i of
// instance w with class b, let c_{i,b'} be the choosers of (w, b') before i.  The
// first H_{w,b} choosers of class b pass the class cap; the admitted ones are those
// passing it while fewer than G_w earlier choosers did: admitted(i) = c_{i,b} < H_{w,b}
// and sum_b' min(c_{i,b'}, H_{w,b'}) < G_w -- exactly the sequential walk of Eq. (6).
__global__ void __launch_bounds__(256) k4_tile_count(RoundArgs a) {
  extern __shared__ int32_t s_cnt[];
  if (block_error(a.err) || !round_live(a)) return;
  const int nb = 3 * a.W;
  for (int k = threadIdx.x; k < nb; k += blockDim.x) s_cnt[k] = 0;
  __syncthreads();
  const int t = blockIdx.x;
  for (int i0 = 0; i0 < kTile; i0 += blockDim.x) {
    // choosers herd to the same (instance, class): one shared add per group of equal keys
    const int i = i0 + (int)threadIdx.x;
    const int r = t * kTile + i;
    int key = -1;
    if (i < kTile && r < a.n && a.rq.status[r] == kStUnresolved) {
      const int c = a.rq.choice[r];
      if (c >= 0) key = c * 3 + a.rq.cls[r];
    }
    const unsigned peers = __match_any_sync(kFull, key);
    if (key >= 0 && (int)(threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&s_cnt[key], __popc(peers));
  }
  __syncthreads();
  int32_t* out = a.tile_counts + (int64_t)t * nb;
  for (int k = threadIdx.x; k < nb; k += blockDim.x) out[k] = s_cnt[k];
}

// Exclusive scan of the tile counts over the tiles, per (instance, class) column: a CTA of
// 32 warps owns 32 columns (lanes); warp k sums a stripe of tiles, the stripe sums are
// scanned across warps, then each warp rewrites its stripe with running prefixes.
__global__ void __launch_bounds__(1024) k4_tile_scan(RoundArgs a) {
  __shared__ int32_t s_sum[32][33];
  if (block_error(a.err) || !round_live(a)) return;
  const int nb = 3 * a.W;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int col = blockIdx.x * 32 + lane;
  const int T = a.n_tiles;
  const int per = (T + 31) / 32;
  const int t0 = wid * per, t1 = min(T, t0 + per);
  int32_t sum = 0;
  if (col < nb)
    for (int t = t0; t < t1; ++t) sum += a.tile_counts[(int64_t)t * nb + col];
  s_sum[wid][lane] = sum;
  __syncthreads();
  if (wid == 0) {
    int32_t acc = 0;
    for (int k = 0; k < 32; ++k) {
      const int32_t v = s_sum[k][lane];
      s_sum[k][lane] = acc;
      acc += v;
    }
  }
  __syncthreads();
  int32_t acc = s_sum[wid][lane];
  if (col < nb)
    for (int t = t0; t < t1; ++t) {
      int32_t* p = a.tile_counts + (int64_t)t * nb + col;
      const int32_t v = *p;
      *p = acc;
      acc += v;
    }
}

// End of a selection round (one warp, after every tile's admissions): admissions leave the
// headroom of their (instance, class), the admitted prefill joins the instance backlog
// (saturating at 2^61), and a round that admitted nobody (no ADMIT_NEW, no ADMIT_CONT) ends
// the rounds: its successors would see the same inputs.
__device__ __forceinline__ void round_fold(const RoundArgs& a, int lane) {
  constexpr int kF = 4;  // instances per lane per pass, all of their loads issued together
  int admitted = 0;
  for (int w0 = 0; w0 < a.W; w0 += 32 * kF) {
    int32_t d[kF][3], ch[kF][3], gh[kF];
    unsigned long long tok[kF];
    int64_t bk[kF], tc[kF];
#pragma unroll
    for (int f = 0; f < kF; ++f) {
      const int w = w0 + 32 * f + lane;
      if (w < a.W) {
#pragma unroll
        for (int b = 0; b < 3; ++b) {
          d[f][b] = __ldcg(&a.ia.delta[w * 3 + b]);
          ch[f][b] = a.ia.ch[w * 3 + b];
        }
        gh[f] = a.ia.gh[w];
        tok[f] = __ldcg(&a.ia.prefill[w]);
        bk[f] = a.ia.backlog_k[w];
        tc[f] = a.tokcost[w];
      }
    }
#pragma unroll
    for (int f = 0; f < kF; ++f) {
      const int w = w0 + 32 * f + lane;
      if (w < a.W) {
        int32_t sum = 0;
#pragma unroll
        for (int b = 0; b < 3; ++b) {
          a.ia.ch[w * 3 + b] = ch[f][b] - d[f][b];
          a.ia.delta[w * 3 + b] = 0;
          sum += d[f][b];
        }
        a.ia.gh[w] = gh[f] - sum;
        admitted |= sum;
        a.ia.prefill[w] = 0;
        const __int128 v = (__int128)bk[f] + (__int128)tc[f] * (__int128)tok[f];
        a.ia.backlog_k[w] = v > kBacklogMax ? kBacklogMax : (int64_t)v;
      }
    }
  }
  const bool any = __any_sync(kFull, admitted != 0);
  if (lane == 0) {
    if (!any && *(volatile int32_t*)&a.ia.live[1] == 0) a.ia.live[0] = 0;
    a.ia.live[1] = 0;
    a.ia.live[2] = 0;  // the next round's tile tickets
  }
}

__global__ void __launch_bounds__(32) k4_admit(RoundArgs a) {
  extern __shared__ int32_t s_cnt[];
  if (block_error(a.err) || !round_live(a)) return;
  const int nb = 3 * a.W;
  const int t = blockIdx.x;
  const int lane = threadIdx.x;
  constexpr int kC = kTile / 32;  // chunks of 32 requests per tile
  if ((nb & 3) == 0) {  // rows start on 16-byte boundaries
    const int4* src = reinterpret_cast<const int4*>(a.tile_counts + (int64_t)t * nb);
    int4* dst = reinterpret_cast<int4*>(s_cnt);
    for (int k = lane; k < (nb >> 2); k += 32) dst[k] = src[k];
  } else {
    for (int k = lane; k < nb; k += 32) s_cnt[k] = a.tile_counts[(int64_t)t * nb + k];
  }
  // every load of the tile is issued before the in-order walk: the choosers, then the
  // headroom of their instances
  bool need[kC];
  int w[kC], b[kC], G[kC], h0[kC], h1[kC], h2[kC];
#pragma unroll
  for (int c = 0; c < kC; ++c) {
    const int r = t * kTile + 32 * c + lane;
    need[c] = false;
    w[c] = -1;
    b[c] = 0;
    if (r < a.n && a.rq.status[r] == kStUnresolved) {
      w[c] = a.rq.choice[r];
      need[c] = w[c] >= 0;
      b[c] = a.rq.cls[r];
    }
  }
#pragma unroll
  for (int c = 0; c < kC; ++c) {
    if (need[c]) {
      G[c] = a.ia.gh[w[c]];
      h0[c] = a.ia.ch[w[c] * 3 + 0];
      h1[c] = a.ia.ch[w[c] * 3 + 1];
      h2[c] = a.ia.ch[w[c] * 3 + 2];
    }
  }
  __syncwarp();
  const uint32_t lt = lanemask_lt();
#pragma unroll
  for (int c = 0; c < kC; ++c) {
    const int r = t * kTile + 32 * c + lane;
    const unsigned peers_w = __match_any_sync(kFull, need[c] ? w[c] : -1 - lane);
    const unsigned m0 = __ballot_sync(kFull, need[c] && b[c] == 0);
    const unsigned m1 = __ballot_sync(kFull, need[c] && b[c] == 1);
    const unsigned m2 = __ballot_sync(kFull, need[c] && b[c] == 2);
    if (need[c]) {
      const int wc = w[c], bc = b[c];
      const int c_0 = s_cnt[wc * 3 + 0] + __popc(peers_w & m0 & lt);
      const int c_1 = s_cnt[wc * 3 + 1] + __popc(peers_w & m1 & lt);
      const int c_2 = s_cnt[wc * 3 + 2] + __popc(peers_w & m2 & lt);
      const int cb = bc == 0 ? c_0 : (bc == 1 ? c_1 : c_2);
      const int hb = bc == 0 ? h0[c] : (bc == 1 ? h1[c] : h2[c]);
      const long long g = (long long)min(c_0, h0[c]) + min(c_1, h1[c]) + min(c_2, h2[c]);
      if (cb < hb && g < G[c]) {
        a.rq.status[r] = kStResolved;
        a.rq.inst[r] = wc;
        a.rq.reason[r] = MISAT_ADMIT_NEW;
        atomicAdd(&a.ia.delta[wc * 3 + bc], 1);
        atomicAdd(&a.ia.prefill[wc], (unsigned long long)(a.rq.L[r] - 16 * (int64_t)a.H[(int64_t)r * a.W + wc]));
      } else {
        a.rq.last_reason[r] = g >= G[c] ? MISAT_HOLD_GLOBAL_CAP : MISAT_HOLD_CLASS_CAP;
      }
    }
    __syncwarp();
    const unsigned peers_wb = __match_any_sync(kFull, need[c] ? w[c] * 3 + b[c] : -1 - lane);
    if (need[c] && lane == __ffs(peers_wb) - 1) s_cnt[w[c] * 3 + b[c]] += __popc(peers_wb);
    __syncwarp();
  }
  // the last tile to finish folds the round's admissions into headroom and backlog (its
  // ticket comes after every other tile's admissions, which the fences make visible)
  __threadfence();
  unsigned ticket = 0;
  if (lane == 0) ticket = atomicAdd(reinterpret_cast<unsigned*>(&a.ia.live[2]), 1u);
  ticket = __shfl_sync(kFull, ticket, 0);
  if (ticket != gridDim.x - 1) return;
  __threadfence();
  round_fold(a, lane);
}

// End of a round: fold this round's admissions into the headroom, and add the admitted
// prefill to the in-batch backlog d_w (saturating), so the next round sees the load.  A
// round that admitted nobody leaves every input of the next round as it was (headroom,
// backlog, statuses), so the next round would repeat it exactly: the remaining rounds
// are then skipped.

void launch_round(const RoundArgs& a, int num_sms, cudaStream_t st) {
  const size_t score_smem = (size_t)32 * (a.W + (a.W >> 3) + 1);
  int G = 4;
  while (G < 32 && G * 16 < a.W) G <<= 1;  // about two 8-instance chunks per lane
  const int64_t threads = (int64_t)a.n * G;
  int64_t score_grid = (threads + 255) / 256;
  if (score_grid > (int64_t)num_sms * 8) score_grid = (int64_t)num_sms * 8;
  if (score_grid < 1) score_grid = 1;
  switch (G) {  // CPL: 8-instance chunks per lane, ceil(ceil(W/8) / G)
    case 4: k3_score<4, 2><<<(int)score_grid, 256, score_smem, st>>>(a); break;
    case 8: k3_score<8, 2><<<(int)score_grid, 256, score_smem, st>>>(a); break;
    case 16: k3_score<16, 2><<<(int)score_grid, 256, score_smem, st>>>(a); break;
    default: k3_score<32, 4><<<(int)score_grid, 256, score_smem, st>>>(a); break;
  }
  const size_t cnt_smem = (size_t)a.W * 3 * sizeof(int32_t);
  k4_tile_count<<<a.n_tiles, 128, cnt_smem, st>>>(a);
  k4_tile_scan<<<(3 * a.W + 31) / 32, 1024, 0, st>>>(a);
  k4_admit<<<a.n_tiles, 32, cnt_smem, st>>>(a);  // its last tile also ends the round
}

// ---------------------------------------------------------------------------
// Finalise: unresolved leaders are held with their last reason, followers copy their
// leader, hit blocks, statistics and the per-instance new-key bound of the commit.
// stats layout: [0..7] reason counts (CONT NEW FOLLOW GLOBAL CLASS NOELIG PREFER LEADER),
// [8..10] admitted by class, [11..13] held by class, [14] hit tokens, [15] query tokens.
__global__ void __launch_bounds__(256) k4_finalize(FinalizeArgs a) {
  __shared__ unsigned long long s_st[16];
  if (block_error(a.err)) return;
  if (threadIdx.x < 16) s_st[threadIdx.x] = 0;
  __syncthreads();
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  const int lane = threadIdx.x & 31;
  int w = -1, hb = 0, b = 0, ri = -1, L = 0;
  if (r < a.n) {
    uint8_t reason;
    const uint8_t stv = a.rq.status[r];
    const int ld = a.rq.leader[r];
    if (stv == kStFollower) {
      w = a.rq.inst[ld];
      reason = w >= 0 ? MISAT_ADMIT_FOLLOW : MISAT_HOLD_LEADER_HELD;
    } else if (stv == kStUnresolved || stv == kStHeld) {
      w = -1;
      reason = a.rq.last_reason[r];
    } else {
      w = a.rq.inst[r];
      reason = a.rq.reason[r];
    }
    hb = w >= 0 ? (int)a.H[(int64_t)r * a.W + w] : (int)(a.rq.hbest[r] >> 16);  // HOLD: max over instances
    if (stv == kStFollower) {
      a.rq.inst[r] = w;
      a.rq.reason[r] = reason;
    } else if (stv == kStUnresolved || stv == kStHeld) {
      a.rq.reason[r] = reason;
    }
    a.out_inst[r] = w;
    a.out_reason[r] = reason;
    a.out_hit[r] = hb;
    ri = reason < 16 ? reason - 1 : 3 + (reason - 16);
    b = a.rq.cls[r];
    if (w >= 0) {
      L = a.rq.L[r];
      atomic_add_i64(&a.U[w], (long long)(a.rq.nb[r] - hb));
    }
  }
  // statistics: warp ballots and sums, one shared-memory add per warp and counter
  unsigned c[16];
#pragma unroll
  for (int v = 0; v < 8; ++v) c[v] = __popc(__ballot_sync(0xffffffffu, ri == v));
#pragma unroll
  for (int v = 0; v < 3; ++v) {
    c[8 + v] = __popc(__ballot_sync(0xffffffffu, ri >= 0 && w >= 0 && b == v));
    c[11 + v] = __popc(__ballot_sync(0xffffffffu, ri >= 0 && w < 0 && b == v));
  }
  c[14] = __reduce_add_sync(0xffffffffu, w >= 0 ? (unsigned)(16 * hb) : 0u);
  c[15] = __reduce_add_sync(0xffffffffu, w >= 0 ? (unsigned)L : 0u);
  if (lane == 0) {
#pragma unroll
    for (int v = 0; v < 16; ++v)
      if (c[v]) atomicAdd(&s_st[v], (unsigned long long)c[v]);
  }
  __syncthreads();
  if (threadIdx.x < 16 && s_st[threadIdx.x]) atomicAdd(&a.stats[threadIdx.x], s_st[threadIdx.x]);
}

void launch_finalize(const FinalizeArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  k4_finalize<<<(a.n + 255) / 256, 256, 0, st>>>(a);
}

}  // namespace misat
