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
    if (ld == r && a.rq.sst[r] != kSessProtected) atomicAdd(&s_cand[a.rq.cls[r]], 1ull);
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
    // conservative reference length kbar_w: demand-weighted class footprint, rounded up
    int64_t kw;
    if (sumN > 0) {
      __int128 num = 0;
      for (int b = 0; b < 3; ++b) num += (__int128)N[b] * a.kbar_b[b];
      kw = (int64_t)((num + sumN - 1) / sumN);
    } else {
      kw = a.kbar_b[0] < a.kbar_b[1] ? a.kbar_b[0] : a.kbar_b[1];
      kw = kw < a.kbar_b[2] ? kw : a.kbar_b[2];
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
        R[b] = (unsigned __int128)N[b] * (unsigned __int128)a.kbar_b[b];
        if (a.mode == MISAT_MODE_MISA_T) R[b] *= (unsigned __int128)a.T_b[b];
        sumR += R[b];
      }
      for (int b = 0; b < 3; ++b) {
        int64_t M;
        if (sumR > 0)
          M = (int64_t)(((unsigned __int128)Cw * R[b]) / sumR);
        else
          M = (int64_t)(((__int128)Cw * a.rho[b]) / 1000000);
        const int64_t k = M / a.kbar_b[b];
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

// ---------------------------------------------------------------------------
// K3b score: one warp per unresolved leader.  Cost of Eq. (1) in fixed point,
// cost = backlog_k[w] + (L_r - 16 H_rw) * tokcost[w]; eligibility of Eq. (6) with the
// class cap of Sec. 4.2 (headroom at round start); argmin (cost, w) by warp shuffles.
// A session protected on its choice is admitted here (ADMIT_CONT); a released session
// may prefer to wait for its cached instance (Eq. 7).
__global__ void __launch_bounds__(256) k3_score(RoundArgs a) {
  extern __shared__ unsigned char smem[];
  int64_t* s_bk = reinterpret_cast<int64_t*>(smem);
  int64_t* s_tc = s_bk + a.W;
  int32_t* s_gh = reinterpret_cast<int32_t*>(s_tc + a.W);
  int32_t* s_ch = s_gh + a.W;  // [W*3]
  if (block_error(a.err)) return;
  for (int w = threadIdx.x; w < a.W; w += blockDim.x) {
    s_bk[w] = a.ia.backlog_k[w];
    s_tc[w] = a.tokcost[w];
    s_gh[w] = a.ia.gh[w];
    s_ch[w * 3 + 0] = a.ia.ch[w * 3 + 0];
    s_ch[w * 3 + 1] = a.ia.ch[w * 3 + 1];
    s_ch[w * 3 + 2] = a.ia.ch[w * 3 + 2];
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nwarps = (gridDim.x * blockDim.x) >> 5;
  // the next request's fields and first H values are loaded while this one is reduced
  constexpr int kPre = 4;  // H values per lane prefetched (instances lane + 32 i, i < kPre)
  struct Next {
    uint8_t st, b, sst;
    int sinst;
    int32_t L;
    uint16_t h[kPre];
  };
  auto fetch = [&](int rr, Next& x) {
    x.st = rr < a.n ? a.rq.status[rr] : kStResolved;
    if (x.st != kStUnresolved) return;
    x.b = a.rq.cls[rr];
    x.sst = a.rq.sst[rr];
    x.sinst = a.rq.sinst[rr];
    x.L = a.rq.L[rr];
    const uint16_t* Hr = a.H + (int64_t)rr * a.W;
#pragma unroll
    for (int i = 0; i < kPre; ++i) x.h[i] = (lane + 32 * i < a.W) ? Hr[lane + 32 * i] : 0;
  };
  Next nx;
  fetch(warp, nx);
  for (int r = warp; r < a.n; r += nwarps) {
    const Next cur = nx;
    fetch(r + nwarps, nx);
    if (cur.st != kStUnresolved) continue;
    const int b = cur.b;
    const uint8_t sst = cur.sst;
    const int pw = sst == kSessProtected ? cur.sinst : -1;
    const int64_t Lr = cur.L;
    const uint16_t* Hr = a.H + (int64_t)r * a.W;
    int64_t best_c = INT64_MAX;
    int best_w = INT32_MAX;
    int hmax = -1, whit = INT32_MAX;
    auto visit = [&](int w, int h) {
      const bool elig = (w == pw) || (s_gh[w] > 0 && s_ch[w * 3 + b] > 0);
      if (elig) {
        const int64_t cost = s_bk[w] + (Lr - 16 * (int64_t)h) * s_tc[w];
        if (cost < best_c) {
          best_c = cost;
          best_w = w;
        }
      }
      if (h > hmax) {
        hmax = h;
        whit = w;
      }
    };
#pragma unroll
    for (int i = 0; i < kPre; ++i)
      if (lane + 32 * i < a.W) visit(lane + 32 * i, cur.h[i]);
    for (int w = lane + 32 * kPre; w < a.W; w += 32) visit(w, Hr[w]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const int64_t oc = __shfl_xor_sync(kFull, best_c, o);
      const int ow = __shfl_xor_sync(kFull, best_w, o);
      if (oc < best_c || (oc == best_c && ow < best_w)) {
        best_c = oc;
        best_w = ow;
      }
      const int oh = __shfl_xor_sync(kFull, hmax, o);
      const int owh = __shfl_xor_sync(kFull, whit, o);
      if (oh > hmax || (oh == hmax && owh < whit)) {
        hmax = oh;
        whit = owh;
      }
    }
    if (lane == 0) {
      a.rq.hmax[r] = hmax < 0 ? 0 : hmax;
      int choice = -1;
      uint8_t reason = 0;
      if (best_w == INT32_MAX) {
        reason = MISAT_HOLD_NO_ELIGIBLE;
      } else {
        choice = best_w;
        if (sst == kSessReleased && hmax > 0) {
          const bool elig_hit = s_gh[whit] > 0 && s_ch[whit * 3 + b] > 0;
          if (!elig_hit) {
            const int64_t lhs = a.hold_delay_q + s_bk[whit] - s_bk[best_w];
            const int64_t rhs = 16 * (int64_t)hmax * s_tc[whit];
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
        atomicAdd(&a.ia.prefill[choice], (unsigned long long)(Lr - 16 * (int64_t)Hr[choice]));
      } else {
        a.rq.choice[r] = choice;
        if (choice < 0) a.rq.last_reason[r] = reason;
      }
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
  if (block_error(a.err)) return;
  const int nb = 3 * a.W;
  for (int k = threadIdx.x; k < nb; k += blockDim.x) s_cnt[k] = 0;
  __syncthreads();
  const int t = blockIdx.x;
  for (int i = threadIdx.x; i < kTile; i += blockDim.x) {
    const int r = t * kTile + i;
    if (r < a.n && a.rq.status[r] == kStUnresolved) {
      const int c = a.rq.choice[r];
      if (c >= 0) atomicAdd(&s_cnt[c * 3 + a.rq.cls[r]], 1);
    }
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
  if (block_error(a.err)) return;
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

__global__ void __launch_bounds__(32) k4_admit(RoundArgs a) {
  extern __shared__ int32_t s_cnt[];
  if (block_error(a.err)) return;
  const int nb = 3 * a.W;
  const int t = blockIdx.x;
  const int lane = threadIdx.x;
  for (int k = lane; k < nb; k += 32) s_cnt[k] = a.tile_counts[(int64_t)t * nb + k];
  __syncwarp();
  const uint32_t lt = lanemask_lt();
  for (int c0 = 0; c0 < kTile; c0 += 32) {
    const int r = t * kTile + c0 + lane;
    bool need = false;
    int w = -1, b = 0;
    if (r < a.n && a.rq.status[r] == kStUnresolved) {
      w = a.rq.choice[r];
      need = w >= 0;
      b = a.rq.cls[r];
    }
    const unsigned peers_w = __match_any_sync(kFull, need ? w : -1 - lane);
    const unsigned m0 = __ballot_sync(kFull, need && b == 0);
    const unsigned m1 = __ballot_sync(kFull, need && b == 1);
    const unsigned m2 = __ballot_sync(kFull, need && b == 2);
    if (need) {
      const int c_0 = s_cnt[w * 3 + 0] + __popc(peers_w & m0 & lt);
      const int c_1 = s_cnt[w * 3 + 1] + __popc(peers_w & m1 & lt);
      const int c_2 = s_cnt[w * 3 + 2] + __popc(peers_w & m2 & lt);
      const int h0 = a.ia.ch[w * 3 + 0], h1 = a.ia.ch[w * 3 + 1], h2 = a.ia.ch[w * 3 + 2];
      const int G = a.ia.gh[w];
      const int cb = b == 0 ? c_0 : (b == 1 ? c_1 : c_2);
      const int hb = b == 0 ? h0 : (b == 1 ? h1 : h2);
      const long long g = (long long)min(c_0, h0) + min(c_1, h1) + min(c_2, h2);
      if (cb < hb && g < G) {
        a.rq.status[r] = kStResolved;
        a.rq.inst[r] = w;
        a.rq.reason[r] = MISAT_ADMIT_NEW;
        atomicAdd(&a.ia.delta[w * 3 + b], 1);
        atomicAdd(&a.ia.prefill[w], (unsigned long long)(a.rq.L[r] - 16 * (int64_t)a.H[(int64_t)r * a.W + w]));
      } else {
        a.rq.last_reason[r] = g >= G ? MISAT_HOLD_GLOBAL_CAP : MISAT_HOLD_CLASS_CAP;
      }
    }
    __syncwarp();
    const unsigned peers_wb = __match_any_sync(kFull, need ? w * 3 + b : -1 - lane);
    if (need && lane == __ffs(peers_wb) - 1) s_cnt[w * 3 + b] += __popc(peers_wb);
    __syncwarp();
  }
}

// End of a round: fold this round's admissions into the headroom, and add the admitted
// prefill to the in-batch backlog d_w (saturating), so the next round sees the load.
__global__ void __launch_bounds__(1024) k4_round_end(RoundArgs a) {
  if (block_error(a.err)) return;
  for (int w = threadIdx.x; w < a.W; w += blockDim.x) {
    int32_t sum = 0;
    for (int b = 0; b < 3; ++b) {
      const int32_t d = a.ia.delta[w * 3 + b];
      a.ia.ch[w * 3 + b] -= d;
      a.ia.delta[w * 3 + b] = 0;
      sum += d;
    }
    a.ia.gh[w] -= sum;
    const unsigned long long tok = a.ia.prefill[w];
    a.ia.prefill[w] = 0;
    const __int128 v = (__int128)a.ia.backlog_k[w] + (__int128)a.tokcost[w] * (__int128)tok;
    a.ia.backlog_k[w] = v > kBacklogMax ? kBacklogMax : (int64_t)v;
  }
}

void launch_round(const RoundArgs& a, int num_sms, cudaStream_t st) {
  const size_t score_smem = (size_t)a.W * (8 + 8 + 4 + 12);
  int score_grid = (a.n + 7) / 8;
  if (score_grid > num_sms * 8) score_grid = num_sms * 8;
  if (score_grid < 1) score_grid = 1;
  k3_score<<<score_grid, 256, score_smem, st>>>(a);
  const size_t cnt_smem = (size_t)a.W * 3 * sizeof(int32_t);
  k4_tile_count<<<a.n_tiles, 128, cnt_smem, st>>>(a);
  k4_tile_scan<<<(3 * a.W + 31) / 32, 1024, 0, st>>>(a);
  k4_admit<<<a.n_tiles, 32, cnt_smem, st>>>(a);
  k4_round_end<<<1, 1024, 0, st>>>(a);
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
  if (r < a.n) {
    int w;
    uint8_t reason;
    const uint8_t stv = a.rq.status[r];
    if (stv == kStFollower) {
      w = a.rq.inst[a.rq.leader[r]];
      reason = w >= 0 ? MISAT_ADMIT_FOLLOW : MISAT_HOLD_LEADER_HELD;
    } else if (stv == kStUnresolved) {
      w = -1;
      reason = a.rq.last_reason[r];
    } else {
      w = a.rq.inst[r];
      reason = a.rq.reason[r];
    }
    const uint16_t* Hr = a.H + (int64_t)r * a.W;
    int hb = 0;
    if (w >= 0) {
      hb = Hr[w];
    } else if (stv != kStFollower) {
      hb = a.rq.hmax[r];  // every leader was scored at least once
    } else {
      for (int x = 0; x < a.W; ++x) hb = Hr[x] > hb ? Hr[x] : hb;
    }
    if (stv == kStFollower) {
      a.rq.inst[r] = w;
      a.rq.reason[r] = reason;
    } else if (stv == kStUnresolved) {
      a.rq.reason[r] = reason;
    }
    a.out_inst[r] = w;
    a.out_reason[r] = reason;
    a.out_hit[r] = hb;
    const int ri = reason < 16 ? reason - 1 : 3 + (reason - 16);
    atomicAdd(&s_st[ri], 1ull);
    const int b = a.rq.cls[r];
    if (w >= 0) {
      atomicAdd(&s_st[8 + b], 1ull);
      atomicAdd(&s_st[14], (unsigned long long)(16 * hb));
      atomicAdd(&s_st[15], (unsigned long long)a.rq.L[r]);
      atomic_add_i64(&a.U[w], (long long)(a.rq.nb[r] - hb));
    } else {
      atomicAdd(&s_st[11 + b], 1ull);
    }
  }
  __syncthreads();
  if (threadIdx.x < 16 && s_st[threadIdx.x]) atomicAdd(&a.stats[threadIdx.x], s_st[threadIdx.x]);
}

void launch_finalize(const FinalizeArgs& a, cudaStream_t st) {
  if (a.n <= 0) return;
  k4_finalize<<<(a.n + 255) / 256, 256, 0, st>>>(a);
}

}  // namespace misat
