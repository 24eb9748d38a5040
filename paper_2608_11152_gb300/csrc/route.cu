// Route kernels: batch validation and session snapshot, caps (K3a) and finalisation.
// The placement and admission of the leaders (K3b, K4a) are in select.cu.
#include "common.cuh"
#include "kernels.h"

namespace misat {

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
    }
    a.ia.U[w] = 0;
  }
}

void launch_caps(const CapsArgs& a, cudaStream_t st) { k3_caps<<<1, 1024, 0, st>>>(a); }

__global__ void k_route_params(RouteParams p, int64_t* dst) {
  if (threadIdx.x < 9) dst[threadIdx.x] = p.v[threadIdx.x];
}

void launch_route_params(const RouteParams& p, int64_t* dst, cudaStream_t st) { k_route_params<<<1, 32, 0, st>>>(p, dst); }

// ---------------------------------------------------------------------------
// Finalise: held leaders keep the reason the selection gave them, followers copy their
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
      const int nbr = a.rq.nb[r];
      atomic_add_i64(&a.U[w], (long long)(nbr - hb));
      if (a.grp && nbr > 0) grp_note(a.grp, a.grp_log2, a.keys[a.rq.kbase[r]], w, r);
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
