// MISA-T batched routing decision -- CPU ORACLE (test infrastructure).
//
// This file is test infrastructure, not product code.  Only tests/,
// __graft_entry__.smoke() and bench.py's cpu_baseline / reference leg may load
// it.  It is a plain, slow, single-threaded restatement of the routing policy of
// "Scheduling Mixed RL Rollouts Beyond Prefix Locality" (MISA-T), written with
// std containers, linear scans and arrival-order loops so that each step can be
// checked against the paper by eye.  It shares no source with the CUDA library.
//
// Paper passages followed (section / equation):
//   Sec. 3.2 Eq. (1)   prefill-cost placement  c = d_w + (L_r - H_rw) / mu_w
//   Sec. 4.4           H_rw = longest matching prompt-block hash on instance w;
//                      eviction / reset removes hashes
//   Sec. 4.1 Eq. (6)   Admit(r,w): continuation admitted, new session only with
//                      headroom |O_w|+|P_w| < K_w, otherwise HOLD
//   Sec. 4.1 Eq. (7)   hold-vs-cold rule for a continuation that must be admitted
//                      again
//   Sec. 4.1           K_w^base = floor(C_w / kbar_w), operational K_w <= K_w^base
//   Sec. 4.2 Eqs. (9)-(10)  MISA spatial quota and class cap
//   Sec. 4.3 Eqs. (11),(13) MISA-T block-time quota and class cap
//   Sec. 4.2           N_wb counts active, pending, held and candidate sessions;
//                      a new session needs global and class headroom
//   Sec. 3.3           D_TV(p, q) = 1/2 |p - q|_1
//
// Where the paper is silent (hash function, index eviction order, the order in
// which the requests of one batch are decided, fixed-point units) the oracle
// follows the readings listed in the design notes of this repository; each such
// place is marked "reading:" below.
//
// Parity status: every function below is pinned by the -m "not gpu" tests
// (published SplitMix64 vectors, token-by-token brute force of H, hand-worked
// quota example of Eqs. 9-13, closed forms and invariants).  The overload
// controller of Sec. 4.1 (Eq. 8) is not part of the path; it enters only as the
// integer input cap_contraction_w.

#include <algorithm>
#include <array>
#include <cstdint>
#include <cstring>
#include <deque>
#include <unordered_map>
#include <unordered_set>
#include <vector>

namespace {

// ---- error codes, modes, reasons (values fixed by the library contract) ----
constexpr int OK = 0;
constexpr int ERR_INVALID_ARG = -1;
constexpr int ERR_STATE = -4;

constexpr int MODE_MISA_T = 0;
constexpr int MODE_MISA = 1;
constexpr int MODE_SESSION_ADMISSION = 2;
constexpr int MODE_PLACEMENT_ONLY = 3;

constexpr uint8_t ADMIT_CONT = 1;
constexpr uint8_t ADMIT_NEW = 2;
constexpr uint8_t ADMIT_FOLLOW = 3;
constexpr uint8_t HOLD_GLOBAL_CAP = 16;
constexpr uint8_t HOLD_CLASS_CAP = 17;
constexpr uint8_t HOLD_NO_ELIGIBLE = 18;  // reserved: the serial selection never produces it
constexpr uint8_t HOLD_PREFER_CACHE = 19;
constexpr uint8_t HOLD_LEADER_HELD = 20;

constexpr int SESS_PROTECTED = 1;   // s in O_w u P_w on instance `inst`
constexpr int SESS_RELEASED = 2;    // admitted before, protected nowhere now

constexpr int64_t CAP_INF = 2147483647;           // "no cap"
constexpr int64_t BACKLOG_MAX = (int64_t)1 << 61;   // largest backlog d_w and hold delay
constexpr int64_t TOKCOST_MAX = (int64_t)1 << 32;
constexpr int64_t MAX_PROMPT_TOKENS = (int64_t)1 << 20;
constexpr int BLOCK = 16;  // tokens per KV block

// ---- block hash (reading: the engine's block hash is not specified, Sec. 4.4) ----
// SplitMix64 finaliser (Steele, Lea & Flood 2014), golden-ratio increment G.
constexpr uint64_t G = 0x9e3779b97f4a7c15ULL;

uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
  z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
  return z ^ (z >> 31);
}

// Odd word multiplier of the content hash: the second SplitMix64 multiplier.
constexpr uint64_t WORD_MUL = 0x94d049bb133111ebULL;

// Content hash of one full block of 16 token ids: the 16 ids are read as eight
// 64-bit words (even id in the low half), each word is offset by its position
// times G and multiplied by the odd constant WORD_MUL (a bijection of the word), the
// eight products are XOR-ed and mixed once.
uint64_t block_content_hash(const int32_t* t) {
  uint64_t acc = 0;
  for (int i = 0; i < 8; ++i) {
    uint64_t lo = (uint32_t)t[2 * i];
    uint64_t hi = (uint32_t)t[2 * i + 1];
    uint64_t x = lo | (hi << 32);
    acc ^= (x + (uint64_t)(i + 1) * G) * WORD_MUL;
  }
  return mix64(acc);
}

// Chained key of every full block of a prompt: a_j = a_{j-1} * G + c_j with
// a_{-1} = seed, key_j = mix64(a_j ^ (j + 1)), keys 0 and 1 are reserved.
// A trailing partial block is not hashed.
std::vector<uint64_t> hash_prompt(const int32_t* tok, int64_t L, uint64_t seed) {
  std::vector<uint64_t> keys;
  int64_t nb = L / BLOCK;
  uint64_t a = seed;
  for (int64_t j = 0; j < nb; ++j) {
    uint64_t c = block_content_hash(tok + j * BLOCK);
    a = a * G + c;
    uint64_t k = mix64(a ^ (uint64_t)(j + 1));
    if (k < 2) k += 2;
    keys.push_back(k);
  }
  return keys;
}

// ---- index entry metadata (reading: LRU by commit tick, deepest first) ----
// meta = seq << 36 | arrival << 16 | (65535 - depth): ascending meta is the
// eviction order (oldest tick first, deeper block first among equal ticks).
uint64_t pack_meta(uint64_t seq, uint64_t arrival, uint64_t depth) {
  return (seq << 36) | (arrival << 16) | (uint64_t)(65535 - depth);
}

struct Entry {
  uint64_t meta;
  uint64_t parent;  // key of block depth-1 of the chain that inserted it; 0 if none/unknown
};

struct Session {
  int state;
  int inst;
  int cls;
};

struct Oracle {
  // configuration
  int32_t W = 0;
  std::vector<int64_t> cap;
  int32_t pf_q16 = 0;
  int32_t mode = 0;
  int64_t hold_delay_q = 0;
  int32_t hist_window = 256;
  int32_t min_obs = 8;
  int64_t prior_kbar[3] = {1, 1, 1};
  int64_t prior_T = 1;
  uint64_t hash_seed = G;

  // per-instance state
  std::vector<std::unordered_map<uint64_t, Entry>> index;
  std::vector<int64_t> backlog_q, tokcost_q;
  std::vector<int32_t> contraction;
  std::vector<std::array<int64_t, 3>> prot;  // protected sessions per (w, b)
  std::unordered_map<uint64_t, Session> sessions;
  std::deque<int64_t> hist_blocks[3], hist_res[3];
  uint32_t rho[3] = {333334, 333333, 333333};
  uint64_t seq = 0;

  // last route
  bool routed = false;
  int32_t n = 0;
  std::vector<uint8_t> cls;
  std::vector<uint64_t> sess;
  std::vector<int64_t> L;
  std::vector<std::vector<uint64_t>> keys;
  std::vector<uint16_t> H;  // [n][W]
  std::vector<int32_t> out_inst, out_hit, leader;
  std::vector<uint8_t> out_reason;
  std::vector<int64_t> K_w, K_wb, N_wb, kbar_w;
  int64_t kbar_b[3] = {0, 0, 0}, T_b[3] = {0, 0, 0}, cand[3] = {0, 0, 0};
  int64_t stats[32] = {0};
  int64_t commit_new_keys = 0, commit_evicted = 0;
};

int64_t index_size(const Oracle& o, int w) { return (int64_t)o.index[w].size(); }

// Insert one block with max-merge of its meta (a re-inserted block keeps the
// newest tick).  Returns 1 if the key was new.
int insert_block(Oracle& o, int w, uint64_t key, uint64_t meta, uint64_t parent) {
  auto it = o.index[w].find(key);
  if (it != o.index[w].end()) {
    if (meta > it->second.meta) it->second.meta = meta;
    return 0;
  }
  o.index[w][key] = Entry{meta, parent};
  return 1;
}

// Evict down to capacity: remove the smallest (meta, key) pairs, i.e. least
// recently committed first, deepest block first among equal ticks, key as the
// last tie-break (reading: eviction policy unspecified, Sec. 4.4).
int64_t evict_to_cap(Oracle& o, int w) {
  int64_t sz = index_size(o, w);
  if (sz <= o.cap[w]) return 0;
  std::vector<std::pair<uint64_t, uint64_t>> order;
  order.reserve(sz);
  for (auto& kv : o.index[w]) order.push_back({kv.second.meta, kv.first});
  std::sort(order.begin(), order.end());
  int64_t e = sz - o.cap[w];
  for (int64_t i = 0; i < e; ++i) o.index[w].erase(order[i].second);
  return e;
}

// ---- class estimators (Sec. 4.1 and Sec. 4.3; reading: p90 and window mean) ----
int64_t estimate_kbar(const Oracle& o, int b) {
  const auto& h = o.hist_blocks[b];
  if (h.empty()) return o.prior_kbar[b];
  std::vector<int64_t> v(h.begin(), h.end());
  std::sort(v.begin(), v.end());
  int64_t m = (int64_t)v.size();
  int64_t rank = (9 * m + 9) / 10;  // nearest-rank 90th percentile, ceil(0.9 m)
  int64_t p90 = v[rank - 1];
  return std::max(o.prior_kbar[b], p90);
}

int64_t estimate_T(const Oracle& o, int b) {
  const auto& h = o.hist_res[b];
  if ((int64_t)h.size() < o.min_obs) return o.prior_T;  // shared neutral prior
  int64_t s = 0;
  for (int64_t x : h) s += x;
  return s / (int64_t)h.size();
}

// ---- caps of one instance: Sec. 4.1 (K_w), Eqs. (9)-(10) MISA, (11),(13) MISA-T ----
void instance_caps(const Oracle& o, int w, const int64_t N[3], const int64_t kb[3],
                   const int64_t Tb[3], int64_t* Kw_out, int64_t Kwb_out[3],
                   int64_t* kbar_w_out) {
  // reference footprint of the instance: demand-weighted mean footprint, rounded up
  int64_t sumN = N[0] + N[1] + N[2];
  int64_t kw;
  if (sumN > 0) {
    __int128 num = 0;
    for (int b = 0; b < 3; ++b) num += (__int128)N[b] * kb[b];
    kw = (int64_t)((num + sumN - 1) / sumN);
  } else {
    kw = std::min(kb[0], std::min(kb[1], kb[2]));
  }
  *kbar_w_out = kw;
  // protected budget C_w and the base cap
  int64_t Cw = (int64_t)(((__int128)o.cap[w] * o.pf_q16) >> 16);
  int64_t Kbase = Cw / kw;
  int64_t Kw = std::max<int64_t>(1, Kbase - o.contraction[w]);
  if (o.mode == MODE_PLACEMENT_ONLY) Kw = CAP_INF;
  *Kw_out = Kw;
  if (o.mode == MODE_SESSION_ADMISSION || o.mode == MODE_PLACEMENT_ONLY) {
    for (int b = 0; b < 3; ++b) Kwb_out[b] = CAP_INF;
    return;
  }
  // block(-time) demand R_wb and proportional quota M_wb
  unsigned __int128 R[3], sumR = 0;
  for (int b = 0; b < 3; ++b) {
    R[b] = (unsigned __int128)N[b] * (unsigned __int128)kb[b];
    if (o.mode == MODE_MISA_T) R[b] *= (unsigned __int128)Tb[b];
    sumR += R[b];
  }
  for (int b = 0; b < 3; ++b) {
    int64_t M;
    if (sumR > 0)
      M = (int64_t)(((unsigned __int128)Cw * R[b]) / sumR);
    else  // reading: no demand at all -> split the budget by the trainer mixture
      M = (int64_t)(((__int128)Cw * o.rho[b]) / 1000000);
    Kwb_out[b] = std::max<int64_t>(1, M / kb[b]);
  }
}

int validate_config(int32_t W, const int64_t* cap, int32_t pf, int32_t mode, int64_t hold,
                    int32_t win, int32_t min_obs, const int64_t* pk, int64_t T0) {
  if (W < 1 || W > 1024) return ERR_INVALID_ARG;
  for (int w = 0; w < W; ++w)
    if (cap[w] < 1 || cap[w] > ((int64_t)1 << 26)) return ERR_INVALID_ARG;
  if (pf < 1 || pf > 65536) return ERR_INVALID_ARG;
  if (mode < 0 || mode > 3) return ERR_INVALID_ARG;
  if (hold < 0 || hold > BACKLOG_MAX) return ERR_INVALID_ARG;
  if (win < 1 || win > 4096 || min_obs < 1) return ERR_INVALID_ARG;
  for (int b = 0; b < 3; ++b)
    if (pk[b] < 1 || pk[b] > ((int64_t)1 << 30)) return ERR_INVALID_ARG;
  if (T0 < 0 || T0 > ((int64_t)1 << 40)) return ERR_INVALID_ARG;
  return OK;
}

}  // namespace

extern "C" {

uint64_t oracle_mix64(uint64_t z) { return mix64(z); }

int64_t oracle_hash_prompt(const int32_t* tokens, int64_t L, uint64_t seed, uint64_t* out) {
  std::vector<uint64_t> k = hash_prompt(tokens, L, seed);
  for (size_t j = 0; j < k.size(); ++j) out[j] = k[j];
  return (int64_t)k.size();
}

// Quota arithmetic of one instance in isolation (used by the hand-worked
// example test): C_w, N_b, kbar_b, T_b -> M_b and K_b.  mode 0 = MISA-T, 1 = MISA.
int oracle_caps_eval(int64_t Cw, const int64_t* N, const int64_t* kb, const int64_t* Tb,
                     int32_t mode, const uint32_t* rho, int64_t* M_out, int64_t* K_out) {
  unsigned __int128 R[3], sumR = 0;
  for (int b = 0; b < 3; ++b) {
    if (kb[b] < 1) return ERR_INVALID_ARG;
    R[b] = (unsigned __int128)N[b] * (unsigned __int128)kb[b];
    if (mode == MODE_MISA_T) R[b] *= (unsigned __int128)Tb[b];
    sumR += R[b];
  }
  for (int b = 0; b < 3; ++b) {
    int64_t M = sumR > 0 ? (int64_t)(((unsigned __int128)Cw * R[b]) / sumR)
                         : (int64_t)(((__int128)Cw * rho[b]) / 1000000);
    M_out[b] = M;
    K_out[b] = std::max<int64_t>(1, M / kb[b]);
  }
  return OK;
}

void* oracle_create(int32_t W, const int64_t* cap, int32_t pf_q16, int32_t mode,
                    int64_t hold_delay_q, int32_t hist_window, int32_t min_obs,
                    const int64_t* prior_kbar, int64_t prior_T_us, uint64_t hash_seed) {
  if (validate_config(W, cap, pf_q16, mode, hold_delay_q, hist_window, min_obs, prior_kbar,
                      prior_T_us) != OK)
    return nullptr;
  Oracle* o = new Oracle();
  o->W = W;
  o->cap.assign(cap, cap + W);
  o->pf_q16 = pf_q16;
  o->mode = mode;
  o->hold_delay_q = hold_delay_q;
  o->hist_window = hist_window;
  o->min_obs = min_obs;
  for (int b = 0; b < 3; ++b) o->prior_kbar[b] = prior_kbar[b];
  o->prior_T = prior_T_us;
  o->hash_seed = hash_seed;
  o->index.resize(W);
  o->backlog_q.assign(W, 0);
  o->tokcost_q.assign(W, 0);
  o->contraction.assign(W, 0);
  o->prot.assign(W, {0, 0, 0});
  return o;
}

void oracle_destroy(void* h) { delete (Oracle*)h; }

int oracle_set_mixture(void* h, const uint32_t* rho_ppm) {
  Oracle* o = (Oracle*)h;
  if ((uint64_t)rho_ppm[0] + rho_ppm[1] + rho_ppm[2] != 1000000) return ERR_INVALID_ARG;
  for (int b = 0; b < 3; ++b) o->rho[b] = rho_ppm[b];
  return OK;
}

int oracle_set_instance_state(void* h, const int64_t* backlog_q, const int64_t* tokcost_q,
                              const int32_t* contraction) {
  Oracle* o = (Oracle*)h;
  for (int w = 0; w < o->W; ++w) {
    if (backlog_q && (backlog_q[w] < 0 || backlog_q[w] > BACKLOG_MAX)) return ERR_INVALID_ARG;
    if (tokcost_q && (tokcost_q[w] < 0 || tokcost_q[w] > TOKCOST_MAX)) return ERR_INVALID_ARG;
    if (contraction && contraction[w] < 0) return ERR_INVALID_ARG;
  }
  for (int w = 0; w < o->W; ++w) {
    if (backlog_q) o->backlog_q[w] = backlog_q[w];
    if (tokcost_q) o->tokcost_q[w] = tokcost_q[w];
    if (contraction) o->contraction[w] = contraction[w];
  }
  return OK;
}

// Route one batch against the state at batch start.  Outputs per request:
// instance (-1 = HOLD), reason code, and hit blocks.
int oracle_route(void* h, int32_t n, const uint8_t* cls, const uint64_t* session,
                 const int64_t* tok_off, const int32_t* tokens, int32_t* out_inst,
                 uint8_t* out_reason, int32_t* out_hit) {
  Oracle* o = (Oracle*)h;
  const int W = o->W;
  if (n < 0 || n > (1 << 20)) return ERR_INVALID_ARG;
  if (n > 0 && tok_off[0] != 0) return ERR_INVALID_ARG;
  for (int r = 0; r < n; ++r) {
    if (cls[r] > 2 || session[r] == 0) return ERR_INVALID_ARG;
    int64_t len = tok_off[r + 1] - tok_off[r];
    if (len < 0 || len >= MAX_PROMPT_TOKENS) return ERR_INVALID_ARG;
  }
  o->routed = false;
  o->n = n;
  o->cls.assign(cls, cls + n);
  o->sess.assign(session, session + n);
  o->L.assign(n, 0);
  o->keys.assign(n, {});
  for (int r = 0; r < n; ++r) {
    o->L[r] = tok_off[r + 1] - tok_off[r];
    o->keys[r] = hash_prompt(tokens + tok_off[r], o->L[r], o->hash_seed);
  }

  // H_rw: number of leading blocks of r resident on w, by linear scan (Sec. 4.4)
  o->H.assign((size_t)n * W, 0);
  int64_t lookups = 0;
  for (int r = 0; r < n; ++r) {
    for (int w = 0; w < W; ++w) {
      int64_t hcount = 0;
      while (hcount < (int64_t)o->keys[r].size() && o->index[w].count(o->keys[r][hcount])) {
        ++hcount;
        ++lookups;
      }
      o->H[(size_t)r * W + w] = (uint16_t)hcount;
    }
  }

  // leaders: first request of each session in arrival order
  o->leader.assign(n, 0);
  {
    std::unordered_map<uint64_t, int> first;
    for (int r = 0; r < n; ++r) {
      auto it = first.find(session[r]);
      if (it == first.end()) {
        first[session[r]] = r;
        o->leader[r] = r;
      } else {
        o->leader[r] = it->second;
      }
    }
  }

  // session snapshot at batch start (O_w u P_w merged; Sec. 4.1)
  std::vector<int> st_state(n, 0), st_inst(n, -1);
  for (int r = 0; r < n; ++r) {
    auto it = o->sessions.find(session[r]);
    if (it != o->sessions.end()) {
      st_state[r] = it->second.state;
      st_inst[r] = it->second.inst;
    }
  }

  // class footprint and residency estimates (Sec. 4.1, Sec. 4.3)
  for (int b = 0; b < 3; ++b) {
    o->kbar_b[b] = estimate_kbar(*o, b);
    o->T_b[b] = estimate_T(*o, b);
    o->cand[b] = 0;
  }
  // candidate sessions: distinct sessions in the batch protected nowhere (Sec. 4.2)
  for (int r = 0; r < n; ++r)
    if (o->leader[r] == r && st_state[r] != SESS_PROTECTED) o->cand[cls[r]] += 1;

  // caps per instance
  o->K_w.assign(W, 0);
  o->K_wb.assign((size_t)W * 3, 0);
  o->N_wb.assign((size_t)W * 3, 0);
  o->kbar_w.assign(W, 0);
  std::vector<int64_t> tot(W, 0);
  for (int w = 0; w < W; ++w) {
    int64_t N[3];
    for (int b = 0; b < 3; ++b) {
      N[b] = o->prot[w][b] + o->cand[b];
      o->N_wb[(size_t)w * 3 + b] = N[b];
      tot[w] += o->prot[w][b];
    }
    int64_t Kwb[3];
    instance_caps(*o, w, N, o->kbar_b, o->T_b, &o->K_w[w], Kwb, &o->kbar_w[w]);
    for (int b = 0; b < 3; ++b) o->K_wb[(size_t)w * 3 + b] = Kwb[b];
  }

  // selection (reading: the batch's leaders are decided one at a time in arrival order,
  // as the online router of Sec. 4 decides requests.  Each one sees the snapshot taken at
  // batch start -- caches, sessions, backlog d_w and throughput mu_w -- and the admissions
  // of the leaders before it: an admitted session is recorded at once as pending on its
  // instance (P_w, Sec. 4.1-4.2), so it takes headroom from everyone after it.  A leader is
  // therefore held only when no instance has headroom for it at its turn.)
  std::vector<int64_t> adm(W, 0);
  std::vector<std::array<int64_t, 3>> admb(W, {0, 0, 0});
  const std::vector<int64_t>& bk = o->backlog_q;
  o->out_inst.assign(n, -1);
  o->out_reason.assign(n, 0);

  auto eligible = [&](int r, int w) {
    int b = cls[r];
    bool protected_here = st_state[r] == SESS_PROTECTED && st_inst[r] == w;
    if (protected_here) return true;  // Eq. (6), first case
    return tot[w] + adm[w] < o->K_w[w] &&
           o->prot[w][b] + admb[w][b] < o->K_wb[(size_t)w * 3 + b];  // Eq. (6) + Sec. 4.2
  };

  for (int r = 0; r < n; ++r) {
    if (o->leader[r] != r) continue;
    const int b = cls[r];
    // placement among the instances where Admit(r, w) holds (Sec. 4.4: filter by
    // headroom, then cache-aware placement): argmin of Eq. (1), ties to the lower w
    int best = -1;
    int64_t best_cost = 0;
    for (int w = 0; w < W; ++w) {
      if (!eligible(r, w)) continue;
      int64_t cost = bk[w] + (o->L[r] - BLOCK * (int64_t)o->H[(size_t)r * W + w]) * o->tokcost_q[w];
      if (best < 0 || cost < best_cost) {
        best = w;
        best_cost = cost;
      }
    }
    if (best < 0) {
      // HOLD: the global cap binds everywhere, or the class cap binds on every instance
      // that still has global headroom
      bool global_room = false;
      for (int w = 0; w < W; ++w)
        if (tot[w] + adm[w] < o->K_w[w]) global_room = true;
      o->out_reason[r] = global_room ? HOLD_CLASS_CAP : HOLD_GLOBAL_CAP;
      continue;
    }
    // Eq. (7): a continuation that must be admitted again may prefer to wait
    if (st_state[r] == SESS_RELEASED) {
      int wh = 0;
      for (int w = 1; w < W; ++w)
        if (o->H[(size_t)r * W + w] > o->H[(size_t)r * W + wh]) wh = w;
      int64_t Hh = o->H[(size_t)r * W + wh];
      if (Hh > 0 && !eligible(r, wh)) {
        int64_t lhs = o->hold_delay_q + bk[wh] - bk[best];
        int64_t rhs = BLOCK * Hh * o->tokcost_q[wh];
        if (lhs < rhs) {
          o->out_reason[r] = HOLD_PREFER_CACHE;
          continue;
        }
      }
    }
    bool protected_here = st_state[r] == SESS_PROTECTED && st_inst[r] == best;
    o->out_inst[r] = best;
    if (protected_here) {
      o->out_reason[r] = ADMIT_CONT;  // no headroom consumed
    } else {
      o->out_reason[r] = ADMIT_NEW;   // pending on `best` from now on
      adm[best] += 1;
      admb[best][b] += 1;
    }
  }
  // followers: later requests of a session in the batch follow their leader
  for (int r = 0; r < n; ++r) {
    int ld = o->leader[r];
    if (ld == r) continue;
    if (o->out_inst[ld] >= 0) {
      o->out_inst[r] = o->out_inst[ld];
      o->out_reason[r] = ADMIT_FOLLOW;
    } else {
      o->out_inst[r] = -1;
      o->out_reason[r] = HOLD_LEADER_HELD;
    }
  }
  // hit blocks and statistics
  o->out_hit.assign(n, 0);
  std::memset(o->stats, 0, sizeof(o->stats));
  int64_t* S = o->stats;
  S[0] = n;
  for (int r = 0; r < n; ++r) {
    int w = o->out_inst[r];
    int64_t hb = 0;
    if (w >= 0) {
      hb = o->H[(size_t)r * W + w];
    } else {
      for (int x = 0; x < W; ++x) hb = std::max<int64_t>(hb, o->H[(size_t)r * W + x]);
    }
    o->out_hit[r] = (int32_t)hb;
    uint8_t rs = o->out_reason[r];
    int ri = rs < 16 ? rs - 1 : 3 + (rs - 16);
    S[3 + ri] += 1;
    if (w >= 0) {
      S[1] += 1;
      S[11 + cls[r]] += 1;
      S[17] += BLOCK * hb;
      S[18] += o->L[r];
    } else {
      S[2] += 1;
      S[14 + cls[r]] += 1;
    }
  }
  // D_TV between the admitted class mix and the trainer mixture, in ppm (Sec. 3.3)
  int64_t A = S[1];
  if (A > 0) {
    __int128 acc = 0;
    for (int b = 0; b < 3; ++b) {
      __int128 d = (__int128)1000000 * S[11 + b] - (__int128)o->rho[b] * A;
      acc += d < 0 ? -d : d;
    }
    S[19] = (int64_t)(acc / (2 * (__int128)A));
  } else {
    S[19] = -1;
  }
  S[20] = lookups;
  for (int r = 0; r < n; ++r) {
    out_inst[r] = o->out_inst[r];
    out_reason[r] = o->out_reason[r];
    out_hit[r] = o->out_hit[r];
  }
  o->routed = true;
  return OK;
}

int oracle_get_H(void* h, uint16_t* out) {
  Oracle* o = (Oracle*)h;
  std::memcpy(out, o->H.data(), o->H.size() * sizeof(uint16_t));
  return OK;
}

// Keys of the last routed batch in request order (compact: request 0's blocks,
// then request 1's, ...).
int oracle_get_keys(void* h, uint64_t* out, int64_t cap, int64_t* n_out) {
  Oracle* o = (Oracle*)h;
  int64_t k = 0;
  for (auto& v : o->keys) {
    for (uint64_t x : v) {
      if (k >= cap) return ERR_INVALID_ARG;
      out[k++] = x;
    }
  }
  *n_out = k;
  return OK;
}

// Caps of the last route: K_w [W], K_wb [W*3], N_wb [W*3], kbar_w [W],
// and per class kbar_b [3], T_b [3].
int oracle_get_caps(void* h, int64_t* Kw, int64_t* Kwb, int64_t* Nwb, int64_t* kbw, int64_t* kb,
                    int64_t* Tb) {
  Oracle* o = (Oracle*)h;
  for (int w = 0; w < o->W; ++w) {
    Kw[w] = o->K_w[w];
    kbw[w] = o->kbar_w[w];
    for (int b = 0; b < 3; ++b) {
      Kwb[w * 3 + b] = o->K_wb[(size_t)w * 3 + b];
      Nwb[w * 3 + b] = o->N_wb[(size_t)w * 3 + b];
    }
  }
  for (int b = 0; b < 3; ++b) {
    kb[b] = o->kbar_b[b];
    Tb[b] = o->T_b[b];
  }
  return OK;
}

// Stats of the last route (layout: see the Python wrapper).
int oracle_get_stats(void* h, int64_t* out) {
  Oracle* o = (Oracle*)h;
  for (int i = 0; i < 32; ++i) out[i] = o->stats[i];
  out[21] = o->commit_new_keys;
  out[22] = o->commit_evicted;
  out[23] = (int64_t)o->seq;
  return OK;
}

// Apply the last route: index inserts (tick = commit seq and arrival index,
// depth = block index), session table and protected counts, then eviction.
int oracle_commit(void* h) {
  Oracle* o = (Oracle*)h;
  if (!o->routed) return ERR_STATE;
  uint64_t seq_c = o->seq + 1;
  int64_t new_keys = 0;
  for (int r = 0; r < o->n; ++r) {
    int w = o->out_inst[r];
    if (w < 0) continue;
    const auto& k = o->keys[r];
    for (size_t j = 0; j < k.size(); ++j)
      new_keys += insert_block(*o, w, k[j], pack_meta(seq_c, (uint64_t)r, j), j ? k[j - 1] : 0);
  }
  // newly admitted sessions become pending/protected on their instance (Sec. 4.1);
  // a rebound session leaves the protected count of its previous instance
  for (int r = 0; r < o->n; ++r) {
    if (o->leader[r] != r || o->out_reason[r] != ADMIT_NEW) continue;
    uint64_t s = o->sess[r];
    auto it = o->sessions.find(s);
    if (it != o->sessions.end() && it->second.state == SESS_PROTECTED)
      o->prot[it->second.inst][it->second.cls] -= 1;
    o->sessions[s] = Session{SESS_PROTECTED, o->out_inst[r], o->cls[r]};
    o->prot[o->out_inst[r]][o->cls[r]] += 1;
  }
  int64_t ev = 0;
  for (int w = 0; w < o->W; ++w) ev += evict_to_cap(*o, w);
  o->commit_new_keys = new_keys;
  o->commit_evicted = ev;
  o->seq = seq_c;
  o->routed = false;
  return OK;
}

// Completion events: done=1 finishes the session (histories, leaves the
// protected set, forgotten); done=0 releases its protection but remembers it
// (a later request is a continuation that must be admitted again, Eq. 7).
int oracle_complete(void* h, int32_t n, const uint64_t* session, const uint8_t* cls,
                    const int32_t* total_blocks, const int64_t* residency_us,
                    const uint8_t* done) {
  Oracle* o = (Oracle*)h;
  std::unordered_set<uint64_t> seen;
  for (int i = 0; i < n; ++i) {
    if (cls[i] > 2 || total_blocks[i] < 0 || residency_us[i] < 0 || session[i] == 0)
      return ERR_INVALID_ARG;
    if (!seen.insert(session[i]).second) return ERR_INVALID_ARG;
  }
  for (int i = 0; i < n; ++i) {
    if (done[i]) {
      int b = cls[i];
      o->hist_blocks[b].push_back(total_blocks[i]);
      o->hist_res[b].push_back(residency_us[i]);
      while ((int32_t)o->hist_blocks[b].size() > o->hist_window) o->hist_blocks[b].pop_front();
      while ((int32_t)o->hist_res[b].size() > o->hist_window) o->hist_res[b].pop_front();
    }
    auto it = o->sessions.find(session[i]);
    if (it == o->sessions.end()) continue;
    if (it->second.state == SESS_PROTECTED) o->prot[it->second.inst][it->second.cls] -= 1;
    if (done[i])
      o->sessions.erase(it);
    else
      it->second.state = SESS_RELEASED;
  }
  return OK;
}

// Engine removal events (Sec. 4.4): remove the listed keys of instance w.
int oracle_evict(void* h, int32_t w, const uint64_t* keys, int64_t n) {
  Oracle* o = (Oracle*)h;
  if (w < 0 || w >= o->W || n < 0) return ERR_INVALID_ARG;
  for (int64_t i = 0; i < n; ++i) o->index[w].erase(keys[i]);
  return OK;
}

// Cache reset after a weight sync: the instance's index becomes empty.
int oracle_reset_instance(void* h, int32_t w) {
  Oracle* o = (Oracle*)h;
  if (w < 0 || w >= o->W) return ERR_INVALID_ARG;
  o->index[w].clear();
  return OK;
}

int oracle_load_entries(void* h, int32_t w, const uint64_t* keys, const uint64_t* metas,
                        int64_t n) {
  Oracle* o = (Oracle*)h;
  if (w < 0 || w >= o->W || n < 0) return ERR_INVALID_ARG;
  for (int64_t i = 0; i < n; ++i)
    if (keys[i] < 2 || (metas[i] & 0xFFFF) == 0) return ERR_INVALID_ARG;
  for (int64_t i = 0; i < n; ++i) insert_block(*o, w, keys[i], metas[i], 0);
  evict_to_cap(*o, w);
  return OK;
}

// Warm chains: hash each chain's tokens and insert its first min(n_blocks,
// max_blocks[c]) blocks on inst[c] with tick (seq[c], arr[c]); then evict.
int oracle_load_chains(void* h, int32_t n_chains, const int64_t* tok_off, const int32_t* tokens,
                       const int32_t* inst, const uint64_t* seq, const uint32_t* arr,
                       const int32_t* max_blocks) {
  Oracle* o = (Oracle*)h;
  for (int c = 0; c < n_chains; ++c) {
    if (inst[c] < 0 || inst[c] >= o->W || seq[c] >= ((uint64_t)1 << 28) ||
        arr[c] >= (1u << 20) || max_blocks[c] < 0)
      return ERR_INVALID_ARG;
    int64_t len = tok_off[c + 1] - tok_off[c];
    if (len < 0 || len >= MAX_PROMPT_TOKENS) return ERR_INVALID_ARG;
  }
  for (int c = 0; c < n_chains; ++c) {
    std::vector<uint64_t> k = hash_prompt(tokens + tok_off[c], tok_off[c + 1] - tok_off[c],
                                          o->hash_seed);
    int64_t m = std::min<int64_t>((int64_t)k.size(), max_blocks[c]);
    for (int64_t j = 0; j < m; ++j)
      insert_block(*o, inst[c], k[j], pack_meta(seq[c], arr[c], (uint64_t)j), j ? k[j - 1] : 0);
  }
  for (int w = 0; w < o->W; ++w) evict_to_cap(*o, w);
  return OK;
}

int64_t oracle_index_size(void* h, int32_t w) { return index_size(*(Oracle*)h, w); }

int oracle_dump_index(void* h, int32_t w, uint64_t* keys, uint64_t* metas, int64_t cap,
                      int64_t* n_out) {
  Oracle* o = (Oracle*)h;
  if (w < 0 || w >= o->W) return ERR_INVALID_ARG;
  std::vector<std::pair<uint64_t, uint64_t>> v;
  for (auto& kv : o->index[w]) v.push_back({kv.first, kv.second.meta});
  std::sort(v.begin(), v.end());
  if ((int64_t)v.size() > cap) return ERR_INVALID_ARG;
  for (size_t i = 0; i < v.size(); ++i) {
    keys[i] = v[i].first;
    metas[i] = v[i].second;
  }
  *n_out = (int64_t)v.size();
  return OK;
}

int oracle_get_counts(void* h, int32_t* prot) {
  Oracle* o = (Oracle*)h;
  for (int w = 0; w < o->W; ++w)
    for (int b = 0; b < 3; ++b) prot[w * 3 + b] = (int32_t)o->prot[w][b];
  return OK;
}

int64_t oracle_n_sessions(void* h) { return (int64_t)((Oracle*)h)->sessions.size(); }

int oracle_dump_sessions(void* h, uint64_t* ids, int32_t* state, int32_t* inst, int32_t* cls,
                         int64_t cap, int64_t* n_out) {
  Oracle* o = (Oracle*)h;
  std::vector<uint64_t> v;
  for (auto& kv : o->sessions) v.push_back(kv.first);
  std::sort(v.begin(), v.end());
  if ((int64_t)v.size() > cap) return ERR_INVALID_ARG;
  for (size_t i = 0; i < v.size(); ++i) {
    const Session& s = o->sessions[v[i]];
    ids[i] = v[i];
    state[i] = s.state;
    inst[i] = s.inst;
    cls[i] = s.cls;
  }
  *n_out = (int64_t)v.size();
  return OK;
}

uint64_t oracle_seq(void* h) { return ((Oracle*)h)->seq; }

// Invariants after a commit.  Returns 0 if all hold, else the number of the
// first one broken: 1 size <= Cap, 2 prefix closure (a resident block's parent
// is resident), 3 tick(parent) >= tick(child), 4 protected counts agree with
// the session table, 5 a protected count is negative.
int oracle_check_invariants(void* h) {
  Oracle* o = (Oracle*)h;
  for (int w = 0; w < o->W; ++w) {
    if (index_size(*o, w) > o->cap[w]) return 1;
    for (auto& kv : o->index[w]) {
      uint64_t p = kv.second.parent;
      if (p == 0) continue;
      auto it = o->index[w].find(p);
      if (it == o->index[w].end()) return 2;
      if ((it->second.meta >> 16) < (kv.second.meta >> 16)) return 3;
    }
  }
  std::vector<std::array<int64_t, 3>> cnt(o->W, {0, 0, 0});
  for (auto& kv : o->sessions)
    if (kv.second.state == SESS_PROTECTED) cnt[kv.second.inst][kv.second.cls] += 1;
  for (int w = 0; w < o->W; ++w)
    for (int b = 0; b < 3; ++b) {
      if (o->prot[w][b] < 0) return 5;
      if (cnt[w][b] != o->prot[w][b]) return 4;
    }
  return 0;
}

}  // extern "C"

extern "C" {
// Deep copy of an oracle state (used to restart a timed step from the same state).
void* oracle_clone(void* h) { return new Oracle(*(Oracle*)h); }
}
