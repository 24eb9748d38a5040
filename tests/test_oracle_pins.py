"""Pins of the CPU oracle against what the paper and mathematics fix (no GPU).

Every check here is independent of the oracle's own code: published SplitMix64
outputs, a token-by-token brute-force prefix index, the hand-worked quota example
of Eqs. (9)-(13), closed forms, special cases and invariants.
"""

import os

import numpy as np
import pytest

import oracle
from paper_2608_11152_gb300 import workload as wl
from tests.helpers import ADMITS, HOLDS, BlockModel, make_oracle, scenario_steps

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
G = 0x9E3779B97F4A7C15
M64 = (1 << 64) - 1


def _golden_kv(name):
    out = {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        k, *v = line.split()
        out[k] = [int(x) for x in v]
    return out


# ---------------------------------------------------------------- block hash

def test_mix64_reproduces_published_splitmix64_outputs():
    vals = [int(l, 16) for l in open(os.path.join(GOLDEN, "splitmix64_seed0.txt"))
            if l.strip() and not l.startswith("#")]
    for k, v in enumerate(vals, start=1):
        assert oracle.mix64((k * G) & M64) == v


def test_mix64_is_a_bijection_on_a_sample():
    rng = np.random.default_rng(1)
    xs = rng.integers(0, 2**63, size=20000, dtype=np.int64).astype(np.uint64)
    ys = {oracle.mix64(int(x)) for x in xs}
    assert len(ys) == len(set(int(x) for x in xs))


def test_hash_is_chained_over_the_prefix():
    rng = np.random.default_rng(2)
    a = rng.integers(0, wl.VOCAB, size=16 * 12 + 5, dtype=np.int32)
    ka = oracle.hash_prompt(a)
    assert len(ka) == 12                                   # trailing partial block not hashed
    assert np.all(ka >= 2)                                 # 0 and 1 reserved
    # an extension keeps every earlier key
    ext = np.concatenate([a, rng.integers(0, wl.VOCAB, size=40, dtype=np.int32)])
    assert np.array_equal(oracle.hash_prompt(ext)[:12], ka)
    # changing one token of block 3 changes key 3 and every later key, not earlier ones
    b = a.copy()
    b[16 * 3 + 7] ^= 1
    kb = oracle.hash_prompt(b)
    assert np.array_equal(kb[:3], ka[:3])
    assert np.all(kb[3:] != ka[3:])
    # identical block content at a different depth or after a different prefix gives a different key
    c = np.concatenate([a[16:32], a[16:32]])
    kc = oracle.hash_prompt(c)
    assert kc[0] != kc[1] and kc[0] != ka[1]
    # swapping two tokens inside a block changes the key (position-sensitive content hash)
    d = a.copy()
    d[[0, 1]] = d[[1, 0]]
    if d[0] != d[1]:
        assert oracle.hash_prompt(d)[0] != ka[0]
    # the chain seed matters
    assert np.all(oracle.hash_prompt(a, seed=12345) != ka)


def test_hash_distinct_keys_on_medium_workload():
    sc = wl.config1()
    seen = {}
    for b, _ in scenario_steps(sc):
        for r in range(b.n):
            t = b.tokens[b.tok_off[r]:b.tok_off[r + 1]]
            ks = oracle.hash_prompt(t)
            for j, k in enumerate(ks):
                ident = t[: 16 * (j + 1)].tobytes()
                prev = seen.setdefault(int(k), ident)
                assert prev == ident, "two different prefixes share a key"


# ---------------------------------------------------------------- H and the index, brute force

@pytest.mark.parametrize("seed", list(range(12)))
def test_H_and_index_match_token_level_bruteforce(seed):
    sc = wl.small_random(1000 + seed, W=3, cap=48, n=20, mode=seed % 4, n_warm=3)
    o = make_oracle(sc)
    model = BlockModel(sc.cap_blocks)
    seq = 0
    for b, comp in scenario_steps(sc):
        inst, reason, hit = o.route(b.cls, b.session, b.tok_off, b.tokens)
        assert np.array_equal(o.H(), model.H(b))
        o.commit()
        seq += 1
        model.commit(seq, b, inst)
        assert o.check_invariants() == 0
        for w in range(sc.W):
            k, m = o.dump_index(w)
            assert np.array_equal(np.sort(m), model.metas(w))
            assert np.array_equal(k, model.keys(w))
        if comp is not None:
            o.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)


# ---------------------------------------------------------------- quotas, Eqs. (9)-(13)

def test_quota_hand_example_eqs_9_to_13():
    g = _golden_kv("quota_example.txt")
    M, K = oracle.caps_eval(g["C"][0], g["N"], g["kbar"], g["T"], mode=oracle.MODE_MISA)
    assert list(M) == g["misa_M"] and list(K) == g["misa_K"]
    M, K = oracle.caps_eval(g["C"][0], g["N"], g["kbar"], g["T"], mode=oracle.MODE_MISA_T)
    assert list(M) == g["misat_M"] and list(K) == g["misat_K"]


def _batch(cls, sessions, lens, seed=0):
    rng = np.random.default_rng(seed)
    off = np.zeros(len(cls) + 1, np.int64)
    np.cumsum(lens, out=off[1:])
    toks = rng.integers(0, wl.VOCAB, size=int(off[-1]), dtype=np.int32)
    return wl.Batch(cls=np.array(cls, np.uint8), session=np.array(sessions, np.uint64),
                    group=np.zeros(len(cls), np.uint64), tok_off=off, tokens=toks)


@pytest.mark.parametrize("mode,Kb", [(oracle.MODE_MISA_T, (2, 1, 1)), (oracle.MODE_MISA, (4, 2, 1))])
def test_quota_hand_example_end_to_end(mode, Kb):
    """One instance with C_w = 1000, 8/4/2 new sessions, priors (64, 96, 512) and
    residencies (600, 120, 1800): the route must apply exactly the hand-worked caps."""
    o = oracle.Oracle([1000], protected_frac_q16=65536, mode=mode,
                      prior_kbar=(64, 96, 512), prior_T_us=1, min_obs=1, hist_window=1)
    o.set_mixture((400000, 300000, 300000))
    o.set_instance_state([0], [1], [0])
    # one completed observation per class: residency as in the example, 0 blocks (keeps kbar at the prior)
    o.complete([91, 92, 93], [0, 1, 2], [0, 0, 0], [600, 120, 1800], [1, 1, 1])
    cls = [0] * 8 + [1] * 4 + [2] * 2
    b = _batch(cls, list(range(1, 15)), [32] * 14)
    inst, reason, hit = o.route(b.cls, b.session, b.tok_off, b.tokens)
    caps = o.caps()
    assert list(caps["N_wb"][0]) == [8, 4, 2]
    assert list(caps["kbar_b"]) == [64, 96, 512]
    assert list(caps["K_wb"][0]) == list(Kb)
    # kbar_w = ceil((8*64 + 4*96 + 2*512) / 14) = ceil(137.14) = 138; K_w = floor(1000/138) = 7
    assert caps["kbar_w"][0] == 138 and caps["K_w"][0] == 7
    # admission in arrival order: the first Kb[b] sessions of each class, global cap 7 not binding
    adm = [r for r in range(14) if reason[r] == oracle.ADMIT_NEW]
    exp = [r for b_ in range(3) for r in [i for i in range(14) if cls[i] == b_][: Kb[b_]]]
    assert sorted(adm) == sorted(exp)
    for r in range(14):
        if r not in exp:
            before = sum(1 for x in exp if x < r)
            assert reason[r] == (oracle.HOLD_GLOBAL_CAP if before >= 7 else oracle.HOLD_CLASS_CAP)


def test_serial_selection_hand_example():
    """Sec. 4.1 Eq. (6), Sec. 4.2 and the Sec. 4.4 pipeline on a batch worked by hand
    (tests/golden/serial_selection_example.txt): each leader takes the cheapest instance
    where Admit holds given the sessions admitted before it, and is held only when none has
    headroom for it (class cap while some instance has global headroom, else global cap)."""
    g = _golden_kv("serial_selection_example.txt")
    W = len(g["backlog"])
    o = oracle.Oracle([4096] * W, protected_frac_q16=65536, mode=oracle.MODE_MISA_T,
                      prior_kbar=(2048, 2048, 2048))
    o.set_instance_state(g["backlog"], g["tokcost"], [0] * W)
    n = len(g["cls"])
    b = _batch(g["cls"], list(range(1, n + 1)), [g["prompt_tokens"][0]] * n)
    inst, reason, hit = o.route(b.cls, b.session, b.tok_off, b.tokens)
    caps = o.caps()
    assert list(caps["K_w"]) == g["K_w"]
    assert all(list(caps["K_wb"][w]) == g["K_wb"] for w in range(W))
    assert list(inst) == g["inst"] and list(reason) == g["reason"]


def test_quota_closed_forms_random():
    rng = np.random.default_rng(5)
    for _ in range(2000):
        C = int(rng.integers(1, 10**7))
        N = rng.integers(0, 5000, size=3)
        kb = rng.integers(1, 10**5, size=3)
        T = rng.integers(0, 10**9, size=3)
        for mode in (oracle.MODE_MISA_T, oracle.MODE_MISA):
            M, K = oracle.caps_eval(C, N, kb, T, mode=mode)
            R = [int(N[b]) * int(kb[b]) * (int(T[b]) if mode == 0 else 1) for b in range(3)]
            S = sum(R)
            assert np.all(K >= 1)
            if S == 0:
                continue
            # Eq. (3): quotas never exceed the protected budget; floors lose < 1 block per class
            assert C - 2 <= int(M.sum()) <= C
            # Eq. (12): every class's drain time R_b / M_b is at least sum R / C
            for b in range(3):
                if M[b] > 0:
                    assert R[b] * C >= int(M[b]) * S
        # equal residency makes MISA-T quotas equal the MISA quotas (Eq. 13 vs Eq. 10)
        Tq = np.full(3, int(rng.integers(1, 10**6)))
        assert np.array_equal(oracle.caps_eval(C, N, kb, Tq, 0)[0], oracle.caps_eval(C, N, kb, Tq, 1)[0])


# ---------------------------------------------------------------- special cases

def test_one_instance_no_cache_admits_in_arrival_order():
    o = oracle.Oracle([4096], prior_kbar=(16, 16, 16))
    o.set_instance_state([0], [10], [0])
    rng = np.random.default_rng(3)
    cls = list(rng.integers(0, 3, size=200))
    b = _batch(cls, list(range(1, 201)), list(rng.integers(0, 300, size=200)))
    inst, reason, hit = o.route(b.cls, b.session, b.tok_off, b.tokens)
    caps = o.caps()
    Kw, Kwb = caps["K_w"][0], caps["K_wb"][0]
    tot, per = 0, [0, 0, 0]
    for r in range(200):
        c = cls[r]
        if tot < Kw and per[c] < Kwb[c]:
            assert reason[r] == oracle.ADMIT_NEW and inst[r] == 0
            tot += 1
            per[c] += 1
        else:
            assert inst[r] == -1
            assert reason[r] == (oracle.HOLD_GLOBAL_CAP if tot >= Kw else oracle.HOLD_CLASS_CAP)
    assert np.all(hit == 0)


def test_placement_only_without_token_cost_picks_least_backlog():
    W = 6
    o = oracle.Oracle([512] * W, mode=oracle.MODE_PLACEMENT_ONLY)
    bk = [50, 20, 70, 20, 90, 30]
    o.set_instance_state(bk, [0] * W, [0] * W)
    b = _batch([0, 1, 2] * 10, list(range(1, 31)), [64] * 30)
    inst, reason, _ = o.route(b.cls, b.session, b.tok_off, b.tokens)
    assert np.all(inst == 1) and np.all(reason == oracle.ADMIT_NEW)


def test_placement_only_with_equal_backlogs_picks_longest_prefix():
    W = 5
    o = oracle.Oracle([4096] * W, mode=oracle.MODE_PLACEMENT_ONLY)
    rng = np.random.default_rng(9)
    base = rng.integers(0, wl.VOCAB, size=16 * 20, dtype=np.int32)
    # warm instance w with the first 4*w blocks of `base` (w = 1..4)
    lens = [64 * w for w in range(1, 5)]
    off = np.zeros(5, np.int64)
    np.cumsum(lens, out=off[1:])
    toks = np.concatenate([base[:l] for l in lens])
    o.load_chains(off, toks, [1, 2, 3, 4], [0] * 4, [0] * 4, [1 << 20] * 4)
    o.set_instance_state([7] * W, [100] * W, [0] * W)
    b = wl.Batch(cls=np.array([0, 1], np.uint8), session=np.array([5, 6], np.uint64),
                 group=np.zeros(2, np.uint64), tok_off=np.array([0, 320, 320 + 96], np.int64),
                 tokens=np.concatenate([base, base[:96]]))
    inst, reason, hit = o.route(b.cls, b.session, b.tok_off, b.tokens)
    H = o.H()
    assert list(H[0]) == [0, 4, 8, 12, 16] and list(H[1]) == [0, 4, 6, 6, 6]
    assert inst[0] == 4 and hit[0] == 16
    assert inst[1] == 2 and hit[1] == 6          # ties of H go to the lowest index (lowest cost)


def test_equal_residency_makes_misat_equal_misa():
    for seed in range(6):
        sc = wl.small_random(2000 + seed, W=4, cap=96, n=30, mode=0, n_warm=0)
        res = []
        for mode in (oracle.MODE_MISA_T, oracle.MODE_MISA):
            o = make_oracle(sc, mode=mode)
            b = sc.batch
            res.append(o.route(b.cls, b.session, b.tok_off, b.tokens))
            res.append(o.caps()["K_wb"])
        for x, y in zip(res[0], res[2]):
            assert np.array_equal(x, y)
        assert np.array_equal(res[1], res[3])


# ---------------------------------------------------------------- invariants on random scenarios

def _check_route_invariants(o, b, inst, reason, hit, prot_before, sess_before):
    n, W = b.n, o.W
    caps = o.caps()
    H = o.H()
    assert len(inst) == n                                     # none dropped
    for r in range(n):
        if inst[r] >= 0:
            assert reason[r] in ADMITS and hit[r] == H[r, inst[r]]
        else:
            assert reason[r] in HOLDS and hit[r] == H[r].max()
    # followers copy their session leader
    first = {}
    for r in range(n):
        s = int(b.session[r])
        if s in first:
            ld = first[s]
            assert inst[r] == inst[ld]
            assert reason[r] == (oracle.ADMIT_FOLLOW if inst[ld] >= 0 else oracle.HOLD_LEADER_HELD)
        else:
            first[s] = r
    # continuations only where the session was protected; new sessions within both caps
    new = np.zeros((W, 3), np.int64)
    for r in range(n):
        if reason[r] == oracle.ADMIT_CONT:
            st = sess_before.get(int(b.session[r]))
            assert st is not None and st[0] == 1 and st[1] == inst[r]
        if reason[r] == oracle.ADMIT_NEW:
            new[inst[r], b.cls[r]] += 1
    for w in range(W):
        tot = prot_before[w].sum()
        assert new[w].sum() <= max(0, caps["K_w"][w] - tot)
        for c in range(3):
            assert new[w, c] <= max(0, caps["K_wb"][w, c] - prot_before[w, c])


def _eligible_after(caps, prot_before, adm, st, w, c):
    """Admit(r, w) of Eq. (6) with the class cap of Sec. 4.2, given the new sessions `adm`
    [W][3] admitted so far in the batch (pending, Sec. 4.1)."""
    if st[0] == 1 and st[1] == w:
        return True
    return (prot_before[w].sum() + adm[w].sum() < caps["K_w"][w]
            and prot_before[w, c] + adm[w, c] < caps["K_wb"][w, c])


def _check_held_have_no_headroom(o, b, inst, reason, prot_before, sess_before):
    """Eq. (6) holds a request only when it cannot get headroom: under the counts after the
    whole batch, a leader held for a cap has no instance where Admit holds."""
    W = o.W
    caps = o.caps()
    adm = np.zeros((W, 3), np.int64)
    for r in range(b.n):
        if reason[r] == oracle.ADMIT_NEW:
            adm[inst[r], b.cls[r]] += 1
    for r in range(b.n):
        if reason[r] in (oracle.HOLD_GLOBAL_CAP, oracle.HOLD_CLASS_CAP, oracle.HOLD_NO_ELIGIBLE):
            st = sess_before.get(int(b.session[r]), (0, -1))
            assert not any(_eligible_after(caps, prot_before, adm, st, w, b.cls[r]) for w in range(W))
            if reason[r] == oracle.HOLD_GLOBAL_CAP:
                assert all(prot_before[w].sum() + adm[w].sum() >= caps["K_w"][w] for w in range(W))


def _check_serial_order(o, b, inst, reason, prot_before, sess_before, backlog, tokcost, hold):
    """The batch decided one leader at a time in arrival order, checked on the decisions
    alone: with the sessions admitted before a leader counted as pending, an admitted leader
    sits on the cheapest instance of Eq. (1) where Admit holds (Sec. 4.4, ties to the lower
    index); a leader held for a cap had no such instance at its turn; an Eq. (7) hold had its
    cached instance without headroom and a saving above the hold delay."""
    W = o.W
    caps = o.caps()
    H = o.H().astype(np.int64)
    L = np.diff(b.tok_off).astype(np.int64)
    adm = np.zeros((W, 3), np.int64)
    seen = set()
    for r in range(b.n):
        s = int(b.session[r])
        if s in seen:
            continue
        seen.add(s)
        c = int(b.cls[r])
        st = sess_before.get(s, (0, -1))
        E = [w for w in range(W) if _eligible_after(caps, prot_before, adm, st, w, c)]
        if reason[r] in (oracle.HOLD_GLOBAL_CAP, oracle.HOLD_CLASS_CAP):
            assert not E
            room = any(prot_before[w].sum() + adm[w].sum() < caps["K_w"][w] for w in range(W))
            assert reason[r] == (oracle.HOLD_CLASS_CAP if room else oracle.HOLD_GLOBAL_CAP)
            continue
        assert reason[r] != oracle.HOLD_NO_ELIGIBLE and E
        cost = {w: int(backlog[w]) + int(L[r] - 16 * H[r, w]) * int(tokcost[w]) for w in E}
        best = min(E, key=lambda w: (cost[w], w))
        wh = int(np.argmax(H[r]))
        eq7 = (st[0] == 2 and H[r, wh] > 0 and wh not in E
               and hold + int(backlog[wh]) - int(backlog[best]) < 16 * int(H[r, wh]) * int(tokcost[wh]))
        if reason[r] == oracle.HOLD_PREFER_CACHE:
            assert eq7 and inst[r] == -1
            continue
        assert not eq7 and inst[r] == best
        if reason[r] == oracle.ADMIT_CONT:
            assert st == (1, best)
        else:
            assert reason[r] == oracle.ADMIT_NEW and st != (1, best)
            adm[best, c] += 1


@pytest.mark.parametrize("seed", list(range(40)))
def test_invariants_random_small(seed):
    rng = np.random.default_rng(seed)
    sc = wl.small_random(3000 + seed, W=int(rng.integers(1, 6)), cap=int(rng.integers(16, 128)),
                         n=int(rng.integers(1, 40)), mode=seed % 4,
                         n_warm=int(rng.integers(0, 5)))
    o = make_oracle(sc)
    for b, comp in scenario_steps(sc):
        prot_before = o.counts().copy()
        ids, st, ins, cl = o.sessions()
        sess_before = {int(i): (int(s), int(w)) for i, s, w in zip(ids, st, ins)}
        inst, reason, hit = o.route(b.cls, b.session, b.tok_off, b.tokens)
        _check_route_invariants(o, b, inst, reason, hit, prot_before, sess_before)
        _check_held_have_no_headroom(o, b, inst, reason, prot_before, sess_before)
        _check_serial_order(o, b, inst, reason, prot_before, sess_before, sc.backlog_q, sc.tokcost_q,
                            sc.hold_delay_q)
        if sc.mode == oracle.MODE_PLACEMENT_ONLY:
            assert np.all(inst >= 0)
        if sc.mode in (oracle.MODE_SESSION_ADMISSION, oracle.MODE_PLACEMENT_ONLY):
            assert not np.any(reason == oracle.HOLD_CLASS_CAP)
        o.commit()
        assert o.check_invariants() == 0
        if comp is not None:
            # release a few sessions (done=0) as well, so that Eq. (7) continuations occur
            o.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
            ids, st, ins, cl = o.sessions()
            if len(ids):
                pick = ids[rng.random(len(ids)) < 0.3]
                o.complete(pick, np.zeros(len(pick), np.uint8), np.zeros(len(pick), np.int32),
                           np.zeros(len(pick), np.int64), np.zeros(len(pick), np.uint8))
                assert o.check_invariants() == 0


def test_prefer_cache_rule_eq7():
    """A released continuation whose cached instance has no headroom waits when the
    saved prefill beats the hold delay plus the queue difference, else goes cold."""
    for hold, expect in ((0, oracle.HOLD_PREFER_CACHE), (10**12, oracle.ADMIT_NEW)):
        o = oracle.Oracle([4096, 4096], prior_kbar=(4000, 4000, 4000), hold_delay_q=hold,
                          protected_frac_q16=65536)
        o.set_instance_state([100, 100], [1000, 1000], [0, 0])
        # K_w = floor(4096/4000) = 1 on both instances
        rng = np.random.default_rng(4)
        p = rng.integers(0, wl.VOCAB, size=640, dtype=np.int32)
        b1 = wl.Batch(cls=np.array([2], np.uint8), session=np.array([77], np.uint64),
                      group=np.zeros(1, np.uint64), tok_off=np.array([0, 640]), tokens=p)
        inst, reason, _ = o.route(b1.cls, b1.session, b1.tok_off, b1.tokens)
        assert inst[0] == 0 and reason[0] == oracle.ADMIT_NEW
        o.commit()
        o.complete([77], [2], [0], [0], [0])              # released: must be admitted again
        # another session now fills instance 0's single slot
        b2 = _batch([0], [88], [16], seed=5)
        o.route(b2.cls, b2.session, b2.tok_off, b2.tokens)
        o.commit()
        inst, reason, hit = o.route(b1.cls, b1.session, b1.tok_off, b1.tokens)
        assert o.H()[0, 0] == 40 and hit[0] == (40 if expect == oracle.HOLD_PREFER_CACHE else 0)
        assert reason[0] == expect and (inst[0] == -1) == (expect == oracle.HOLD_PREFER_CACHE)


def test_rebound_moves_protection():
    o = oracle.Oracle([4096, 4096], prior_kbar=(8, 8, 8))
    o.set_instance_state([0, 10**9], [1, 1], [0, 0])
    b = _batch([1], [55], [64])
    inst, reason, _ = o.route(b.cls, b.session, b.tok_off, b.tokens)
    assert inst[0] == 0
    o.commit()
    # instance 0 becomes very slow: the continuation rebinds to instance 1 (it has headroom)
    o.set_instance_state([10**12, 0], [1, 1], [0, 0])
    inst, reason, _ = o.route(b.cls, b.session, b.tok_off, b.tokens)
    assert inst[0] == 1 and reason[0] == oracle.ADMIT_NEW
    o.commit()
    assert list(o.counts()[:, 1]) == [0, 1]
    assert o.check_invariants() == 0


def test_external_evict_and_reset():
    o = oracle.Oracle([4096])
    b = _batch([0], [9], [16 * 10])
    o.route(b.cls, b.session, b.tok_off, b.tokens)
    o.commit()
    keys = o.keys(100)
    assert o.index_size(0) == 10
    o.evict(0, keys[6:])                 # suffix-closed removal keeps the prefix property
    assert o.index_size(0) == 6 and o.check_invariants() == 0
    o.route(b.cls, b.session, b.tok_off, b.tokens)
    assert o.H()[0, 0] == 6
    o.evict(0, keys[2:3])                # removing a middle block breaks prefix closure
    assert o.check_invariants() == 2
    o.reset_instance(0)
    assert o.index_size(0) == 0 and o.check_invariants() == 0


def test_held_leaders_have_no_headroom_on_rlvr_heavy_config():
    """The RLVR-heavy workload (32 x 131,072 blocks, 16,384 requests): every leader held for
    a cap has no instance with headroom for it once the batch is decided, and the batch is
    decided in arrival order as the per-turn check describes."""
    sc = wl.config3()
    o = make_oracle(sc)
    for b, comp in sc.warm:
        o.route(b.cls, b.session, b.tok_off, b.tokens)
        o.commit()
        o.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
    prot_before = o.counts().astype(np.int64)
    ids, st, ins, cl = o.sessions()
    sess_before = {int(i): (int(s), int(w)) for i, s, w in zip(ids, st, ins)}
    b = sc.batch
    inst, reason, hit = o.route(b.cls, b.session, b.tok_off, b.tokens)
    _check_held_have_no_headroom(o, b, inst, reason, prot_before, sess_before)
    held = int(np.sum(np.isin(reason, (oracle.HOLD_GLOBAL_CAP, oracle.HOLD_CLASS_CAP))))
    assert held > 0 and int(np.sum(reason == oracle.ADMIT_NEW)) > 3000
