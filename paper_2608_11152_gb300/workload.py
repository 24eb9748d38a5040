"""Seeded synthetic mixed-rollout workloads (inputs only).

This module draws the inputs that both the CUDA path and the CPU oracle
consume: prompt token ids, workload classes, session and group ids, arrival
order, completion events, per-instance load figures and filler cache entries.
It contains none of the routing method's arithmetic (no hashing, no probing,
no caps, no scoring).

The paper's online trace (Table 2) is not available, so every batch is
synthetic, shaped after the workload descriptions of the paper:

* RLVR: short prompts fanned out to several samples that share the prompt
  (grouped rollouts), long lognormal decode tails (Table 1, Table 2).
* RLHF: medium prompts and responses.
* Agentic: multi-turn sessions whose prompt is the accumulated history plus the
  new turn's tool output and reply (Table 1); residency includes the tool gap
  (Table 3).

Lognormal sigmas come from Table 2's p95/p50 output ratios
(ln(p95/p50)/1.645): RLVR 0.61, RLHF 0.73, agentic 1.45.  Residency is decode
tokens x 25 ms per token, divided by 0.773 for agentic sessions (model-request
share of Table 3, Qwen3.6-35B-A3B row).

Five configurations follow the five benchmark workloads (tiny, medium mixed,
RLVR-heavy long tail, agentic-heavy long session, throughput stress sweep).
Every draw uses numpy's PCG64 generator, which gives identical streams on x86
and Arm hosts.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

VOCAB = 151936
BLOCK_TOKENS = 16
RLVR, RLHF, AGENTIC = 0, 1, 2
MS_PER_DECODE_TOKEN = 25
AGENT_MODEL_SHARE = 0.773  # Table 3: model request share of agent task time


def split_classes(n: int, rho_ppm) -> list[int]:
    """Largest-remainder split of n requests by the trainer mixture (ties to the lower class)."""
    exact = [n * r for r in rho_ppm]
    base = [e // 1_000_000 for e in exact]
    rem = [e % 1_000_000 for e in exact]
    left = n - sum(base)
    order = sorted(range(3), key=lambda b: (-rem[b], b))
    for b in order[:left]:
        base[b] += 1
    return base


def entry_meta(seq, arrival, depth):
    """Index entry metadata format of the library's load API: seq<<36 | arrival<<16 | (65535-depth)."""
    seq = np.asarray(seq, np.uint64)
    arrival = np.asarray(arrival, np.uint64)
    depth = np.asarray(depth, np.uint64)
    return (seq << np.uint64(36)) | (arrival << np.uint64(16)) | (np.uint64(65535) - depth)


@dataclass
class Batch:
    cls: np.ndarray        # uint8 [n]
    session: np.ndarray    # uint64 [n], never 0
    group: np.ndarray      # uint64 [n], prompt group id (0 = none)
    tok_off: np.ndarray    # int64 [n+1]
    tokens: np.ndarray     # int32 [n_tokens]

    @property
    def n(self) -> int:
        return int(len(self.cls))

    @property
    def n_tokens(self) -> int:
        return int(self.tok_off[-1])


@dataclass
class DeltaBatch:
    """A batch whose prompts extend earlier prompts of the batch (the host layout of
    misat_stage_host_delta): prompt(r) = prompt(base[r]) ++ delta_tokens[delta_off[r]:delta_off[r+1]]."""
    cls: np.ndarray           # uint8 [n]
    session: np.ndarray       # uint64 [n]
    base: np.ndarray          # int32 [n], -1 or an earlier request
    delta_off: np.ndarray     # int64 [n+1]
    delta_tokens: np.ndarray  # int32

    @property
    def n(self) -> int:
        return int(len(self.cls))


DELTA_MAX_DEPTH = 64


def encode_delta(b: Batch) -> DeltaBatch:
    """Delta layout of a batch: a request's base is the latest earlier request of its session,
    else the first earlier request of its prompt group, whose whole prompt starts its own
    (checked token by token); chains stay within DELTA_MAX_DEPTH."""
    n = b.n
    base = np.full(n, -1, np.int32)
    depth = np.zeros(n, np.int32)
    last_of_session = {}
    first_of_group = {}
    parts, off = [], np.zeros(n + 1, np.int64)
    for r in range(n):
        t = b.tokens[b.tok_off[r]:b.tok_off[r + 1]]
        cands = []
        s = int(b.session[r])
        if s in last_of_session:
            cands.append(last_of_session[s])
        g = int(b.group[r]) if b.group is not None else 0
        if g and g in first_of_group:
            cands.append(first_of_group[g])
        for c in cands:
            pt = b.tokens[b.tok_off[c]:b.tok_off[c + 1]]
            if len(pt) <= len(t) and depth[c] < DELTA_MAX_DEPTH and np.array_equal(pt, t[:len(pt)]):
                base[r] = c
                depth[r] = depth[c] + 1
                t = t[len(pt):]
                break
        else:
            depth[r] = 1
        parts.append(t)
        off[r + 1] = off[r] + len(t)
        last_of_session[s] = r
        if g and g not in first_of_group:
            first_of_group[g] = r
    tok = np.concatenate(parts).astype(np.int32) if parts else np.zeros(0, np.int32)
    return DeltaBatch(cls=b.cls.copy(), session=b.session.copy(), base=base, delta_off=off, delta_tokens=tok)


def decode_delta(d: DeltaBatch) -> tuple:
    """(tok_off, tokens) of the full batch a delta layout describes."""
    n = d.n
    full = []
    off = np.zeros(n + 1, np.int64)
    for r in range(n):
        own = d.delta_tokens[d.delta_off[r]:d.delta_off[r + 1]]
        t = np.concatenate([full[d.base[r]], own]) if d.base[r] >= 0 else own
        full.append(t)
        off[r + 1] = off[r] + len(t)
    tok = np.concatenate(full).astype(np.int32) if full else np.zeros(0, np.int32)
    return off, tok


@dataclass
class Completion:
    session: np.ndarray       # uint64
    cls: np.ndarray           # uint8
    total_blocks: np.ndarray  # int32
    residency_us: np.ndarray  # int64
    done: np.ndarray          # uint8


@dataclass
class Filler:
    """Resident cache entries loaded before the first batch (prefix-closed: depth 0 only)."""
    w: int
    keys: np.ndarray   # uint64, >= 2, distinct
    metas: np.ndarray  # uint64


@dataclass
class ChainBatch:
    """Prompt chains resident before the first batch, in the layout of the load_chains call:
    chain c is tokens[tok_off[c]:tok_off[c+1]]; its first max_blocks[c] full blocks are
    resident on instance inst[c] with the tick (seq[c], arr[c]) -- whole prefixes with one
    tick, so depth orders their eviction."""
    tok_off: np.ndarray     # int64 [m+1]
    tokens: np.ndarray      # int32
    inst: np.ndarray        # int32 [m]
    seq: np.ndarray         # uint64 [m]
    arr: np.ndarray         # uint32 [m]
    max_blocks: np.ndarray  # int32 [m]


@dataclass
class MixSpec:
    rho_ppm: tuple
    rlvr_prompt: tuple
    rlvr_fanout: int
    rlvr_decode_median: int
    rlvr_decode_cap: int
    rlhf_prompt: tuple
    rlhf_decode: tuple            # ("lognormal", median, cap) or ("uniform", lo, hi)
    agent_initial: tuple
    agent_append: tuple
    agent_max_turns: tuple
    agent_hist_cap: int
    agent_sessions: int           # sessions contributing turns to each batch
    agent_decode_median: int = 256
    agent_decode_cap: int = 8192


@dataclass
class Scenario:
    name: str
    W: int
    cap_blocks: np.ndarray
    rho_ppm: tuple
    prior_kbar: tuple
    prior_T_us: int
    backlog_q: np.ndarray
    tokcost_q: np.ndarray
    contraction: np.ndarray
    hold_delay_q: int
    protected_frac_q16: int = 58982   # C_w = 0.9 Cap_w
    mode: int = 0
    fillers: list = field(default_factory=list)  # list of Filler (loaded entries)
    chains: list = field(default_factory=list)   # list of ChainBatch (loaded prompt chains)
    warm: list = field(default_factory=list)   # list of (Batch, Completion)
    batch: Batch | None = None
    batch_completion: Completion | None = None  # completion events of the measured batch's sessions
    batch_delta: DeltaBatch | None = None       # the measured batch in the delta layout
    stream: object = None                       # generator of the batches after the measured one
    max_tokens: int = 0
    max_batch: int = 0


class _AgentSession:
    """Session history kept in one growing buffer; each turn's prompt is a prefix view."""
    __slots__ = ("sid", "buf", "plen", "turn", "max_turns", "decode_sum", "last_decode")

    def __init__(self, sid, first, max_turns, capacity):
        self.sid = sid
        self.buf = np.empty(max(capacity, len(first)), dtype=np.int32)
        self.buf[: len(first)] = first
        self.plen = len(first)
        self.turn = 0
        self.max_turns = max_turns
        self.decode_sum = 0
        self.last_decode = 0

    @property
    def prompt(self):
        return self.buf[: self.plen]

    def append(self, toks):
        self.buf[self.plen: self.plen + len(toks)] = toks
        self.plen += len(toks)


class MixedStream:
    """A stream of mixed batches sharing one agentic session pool."""

    def __init__(self, spec: MixSpec, seed: int, sid_base: int):
        self.spec = spec
        self.rng = np.random.default_rng(seed)
        self.next_sid = sid_base
        self.next_group = sid_base
        self.pool: list[_AgentSession] = []

    def _sid(self):
        self.next_sid += 1
        return self.next_sid

    def _tokens(self, n):
        return self.rng.integers(0, VOCAB, size=int(n), dtype=np.int32)

    def _lognormal(self, median, sigma, cap):
        v = int(round(median * math.exp(sigma * self.rng.standard_normal())))
        return max(1, min(cap, v))

    def seed_sessions(self, histories):
        """Put agentic sessions with the given histories (token arrays) at the front of the pool:
        they continue with their next turn, which appends to the history."""
        s = self.spec
        seeded = []
        for h in histories:
            mt = int(self.rng.integers(max(2, s.agent_max_turns[0]), s.agent_max_turns[1] + 1))
            a = _AgentSession(self._sid(), h, mt, max(len(h), s.agent_hist_cap) + s.agent_append[1])
            a.turn = 1
            seeded.append(a)
        self.pool = seeded + self.pool

    def _new_agent(self):
        s = self.spec
        L0 = int(self.rng.integers(s.agent_initial[0], s.agent_initial[1] + 1))
        mt = int(self.rng.integers(s.agent_max_turns[0], s.agent_max_turns[1] + 1))
        return _AgentSession(self._sid(), self._tokens(L0), mt, s.agent_hist_cap + s.agent_append[1])

    def next_batch(self, n: int, delta: bool = False):
        """The next batch of n requests and the completion events of its sessions; with
        delta=True also the batch in the delta layout, built from what the generator knows
        (an agentic turn extends its session's previous turn in the batch, a fan-out sample
        its group's first sample) without comparing tokens."""
        s = self.spec
        rng = self.rng
        n_rlvr, n_rlhf, n_agent = split_classes(n, s.rho_ppm)
        reqs = []  # (cls, session, group, tokens, agent_key)
        comp = []  # (session, cls, total_blocks, residency_us)
        # RLVR: groups of fan-out samples sharing one prompt, one session per sample
        left = n_rlvr
        while left > 0:
            f = min(s.rlvr_fanout, left)
            self.next_group += 1
            g = self.next_group
            p = self._tokens(rng.integers(s.rlvr_prompt[0], s.rlvr_prompt[1] + 1))
            for _ in range(f):
                sid = self._sid()
                reqs.append((RLVR, sid, g, p, None))
                dec = self._lognormal(s.rlvr_decode_median, 0.61, s.rlvr_decode_cap)
                comp.append((sid, RLVR, -(-(len(p) + dec) // BLOCK_TOKENS), dec * MS_PER_DECODE_TOKEN * 1000))
            left -= f
        # RLHF: independent prompts
        for _ in range(n_rlhf):
            sid = self._sid()
            p = self._tokens(rng.integers(s.rlhf_prompt[0], s.rlhf_prompt[1] + 1))
            reqs.append((RLHF, sid, 0, p, None))
            if s.rlhf_decode[0] == "lognormal":
                dec = self._lognormal(s.rlhf_decode[1], 0.73, s.rlhf_decode[2])
            else:
                dec = int(rng.integers(s.rlhf_decode[1], s.rlhf_decode[2] + 1))
            comp.append((sid, RLHF, -(-(len(p) + dec) // BLOCK_TOKENS), dec * MS_PER_DECODE_TOKEN * 1000))
        # Agentic: turns of pool sessions; a session's turns keep their order
        if n_agent > 0:
            n_sess = max(1, min(s.agent_sessions, n_agent))
            while len(self.pool) < n_sess:
                self.pool.append(self._new_agent())
            active = self.pool[:n_sess]
            base, extra = divmod(n_agent, n_sess)
            ended = []
            for i, a in enumerate(active):
                k = base + (1 if i < extra else 0)
                for t in range(k):
                    if a.turn > 0:
                        a.append(self._tokens(rng.integers(s.agent_append[0], s.agent_append[1] + 1)))
                    a.turn += 1
                    dec = self._lognormal(s.agent_decode_median, 1.45, s.agent_decode_cap)
                    a.decode_sum += dec
                    a.last_decode = dec
                    reqs.append((AGENTIC, a.sid, 0, a.prompt, (a.sid, t)))
                    if a.turn >= a.max_turns or len(a.prompt) + s.agent_append[1] >= s.agent_hist_cap:
                        # the session ends after this turn; later turns of this batch restart it
                        if t < k - 1:
                            ended.append(a)
                            a = self._new_agent()
                            active[i] = a
                if a.turn >= a.max_turns or len(a.prompt) + s.agent_append[1] >= s.agent_hist_cap:
                    ended.append(a)
                    active[i] = None
            for a in ended:
                res = int(round(a.decode_sum * MS_PER_DECODE_TOKEN * 1000 / AGENT_MODEL_SHARE))
                comp.append((a.sid, AGENTIC, -(-(len(a.prompt) + a.last_decode) // BLOCK_TOKENS), res))
            self.pool = [a for a in active if a is not None] + self.pool[n_sess:]
        # arrival order: random permutation, each session's turns kept in turn order
        perm = rng.permutation(len(reqs))
        order = np.empty(len(reqs), dtype=np.int64)
        order[perm] = np.arange(len(reqs))  # order[i] = arrival slot of request i
        by_sess: dict[int, list[int]] = {}
        for i, r in enumerate(reqs):
            if r[4] is not None:
                by_sess.setdefault(r[1], []).append(i)
        for idx in by_sess.values():
            if len(idx) > 1:
                slots = sorted(order[j] for j in idx)
                for j, sl in zip(idx, slots):
                    order[j] = sl
        arrival = np.empty(len(reqs), dtype=np.int64)
        arrival[order] = np.arange(len(reqs))
        reqs = [reqs[i] for i in arrival]
        lens = np.array([len(r[3]) for r in reqs], dtype=np.int64)
        tok_off = np.zeros(len(reqs) + 1, dtype=np.int64)
        np.cumsum(lens, out=tok_off[1:])
        tokens = np.concatenate([r[3] for r in reqs]) if reqs else np.zeros(0, np.int32)
        batch = Batch(
            cls=np.array([r[0] for r in reqs], dtype=np.uint8),
            session=np.array([r[1] for r in reqs], dtype=np.uint64),
            group=np.array([r[2] for r in reqs], dtype=np.uint64),
            tok_off=tok_off,
            tokens=np.ascontiguousarray(tokens, dtype=np.int32),
        )
        completion = Completion(
            session=np.array([c[0] for c in comp], dtype=np.uint64),
            cls=np.array([c[1] for c in comp], dtype=np.uint8),
            total_blocks=np.array([c[2] for c in comp], dtype=np.int32),
            residency_us=np.array([c[3] for c in comp], dtype=np.int64),
            done=np.ones(len(comp), dtype=np.uint8),
        )
        if not delta:
            return batch, completion
        return batch, completion, _structural_delta(reqs, batch)


def _structural_delta(reqs, batch: Batch) -> DeltaBatch:
    """Delta layout of a generated batch from its structure: the base of a request is the
    latest earlier request of its session (agentic turns), else the first earlier request of
    its prompt group (fan-out samples), chains at most DELTA_MAX_DEPTH long."""
    n = len(reqs)
    base = np.full(n, -1, np.int32)
    depth = np.zeros(n, np.int32)
    last_of_session, first_of_group = {}, {}
    lens = np.diff(batch.tok_off)
    parts, off = [], np.zeros(n + 1, np.int64)
    for r, (c, sid, g, prompt, akey) in enumerate(reqs):
        b = -1
        if akey is not None and sid in last_of_session:
            b = last_of_session[sid]
        elif g and g in first_of_group:
            b = first_of_group[g]
        if b >= 0 and depth[b] < DELTA_MAX_DEPTH:
            base[r] = b
            depth[r] = depth[b] + 1
            own = prompt[int(lens[b]):]
        else:
            depth[r] = 1
            own = prompt
        parts.append(own)
        off[r + 1] = off[r] + len(own)
        if akey is not None:
            last_of_session[sid] = r
        if g and g not in first_of_group:
            first_of_group[g] = r
    tok = np.concatenate(parts).astype(np.int32) if parts else np.zeros(0, np.int32)
    return DeltaBatch(cls=batch.cls.copy(), session=batch.session.copy(), base=base, delta_off=off,
                      delta_tokens=tok)


def _prior_kbar(spec: MixSpec) -> tuple:
    """Class footprint priors: (median prompt + median decode) / 16, rounded up."""
    rlvr = (spec.rlvr_prompt[0] + spec.rlvr_prompt[1]) // 2 + spec.rlvr_decode_median
    if spec.rlhf_decode[0] == "lognormal":
        rlhf_dec = spec.rlhf_decode[1]
    else:
        rlhf_dec = (spec.rlhf_decode[1] + spec.rlhf_decode[2]) // 2
    rlhf = (spec.rlhf_prompt[0] + spec.rlhf_prompt[1]) // 2 + rlhf_dec
    agent = (spec.agent_initial[0] + spec.agent_initial[1]) // 2 + spec.agent_decode_median
    return tuple(-(-x // BLOCK_TOKENS) for x in (rlvr, rlhf, agent))


def _instance_state(rng, W):
    backlog = rng.integers(0, 20_000_000, size=W, dtype=np.int64)      # ns of queued prefill
    tokcost = rng.integers(20_000, 40_001, size=W, dtype=np.int64)     # ns per prompt token (1/mu_w)
    return backlog, tokcost, np.zeros(W, dtype=np.int32)


MIX2 = dict(rlvr_prompt=(64, 1024), rlvr_fanout=8, rlvr_decode_median=4096, rlvr_decode_cap=32768,
            rlhf_prompt=(512, 2048), rlhf_decode=("uniform", 256, 2048),
            agent_initial=(1000, 4000), agent_append=(200, 1500), agent_max_turns=(5, 20),
            agent_hist_cap=32768)


CHAIN_BLOCKS = (32, 1024)   # blocks per fill chain, uniform (512 to 16,384 tokens)
CHAIN_TOKENS_PER_LOAD = 1 << 25   # tokens per ChainBatch (the load call's staging limit)
CHAIN_PER_LOAD = 16384            # chains per ChainBatch


def _chain_fill(rng, W, cap, fill, n_sessions):
    """Resident prompt chains filling every instance to `fill` of its capacity: chains of
    CHAIN_BLOCKS random-token blocks, each older than any commit (seq 0, its own arrival
    tick).  The first n_sessions chains are also returned as the histories of agentic sessions
    that continue later; those are resident only 60-90% deep (uniform per chain)."""
    target = int(fill * cap)
    lens, insts = [], []
    for w in range(W):
        left = target
        while left > 0:
            k = min(left, int(rng.integers(CHAIN_BLOCKS[0], CHAIN_BLOCKS[1] + 1)))
            lens.append(k)
            insts.append(w)
            left -= k
    m = len(lens)
    perm = rng.permutation(m)  # the session histories come from every instance
    lens = np.array(lens, np.int64)[perm]
    insts = np.array(insts, np.int32)[perm]
    maxb = lens.astype(np.int32).copy()
    ns = min(n_sessions, m)
    maxb[:ns] = np.maximum(1, (lens[:ns] * rng.uniform(0.6, 0.9, size=ns)).astype(np.int32))
    arr = rng.integers(0, 1 << 20, size=m, dtype=np.int64).astype(np.uint32)
    tok_len = 16 * lens
    batches, histories = [], []
    c0 = 0
    while c0 < m:
        c1 = c0
        t = 0
        while c1 < m and c1 - c0 < CHAIN_PER_LOAD and (t + tok_len[c1] <= CHAIN_TOKENS_PER_LOAD or c1 == c0):
            t += tok_len[c1]
            c1 += 1
        off = np.zeros(c1 - c0 + 1, np.int64)
        np.cumsum(tok_len[c0:c1], out=off[1:])
        toks = rng.integers(0, VOCAB, size=int(off[-1]), dtype=np.int32)
        batches.append(ChainBatch(tok_off=off, tokens=toks, inst=insts[c0:c1].copy(),
                                  seq=np.zeros(c1 - c0, np.uint64), arr=arr[c0:c1].copy(),
                                  max_blocks=maxb[c0:c1].copy()))
        for c in range(c0, min(c1, ns)):
            histories.append(toks[off[c - c0]:off[c - c0 + 1]].copy())
        c0 = c1
    return batches, histories


def _stream_scenario(name, seed, W, cap, n, n_warm, spec: MixSpec, fill=0.0, chain_fill=False):
    rng = np.random.default_rng(seed + 7)
    backlog, tokcost, contraction = _instance_state(rng, W)
    sc = Scenario(name=name, W=W, cap_blocks=np.full(W, cap, dtype=np.int64), rho_ppm=spec.rho_ppm,
                  prior_kbar=_prior_kbar(spec), prior_T_us=30_000_000, backlog_q=backlog,
                  tokcost_q=tokcost, contraction=contraction, hold_delay_q=50_000_000)
    histories = []
    if fill > 0 and chain_fill:
        n_hist = max(1, spec.agent_sessions // 4)
        sc.chains, histories = _chain_fill(rng, W, cap, fill, n_hist)
    elif fill > 0:
        nf = int(fill * cap)
        for w in range(W):
            # full 64-bit keys (like block hashes), 0 and 1 excluded
            keys = rng.integers(2, np.iinfo(np.uint64).max, size=nf + 64, dtype=np.uint64, endpoint=True)
            srt = np.sort(keys)
            dup = np.zeros(len(keys), bool)
            dup[1:] = srt[1:] == srt[:-1]
            if dup.any():  # keep distinct keys only (2^-64 collisions: practically never)
                keys = np.array(sorted(set(keys.tolist())), dtype=np.uint64)
                rng.shuffle(keys)
            keys = keys[:nf]
            arr = rng.integers(0, 1 << 20, size=len(keys), dtype=np.int64)
            sc.fillers.append(Filler(w=w, keys=keys, metas=entry_meta(0, arr, 0)))
    stream = MixedStream(spec, seed, sid_base=(seed % 4096) << 40)
    for _ in range(n_warm):
        sc.warm.append(stream.next_batch(n))
    if histories:
        # agentic sessions whose history is (60-90% deep) resident on some instance continue in
        # the measured batch; the router has not seen them (they are new sessions to it)
        stream.seed_sessions(histories)
    sc.batch, sc.batch_completion, sc.batch_delta = stream.next_batch(n, delta=True)
    sc.stream = stream   # continues with the batches after the measured one
    sc.max_batch = max([b.n for b, _ in sc.warm] + [sc.batch.n] + [len(c.inst) for c in sc.chains])
    sc.max_tokens = max([b.n_tokens for b, _ in sc.warm] + [sc.batch.n_tokens] + [int(c.tok_off[-1]) for c in sc.chains])
    return sc


def config1(seed=20260001) -> Scenario:
    """Tiny batch: 4 x 2,048 blocks, 64 requests (32 RLVR / 16 RLHF / 16 agentic), 256 warm-up requests."""
    spec = MixSpec(rho_ppm=(500000, 250000, 250000), rlvr_prompt=(128, 512), rlvr_fanout=4,
                   rlvr_decode_median=2048, rlvr_decode_cap=8192, rlhf_prompt=(512, 1024),
                   rlhf_decode=("lognormal", 512, 8192), agent_initial=(1024, 4096),
                   agent_append=(100, 400), agent_max_turns=(4, 16), agent_hist_cap=8192,
                   agent_sessions=4)
    return _stream_scenario("cfg1_tiny_4x2048_n64", seed, 4, 2048, 64, 4, spec)


def config2(seed=20260002) -> Scenario:
    """Medium mixed: 16 x 65,536 blocks, 4,096 requests 40/30/30, 16,384 warm-up requests."""
    spec = MixSpec(rho_ppm=(400000, 300000, 300000), agent_sessions=256, **MIX2)
    return _stream_scenario("cfg2_medium_16x65536_n4096", seed, 16, 65536, 4096, 4, spec)


def config3(seed=20260003) -> Scenario:
    """RLVR-heavy long tail: 32 x 131,072 blocks, 16,384 requests 70/15/15, fan-out 16."""
    mix = dict(MIX2)
    mix.update(rlvr_prompt=(64, 512), rlvr_fanout=16, rlvr_decode_median=8192, rlvr_decode_cap=65536)
    spec = MixSpec(rho_ppm=(700000, 150000, 150000), agent_sessions=512, **mix)
    return _stream_scenario("cfg3_rlvr_heavy_32x131072_n16384", seed, 32, 131072, 16384, 2, spec)


def config4(seed=20260004) -> Scenario:
    """Agentic-heavy long sessions: 64 x 262,144 blocks, 1,024 sessions at turns 1-40 (histories up to
    128K tokens, 60-90% resident from a warm-up) mixed with 8,192 RLVR/RLHF requests."""
    rng = np.random.default_rng(seed)
    W, cap = 64, 262144
    spec2 = MixSpec(rho_ppm=(500000, 500000, 0), agent_sessions=1, **MIX2)
    stream = MixedStream(spec2, seed, sid_base=(seed % 4096) << 40)
    backlog, tokcost, contraction = _instance_state(np.random.default_rng(seed + 7), W)
    mix_for_prior = MixSpec(rho_ppm=(200000, 200000, 600000), agent_sessions=1024,
                            **{**MIX2, "agent_initial": (200, 2000), "agent_append": (200, 2000),
                               "agent_max_turns": (1, 40), "agent_hist_cap": 131072})
    sc = Scenario(name="cfg4_agentic_64x262144_n9216", W=W, cap_blocks=np.full(W, cap, dtype=np.int64),
                  rho_ppm=(200000, 200000, 600000), prior_kbar=_prior_kbar(mix_for_prior),
                  prior_T_us=30_000_000, backlog_q=backlog, tokcost_q=tokcost,
                  contraction=contraction, hold_delay_q=50_000_000)
    sid0 = ((seed % 4096) << 40) | (1 << 39)
    hist, cur = [], []
    for i in range(1024):
        turn = int(rng.integers(1, 41))
        parts = [rng.integers(0, VOCAB, size=int(rng.integers(200, 2001)), dtype=np.int32)]
        for _ in range(turn - 1):
            if sum(len(p) for p in parts) + 2000 >= 131072:
                break
            parts.append(rng.integers(0, VOCAB, size=int(rng.integers(200, 2001)), dtype=np.int32))
        h = np.concatenate(parts)
        hist.append(h)
        cur.append(turn)
    # warm-up: each continuing session's earlier turn covered 60-90% of its current history
    def agent_batch(prompts, sids):
        lens = np.array([len(p) for p in prompts], dtype=np.int64)
        off = np.zeros(len(prompts) + 1, dtype=np.int64)
        np.cumsum(lens, out=off[1:])
        return Batch(cls=np.full(len(prompts), AGENTIC, np.uint8), session=np.array(sids, np.uint64),
                     group=np.zeros(len(prompts), np.uint64), tok_off=off,
                     tokens=np.concatenate(prompts) if prompts else np.zeros(0, np.int32))

    warm_p, warm_s = [], []
    for i in range(1024):
        if cur[i] > 1:
            f = rng.uniform(0.6, 0.9)
            warm_p.append(hist[i][: int(f * len(hist[i]))])
            warm_s.append(sid0 + i + 1)
    b_warm_rl, c_warm_rl = stream.next_batch(8192)
    sc.warm.append((_concat_batches([agent_batch(warm_p, warm_s), b_warm_rl], rng), c_warm_rl))
    # measured batch: one current turn per session (history + new turn) and fresh RLVR/RLHF
    turn_p = [np.concatenate([hist[i], rng.integers(0, VOCAB, size=int(rng.integers(200, 2001)), dtype=np.int32)])
              for i in range(1024)]
    b_rl, _ = stream.next_batch(8192)
    sc.batch = _concat_batches([agent_batch(turn_p, [sid0 + i + 1 for i in range(1024)]), b_rl], rng)
    sc.max_batch = max(b.n for b in [sc.warm[0][0], sc.batch])
    sc.max_tokens = max(b.n_tokens for b in [sc.warm[0][0], sc.batch])
    return sc


def _concat_batches(batches, rng):
    """Concatenate batches and interleave their requests in a random arrival order."""
    n = sum(b.n for b in batches)
    prompts, cls, ses, grp = [], [], [], []
    for b in batches:
        for r in range(b.n):
            prompts.append(b.tokens[b.tok_off[r]:b.tok_off[r + 1]])
        cls.append(b.cls)
        ses.append(b.session)
        grp.append(b.group)
    cls, ses, grp = np.concatenate(cls), np.concatenate(ses), np.concatenate(grp)
    perm = rng.permutation(n)
    # keep each session's requests in their original relative order
    pos = {}
    for i in range(n):
        pos.setdefault(int(ses[i]), []).append(i)
    slot = np.empty(n, dtype=np.int64)
    slot[perm] = np.arange(n)
    for idx in pos.values():
        if len(idx) > 1:
            s = sorted(slot[j] for j in idx)
            for j, sl in zip(idx, s):
                slot[j] = sl
    order = np.empty(n, dtype=np.int64)
    order[slot] = np.arange(n)
    lens = np.array([len(prompts[i]) for i in order], dtype=np.int64)
    off = np.zeros(n + 1, dtype=np.int64)
    np.cumsum(lens, out=off[1:])
    return Batch(cls=cls[order], session=ses[order], group=grp[order], tok_off=off,
                 tokens=np.ascontiguousarray(np.concatenate([prompts[i] for i in order]), dtype=np.int32))


def config5(n=65536, fill=0.95, seed=20260005, n_warm=1, instances=128, cap=262144) -> Scenario:
    """Throughput stress: 128 x 262,144 blocks filled to `fill` with resident prompt chains (a
    quarter of the batch's agentic sessions continue histories that are 60-90% resident),
    batches of n requests 40/30/30 (fewer instances only for small profiling captures)."""
    spec = MixSpec(rho_ppm=(400000, 300000, 300000), agent_sessions=max(1, round(0.3 * n / 4.8)), **MIX2)
    return _stream_scenario(f"cfg5_stress_{instances}x{cap}_n{n}_fill{int(fill * 100)}", seed, instances, cap, n,
                            n_warm, spec, fill=fill, chain_fill=True)


def small_random(seed, W=3, cap=64, n=24, mode=0, n_warm=2) -> Scenario:
    """Tiny randomized scenario (small W and capacity so caps and eviction bind often)."""
    rng = np.random.default_rng(seed)
    spec = MixSpec(rho_ppm=(400000, 300000, 300000), rlvr_prompt=(8, 96), rlvr_fanout=int(rng.integers(1, 5)),
                   rlvr_decode_median=64, rlvr_decode_cap=512, rlhf_prompt=(16, 128),
                   rlhf_decode=("uniform", 16, 256), agent_initial=(32, 160), agent_append=(8, 48),
                   agent_max_turns=(2, 6), agent_hist_cap=512, agent_sessions=int(rng.integers(1, 4)))
    sc = _stream_scenario(f"small_{seed}", seed, W, cap, n, n_warm, spec)
    sc.cap_blocks = rng.integers(max(4, cap // 4), cap + 1, size=W).astype(np.int64)
    sc.mode = mode
    sc.hold_delay_q = int(rng.integers(0, 2_000_000))
    sc.backlog_q = rng.integers(0, 2_000_000, size=W, dtype=np.int64)
    sc.tokcost_q = rng.integers(0, 40_000, size=W, dtype=np.int64)
    sc.contraction = rng.integers(0, 3, size=W, dtype=np.int32)
    return sc


CONFIGS = {1: config1, 2: config2, 3: config3, 4: config4, 5: config5}
