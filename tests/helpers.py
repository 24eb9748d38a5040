"""Test helpers: drive a synthetic scenario through the oracle, plus a
token-level brute-force model of the prefix index (no hashing at all)."""

from __future__ import annotations

import numpy as np

import oracle

ADMITS = (oracle.ADMIT_CONT, oracle.ADMIT_NEW, oracle.ADMIT_FOLLOW)
HOLDS = (oracle.HOLD_GLOBAL_CAP, oracle.HOLD_CLASS_CAP, oracle.HOLD_NO_ELIGIBLE,
         oracle.HOLD_PREFER_CACHE, oracle.HOLD_LEADER_HELD)


def make_oracle(sc, **over):
    kw = dict(protected_frac_q16=sc.protected_frac_q16, mode=sc.mode,
              hold_delay_q=sc.hold_delay_q, prior_kbar=sc.prior_kbar, prior_T_us=sc.prior_T_us)
    kw.update(over)
    o = oracle.Oracle(sc.cap_blocks, **kw)
    o.set_mixture(sc.rho_ppm)
    o.set_instance_state(sc.backlog_q, sc.tokcost_q, sc.contraction)
    return o


def load_fill(x, sc):
    """Load a scenario's resident fill (entries and prompt chains) into a router or an oracle."""
    for f in sc.fillers:
        x.load_entries(f.w, f.keys, f.metas)
    for c in sc.chains:
        x.load_chains(c.tok_off, c.tokens, c.inst, c.seq, c.arr, c.max_blocks)


def scenario_steps(sc):
    """Yield ("route", batch, completion_after) for the warm-up batches and the measured batch."""
    for b, c in sc.warm:
        yield b, c
    yield sc.batch, None


class BlockModel:
    """Brute-force prefix index: an entry is the token prefix itself (first 16(j+1) tokens),
    so hashing plays no part.  Same insert / eviction rules as the method's index."""

    def __init__(self, caps):
        self.caps = list(int(c) for c in caps)
        self.d = [dict() for _ in caps]

    @staticmethod
    def _prefixes(tokens):
        nb = len(tokens) // 16
        return [tokens[: 16 * (j + 1)].tobytes() for j in range(nb)]

    def H(self, batch):
        W = len(self.d)
        out = np.zeros((batch.n, W), np.uint16)
        for r in range(batch.n):
            t = batch.tokens[batch.tok_off[r]:batch.tok_off[r + 1]]
            pre = self._prefixes(t)
            for w in range(W):
                h = 0
                while h < len(pre) and pre[h] in self.d[w]:
                    h += 1
                out[r, w] = h
        return out

    def commit(self, seq, batch, inst):
        for r in range(batch.n):
            w = int(inst[r])
            if w < 0:
                continue
            t = batch.tokens[batch.tok_off[r]:batch.tok_off[r + 1]]
            for j, p in enumerate(self._prefixes(t)):
                m = (seq << 36) | (r << 16) | (65535 - j)
                self.d[w][p] = max(self.d[w].get(p, 0), m)
        for w in range(len(self.d)):
            d = self.d[w]
            if len(d) > self.caps[w]:
                order = sorted(d.items(), key=lambda kv: kv[1])
                metas = [m for _, m in order]
                assert len(set(metas)) == len(metas), "commit-only ticks are unique per entry"
                for p, _ in order[: len(d) - self.caps[w]]:
                    del d[p]

    def metas(self, w):
        return np.array(sorted(self.d[w].values()), dtype=np.uint64)

    def keys(self, w, seed=0x9E3779B97F4A7C15):
        ks = []
        for p in self.d[w]:
            t = np.frombuffer(p, dtype=np.int32)
            ks.append(int(oracle.hash_prompt(t, seed)[-1]))
        return np.array(sorted(ks), dtype=np.uint64)
