"""Oracle of the host-side admission controllers -- TEST INFRASTRUCTURE.

Only ``tests/`` imports this module.  Plain Python integers, one loop per window and
instance, written from the paper's description (Sec. 4.1): the operational cap stays below
its base; a confirmed decline of the prefix-cache hit rate relative to recent healthy
windows, G_w = max(0, h*_w - h_w), with confirmation and slope checks, or a persistent
waiting queue contracts it temporarily, and it recovers gradually; for grouped rollouts
the recheck delay of a held request falls as more siblings of its prompt group are
visible.  The paper prints no thresholds, window lengths or step sizes: the ones below
are the library's configuration (its defaults are the same numbers), not the paper's.

Parity pins (tests/test_overload.py): steady health never contracts; a single-window dip
(transient) never contracts; a sustained drop contracts after exactly `confirm` windows by
the stated step; a drop that is already recovering (rising slope) does not contract;
recovery is one session per `recover_after` quiet windows down to zero; the contraction
never passes max_contraction_pct of the base cap; a queue signal alone contracts by
k_base/8; recheck delays reduce to base/v for v visible siblings.
"""

from __future__ import annotations

PPM = 1_000_000

DEFAULTS = dict(ref_windows=8, min_ref=3, gap_ppm=100_000, confirm=2, queue_thresh=64, recover_after=2,
                max_contraction_pct=50)


class OverloadOracle:
    def __init__(self, n_instances, **cfg):
        self.cfg = dict(DEFAULTS)
        self.cfg.update(cfg)
        self.W = n_instances
        self.ref = [[] for _ in range(n_instances)]      # healthy hit rates, oldest first
        self.prev = [None] * n_instances                   # previous observed hit rate
        self.sig_run = [0] * n_instances
        self.ok_run = [0] * n_instances
        self.contraction = [0] * n_instances

    def observe(self, hit, query, waiting, k_base):
        c = self.cfg
        out = []
        for w in range(self.W):
            # observed hit rate of the window, in parts per million
            h = (hit[w] * PPM) // query[w] if query[w] > 0 else None
            # the reference: best hit rate among the recent healthy windows
            href = max(self.ref[w]) if len(self.ref[w]) >= c["min_ref"] else None
            gap = max(0, href - h) if (h is not None and href is not None) else 0
            rising = self.prev[w] is not None and h is not None and h > self.prev[w]
            hit_signal = gap > c["gap_ppm"] and not rising
            queue_signal = waiting[w] > c["queue_thresh"]
            signal = hit_signal or queue_signal
            if signal:
                self.sig_run[w] += 1
                self.ok_run[w] = 0
            else:
                self.sig_run[w] = 0
                self.ok_run[w] += 1
            if signal and self.sig_run[w] >= c["confirm"]:
                steps = []
                if hit_signal:
                    steps.append(max(1, (k_base[w] * gap) // PPM))
                if queue_signal:
                    steps.append(max(1, k_base[w] // 8))
                self.contraction[w] += max(steps)
            elif not signal and self.ok_run[w] >= c["recover_after"] and self.contraction[w] > 0:
                self.contraction[w] -= 1
                self.ok_run[w] = 0
            limit = (k_base[w] * c["max_contraction_pct"]) // 100
            self.contraction[w] = min(max(self.contraction[w], 0), limit)
            if h is not None and gap <= c["gap_ppm"] and not queue_signal:
                self.ref[w].append(h)
                if len(self.ref[w]) > c["ref_windows"]:
                    self.ref[w].pop(0)
            if h is not None:
                self.prev[w] = h
            out.append(self.contraction[w])
        return out


def recheck_delays(group, held, base_delay_us, min_delay_us):
    """Delay before a held request is evaluated again: base / (visible siblings of its group)."""
    visible = {}
    for g in group:
        if g != 0:
            visible[g] = visible.get(g, 0) + 1
    out = []
    for g, h in zip(group, held):
        if not h:
            out.append(0)
        elif g == 0:
            out.append(base_delay_us)
        else:
            out.append(max(min_delay_us, base_delay_us // visible[g]))
    return out
