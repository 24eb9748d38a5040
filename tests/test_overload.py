"""Host-side admission controllers (Sec. 4.1): overload pressure and grouped-rollout recheck
delays.  The oracle (oracle/overload.py) is pinned by hand-worked cases of its stated rules;
the library (misat_overload_*, misat_recheck_delays, no GPU needed) must then agree with it
exactly on random window sequences."""

import numpy as np
import pytest

from oracle import overload as ovo
from paper_2608_11152_gb300 import misat

PPM = 1_000_000


def _run(oracle, seq):
    return [oracle.observe(*win) for win in seq]


def _win(rate_ppm, waiting=0, k_base=100, query=1_000_000):
    """One instance's window: hit tokens for a hit rate (ppm) out of `query` tokens."""
    return ([rate_ppm * query // PPM], [query], [waiting], [k_base])


# ---- pins of the oracle -------------------------------------------------------------------

def test_steady_health_never_contracts():
    o = ovo.OverloadOracle(1)
    assert all(c == [0] for c in _run(o, [_win(900_000)] * 30))


def test_single_window_dip_is_filtered_by_confirmation():
    o = ovo.OverloadOracle(1)
    seq = [_win(900_000)] * 5 + [_win(500_000)] + [_win(900_000)] * 5
    assert all(c == [0] for c in _run(o, seq))


def test_sustained_drop_contracts_after_confirmation_then_recovers_gradually():
    o = ovo.OverloadOracle(1)
    out = _run(o, [_win(900_000)] * 5)
    assert out[-1] == [0]
    # gap 400,000 ppm on k_base 100: step 40 from the second signalling window, capped at 50
    drop = _run(o, [_win(500_000)] * 4)
    assert [c[0] for c in drop] == [0, 40, 50, 50]
    # healthy again (gap 0 against the 900,000 reference): one session every 2 windows
    rec = [c[0] for c in _run(o, [_win(900_000)] * 8)]
    assert rec == [50, 49, 49, 48, 48, 47, 47, 46]


def test_a_drop_that_is_already_recovering_does_not_contract():
    o = ovo.OverloadOracle(1)
    seq = [_win(900_000)] * 5 + [_win(500_000), _win(600_000), _win(700_000), _win(750_000)]
    assert all(c == [0] for c in _run(o, seq))


def test_no_reference_before_min_ref_healthy_windows():
    # two healthy windows: the third has no reference yet, so it is judged healthy and joins
    # it; only then do drops signal (gap 800,000 on k_base 100 -> step 80, capped at 50)
    o = ovo.OverloadOracle(1, min_ref=3)
    seq = [_win(900_000)] * 2 + [_win(100_000)] * 3
    assert [c[0] for c in _run(o, seq)] == [0, 0, 0, 0, 50]


def test_queue_signal_alone_contracts_by_an_eighth_of_the_base():
    o = ovo.OverloadOracle(1, queue_thresh=10)
    seq = [_win(900_000, waiting=50, k_base=80)] * 3
    assert [c[0] for c in _run(o, seq)] == [0, 10, 20]


def test_contraction_stays_within_the_percentage_of_the_base():
    o = ovo.OverloadOracle(1, max_contraction_pct=25, queue_thresh=0)
    out = [c[0] for c in _run(o, [_win(900_000, waiting=5, k_base=40)] * 10)]
    assert max(out) == 10 and out[-1] == 10


def test_windows_without_queries_carry_no_hit_signal():
    o = ovo.OverloadOracle(1)
    seq = [_win(900_000)] * 5 + [([0], [0], [0], [100])] * 4
    assert all(c == [0] for c in _run(o, seq))


def test_recheck_delay_pins():
    group = [0, 7, 7, 7, 7, 9, 9, 3]
    held = [1, 1, 1, 1, 0, 1, 1, 0]
    assert ovo.recheck_delays(group, held, 1000, 100) == [1000, 250, 250, 250, 0, 500, 500, 0]
    assert ovo.recheck_delays([5] * 20, [1] * 20, 1000, 100) == [100] * 20  # floor of 50 clamped to 100


# ---- library parity -----------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(6))
def test_library_matches_oracle_on_random_windows(seed):
    rng = np.random.default_rng(7000 + seed)
    W = 5
    cfg = dict(ref_windows=int(rng.integers(1, 10)), confirm=int(rng.integers(1, 4)),
               gap_ppm=int(rng.integers(0, 300_000)), queue_thresh=int(rng.integers(0, 40)),
               recover_after=int(rng.integers(1, 4)), max_contraction_pct=int(rng.integers(0, 101)))
    cfg["min_ref"] = int(rng.integers(1, cfg["ref_windows"] + 1))
    lib = misat.OverloadController(W, **cfg)
    ora = ovo.OverloadOracle(W, **cfg)
    base = rng.uniform(0.5, 0.98, W)
    for t in range(120):
        # regime changes: healthy, degraded (hit rate falls), queue build-up, idle windows
        rate = np.clip(base - (rng.random(W) < 0.3) * rng.uniform(0, 0.6, W) + rng.normal(0, 0.03, W), 0, 1)
        query = rng.integers(0, 2_000_000, W) * (rng.random(W) > 0.1)
        hit = np.minimum(query, (rate * query).astype(np.int64))
        waiting = rng.integers(0, 60, W) * (rng.random(W) < 0.4)
        k_base = rng.integers(0, 400, W)
        got = lib.observe(hit, query, waiting, k_base)
        want = ora.observe([int(x) for x in hit], [int(x) for x in query], [int(x) for x in waiting],
                           [int(x) for x in k_base])
        assert list(got) == want, f"window {t}"
    lib.close()


def test_library_defaults_are_the_documented_ones():
    assert misat.overload_default_config() == ovo.DEFAULTS


def test_library_rejects_invalid_windows_without_changing_state():
    lib = misat.OverloadController(2)
    ora = ovo.OverloadOracle(2)
    ok = ([900, 800], [1000, 1000], [0, 0], [100, 100])
    assert list(lib.observe(*ok)) == ora.observe(*ok)
    with pytest.raises(misat.MisatError):
        lib.observe([1001, 0], [1000, 1000], [0, 0], [100, 100])  # hit > query
    with pytest.raises(misat.MisatError):
        lib.observe([0, 0], [1000, 1000], [-1, 0], [100, 100])
    for _ in range(6):
        win = ([400, 800], [1000, 1000], [0, 0], [100, 100])
        assert list(lib.observe(*win)) == ora.observe(*win)
    with pytest.raises(misat.MisatError):
        misat.OverloadController(2, ref_windows=0)
    lib.close()


@pytest.mark.parametrize("seed", range(4))
def test_recheck_delays_match_oracle(seed):
    rng = np.random.default_rng(9100 + seed)
    n = int(rng.integers(1, 400))
    group = rng.integers(0, 12, n).astype(np.uint64)
    held = (rng.random(n) < 0.6).astype(np.uint8)
    base = int(rng.integers(1000, 10_000_000))
    mn = int(rng.integers(0, base))
    got = misat.recheck_delays(group, held, base, mn)
    want = ovo.recheck_delays([int(g) for g in group], [int(h) for h in held], base, mn)
    assert list(got) == want
    assert list(misat.recheck_delays(np.zeros(0, np.uint64), np.zeros(0, np.uint8), base, mn)) == []
    with pytest.raises(misat.MisatError):
        misat.recheck_delays(group, held, 10, 20)
