"""CUDA path (through the C ABI) vs the CPU oracle, element by element (bit-exact:
every output of this path is integer or index work).

Covers keys, the H matrix, caps, decisions, reasons, hit blocks, statistics, protected
counts, the session table and the full sorted index of every instance after every
commit; on random small scenarios (all modes, caps and eviction binding often), the five
workload configurations and the edge cases of the API."""

import numpy as np
import pytest

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover
    pytestmark = pytest.mark.skip(reason="needs a CUDA GPU")
else:
    pytestmark = pytest.mark.gpu

import oracle  # noqa: E402
from paper_2608_11152_gb300 import workload as wl  # noqa: E402
from tests.gpu_helpers import assert_equal, compare_state, make_router, route_both, run_parity  # noqa: E402
from tests.helpers import load_fill, make_oracle  # noqa: E402

pytestmark = [pytest.mark.gpu]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()
    from paper_2608_11152_gb300 import misat  # noqa: F401


def _mk(cls, sessions, lens, seed=0, offset_tokens=None):
    rng = np.random.default_rng(seed)
    off = np.zeros(len(cls) + 1, np.int64)
    np.cumsum(lens, out=off[1:])
    toks = offset_tokens if offset_tokens is not None else rng.integers(0, wl.VOCAB, size=int(off[-1]), dtype=np.int32)
    return wl.Batch(cls=np.array(cls, np.uint8), session=np.array(sessions, np.uint64),
                    group=np.zeros(len(cls), np.uint64), tok_off=off, tokens=np.ascontiguousarray(toks, np.int32))


# ------------------------------------------------------------------ random small scenarios

@pytest.mark.parametrize("seed", list(range(40)))
def test_parity_random_small(seed):
    rng = np.random.default_rng(seed)
    sc = wl.small_random(5000 + seed, W=int(rng.integers(1, 9)), cap=int(rng.integers(8, 160)),
                         n=int(rng.integers(1, 80)), mode=seed % 4,
                         n_warm=int(rng.integers(0, 6)))
    r, o = run_parity(sc)
    r.close()


@pytest.mark.parametrize("seed", list(range(10)))
def test_parity_with_releases_and_rebounds(seed):
    """Completions with done=0 release sessions (Eq. 7 continuations); backlogs change
    between batches so continuations rebind; caps are contracted on some instances."""
    sc = wl.small_random(7000 + seed, W=4, cap=96, n=48, mode=0, n_warm=6)
    r, o = make_router(sc), make_oracle(sc)
    rng = np.random.default_rng(seed)
    steps = list(sc.warm) + [(sc.batch, None)]
    for i, (b, comp) in enumerate(steps):
        bk = rng.integers(0, 3_000_000, size=sc.W)
        cont = rng.integers(0, 3, size=sc.W).astype(np.int32)
        for x in (r, o):
            x.set_instance_state(bk, None, cont)
        route_both(r, o, b, sc.W)
        r.commit()
        o.commit()
        compare_state(r, o, sc.W)
        if comp is not None:
            for x in (r, o):
                x.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
        ids, st, ins, cl = o.sessions()
        pick = ids[rng.random(len(ids)) < 0.35]
        if len(pick):
            z8, z32, z64 = np.zeros(len(pick), np.uint8), np.zeros(len(pick), np.int32), np.zeros(len(pick), np.int64)
            for x in (r, o):
                x.complete(pick, z8, z32, z64, z8)
        compare_state(r, o, sc.W, index=False)
    r.close()


# ------------------------------------------------------------------ workload configurations

# both block-0 probe layouts: 0 = through the global index, 1 = per-instance tables with the
# lookups shared by the requests that start with the same block (the benchmark's layout)
LAYOUTS = [0, 1]


@pytest.mark.parametrize("prefix_index", LAYOUTS)
@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_parity_config(cfg, prefix_index):
    sc = wl.CONFIGS[cfg]()
    r, o = run_parity(sc, index_every_step=cfg == 1, prefix_index=prefix_index)
    r.close()


@pytest.mark.parametrize("prefix_index", LAYOUTS)
def test_parity_config4_agentic_long_sessions(prefix_index):
    sc = wl.config4()
    r, o = run_parity(sc, index_every_step=False, prefix_index=prefix_index)
    r.close()


@pytest.mark.parametrize("prefix_index", LAYOUTS)
def test_parity_config5_reduced(prefix_index):
    sc = wl.config5(n=4096, fill=0.5)
    r, o = run_parity(sc, index_every_step=False, prefix_index=prefix_index)
    r.close()


@pytest.mark.parametrize("prefix_index", LAYOUTS)
def test_parity_config5_full_size(prefix_index):
    """The benchmark workload itself: 128 x 262,144 blocks at 95% fill (resident prompt chains,
    some of them histories that agentic sessions of the batch continue), 65,536 requests, in
    the launch configuration the benchmark times (per-instance tables; the global index as
    well): the measured batch is routed as the benchmark routes it (same buffers every call,
    so the route is launched directly, then captured, then replayed from its CUDA graph) and
    every one of those routes must give the oracle's decisions; then the commit and every
    instance's index are compared."""
    import torch

    sc = wl.config5(n=65536, fill=0.95)
    r = make_router(sc, prefix_index=prefix_index)
    o = make_oracle(sc)
    try:
        load_fill(r, sc)
        load_fill(o, sc)
        for b, comp in sc.warm:
            route_both(r, o, b, sc.W, check_H=False, check_keys=False)
            r.commit()
            o.commit()
            if comp is not None:
                for x in (r, o):
                    x.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
        b = sc.batch
        route_both(r, o, b, sc.W, check_H=True, check_keys=True)  # H and keys against the oracle
        oi, orr, oh = o.route(b.cls, b.session, b.tok_off, b.tokens)
        db, out = r.device_batch(b), r.alloc_decisions(b.n)
        for rep in range(3):
            out["inst"].fill_(-7)
            r.route(db, out)
            torch.cuda.synchronize()
            assert_equal(f"inst (bench call {rep})", out["inst"][: b.n].cpu().numpy(), oi)
            assert_equal(f"reason (bench call {rep})", out["reason"][: b.n].cpu().numpy(), orr)
            assert_equal(f"hit blocks (bench call {rep})", out["hit_blocks"][: b.n].cpu().numpy(), oh)
        r.commit()
        o.commit()
        compare_state(r, o, sc.W, index=True)
        s, os_ = r.stats(), o.stats()
        assert s.new_keys == os_[21] and s.evicted == os_[22]
        assert o.check_invariants() == 0
        r.sync()
    finally:
        r.close()


# ------------------------------------------------------------------ edge cases

def test_empty_batch_and_commit_state():
    from paper_2608_11152_gb300 import misat

    sc = wl.small_random(11, n_warm=1)
    r, o = make_router(sc), make_oracle(sc)
    with pytest.raises(misat.MisatError) as e:
        r.commit()
    assert e.value.code == misat.ERR_STATE
    empty = _mk([], [], [])
    route_both(r, o, empty, sc.W)
    r.commit()
    o.commit()
    assert r.stats().seq == o.seq() == 1
    b, c = sc.warm[0]
    route_both(r, o, b, sc.W)
    r.commit()
    o.commit()
    compare_state(r, o, sc.W)
    r.close()


def test_short_prompts_alignments_and_partial_blocks():
    """Prompts of 0..40 tokens (no full block, exactly one, a trailing partial block) at every
    16-byte misalignment of their first token."""
    lens = [0, 1, 3, 15, 16, 17, 31, 32, 33, 40, 5, 16, 47, 48, 2, 64]
    n = len(lens)
    sc = wl.small_random(12, W=3, cap=64, n=4, n_warm=0)
    r, o = make_router(sc, max_batch=64, max_tokens=4096), make_oracle(sc)
    rng = np.random.default_rng(3)
    shared = rng.integers(0, wl.VOCAB, size=64, dtype=np.int32)
    toks = np.concatenate([shared[:L] for L in lens])
    b = _mk([i % 3 for i in range(n)], list(range(1, n + 1)), lens, offset_tokens=toks)
    for _ in range(3):
        route_both(r, o, b, sc.W)
        r.commit()
        o.commit()
        compare_state(r, o, sc.W)
    r.close()


def test_longest_prompt_65535_blocks():
    sc = wl.small_random(13, W=2, cap=70000, n=2, n_warm=0)
    sc.cap_blocks = np.array([70000, 70000], np.int64)
    L = (1 << 20) - 1
    r, o = make_router(sc, max_batch=4, max_tokens=2 * L), make_oracle(sc)
    rng = np.random.default_rng(4)
    t = rng.integers(0, wl.VOCAB, size=L, dtype=np.int32)
    b = _mk([2, 2], [7, 8], [L, L], offset_tokens=np.concatenate([t, t]))
    route_both(r, o, b, sc.W)
    r.commit()
    o.commit()
    compare_state(r, o, sc.W)
    # the same prompt again: fully cached on its instance (H = 65535)
    b2 = _mk([2], [7], [L], offset_tokens=t)
    out = route_both(r, o, b2, sc.W)
    assert int(out["hit_blocks"][0]) == 65535
    r.close()


@pytest.mark.parametrize("prefix_index", LAYOUTS)
def test_many_instances_w1024(prefix_index):
    sc = wl.small_random(14, W=1024, cap=32, n=300, n_warm=2)
    r, o = run_parity(sc, prefix_index=prefix_index)
    r.close()


@pytest.mark.parametrize("prefix_index", LAYOUTS)
def test_one_instance(prefix_index):
    sc = wl.small_random(15, W=1, cap=256, n=60, n_warm=3)
    r, o = run_parity(sc, prefix_index=prefix_index)
    r.close()


def test_shared_block0_lookups_count_the_distinct_first_blocks():
    """Per-instance tables: every distinct block-0 key of a batch is probed once per instance.
    The statistics must report the number of distinct first blocks (16-token prefixes,
    counted on the host from the tokens) and exactly that many probes per instance, and
    the decisions and H rows must still equal the oracle's (route_both)."""
    sc = wl.config3()
    r = make_router(sc, prefix_index=1)
    o = make_oracle(sc)
    try:
        load_fill(r, sc)
        load_fill(o, sc)
        for b, comp in list(sc.warm) + [(sc.batch, None)]:
            route_both(r, o, b, sc.W)
            s = r.stats()
            L = np.diff(b.tok_off)
            firsts = {b.tokens[b.tok_off[i]:b.tok_off[i] + 16].tobytes() for i in range(b.n) if L[i] >= 16}
            assert s.first_block_keys == len(firsts), (s.first_block_keys, len(firsts))
            assert s.probes_first == len(firsts) * sc.W
            assert s.first_block_lookups == int((L >= 16).sum())
            assert len(firsts) < int((L >= 16).sum())  # the workload does share first blocks
            r.commit()
            o.commit()
            if comp is not None:
                for x in (r, o):
                    x.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
        compare_state(r, o, sc.W, index=True)
    finally:
        r.close()


def test_table_growth_and_session_rebuild():
    """Tiny tables and a tiny session table: growth and rebuild paths run and stay exact."""
    sc = wl.small_random(16, W=3, cap=8, n=70, mode=3, n_warm=5)
    r, o = run_parity(sc, max_sessions=1, table_load=0.25)
    r.close()


def test_batch_too_large_and_invalid_device_input():
    from paper_2608_11152_gb300 import misat

    sc = wl.small_random(17, W=2, cap=64, n=8, n_warm=0)
    r = make_router(sc, max_batch=8, max_tokens=2048)
    big = _mk([0] * 9, list(range(1, 10)), [16] * 9)
    with pytest.raises(misat.MisatError) as e:
        r.route(r.device_batch(big))
    assert e.value.code == misat.ERR_BATCH_TOO_LARGE
    # a zero session id and a class id of 7 are found on the device: sticky error, no state change
    bad = _mk([0, 7], [0, 5], [32, 32])
    r.route(r.device_batch(bad))
    with pytest.raises(misat.MisatError) as e:
        r.sync()
    assert e.value.code == misat.ERR_INVALID_ARG
    # non-monotone offsets
    bad2 = _mk([0, 1], [4, 5], [32, 32])
    bad2.tok_off[1] = 40
    bad2.tok_off[2] = 32
    r.route(r.device_batch(bad2))
    with pytest.raises(misat.MisatError):
        r.sync()
    # the context is usable again and still matches the oracle
    o = make_oracle(sc)
    good = _mk([0, 1, 2], [4, 5, 6], [48, 40, 33])
    route_both(r, o, good, sc.W)
    r.commit()
    o.commit()
    compare_state(r, o, sc.W)
    r.close()


def test_route_host_matches_device_route():
    sc = wl.config1()
    r1, r2, o = make_router(sc), make_router(sc), make_oracle(sc)
    for b, comp in list(sc.warm) + [(sc.batch, None)]:
        dev = route_both(r1, o, b, sc.W)
        host = r2.route_host(b)
        for k in ("inst", "reason", "hit_blocks"):
            assert_equal(k, host[k][: b.n], dev[k][: b.n].cpu().numpy())
        for x in (r1, r2, o):
            x.commit()
        if comp is not None:
            for x in (r1, r2, o):
                x.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
    for w in range(sc.W):
        assert_equal("index", r1.dump_index(w)[1], r2.dump_index(w)[1])
    r1.close()
    r2.close()


def _pinned_batch(b):
    def pin(a):
        t = torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
        return t.numpy()

    return wl.Batch(cls=pin(b.cls), session=pin(b.session.view(np.int64)).view(np.uint64), group=b.group,
                    tok_off=pin(b.tok_off), tokens=pin(b.tokens))


@pytest.mark.parametrize("cfg", [1, 2])
def test_pipelined_host_staging_matches_the_oracle(cfg):
    """Batch k+1 is staged (copy stream) before batch k is routed from the other slot; every
    decision and the index after every commit equal the oracle's."""
    sc = {1: wl.config1, 2: wl.config2}[cfg]()
    r, o = make_router(sc), make_oracle(sc)
    steps = list(sc.warm) + [(sc.batch, None)]
    pinned = [_pinned_batch(b) for b, _ in steps]
    r.stage_host(pinned[0], 0)
    for k, (b, comp) in enumerate(steps):
        if k + 1 < len(steps):
            r.stage_host(pinned[k + 1], (k + 1) % 2)
        got = r.route_staged(k % 2)
        oi, orr, oh = o.route(b.cls, b.session, b.tok_off, b.tokens)
        assert_equal("inst", got["inst"][: b.n], oi)
        assert_equal("reason", got["reason"][: b.n], orr)
        assert_equal("hit_blocks", got["hit_blocks"][: b.n], oh)
        r.commit()
        o.commit()
        compare_state(r, o, sc.W)
        if comp is not None:
            for x in (r, o):
                x.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
    r.sync()
    r.close()


def _pinned_delta(d):
    def pin(a):
        return torch.from_numpy(np.ascontiguousarray(a)).pin_memory().numpy()

    return wl.DeltaBatch(cls=pin(d.cls), session=pin(d.session.view(np.int64)).view(np.uint64), base=pin(d.base),
                         delta_off=pin(d.delta_off), delta_tokens=pin(d.delta_tokens))


@pytest.mark.parametrize("cfg", [1, 2, 3])
def test_delta_staging_matches_the_oracle(cfg):
    """Batches sent in the delta layout (each prompt as an extension of an earlier prompt of
    the batch), rebuilt on the GPU and routed through the pipelined slots: every decision,
    every block key and the state after every commit equal the oracle's on the full batch."""
    sc = {1: wl.config1, 2: wl.config2, 3: wl.config3}[cfg]()
    r, o = make_router(sc), make_oracle(sc)
    steps = list(sc.warm) + [(sc.batch, None)]
    encs = [_pinned_delta(wl.encode_delta(b)) for b, _ in steps]
    r.stage_host_delta(encs[0], 0)
    for k, (b, comp) in enumerate(steps):
        if k + 1 < len(steps):
            r.stage_host_delta(encs[k + 1], (k + 1) % 2)
        got = r.route_staged(k % 2)
        oi, orr, oh = o.route(b.cls, b.session, b.tok_off, b.tokens)
        assert_equal("inst", got["inst"][: b.n], oi)
        assert_equal("reason", got["reason"][: b.n], orr)
        assert_equal("hit_blocks", got["hit_blocks"][: b.n], oh)
        cap = b.n_tokens // 16 + 1
        assert_equal("keys", r.dump_keys(cap), o.keys(cap))
        r.commit()
        o.commit()
        compare_state(r, o, sc.W)
        if comp is not None:
            for x in (r, o):
                x.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
    r.sync()
    r.close()


def test_delta_staging_rejects_malformed_layouts():
    """A base that is not an earlier request, a chain deeper than the limit and offsets that
    do not start at zero are refused before anything is copied; the slot stays free."""
    from paper_2608_11152_gb300 import misat

    sc = wl.config1()
    r = make_router(sc, max_batch=128)
    b = sc.warm[0][0]
    good = wl.encode_delta(b)

    def variant(**kw):
        f = dict(cls=good.cls, session=good.session, base=good.base.copy(), delta_off=good.delta_off.copy(),
                 delta_tokens=good.delta_tokens)
        f.update(kw)
        return wl.DeltaBatch(**f)

    bad_base = good.base.copy()
    bad_base[3] = 3
    deep = 70
    chain = wl.DeltaBatch(cls=np.zeros(deep, np.uint8), session=np.arange(1, deep + 1, dtype=np.uint64),
                          base=np.arange(-1, deep - 1, dtype=np.int32), delta_off=np.arange(0, 16 * deep + 1, 16,
                                                                                            dtype=np.int64),
                          delta_tokens=np.ones(16 * deep, np.int32))
    shifted = good.delta_off.copy() + 1
    for enc in (variant(base=bad_base), chain, variant(delta_off=shifted)):
        with pytest.raises(misat.MisatError) as e:
            r.stage_host_delta(enc, 0)
        assert e.value.code == misat.ERR_INVALID_ARG
    r.stage_host_delta(good, 0)  # the slot is still free
    got = r.route_staged(0)
    ref = r.route_host(b)
    for k in ("inst", "reason", "hit_blocks"):
        assert_equal(k, got[k][: b.n], ref[k][: b.n])
    r.sync()
    r.close()


def test_pipelined_staging_slot_states_and_graph_replay():
    """A slot holds one batch until it is routed; routing an empty slot is refused.  The same
    batch routed from alternating slots after a state restore (graphs captured per slot and
    replayed) gives the same decisions every time."""
    from paper_2608_11152_gb300 import misat

    sc = wl.config2()
    r = make_router(sc)
    for b, comp in sc.warm:
        r.route_host(b)
        r.commit()
        if comp is not None:
            r.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
    pb = _pinned_batch(sc.batch)
    with pytest.raises(misat.MisatError) as e:
        r.route_staged(0)
    assert e.value.code == misat.ERR_STATE
    r.stage_host(pb, 0)
    with pytest.raises(misat.MisatError) as e:
        r.stage_host(pb, 0)
    assert e.value.code == misat.ERR_STATE
    with pytest.raises(misat.MisatError) as e:
        r.stage_host(pb, 2)
    assert e.value.code == misat.ERR_INVALID_ARG
    ckpt = r.checkpoint_save()
    ref = r.route_host(sc.batch)
    ref = {k: v[: sc.batch.n].copy() for k, v in ref.items()}

    def slot(k):  # 1, 0, 1, 0, ...
        return (k + 1) % 2

    first = r.route_staged(0)  # the batch staged above, routed from the same state
    for name in ("inst", "reason", "hit_blocks"):
        assert_equal(name, first[name][: sc.batch.n], ref[name])
    r.stage_host(pb, slot(0))
    for k in range(6):
        r.checkpoint_restore(ckpt)
        if k + 1 < 6:
            r.stage_host(pb, slot(k + 1))
        got = r.route_staged(slot(k))
        for name in ("inst", "reason", "hit_blocks"):
            assert_equal(f"{name} (route {k})", got[name][: sc.batch.n], ref[name])
    r.commit()
    r.sync()
    ckpt.free()
    r.close()


def test_external_evict_reset_and_load_chains():
    sc = wl.small_random(18, W=3, cap=200, n=20, n_warm=2)
    r, o = run_parity(sc)
    # engine removal events: drop a suffix of one resident chain on every instance
    for w in range(sc.W):
        gk, gm = r.dump_index(w)
        if len(gk) == 0:
            continue
        depth = 65535 - (gm & 0xFFFF).astype(np.int64)
        drop = gk[depth >= max(1, int(depth.max()) - 1)]
        r.evict(w, drop)
        o.evict(w, drop)
    compare_state(r, o, sc.W)
    assert o.check_invariants() == 0
    # cache reset of one instance (weight sync)
    r.reset_instance(1)
    o.reset_instance(1)
    compare_state(r, o, sc.W)
    # warm chains with explicit ticks and block limits
    rng = np.random.default_rng(5)
    lens = [100, 35, 300, 16, 0, 77]
    off = np.zeros(len(lens) + 1, np.int64)
    np.cumsum(lens, out=off[1:])
    toks = rng.integers(0, wl.VOCAB, size=int(off[-1]), dtype=np.int32)
    inst, seq, arr, mb = [0, 1, 2, 1, 0, 2], [1, 1, 2, 0, 1, 3], [5, 6, 7, 8, 9, 10], [3, 100, 12, 1, 4, 0]
    r.load_chains(off, toks, inst, seq, arr, mb)
    o.load_chains(off, toks, inst, seq, arr, mb)
    compare_state(r, o, sc.W)
    route_both(r, o, sc.batch, sc.W)
    r.commit()
    o.commit()
    compare_state(r, o, sc.W)
    r.close()


def test_all_four_modes_on_config1():
    for mode in range(4):
        sc = wl.config1()
        sc.mode = mode
        r, o = run_parity(sc)
        r.close()


@pytest.mark.parametrize("seed,W", [(0, 64), (1, 300), (2, 37), (3, 5)])
def test_serial_selection_many_windows_and_fills(seed, W):
    """Batches of a few thousand leaders (several selection windows) against small caps, so
    that instances run out of global and class headroom inside windows and envelopes lose
    many lines; released sessions make Eq. (7) leaders.  Decisions, caps and committed state
    equal the oracle's after every batch."""
    sc = wl.small_random(9100 + seed, W=W, cap=200, n=3000, mode=seed % 2, n_warm=3)
    r, o = make_router(sc), make_oracle(sc)
    rng = np.random.default_rng(seed)
    held = admitted = 0
    for b, comp in list(sc.warm) + [(sc.batch, None)]:
        route_both(r, o, b, W)
        st = o.stats()
        held += int(st[oracle.STAT_HELD])
        admitted += int(st[oracle.STAT_ADMITTED])
        r.commit()
        o.commit()
        compare_state(r, o, W, index=False)
        if comp is not None:
            for x in (r, o):
                x.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
        ids, _, _, _ = o.sessions()
        pick = ids[rng.random(len(ids)) < 0.3]
        if len(pick):
            z8, z32, z64 = np.zeros(len(pick), np.uint8), np.zeros(len(pick), np.int32), np.zeros(len(pick), np.int64)
            for x in (r, o):
                x.complete(pick, z8, z32, z64, z8)
    compare_state(r, o, W)
    assert held > 0 and admitted > 0
    r.close()


def test_per_class_and_joint_selection_paths_match_the_oracle():
    """While no instance runs out of global headroom, the per-class chains decide a batch;
    otherwise the joint chain over all classes decides it again.  Across these scenarios both
    paths decide some batches (session admission, which has no class caps, makes the global cap
    bind), and every batch equals the oracle's decisions and committed state."""
    seen = {0: 0, 1: 0}
    for seed in range(12):
        rng = np.random.default_rng(300 + seed)
        W = int(rng.integers(2, 9))
        sc = wl.small_random(9300 + seed, W=W, cap=int(rng.integers(40, 200)), n=int(rng.integers(100, 600)),
                             mode=seed % 4, n_warm=3)
        r, o = make_router(sc), make_oracle(sc)
        for b, comp in list(sc.warm) + [(sc.batch, None)]:
            route_both(r, o, b, W)
            seen[int(r.stats().joint_selection)] += 1
            r.commit()
            o.commit()
            compare_state(r, o, W, index=False)
            if comp is not None:
                for x in (r, o):
                    x.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
        compare_state(r, o, W)
        r.close()
    assert seen[0] > 0 and seen[1] > 0, seen


def test_checkpoint_restore_replays_identically():
    """A restored checkpoint gives the same decisions and the same committed state again,
    including after a commit that grew a table (the restore shrinks it back)."""
    sc = wl.small_random(19, W=3, cap=16, n=60, mode=3, n_warm=2)
    r, o = run_parity(sc, table_load=0.25)
    ck = r.checkpoint_save()
    o2 = o.clone()
    outs = []
    for _ in range(2):
        r.checkpoint_restore(ck)
        oc = o2.clone()
        out = route_both(r, oc, sc.batch, sc.W)
        outs.append({k: v[: sc.batch.n].cpu().numpy() for k, v in out.items()})
        r.commit()
        oc.commit()
        compare_state(r, oc, sc.W)
        oc.close()
    for k in outs[0]:
        assert_equal(k, outs[0][k], outs[1][k])
    r.set_timing(True)
    r.checkpoint_restore(ck)
    r.route(r.device_batch(sc.batch))
    r.commit()
    ph = r.phase_times()
    assert set(ph) >= {"hash", "probe_first", "evict"} and all(v >= 0 for v in ph.values())
    ck.free()
    o2.close()
    r.close()


def test_route_graph_capture_and_replay_match_the_oracle():
    """The route is launched directly the first time a set of buffers is seen, captured the
    second time and replayed from then on; with phase timing on it is launched directly.  All
    of these give the oracle's decisions (the same batch routed repeatedly before its commit
    replaces the pending route on both sides)."""
    import torch

    sc = wl.config2()
    r = make_router(sc)
    o = make_oracle(sc)
    try:
        for i, (b, comp) in enumerate(list(sc.warm) + [(sc.batch, None)]):
            db = r.device_batch(b)
            out = r.alloc_decisions(b.n)
            oi, orr, oh = o.route(b.cls, b.session, b.tok_off, b.tokens)
            for rep in range(4):
                r.set_timing(rep == 3)
                r.route(db, out)
                torch.cuda.synchronize()
                assert_equal(f"inst batch {i} call {rep}", out["inst"][: b.n].cpu().numpy(), oi)
                assert_equal(f"reason batch {i} call {rep}", out["reason"][: b.n].cpu().numpy(), orr)
                assert_equal(f"hit batch {i} call {rep}", out["hit_blocks"][: b.n].cpu().numpy(), oh)
            r.set_timing(False)
            r.commit()
            o.commit()
            compare_state(r, o, sc.W, index=(i == len(sc.warm)))
            if comp is not None:
                r.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
                o.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
        r.sync()
    finally:
        r.close()


def test_route_graph_cache_rotation_over_more_buffer_sets_than_it_keeps():
    """Six copies of one batch, each routed twice in a row (launched directly, then captured)
    and visited in rotation, so that the cache (four graphs) drops the least recently used
    graphs and captures them again; then the last four copies in rotation (replayed).  Every
    route before the commit gives the oracle's decisions."""
    import torch

    sc = wl.config1()
    r = make_router(sc)
    o = make_oracle(sc)
    try:
        for b, comp in sc.warm:
            route_both(r, o, b, sc.W, check_H=False, check_keys=False)
            r.commit()
            o.commit()
            if comp is not None:
                r.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
                o.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
        b = sc.batch
        oi, orr, oh = o.route(b.cls, b.session, b.tok_off, b.tokens)
        copies = [(r.device_batch(b), r.alloc_decisions(b.n)) for _ in range(6)]
        order = [j for _ in range(3) for j in range(6) for _ in range(2)] + [2, 3, 4, 5] * 3
        for step, j in enumerate(order):
            db, out = copies[j]
            out["inst"].fill_(-7)
            r.route(db, out)
            torch.cuda.synchronize()
            assert_equal(f"inst copy {j} step {step}", out["inst"][: b.n].cpu().numpy(), oi)
            assert_equal(f"reason copy {j} step {step}", out["reason"][: b.n].cpu().numpy(), orr)
            assert_equal(f"hit copy {j} step {step}", out["hit_blocks"][: b.n].cpu().numpy(), oh)
        r.commit()
        o.commit()
        compare_state(r, o, sc.W)
        r.sync()
    finally:
        r.close()
