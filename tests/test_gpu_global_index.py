"""Global prefix index (Sec. 4.4: the router maps each prefix block hash to the set of
instances that cache it) against the oracle's per-instance indexes.

The CUDA path keeps a key -> instance-bitmask table next to the per-instance tables and
answers the block-0 probe from it.  These tests check that (a) the decisions and the H
matrix are bit-exact with the oracle in both probe layouts, and (b) after every kind of
index change (commit inserts, eviction, engine removals, cache reset, warm loads,
checkpoint restore, rebuilds) the global index holds exactly the keys of the oracle's
instance indexes, each with exactly the set of instances holding it."""

import numpy as np
import pytest

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover
    pytestmark = pytest.mark.skip(reason="needs a CUDA GPU")
else:
    pytestmark = pytest.mark.gpu

from paper_2608_11152_gb300 import workload as wl  # noqa: E402
from tests.gpu_helpers import compare_state, make_router, route_both, run_parity  # noqa: E402
from tests.helpers import make_oracle  # noqa: E402

pytestmark = [pytest.mark.gpu]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def expected_masks(o, W):
    """key -> instance bitmask (Python int) from the oracle's instance indexes."""
    exp = {}
    for w in range(W):
        keys, _ = o.dump_index(w)
        for k in keys.tolist():
            exp[k] = exp.get(k, 0) | (1 << w)
    return exp


def check_global(r, o, W):
    keys, masks = r.global_dump()
    got = {}
    for k, row in zip(keys.tolist(), masks.tolist()):
        assert k not in got, f"key {k:#x} listed twice in the global index"
        m = 0
        for i, word in enumerate(row):
            m |= int(word) << (64 * i)
        got[k] = m
    exp = expected_masks(o, W)
    assert set(got) == set(exp), f"global index keys: {len(set(got) - set(exp))} extra, {len(set(exp) - set(got))} missing"
    bad = [k for k in exp if got[k] != exp[k]]
    assert not bad, f"{len(bad)} keys with a wrong instance mask, e.g. {bad[0]:#x}: {got[bad[0]]:#x} vs {exp[bad[0]]:#x}"


@pytest.mark.parametrize("seed", list(range(12)))
@pytest.mark.parametrize("prefix_index", [0, 1])
def test_parity_random_small_both_layouts(seed, prefix_index):
    rng = np.random.default_rng(100 + seed)
    sc = wl.small_random(9000 + seed, W=int(rng.integers(1, 9)), cap=int(rng.integers(8, 160)),
                         n=int(rng.integers(1, 80)), mode=seed % 4,
                         n_warm=int(rng.integers(0, 6)))
    r, o = run_parity(sc, prefix_index=prefix_index)
    if prefix_index == 0:
        check_global(r, o, sc.W)
    r.close()


def test_parity_config2_per_instance_layout():
    sc = wl.config2()
    r, o = run_parity(sc, index_every_step=False, prefix_index=1)
    r.close()


def test_parity_config5_reduced_per_instance_layout():
    sc = wl.config5(n=4096, fill=0.5)
    r, o = run_parity(sc, index_every_step=False, prefix_index=1)
    r.close()


def test_global_index_mirrors_every_kind_of_change():
    sc = wl.small_random(31, W=5, cap=120, n=40, mode=0, n_warm=4)
    r, o = run_parity(sc)
    check_global(r, o, sc.W)
    # engine removal events: drop a suffix of the deepest chain on every instance
    for w in range(sc.W):
        gk, gm = r.dump_index(w)
        if len(gk) == 0:
            continue
        depth = 65535 - (gm & 0xFFFF).astype(np.int64)
        drop = gk[depth >= max(1, int(depth.max()) - 2)]
        r.evict(w, drop)
        o.evict(w, drop)
    compare_state(r, o, sc.W)
    check_global(r, o, sc.W)
    # cache reset of one instance
    r.reset_instance(2)
    o.reset_instance(2)
    check_global(r, o, sc.W)
    # warm chains and raw entries (a key shared by two instances)
    rng = np.random.default_rng(3)
    lens = [90, 48, 200, 17]
    off = np.zeros(len(lens) + 1, np.int64)
    np.cumsum(lens, out=off[1:])
    toks = rng.integers(0, wl.VOCAB, size=int(off[-1]), dtype=np.int32)
    inst, seq, arr, mb = [0, 2, 2, 4], [1, 2, 2, 3], [1, 2, 3, 4], [100, 2, 100, 1]
    for x in (r, o):
        x.load_chains(off, toks, inst, seq, arr, mb)
    check_global(r, o, sc.W)
    ek = np.array([0x1234567890ABCDEF, 0x0FEDCBA987654321], np.uint64)
    em = np.array([(1 << 36) | (5 << 16) | 65535, (1 << 36) | (6 << 16) | 65535], np.uint64)
    for w in (1, 3):
        r.load_entries(w, ek, em)
        o.load_entries(w, ek, em)
    check_global(r, o, sc.W)
    # a further batch through route and commit
    route_both(r, o, sc.batch, sc.W)
    r.commit()
    o.commit()
    compare_state(r, o, sc.W)
    check_global(r, o, sc.W)
    # checkpoint, change, restore
    ck = r.checkpoint_save()
    o2 = o.clone()
    r.reset_instance(0)
    r.global_rebuild()
    r.checkpoint_restore(ck)
    check_global(r, o2, sc.W)
    route_both(r, o2, sc.batch, sc.W)
    r.commit()
    o2.commit()
    check_global(r, o2, sc.W)
    # an explicit rebuild changes nothing observable
    r.global_rebuild()
    check_global(r, o2, sc.W)
    ck.free()
    o2.close()
    r.close()


def test_global_index_rebuilds_when_claimed_slots_accumulate():
    """Keys whose instances all evicted them keep their slot until the library rebuilds the
    index from the instance tables; many small commits must trigger such rebuilds and stay
    bit-exact throughout."""
    sc = wl.small_random(47, W=4, cap=64, n=60, mode=3, n_warm=40)
    r, o = make_router(sc), make_oracle(sc)
    _, slots, _ = r.global_info()
    claimed_seen = []
    for b, comp in list(sc.warm) + [(sc.batch, None)]:
        route_both(r, o, b, sc.W)
        r.commit()
        o.commit()
        compare_state(r, o, sc.W)
        claimed_seen.append(r.global_info()[2])
        if comp is not None:
            for x in (r, o):
                x.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
    check_global(r, o, sc.W)
    assert max(claimed_seen) <= 0.7 * slots + 64 * 60, "claimed slots exceeded the rebuild bound"
    assert any(b < a for a, b in zip(claimed_seen, claimed_seen[1:])), \
        f"no rebuild happened (claimed slots {claimed_seen}, {slots} slots)"
    r.close()
