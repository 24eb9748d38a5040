"""The allocation-free block-hash entry point (misat_block_hash_noalloc).

It exists for callers that cannot allocate device memory (an engine whose free HBM
already belongs to its KV-cache pool, or code running inside another framework's
allocator scope).  Its keys must equal those of the regular routing entry point
(misat_route, read back with misat_dump_keys) and, request by request, the oracle's chained
block keys, bit for bit -- the tolerance of every integer output in these tests -- on two
calls in a row, which share the library's one scratch array.  This file is collected last
on purpose."""

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _batches():
    from paper_2608_11152_gb300 import workload as wl

    sc = wl.config1()
    out = [sc.warm[0][0], sc.batch]
    # more requests than one tile of the offsets scan (1,024), lengths around block edges
    rng0 = np.random.default_rng(22)
    lens0 = rng0.integers(0, 70, size=2500)
    off0 = np.zeros(len(lens0) + 1, np.int64)
    np.cumsum(lens0, out=off0[1:])
    out.append(wl.Batch(cls=np.zeros(len(lens0), np.uint8), session=np.arange(1, len(lens0) + 1, dtype=np.uint64),
                        group=np.zeros(len(lens0), np.uint64), tok_off=off0,
                        tokens=rng0.integers(0, wl.VOCAB, size=int(off0[-1]), dtype=np.int32)))
    # short and misaligned prompts, one without any full block
    rng = np.random.default_rng(21)
    lens = [0, 5, 16, 17, 33, 100, 1000, 31, 2048, 3]
    off = np.zeros(len(lens) + 1, np.int64)
    np.cumsum(lens, out=off[1:])
    out.append(wl.Batch(cls=np.zeros(len(lens), np.uint8), session=np.arange(1, len(lens) + 1, dtype=np.uint64),
                        group=np.zeros(len(lens), np.uint64), tok_off=off,
                        tokens=rng.integers(0, wl.VOCAB, size=int(off[-1]), dtype=np.int32)))
    return sc, out


def test_noalloc_hash_matches_routing_keys_and_oracle_twice():
    import __graft_entry__

    __graft_entry__.build()
    import oracle
    from paper_2608_11152_gb300 import misat

    torch.cuda.set_device(0)
    sc, batches = _batches()
    r = misat.Router(sc.cap_blocks, max_batch=max(b.n for b in batches), max_tokens=max(b.n_tokens for b in batches),
                     prior_kbar=sc.prior_kbar)
    for b in batches:
        db = r.device_batch(b)
        r.route(db)
        torch.cuda.synchronize()
        expect = r.dump_keys(b.n_tokens // 16 + 1)
        # the oracle's keys of every request, in request order (its compact layout)
        ref = [oracle.hash_prompt(b.tokens[b.tok_off[q]:b.tok_off[q + 1]]) for q in range(b.n)]
        ref = np.concatenate(ref) if ref else np.zeros(0, np.uint64)
        assert np.array_equal(expect, ref)
        for _ in range(2):  # two calls in a row share (and must clear) the scratch array
            keys = torch.full((len(expect) + 7,), -1, dtype=torch.int64, device="cuda")
            misat.block_hash_noalloc(db["tok_off"], db["tokens"], b.n, b.n_tokens, keys)
            got = keys.cpu().numpy().view(np.uint64)
            assert np.array_equal(got[: len(expect)], expect)
            assert np.array_equal(got[: len(ref)], ref)
            assert np.all(keys.cpu().numpy()[len(expect):] == -1)  # nothing written past the keys
    r.close()


def test_noalloc_rejects_batches_beyond_its_scratch():
    from paper_2608_11152_gb300 import misat

    n = misat.NOALLOC_MAX_REQUESTS + 1
    off = torch.zeros(n + 1, dtype=torch.int64, device="cuda")
    toks = torch.zeros(16, dtype=torch.int32, device="cuda")
    keys = torch.zeros(16, dtype=torch.int64, device="cuda")
    with pytest.raises(misat.MisatError) as e:
        misat.block_hash_noalloc(off, toks, n, 0, keys)
    assert e.value.code == misat.ERR_BATCH_TOO_LARGE
    # keys_cap smaller than the number of full blocks: rejected on the device, nothing written
    off = torch.tensor([0, 64], dtype=torch.int64, device="cuda")
    toks = torch.zeros(64, dtype=torch.int32, device="cuda")
    small = torch.full((2,), 7, dtype=torch.int64, device="cuda")
    with pytest.raises(misat.MisatError) as e:
        misat.block_hash_noalloc(off, toks, 1, 64, small)
    assert e.value.code == misat.ERR_INVALID_ARG
    assert small.cpu().tolist() == [7, 7]
