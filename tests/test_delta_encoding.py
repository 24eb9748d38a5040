"""Delta layout of host batches (input encoding, no GPU): every batch of the workloads is
rebuilt exactly from its layout, bases point to earlier requests whose whole prompt starts
the request's prompt, chains stay within the depth limit, and the layout is much smaller
than the batch where sessions and prompt groups repeat their prompts."""

import numpy as np
import pytest

from paper_2608_11152_gb300 import workload as wl


def _batches():
    for sc in (wl.config1(), wl.config2(), wl.small_random(3, n=40, n_warm=3)):
        yield from [b for b, _ in sc.warm] + [sc.batch]


def test_layout_round_trip_and_bases():
    for b in _batches():
        d = wl.encode_delta(b)
        off, tok = wl.decode_delta(d)
        assert np.array_equal(off, b.tok_off) and np.array_equal(tok, b.tokens)
        depth = np.zeros(b.n, np.int64)
        for r in range(b.n):
            c = d.base[r]
            assert -1 <= c < r
            if c >= 0:
                pc = b.tokens[b.tok_off[c]:b.tok_off[c + 1]]
                assert np.array_equal(pc, b.tokens[b.tok_off[r]:b.tok_off[r] + len(pc)])
                depth[r] = depth[c] + 1
            assert depth[r] < wl.DELTA_MAX_DEPTH


def test_layout_is_smaller_where_prompts_repeat():
    sc = wl.config2()
    d = wl.encode_delta(sc.batch)
    assert d.delta_off[-1] < 0.6 * sc.batch.n_tokens  # agentic histories and fan-out prompts
    assert (d.base >= 0).sum() > 0.3 * sc.batch.n


def test_decode_follows_chains():
    d = wl.DeltaBatch(cls=np.zeros(4, np.uint8), session=np.arange(1, 5, dtype=np.uint64),
                      base=np.array([-1, 0, 1, 0], np.int32), delta_off=np.array([0, 3, 5, 6, 6], np.int64),
                      delta_tokens=np.array([1, 2, 3, 4, 5, 6], np.int32))
    off, tok = wl.decode_delta(d)
    assert off.tolist() == [0, 3, 8, 14, 17]
    assert tok.tolist() == [1, 2, 3, 1, 2, 3, 4, 5, 1, 2, 3, 4, 5, 6, 1, 2, 3]


def test_generator_layout_equals_token_comparison():
    """The layout the generator emits from its structure (turns extend their session's
    previous turn, fan-out samples their group's first sample) is the one found by comparing
    tokens, and rebuilds the batch exactly."""
    for sc in (wl.config1(), wl.config2(), wl.small_random(5, n=60, n_warm=2)):
        for _ in range(2):
            b, _, d = sc.stream.next_batch(sc.batch.n, delta=True)
            e = wl.encode_delta(b)
            assert np.array_equal(d.base, e.base)
            assert np.array_equal(d.delta_off, e.delta_off) and np.array_equal(d.delta_tokens, e.delta_tokens)
            off, tok = wl.decode_delta(d)
            assert np.array_equal(off, b.tok_off) and np.array_equal(tok, b.tokens)
        e = wl.encode_delta(sc.batch)
        assert np.array_equal(sc.batch_delta.base, e.base)
        assert np.array_equal(sc.batch_delta.delta_tokens, e.delta_tokens)
