"""The overload controller in the routing loop, on the GPU: after every batch each side
computes its per-instance window (hit and prompt tokens of its admitted requests, held
requests, base cap floor(C_w / kbar_w) from its own caps), feeds its own controller (the
library's misat_overload_* for the GPU router, the plain-Python oracle for the CPU oracle)
and applies the contraction to its router; decisions, caps and indexes must stay equal."""

import numpy as np
import pytest
import torch

from oracle import overload as ovo
from paper_2608_11152_gb300 import misat
from paper_2608_11152_gb300 import workload as wl
from tests.gpu_helpers import assert_equal, compare_state, make_router
from tests.helpers import load_fill, make_oracle

# reactive thresholds so that contractions happen within a few batches
CFG = dict(ref_windows=4, min_ref=1, gap_ppm=0, confirm=1, queue_thresh=2, recover_after=1, max_contraction_pct=60)


def _window(inst, hit_blocks, L, W):
    hit = np.zeros(W, np.int64)
    query = np.zeros(W, np.int64)
    adm = inst >= 0
    np.add.at(hit, inst[adm], 16 * hit_blocks[adm].astype(np.int64))
    np.add.at(query, inst[adm], L[adm].astype(np.int64))
    waiting = np.full(W, int((~adm).sum()) // W, np.int64)
    return hit, query, waiting


def _k_base(caps, cap_blocks, pf_q16):
    C = (np.asarray(cap_blocks, np.int64) * pf_q16) >> 16
    return C // np.maximum(caps["kbar_w"], 1)


def _run(sc):
    W = sc.W
    r = make_router(sc)
    o = make_oracle(sc)
    ctl_g = misat.OverloadController(W, **CFG)
    ctl_o = ovo.OverloadOracle(W, **CFG)
    contracted = 0
    try:
        for x in (r, o):
            load_fill(x, sc)
        for b, comp in list(sc.warm) + [(sc.batch, None)]:
            out = r.route(r.device_batch(b))
            torch.cuda.synchronize()
            oi, orr, oh = o.route(b.cls, b.session, b.tok_off, b.tokens)
            n = b.n
            gi = out["inst"][:n].cpu().numpy()
            gh = out["hit_blocks"][:n].cpu().numpy()
            assert_equal("inst", gi, oi)
            assert_equal("reason", out["reason"][:n].cpu().numpy(), orr)
            assert_equal("hit_blocks", gh, oh)
            gc, oc = r.dump_caps(), o.caps()
            for k in ("K_w", "K_wb", "kbar_w"):
                assert_equal(k, gc[k], oc[k])
            r.commit()
            o.commit()
            L = np.diff(b.tok_off)
            # each side's window from its own outputs
            g_win = _window(gi, gh, L, W)
            o_win = _window(np.asarray(oi), np.asarray(oh), L, W)
            c_g = ctl_g.observe(*g_win, _k_base(gc, sc.cap_blocks, sc.protected_frac_q16))
            c_o = ctl_o.observe(*[list(map(int, x)) for x in o_win],
                                list(map(int, _k_base(oc, sc.cap_blocks, sc.protected_frac_q16))))
            assert list(c_g) == c_o
            contracted += int(np.count_nonzero(c_g))
            r.set_instance_state(contraction=c_g.astype(np.int32))
            o.set_instance_state(contraction=np.asarray(c_o, np.int32))
            if comp is not None:
                r.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
                o.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
        compare_state(r, o, W)
        r.sync()
    finally:
        r.close()
        ctl_g.close()
    return contracted


@pytest.mark.gpu
def test_controller_loop_config2():
    assert _run(wl.config2()) > 0


@pytest.mark.gpu
@pytest.mark.parametrize("seed", range(3))
def test_controller_loop_small_random(seed):
    sc = wl.small_random(800 + seed, W=4, cap=96, n=32, n_warm=10)
    _run(sc)
