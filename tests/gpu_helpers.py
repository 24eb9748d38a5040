"""GPU-vs-oracle drivers for the parity tests: one scenario is run step by step through
the CUDA library (C ABI via the binding) and through the CPU oracle on the same seeded
inputs, and every output is compared element by element."""

from __future__ import annotations

import os
import time

import numpy as np

import oracle
from tests.helpers import load_fill, make_oracle


def make_router(sc, **over):
    from paper_2608_11152_gb300 import misat

    kw = dict(max_batch=max(1, sc.max_batch), max_tokens=max(16, sc.max_tokens),
              protected_frac_q16=sc.protected_frac_q16, mode=sc.mode,
              hold_delay_q=sc.hold_delay_q, prior_kbar=sc.prior_kbar, prior_T_us=sc.prior_T_us)
    kw.update(over)
    r = misat.Router(sc.cap_blocks, **kw)
    r.set_mixture(sc.rho_ppm)
    r.set_instance_state(sc.backlog_q, sc.tokcost_q, sc.contraction)
    return r


def assert_equal(name, got, exp):
    got, exp = np.asarray(got), np.asarray(exp)
    assert got.shape == exp.shape, f"{name}: shape {got.shape} vs {exp.shape}"
    if not np.array_equal(got, exp):
        bad = np.argwhere(got != exp)
        i = tuple(bad[0])
        raise AssertionError(f"{name}: {len(bad)} mismatches, first at {i}: gpu {got[i]} oracle {exp[i]}")


def route_both(r, o, b, W, check_H=True, check_keys=True):
    import torch

    db = r.device_batch(b)
    H = torch.empty(max(1, b.n * W), dtype=torch.int16, device="cuda") if check_H else None
    out = r.route(db, out_H=H)
    torch.cuda.synchronize()
    oi, orr, oh = o.route(b.cls, b.session, b.tok_off, b.tokens)
    n = b.n
    assert_equal("inst", out["inst"][:n].cpu().numpy(), oi)
    assert_equal("reason", out["reason"][:n].cpu().numpy(), orr)
    assert_equal("hit_blocks", out["hit_blocks"][:n].cpu().numpy(), oh)
    if check_H and n:
        assert_equal("H", H[: n * W].cpu().numpy().view(np.uint16).reshape(n, W), o.H())
    if check_keys:
        cap = b.n_tokens // 16 + 1
        assert_equal("keys", r.dump_keys(cap), o.keys(cap))
    gc, oc = r.dump_caps(), o.caps()
    for k in ("K_w", "K_wb", "N_wb", "kbar_w", "kbar_b", "T_b"):
        assert_equal(k, gc[k], oc[k])
    s = r.stats()
    os_ = o.stats()
    assert_equal("reason counts", list(s.by_reason), os_[3:11])
    assert_equal("admitted by class", list(s.admitted_by_class), os_[11:14])
    assert s.hit_tokens == os_[17] and s.query_tokens == os_[18] and s.dtv_ppm == os_[19]
    return out


def compare_state(r, o, W, index=True):
    assert_equal("protected counts", r.dump_counts(), o.counts())
    gi, gs, gw, gcl = r.dump_sessions()
    oi, os_, ow, ocl = o.sessions()
    assert_equal("session ids", gi, oi)
    assert_equal("session state", gs, os_)
    assert_equal("session inst", gw, ow)
    assert_equal("session class", gcl, ocl)
    for w in range(W):
        assert r.index_size(w) == o.index_size(w), f"index size of instance {w}"
        if index:
            gk, gm = r.dump_index(w)
            ok_, om = o.dump_index(w)
            assert_equal(f"index keys w={w}", gk, ok_)
            assert_equal(f"index metas w={w}", gm, om)


_T0 = time.perf_counter()


def progress(msg):
    if os.environ.get("MISAT_TEST_VERBOSE"):
        print(f"[{time.perf_counter() - _T0:8.1f}s] {msg}", flush=True)


def run_parity(sc, index_every_step=True, check_H=True, check_keys=True, final_index=True, **router_over):
    """Run a whole scenario through both implementations, comparing every step."""
    r = make_router(sc, **router_over)
    o = make_oracle(sc)
    try:
        load_fill(r, sc)
        progress("gpu fill loaded")
        load_fill(o, sc)
        progress("oracle fill loaded")
        steps = list(sc.warm) + [(sc.batch, None)]
        for i, (b, comp) in enumerate(steps):
            route_both(r, o, b, sc.W, check_H=check_H, check_keys=check_keys)
            progress(f"batch {i} routed and compared")
            r.commit()
            progress(f"batch {i} gpu commit")
            o.commit()
            progress(f"batch {i} oracle commit")
            last = i == len(steps) - 1
            compare_state(r, o, sc.W, index=index_every_step or (final_index and last))
            progress(f"batch {i} state compared")
            s = r.stats()
            os_ = o.stats()
            assert s.new_keys == os_[21], f"new keys {s.new_keys} vs {os_[21]}"
            assert s.evicted == os_[22], f"evicted {s.evicted} vs {os_[22]}"
            assert o.check_invariants() == 0
            if comp is not None:
                r.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
                o.complete(comp.session, comp.cls, comp.total_blocks, comp.residency_us, comp.done)
        r.sync()
        return r, o
    except Exception:
        r.close()
        raise
