"""Thin ctypes binding of the MISA-T routing library (``include/misat.h``).

Argument marshalling only: every step of the routing decision runs in the CUDA
kernels of ``libmisat.so``.  There is no CPU fallback -- importing this module
without the built library raises.  Device buffers are torch CUDA tensors (PyTorch
is used for device memory and streams only).
"""

from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmisat.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(
        f"{LIB_PATH} is missing: build the CUDA library first "
        "(python -c 'import __graft_entry__ as g; g.build()').  There is no CPU fallback."
    )

_lib = C.CDLL(LIB_PATH)

OK = 0
ERR_INVALID_ARG, ERR_OOM, ERR_CUDA, ERR_STATE, ERR_TABLE_FULL, ERR_BATCH_TOO_LARGE = -1, -2, -3, -4, -5, -6
ERR_INTERNAL = -7
MODE_MISA_T, MODE_MISA, MODE_SESSION_ADMISSION, MODE_PLACEMENT_ONLY = 0, 1, 2, 3
PREFIX_GLOBAL, PREFIX_PER_INSTANCE = 0, 1
ADMIT_CONT, ADMIT_NEW, ADMIT_FOLLOW = 1, 2, 3
HOLD_GLOBAL_CAP, HOLD_CLASS_CAP, HOLD_NO_ELIGIBLE, HOLD_PREFER_CACHE, HOLD_LEADER_HELD = 16, 17, 18, 19, 20

_p = C.c_void_p


class misat_config(C.Structure):
    _fields_ = [("n_instances", C.c_int32), ("cap_blocks", _p), ("protected_frac_q16", C.c_int32),
                ("mode", C.c_int32), ("max_batch", C.c_int32), ("max_tokens", C.c_int64),
                ("max_sessions", C.c_int32), ("hist_window", C.c_int32), ("min_obs", C.c_int32),
                ("hold_delay_q", C.c_int64), ("prior_kbar_blocks", C.c_int64 * 3), ("prior_T_us", C.c_int64),
                ("hash_seed", C.c_uint64), ("table_load", C.c_double), ("prefix_index", C.c_int32)]


class misat_batch(C.Structure):
    _fields_ = [("n", C.c_int32), ("n_tokens", C.c_int64), ("cls", _p), ("session", _p), ("group", _p),
                ("tok_off", _p), ("tokens", _p), ("out_H", _p)]


class misat_batch_delta(C.Structure):
    _fields_ = [("n", C.c_int32), ("cls", _p), ("session", _p), ("base", _p), ("delta_off", _p),
                ("delta_tokens", _p)]


class misat_decisions(C.Structure):
    _fields_ = [("inst", _p), ("reason", _p), ("hit_blocks", _p)]


class misat_entry(C.Structure):
    _fields_ = [("key", C.c_uint64), ("meta", C.c_uint64)]


class misat_batch_stats(C.Structure):
    _fields_ = [("n_requests", C.c_int64), ("n_admitted", C.c_int64), ("n_held", C.c_int64),
                ("by_reason", C.c_int64 * 8), ("admitted_by_class", C.c_int64 * 3),
                ("held_by_class", C.c_int64 * 3), ("hit_tokens", C.c_int64), ("query_tokens", C.c_int64),
                ("dtv_ppm", C.c_int64), ("probes", C.c_int64), ("bucket_reads", C.c_int64),
                ("probes_first", C.c_int64), ("bucket_reads_first", C.c_int64),
                ("new_keys", C.c_int64), ("evicted", C.c_int64), ("seq", C.c_int64),
                ("insert_ops", C.c_int64), ("joint_selection", C.c_int64),
                ("first_block_keys", C.c_int64), ("first_block_lookups", C.c_int64)]


class misat_overload_config(C.Structure):
    _fields_ = [("ref_windows", C.c_int32), ("min_ref", C.c_int32), ("gap_ppm", C.c_int32), ("confirm", C.c_int32),
                ("queue_thresh", C.c_int64), ("recover_after", C.c_int32), ("max_contraction_pct", C.c_int32)]


PHASES = ("prologue", "hash", "caps", "probe_first", "probe_search", "select", "finalize", "insert",
          "sessions", "evict", "gix_insert", "evict_estimate", "evict_collect", "evict_select", "evict_delete",
          "evict_shift")


_SIG = {
    "misat_create": [C.POINTER(misat_config), _p, C.POINTER(_p)],
    "misat_destroy": [_p],
    "misat_set_mixture": [_p, _p],
    "misat_set_instance_state": [_p, _p, _p, _p],
    "misat_route": [_p, C.POINTER(misat_batch), C.POINTER(misat_decisions)],
    "misat_route_host": [_p, C.POINTER(misat_batch), C.POINTER(misat_decisions)],
    "misat_stage_host": [_p, C.POINTER(misat_batch), C.c_int32],
    "misat_route_staged": [_p, C.c_int32, C.POINTER(misat_decisions)],
    "misat_stage_host_delta": [_p, C.POINTER(misat_batch_delta), C.c_int32],
    "misat_commit": [_p],
    "misat_complete": [_p, C.c_int32, _p, _p, _p, _p, _p],
    "misat_evict": [_p, C.c_int32, _p, C.c_int64],
    "misat_reset_instance": [_p, C.c_int32],
    "misat_load_chains": [_p, C.c_int32, _p, _p, _p, _p, _p, _p],
    "misat_load_entries": [_p, C.c_int32, _p, C.c_int64],
    "misat_index_size": [_p, C.c_int32, C.POINTER(C.c_int64)],
    "misat_index_buckets": [_p, C.c_int32, C.POINTER(C.c_int64)],
    "misat_dump_index": [_p, C.c_int32, _p, C.c_int64, C.POINTER(C.c_int64)],
    "misat_dump_keys": [_p, _p, C.c_int64, C.POINTER(C.c_int64)],
    "misat_dump_caps": [_p, _p, _p, _p, _p, _p, _p],
    "misat_dump_counts": [_p, _p],
    "misat_dump_sessions": [_p, _p, _p, _p, _p, C.c_int64, C.POINTER(C.c_int64)],
    "misat_stats": [_p, C.POINTER(misat_batch_stats)],
    "misat_global_info": [_p, C.POINTER(C.c_int32), C.POINTER(C.c_int64), C.POINTER(C.c_int64)],
    "misat_global_dump": [_p, _p, _p, C.c_int64, C.POINTER(C.c_int64)],
    "misat_global_rebuild": [_p],
    "misat_sync": [_p],
    "misat_checkpoint_save": [_p, C.POINTER(_p)],
    "misat_checkpoint_restore": [_p, _p],
    "misat_checkpoint_free": [_p],
    "misat_set_timing": [_p, C.c_int],
    "misat_phase_times": [_p, _p],
    "misat_block_hash_noalloc": [_p, _p, C.c_int32, C.c_int64, C.c_uint64, _p, C.c_int64, _p],
    "misat_overload_create": [C.c_int32, C.POINTER(misat_overload_config), C.POINTER(_p)],
    "misat_overload_destroy": [_p],
    "misat_overload_observe": [_p, _p, _p, _p, _p, _p],
    "misat_recheck_delays": [C.c_int32, _p, _p, C.c_int64, C.c_int64, _p],
}
NOALLOC_MAX_REQUESTS = 65536


def block_hash_noalloc(tok_off, tokens, n, n_tokens, keys_out, seed=0x9E3779B97F4A7C15, stream=None):
    """Chained block keys of a device batch, written in request order into the device tensor
    ``keys_out``, without any device allocation (misat_block_hash_noalloc)."""
    import torch

    st = stream if stream is not None else torch.cuda.current_stream()
    _ck(_lib.misat_block_hash_noalloc(_tptr(tok_off), _tptr(tokens), int(n), int(n_tokens), seed,
                                      _tptr(keys_out), int(keys_out.numel()), _p(st.cuda_stream)),
        "misat_block_hash_noalloc")
for _name, _args in _SIG.items():
    _f = getattr(_lib, _name)
    _f.argtypes = _args
    _f.restype = C.c_int
_lib.misat_strerror.argtypes = [C.c_int]
_lib.misat_strerror.restype = C.c_char_p

_lib.misat_overload_default_config.argtypes = [C.POINTER(misat_overload_config)]
_lib.misat_overload_default_config.restype = None
EXPORTS = sorted(list(_SIG) + ["misat_strerror", "misat_overload_default_config"])


class MisatError(RuntimeError):
    def __init__(self, code, where):
        self.code = code
        super().__init__(f"{where}: {_lib.misat_strerror(code).decode()} ({code})")


def _ck(code, where):
    if code != OK:
        raise MisatError(code, where)


def _np(x, dtype):
    return np.ascontiguousarray(np.asarray(x, dtype=dtype))


def _nptr(a):
    return None if a is None else a.ctypes.data_as(_p)


def _tptr(t):
    return None if t is None else _p(t.data_ptr())


def pack_meta(seq, arrival, depth):
    """Index entry metadata: seq<<36 | arrival<<16 | (65535 - depth)."""
    return (int(seq) << 36) | (int(arrival) << 16) | (65535 - int(depth))


class Router:
    """One MISA-T routing context on the current CUDA device (see include/misat.h)."""

    def __init__(self, cap_blocks, *, max_batch, max_tokens, max_sessions=None, protected_frac_q16=58982,
                 mode=MODE_MISA_T, hold_delay_q=0, hist_window=256, min_obs=8,
                 prior_kbar=(64, 64, 64), prior_T_us=30_000_000, hash_seed=0x9E3779B97F4A7C15,
                 table_load=0.75, prefix_index=None, stream=None):
        import torch

        self._torch = torch
        cap = _np(cap_blocks, np.int64)
        self.W = len(cap)
        self._cap = cap
        cfg = misat_config()
        cfg.n_instances = self.W
        cfg.cap_blocks = _nptr(cap)
        cfg.protected_frac_q16 = protected_frac_q16
        cfg.mode = mode
        cfg.max_batch = int(max_batch)
        cfg.max_tokens = int(max(16, max_tokens))
        cfg.max_sessions = int(max_sessions or max(1024, 4 * max_batch))
        cfg.hist_window = hist_window
        cfg.min_obs = min_obs
        cfg.hold_delay_q = int(hold_delay_q)
        for b in range(3):
            cfg.prior_kbar_blocks[b] = int(prior_kbar[b])
        cfg.prior_T_us = int(prior_T_us)
        cfg.hash_seed = hash_seed
        cfg.table_load = table_load
        cfg.prefix_index = PREFIX_GLOBAL if prefix_index is None else int(prefix_index)
        self.prefix_index = cfg.prefix_index
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        h = _p()
        _ck(_lib.misat_create(C.byref(cfg), _p(self.stream.cuda_stream), C.byref(h)), "misat_create")
        self._h = h
        self.max_batch = int(max_batch)

    def close(self):
        if getattr(self, "_h", None):
            _lib.misat_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ---- configuration / state inputs
    def set_mixture(self, rho_ppm):
        _ck(_lib.misat_set_mixture(self._h, _nptr(_np(rho_ppm, np.uint32))), "misat_set_mixture")

    def set_instance_state(self, backlog_q=None, tokcost_q=None, contraction=None):
        b = None if backlog_q is None else _np(backlog_q, np.int64)
        t = None if tokcost_q is None else _np(tokcost_q, np.int64)
        c = None if contraction is None else _np(contraction, np.int32)
        _ck(_lib.misat_set_instance_state(self._h, _nptr(b), _nptr(t), _nptr(c)), "misat_set_instance_state")

    # ---- routing
    def device_batch(self, batch, device="cuda"):
        """Copy a workload Batch (numpy) to device tensors."""
        torch = self._torch
        return dict(
            n=batch.n, n_tokens=batch.n_tokens,
            cls=torch.from_numpy(batch.cls).to(device),
            session=torch.from_numpy(batch.session.view(np.int64)).to(device),
            tok_off=torch.from_numpy(batch.tok_off).to(device),
            tokens=torch.from_numpy(batch.tokens).to(device) if batch.n_tokens else
            torch.zeros(4, dtype=torch.int32, device=device),
        )

    def alloc_decisions(self, n, device="cuda"):
        torch = self._torch
        return dict(inst=torch.empty(max(1, n), dtype=torch.int32, device=device),
                    reason=torch.empty(max(1, n), dtype=torch.uint8, device=device),
                    hit_blocks=torch.empty(max(1, n), dtype=torch.int32, device=device))

    def route(self, db, out=None, out_H=None):
        """Route a device batch (dict of tensors from device_batch).  Async on the stream."""
        n = db["n"]
        if out is None:
            out = self.alloc_decisions(n)
        b = misat_batch(n, db["n_tokens"], _tptr(db["cls"]), _tptr(db["session"]), None, _tptr(db["tok_off"]),
                        _tptr(db["tokens"]), _tptr(out_H))
        d = misat_decisions(_tptr(out["inst"]), _tptr(out["reason"]), _tptr(out["hit_blocks"]))
        _ck(_lib.misat_route(self._h, C.byref(b), C.byref(d)), "misat_route")
        return out

    def route_host(self, batch, out=None):
        """Route a host batch (numpy arrays, pinned recommended); returns numpy decisions."""
        n = batch.n
        if out is None:
            out = dict(inst=np.empty(max(1, n), np.int32), reason=np.empty(max(1, n), np.uint8),
                       hit_blocks=np.empty(max(1, n), np.int32))
        cls, ses, off, tok = batch.cls, batch.session, batch.tok_off, batch.tokens
        b = misat_batch(n, batch.n_tokens, _nptr(cls), _nptr(ses), None, _nptr(off), _nptr(tok), None)
        d = misat_decisions(_nptr(out["inst"]), _nptr(out["reason"]), _nptr(out["hit_blocks"]))
        _ck(_lib.misat_route_host(self._h, C.byref(b), C.byref(d)), "misat_route_host")
        return out

    def stage_host(self, batch, slot):
        """Start the copy of a host batch (numpy arrays, pinned for asynchrony) into staging
        slot 0 or 1; returns at once.  The arrays are kept referenced until the slot is routed."""
        cls, ses, off, tok = batch.cls, batch.session, batch.tok_off, batch.tokens
        b = misat_batch(batch.n, batch.n_tokens, _nptr(cls), _nptr(ses), None, _nptr(off), _nptr(tok), None)
        _ck(_lib.misat_stage_host(self._h, C.byref(b), int(slot)), "misat_stage_host")
        if not hasattr(self, "_staged"):
            self._staged = {}
        self._staged[int(slot)] = (batch.n, cls, ses, off, tok)

    def stage_host_delta(self, enc, slot):
        """stage_host for a delta-encoded batch (workload.DeltaBatch: numpy arrays, pinned for
        asynchrony); the arrays are kept referenced until the slot is routed."""
        b = misat_batch_delta(enc.n, _nptr(enc.cls), _nptr(enc.session), _nptr(enc.base), _nptr(enc.delta_off),
                              _nptr(enc.delta_tokens))
        _ck(_lib.misat_stage_host_delta(self._h, C.byref(b), int(slot)), "misat_stage_host_delta")
        if not hasattr(self, "_staged"):
            self._staged = {}
        self._staged[int(slot)] = (enc.n, enc.cls, enc.session, enc.base, enc.delta_off, enc.delta_tokens)

    def route_staged(self, slot, out=None):
        """Route the batch staged in `slot`; returns numpy decisions (written into `out` if given)."""
        n = self._staged[int(slot)][0] if getattr(self, "_staged", None) and int(slot) in self._staged else 0
        if out is None:
            out = dict(inst=np.empty(max(1, n), np.int32), reason=np.empty(max(1, n), np.uint8),
                       hit_blocks=np.empty(max(1, n), np.int32))
        d = misat_decisions(_nptr(out["inst"]), _nptr(out["reason"]), _nptr(out["hit_blocks"]))
        try:
            _ck(_lib.misat_route_staged(self._h, int(slot), C.byref(d)), "misat_route_staged")
        finally:
            if getattr(self, "_staged", None):
                self._staged.pop(int(slot), None)
        return out

    def commit(self):
        _ck(_lib.misat_commit(self._h), "misat_commit")

    def complete(self, session, cls, total_blocks, residency_us, done):
        s, c = _np(session, np.uint64), _np(cls, np.uint8)
        tb, ru, dn = _np(total_blocks, np.int32), _np(residency_us, np.int64), _np(done, np.uint8)
        _ck(_lib.misat_complete(self._h, len(s), _nptr(s), _nptr(c), _nptr(tb), _nptr(ru), _nptr(dn)),
            "misat_complete")

    def evict(self, w, keys):
        k = _np(keys, np.uint64)
        _ck(_lib.misat_evict(self._h, w, _nptr(k), len(k)), "misat_evict")

    def reset_instance(self, w):
        _ck(_lib.misat_reset_instance(self._h, w), "misat_reset_instance")

    def load_chains(self, tok_off, tokens, inst, seq, arr, max_blocks):
        off, tok = _np(tok_off, np.int64), _np(tokens, np.int32)
        i, s, a, mb = _np(inst, np.int32), _np(seq, np.uint64), _np(arr, np.uint32), _np(max_blocks, np.int32)
        _ck(_lib.misat_load_chains(self._h, len(i), _nptr(off), _nptr(tok), _nptr(i), _nptr(s), _nptr(a),
                                   _nptr(mb)), "misat_load_chains")

    def load_entries(self, w, keys, metas):
        e = np.empty(len(keys), dtype=[("key", np.uint64), ("meta", np.uint64)])
        e["key"] = _np(keys, np.uint64)
        e["meta"] = _np(metas, np.uint64)
        _ck(_lib.misat_load_entries(self._h, w, _nptr(e), len(e)), "misat_load_entries")

    # ---- state dumps
    def index_size(self, w):
        v = C.c_int64(0)
        _ck(_lib.misat_index_size(self._h, w, C.byref(v)), "misat_index_size")
        return v.value

    def table_buckets(self, w):
        v = C.c_int64(0)
        _ck(_lib.misat_index_buckets(self._h, w, C.byref(v)), "misat_index_buckets")
        return int(v.value)

    def dump_index(self, w):
        cap = self.index_size(w) + 16
        e = np.empty(cap, dtype=[("key", np.uint64), ("meta", np.uint64)])
        n = C.c_int64(0)
        _ck(_lib.misat_dump_index(self._h, w, _nptr(e), cap, C.byref(n)), "misat_dump_index")
        e = e[: n.value]
        return np.ascontiguousarray(e["key"]), np.ascontiguousarray(e["meta"])

    def dump_keys(self, cap):
        out = np.empty(max(1, cap), np.uint64)
        n = C.c_int64(0)
        _ck(_lib.misat_dump_keys(self._h, _nptr(out), cap, C.byref(n)), "misat_dump_keys")
        return out[: n.value]

    def dump_caps(self):
        W = self.W
        Kw, kbw = np.empty(W, np.int64), np.empty(W, np.int64)
        Kwb, Nwb = np.empty(W * 3, np.int64), np.empty(W * 3, np.int64)
        kb, Tb = np.empty(3, np.int64), np.empty(3, np.int64)
        _ck(_lib.misat_dump_caps(self._h, _nptr(Kw), _nptr(Kwb), _nptr(Nwb), _nptr(kbw), _nptr(kb), _nptr(Tb)),
            "misat_dump_caps")
        return dict(K_w=Kw, K_wb=Kwb.reshape(W, 3), N_wb=Nwb.reshape(W, 3), kbar_w=kbw, kbar_b=kb, T_b=Tb)

    def dump_counts(self):
        out = np.empty(self.W * 3, np.int32)
        _ck(_lib.misat_dump_counts(self._h, _nptr(out)), "misat_dump_counts")
        return out.reshape(self.W, 3)

    def dump_sessions(self, cap=None):
        cap = cap or 4 * self.max_batch + 1024
        while True:
            ids = np.empty(cap, np.uint64)
            st, ins, cl = (np.empty(cap, np.int32) for _ in range(3))
            n = C.c_int64(0)
            rc = _lib.misat_dump_sessions(self._h, _nptr(ids), _nptr(st), _nptr(ins), _nptr(cl), cap, C.byref(n))
            if rc == ERR_INVALID_ARG and n.value > cap:
                cap = n.value
                continue
            _ck(rc, "misat_dump_sessions")
            k = n.value
            return ids[:k], st[:k], ins[:k], cl[:k]

    def stats(self):
        s = misat_batch_stats()
        _ck(_lib.misat_stats(self._h, C.byref(s)), "misat_stats")
        return s

    # ---- global prefix index (Sec. 4.4: block hash -> instances caching it)
    def global_info(self):
        """(mask words per key, slots, claimed slots) of the global prefix index."""
        mw, slots, used = C.c_int32(0), C.c_int64(0), C.c_int64(0)
        _ck(_lib.misat_global_info(self._h, C.byref(mw), C.byref(slots), C.byref(used)), "misat_global_info")
        return mw.value, slots.value, used.value

    def global_dump(self):
        """Keys with a non-empty instance mask and their masks [n, mask words] (unordered)."""
        mw = self.global_info()[0]
        n = C.c_int64(0)
        _ck(_lib.misat_global_dump(self._h, None, None, 0, C.byref(n)), "misat_global_dump")
        cap = n.value + 16
        keys = np.empty(cap, np.uint64)
        masks = np.empty(cap * mw, np.uint64)
        _ck(_lib.misat_global_dump(self._h, _nptr(keys), _nptr(masks), cap, C.byref(n)), "misat_global_dump")
        k = n.value
        return keys[:k], masks[: k * mw].reshape(k, mw)

    def global_rebuild(self):
        _ck(_lib.misat_global_rebuild(self._h), "misat_global_rebuild")

    def sync(self):
        _ck(_lib.misat_sync(self._h), "misat_sync")

    # ---- checkpoint / timing
    def checkpoint_save(self):
        k = _p()
        _ck(_lib.misat_checkpoint_save(self._h, C.byref(k)), "misat_checkpoint_save")
        return Checkpoint(k)

    def checkpoint_restore(self, ckpt):
        _ck(_lib.misat_checkpoint_restore(self._h, ckpt._k), "misat_checkpoint_restore")

    def set_timing(self, enable=True):
        _ck(_lib.misat_set_timing(self._h, 1 if enable else 0), "misat_set_timing")

    def phase_times(self):
        out = np.zeros(len(PHASES), np.float32)
        _ck(_lib.misat_phase_times(self._h, _nptr(out)), "misat_phase_times")
        return dict(zip(PHASES, out.tolist()))


class Checkpoint:
    """Device-resident router state snapshot (misat_checkpoint_*)."""

    def __init__(self, k):
        self._k = k

    def free(self):
        if getattr(self, "_k", None):
            _lib.misat_checkpoint_free(self._k)
            self._k = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def _np_ptr(a):
    return _p(a.ctypes.data)


def overload_default_config() -> dict:
    """The library's default overload-controller thresholds (misat_overload_default_config)."""
    c = misat_overload_config()
    _lib.misat_overload_default_config(C.byref(c))
    return {f: getattr(c, f) for f, _ in misat_overload_config._fields_}


class OverloadController:
    """Per-instance overload pressure (Sec. 4.1) on the host: one observe() per window returns
    the cap contraction to pass to Router.set_instance_state (misat_overload_*)."""

    def __init__(self, n_instances: int, **cfg):
        conf = overload_default_config()
        conf.update(cfg)
        c = misat_overload_config(**conf)
        self.W = int(n_instances)
        h = _p()
        _ck(_lib.misat_overload_create(self.W, C.byref(c), C.byref(h)), "misat_overload_create")
        self._h = h

    def observe(self, hit_tokens, query_tokens, waiting, k_base) -> np.ndarray:
        arrs = [np.ascontiguousarray(x, dtype=np.int64) for x in (hit_tokens, query_tokens, waiting, k_base)]
        for x in arrs:
            if x.shape != (self.W,):
                raise ValueError("observe: every array must have one entry per instance")
        out = np.zeros(self.W, dtype=np.int32)
        _ck(_lib.misat_overload_observe(self._h, *[_np_ptr(x) for x in arrs], _np_ptr(out)), "misat_overload_observe")
        return out

    def close(self):
        if self._h:
            _lib.misat_overload_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def recheck_delays(group, held, base_delay_us: int, min_delay_us: int) -> np.ndarray:
    """Recheck delay per request of the scheduler's current view (misat_recheck_delays)."""
    g = np.ascontiguousarray(group, dtype=np.uint64)
    h = np.ascontiguousarray(held, dtype=np.uint8)
    if g.shape != h.shape or g.ndim != 1:
        raise ValueError("recheck_delays: group and held must be 1-d arrays of one length")
    out = np.zeros(g.shape[0], dtype=np.int64)
    _ck(_lib.misat_recheck_delays(int(g.shape[0]), _np_ptr(g), _np_ptr(h), int(base_delay_us), int(min_delay_us),
                                  _np_ptr(out)), "misat_recheck_delays")
    return out
