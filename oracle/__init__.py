"""CPU oracle of the MISA-T batched routing decision -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s cpu_baseline /
reference leg may import this package.  The product path (the CUDA library and
its binding) never imports it and has no CPU fallback.

The oracle itself is plain single-threaded C++ (``misat_oracle.cpp``) built with
g++ into ``libmisat_oracle.so`` and driven through ctypes with numpy arrays.
It shares no source with the CUDA library.  Paper passages followed are listed
in the header of ``misat_oracle.cpp``.
"""

from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "misat_oracle.cpp")
_LIB = os.path.join(_HERE, "libmisat_oracle.so")
_lock = threading.Lock()
_lib = None

# error codes / modes / reasons (same numeric contract as include/misat.h)
OK = 0
ERR_INVALID_ARG = -1
ERR_STATE = -4

MODE_MISA_T, MODE_MISA, MODE_SESSION_ADMISSION, MODE_PLACEMENT_ONLY = 0, 1, 2, 3

ADMIT_CONT, ADMIT_NEW, ADMIT_FOLLOW = 1, 2, 3
HOLD_GLOBAL_CAP, HOLD_CLASS_CAP, HOLD_NO_ELIGIBLE, HOLD_PREFER_CACHE, HOLD_LEADER_HELD = 16, 17, 18, 19, 20

# stats vector layout
STAT_N, STAT_ADMITTED, STAT_HELD = 0, 1, 2
STAT_REASON0 = 3            # 8 reason counters, order CONT NEW FOLLOW GLOBAL CLASS NOELIG PREFER LEADERHELD
STAT_ADM_CLASS0 = 11
STAT_HELD_CLASS0 = 14
STAT_HIT_TOKENS, STAT_QUERY_TOKENS, STAT_DTV_PPM, STAT_LOOKUPS = 17, 18, 19, 20
STAT_NEW_KEYS, STAT_EVICTED, STAT_SEQ = 21, 22, 23


def build(force: bool = False) -> str:
    """Compile the oracle with g++ (portable flags; no -march)."""
    with _lock:
        if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
            return _LIB
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-o", tmp, _SRC])
        os.replace(tmp, _LIB)
        return _LIB


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = C.CDLL(_LIB)
    p, i32, i64, u64 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64
    sig = {
        "oracle_mix64": (u64, [u64]),
        "oracle_hash_prompt": (i64, [p, i64, u64, p]),
        "oracle_caps_eval": (C.c_int, [i64, p, p, p, i32, p, p, p]),
        "oracle_create": (p, [i32, p, i32, i32, i64, i32, i32, p, i64, u64]),
        "oracle_destroy": (None, [p]),
        "oracle_set_mixture": (C.c_int, [p, p]),
        "oracle_set_instance_state": (C.c_int, [p, p, p, p]),
        "oracle_route": (C.c_int, [p, i32, p, p, p, p, p, p, p]),
        "oracle_get_H": (C.c_int, [p, p]),
        "oracle_get_keys": (C.c_int, [p, p, i64, p]),
        "oracle_get_caps": (C.c_int, [p, p, p, p, p, p, p]),
        "oracle_get_stats": (C.c_int, [p, p]),
        "oracle_commit": (C.c_int, [p]),
        "oracle_complete": (C.c_int, [p, i32, p, p, p, p, p]),
        "oracle_evict": (C.c_int, [p, i32, p, i64]),
        "oracle_reset_instance": (C.c_int, [p, i32]),
        "oracle_load_entries": (C.c_int, [p, i32, p, p, i64]),
        "oracle_load_chains": (C.c_int, [p, i32, p, p, p, p, p, p]),
        "oracle_index_size": (i64, [p, i32]),
        "oracle_dump_index": (C.c_int, [p, i32, p, p, i64, p]),
        "oracle_get_counts": (C.c_int, [p, p]),
        "oracle_n_sessions": (i64, [p]),
        "oracle_dump_sessions": (C.c_int, [p, p, p, p, p, i64, p]),
        "oracle_seq": (u64, [p]),
        "oracle_check_invariants": (C.c_int, [p]),
        "oracle_clone": (p, [p]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _arr(x, dtype):
    return np.ascontiguousarray(np.asarray(x, dtype=dtype))


def mix64(z: int) -> int:
    return int(_load().oracle_mix64(C.c_uint64(z & 0xFFFFFFFFFFFFFFFF)))


def hash_prompt(tokens, seed: int = 0x9E3779B97F4A7C15) -> np.ndarray:
    t = _arr(tokens, np.int32)
    out = np.zeros(max(1, len(t) // 16), dtype=np.uint64)
    n = _load().oracle_hash_prompt(_ptr(t), len(t), C.c_uint64(seed), _ptr(out))
    return out[:n]


def caps_eval(Cw, N, kbar, T, mode=MODE_MISA_T, rho=(333334, 333333, 333333)):
    N, kb, Tb = _arr(N, np.int64), _arr(kbar, np.int64), _arr(T, np.int64)
    rh = _arr(rho, np.uint32)
    M = np.zeros(3, np.int64)
    K = np.zeros(3, np.int64)
    rc = _load().oracle_caps_eval(int(Cw), _ptr(N), _ptr(kb), _ptr(Tb), mode, _ptr(rh), _ptr(M), _ptr(K))
    if rc != OK:
        raise ValueError(rc)
    return M, K


class Oracle:
    """Owning handle of one oracle router state (host memory)."""

    def __init__(self, cap_blocks, protected_frac_q16=58982, mode=MODE_MISA_T,
                 hold_delay_q=0, hist_window=256, min_obs=8, prior_kbar=(64, 64, 64),
                 prior_T_us=30_000_000, hash_seed=0x9E3779B97F4A7C15):
        lib = _load()
        cap = _arr(cap_blocks, np.int64)
        pk = _arr(prior_kbar, np.int64)
        self.W = len(cap)
        self._h = lib.oracle_create(self.W, _ptr(cap), protected_frac_q16, mode, hold_delay_q,
                                    hist_window, min_obs, _ptr(pk), prior_T_us, C.c_uint64(hash_seed))
        if not self._h:
            raise ValueError("invalid oracle configuration")
        self._lib = lib
        self.n = 0

    def close(self):
        if getattr(self, "_h", None):
            self._lib.oracle_destroy(self._h)
            self._h = None

    __del__ = close

    def _check(self, rc):
        if rc != OK:
            raise RuntimeError(f"oracle error {rc}")

    def set_mixture(self, rho_ppm):
        self._check(self._lib.oracle_set_mixture(self._h, _ptr(_arr(rho_ppm, np.uint32))))

    def set_instance_state(self, backlog_q=None, tokcost_q=None, contraction=None):
        b = None if backlog_q is None else _arr(backlog_q, np.int64)
        t = None if tokcost_q is None else _arr(tokcost_q, np.int64)
        c = None if contraction is None else _arr(contraction, np.int32)
        self._check(self._lib.oracle_set_instance_state(self._h, _ptr(b), _ptr(t), _ptr(c)))

    def route(self, cls, session, tok_off, tokens):
        cls, ses = _arr(cls, np.uint8), _arr(session, np.uint64)
        off, tok = _arr(tok_off, np.int64), _arr(tokens, np.int32)
        n = len(cls)
        inst = np.zeros(n, np.int32)
        reason = np.zeros(n, np.uint8)
        hit = np.zeros(n, np.int32)
        rc = self._lib.oracle_route(self._h, n, _ptr(cls), _ptr(ses), _ptr(off), _ptr(tok),
                                    _ptr(inst), _ptr(reason), _ptr(hit))
        self._check(rc)
        self.n = n
        return inst, reason, hit

    def H(self):
        out = np.zeros((self.n, self.W), np.uint16)
        self._check(self._lib.oracle_get_H(self._h, _ptr(out)))
        return out

    def keys(self, cap):
        out = np.zeros(max(1, cap), np.uint64)
        n = C.c_int64(0)
        self._check(self._lib.oracle_get_keys(self._h, _ptr(out), cap, C.byref(n)))
        return out[: n.value]

    def caps(self):
        W = self.W
        Kw, kbw = np.zeros(W, np.int64), np.zeros(W, np.int64)
        Kwb, Nwb = np.zeros(W * 3, np.int64), np.zeros(W * 3, np.int64)
        kb, Tb = np.zeros(3, np.int64), np.zeros(3, np.int64)
        self._check(self._lib.oracle_get_caps(self._h, _ptr(Kw), _ptr(Kwb), _ptr(Nwb), _ptr(kbw),
                                              _ptr(kb), _ptr(Tb)))
        return dict(K_w=Kw, K_wb=Kwb.reshape(W, 3), N_wb=Nwb.reshape(W, 3), kbar_w=kbw,
                    kbar_b=kb, T_b=Tb)

    def stats(self):
        out = np.zeros(32, np.int64)
        self._check(self._lib.oracle_get_stats(self._h, _ptr(out)))
        return out

    def commit(self):
        self._check(self._lib.oracle_commit(self._h))

    def complete(self, session, cls, total_blocks, residency_us, done):
        ses, c = _arr(session, np.uint64), _arr(cls, np.uint8)
        tb, ru, d = _arr(total_blocks, np.int32), _arr(residency_us, np.int64), _arr(done, np.uint8)
        self._check(self._lib.oracle_complete(self._h, len(ses), _ptr(ses), _ptr(c), _ptr(tb),
                                              _ptr(ru), _ptr(d)))

    def evict(self, w, keys):
        k = _arr(keys, np.uint64)
        self._check(self._lib.oracle_evict(self._h, w, _ptr(k), len(k)))

    def reset_instance(self, w):
        self._check(self._lib.oracle_reset_instance(self._h, w))

    def load_entries(self, w, keys, metas):
        k, m = _arr(keys, np.uint64), _arr(metas, np.uint64)
        self._check(self._lib.oracle_load_entries(self._h, w, _ptr(k), _ptr(m), len(k)))

    def load_chains(self, tok_off, tokens, inst, seq, arr, max_blocks):
        off, tok = _arr(tok_off, np.int64), _arr(tokens, np.int32)
        i, s = _arr(inst, np.int32), _arr(seq, np.uint64)
        a, mb = _arr(arr, np.uint32), _arr(max_blocks, np.int32)
        self._check(self._lib.oracle_load_chains(self._h, len(i), _ptr(off), _ptr(tok), _ptr(i),
                                                 _ptr(s), _ptr(a), _ptr(mb)))

    def index_size(self, w):
        return int(self._lib.oracle_index_size(self._h, w))

    def dump_index(self, w):
        n = self.index_size(w)
        k, m = np.zeros(max(1, n), np.uint64), np.zeros(max(1, n), np.uint64)
        nn = C.c_int64(0)
        self._check(self._lib.oracle_dump_index(self._h, w, _ptr(k), _ptr(m), max(1, n), C.byref(nn)))
        return k[: nn.value], m[: nn.value]

    def counts(self):
        out = np.zeros(self.W * 3, np.int32)
        self._check(self._lib.oracle_get_counts(self._h, _ptr(out)))
        return out.reshape(self.W, 3)

    def sessions(self):
        n = int(self._lib.oracle_n_sessions(self._h))
        ids = np.zeros(max(1, n), np.uint64)
        st, ins, cl = (np.zeros(max(1, n), np.int32) for _ in range(3))
        nn = C.c_int64(0)
        self._check(self._lib.oracle_dump_sessions(self._h, _ptr(ids), _ptr(st), _ptr(ins), _ptr(cl),
                                                   max(1, n), C.byref(nn)))
        k = nn.value
        return ids[:k], st[:k], ins[:k], cl[:k]

    def seq(self):
        return int(self._lib.oracle_seq(self._h))

    def clone(self):
        """Deep copy of this oracle state."""
        o = object.__new__(Oracle)
        o._lib = self._lib
        o.W = self.W
        o.n = self.n
        o._h = self._lib.oracle_clone(self._h)
        return o

    def check_invariants(self):
        return int(self._lib.oracle_check_invariants(self._h))
