"""The C-ABI library builds for sm_103a, loads and exports every entry point that
include/misat.h declares (no compute calls: runs without a GPU)."""

import ctypes
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    txt = open(os.path.join(ROOT, "include", "misat.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(misat_[a-z_]+)\s*\(", txt)))


def test_header_declares_the_boundary():
    names = _declared()
    for must in ("misat_create", "misat_destroy", "misat_set_mixture", "misat_set_instance_state", "misat_route",
                 "misat_route_host", "misat_stage_host", "misat_route_staged", "misat_stage_host_delta",
                 "misat_commit", "misat_complete",
                 "misat_evict", "misat_reset_instance",
                 "misat_load_chains", "misat_load_entries", "misat_dump_index", "misat_stats", "misat_sync",
                 "misat_strerror"):
        assert must in names


def test_library_builds_loads_and_exports_every_declared_symbol():
    from paper_2608_11152_gb300 import build

    lib_path = build.build()
    lib = ctypes.CDLL(lib_path)
    for name in _declared():
        assert hasattr(lib, name), f"{name} declared in misat.h but not exported"
    from paper_2608_11152_gb300 import misat

    assert set(_declared()) == set(misat.EXPORTS)
    lib.misat_strerror.restype = ctypes.c_char_p
    assert lib.misat_strerror(-5) == b"table full"


def test_binding_rejects_bad_config_without_touching_the_gpu():
    """misat_create validates its arguments before any CUDA call."""
    from paper_2608_11152_gb300 import misat

    cfg = misat.misat_config()
    cfg.n_instances = 0
    h = ctypes.c_void_p()
    assert misat._lib.misat_create(ctypes.byref(cfg), None, ctypes.byref(h)) == misat.ERR_INVALID_ARG
    assert misat._lib.misat_commit(None) == misat.ERR_INVALID_ARG
