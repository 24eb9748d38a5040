import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running oracle case")
    # test modules import the binding, which needs the in-tree library: build it (nvcc
    # cross-compiles without a GPU) when it is missing or older than its sources, so that a
    # fresh checkout collects; a failed build leaves the binding's own import error to report
    try:
        from paper_2608_11152_gb300 import build

        build.build()
    except Exception as e:  # pragma: no cover
        sys.stderr.write(f"[conftest] building the CUDA library failed: {e}\n")
