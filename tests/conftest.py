import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


def pytest_sessionstart(session):
    # A fresh checkout holds no binaries: build the C-ABI library (nvcc, sm_103a) and the
    # oracle's C part from source when they are missing or older than their sources.
    from paper_2004_09362_gb300 import build
    build.build()
    from oracle import column_reduce
    column_reduce.build()
