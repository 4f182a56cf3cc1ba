"""Test configuration: the ``gpu`` marker, and the repository root and this
directory on sys.path (for ``oracle``, the package and ``oracle_pins``)."""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
for p in (ROOT, HERE):
    if p not in sys.path:
        sys.path.insert(0, p)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libblr.so")
