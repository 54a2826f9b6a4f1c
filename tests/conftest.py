"""pytest configuration: the `gpu` marker and shared helpers.

Tests marked `gpu` need a CUDA device and the compiled library; everything
else runs on a CPU-only machine (`pytest -m "not gpu"`).
"""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU and the compiled sm_103a library")
    config.addinivalue_line("markers", "slow: full-size parity cases (seconds to minutes)")


def pytest_collection_modifyitems(config, items):
    """GPU tests fail loudly (not skip) when no device is present and they were asked for."""
    return None
