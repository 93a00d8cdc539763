"""Shared pytest configuration.

Tests marked ``gpu`` need a CUDA device (a GB300) and the package's compiled
library; everything else runs on the CPU. Markers are registered here so
``pytest -m gpu`` / ``-m "not gpu"`` select the two suites.
"""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line(
        "markers", "gpu: needs a CUDA GPU and the compiled CUDA library")
