"""Shared pytest configuration.

Tests marked ``gpu`` need a CUDA device and the compiled RTCC library; every
other test runs on the CPU (oracle pins, host-side controller logic, symbol
export of the C library).
"""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU and the compiled library")
    config.addinivalue_line("markers", "slow: long-running CPU test")
