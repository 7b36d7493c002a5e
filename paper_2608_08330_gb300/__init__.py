"""GB300-native RTCC runtime: release-triggered communication-computation
coupling for multi-agent cooperative perception (arXiv 2608.08330).

The compute path is the C-ABI library built from ``csrc/`` (hand-written
sm_103a CUDA kernels plus a C++ host runtime); :mod:`.rtcc` is a thin ctypes
binding with the same names as ``include/rtcc.h``.  Importing the package does
not load the library; the binding loads it on first use and raises if it is
missing -- there is no CPU fallback.
"""
from . import build  # noqa: F401

__all__ = ["build", "rtcc"]
