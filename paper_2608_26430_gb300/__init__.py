"""GB300-native FrameFT adapter hot path (arxiv 2608.26430).

libframefb.so (C ABI, include/framefb.h) holds the frame and support
construction on the host and the sm_103a kernels; ``framefb`` is its thin
ctypes binding, ``batch`` assembles batched inputs and ``workloads`` defines
the seeded synthetic configurations.
"""
from . import framefb, workloads  # noqa: F401
