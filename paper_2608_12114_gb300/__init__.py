"""File-backed weight ingest and the bandwidth-bound GEMV pass on GB300 (sm_103a).

``wt``     ctypes binding of libwt.so, the C ABI declared in include/wt.h
``build``  compiles libwt.so in-tree with nvcc
``synth``  seeded synthetic checkpoints (input generation only)
"""
from . import build, wt  # noqa: F401
