"""GB300 (sm_103a) library for forced-weight subset evaluation
("Trust the Mass: Forced Weights in KV-Cache Eviction").

The computation lives in libfw.so (CUDA kernels behind the C ABI declared in
include/fw.h); ``paper_2608_25230_gb300.fw`` is its ctypes binding.
"""
from ._build import build  # noqa: F401
