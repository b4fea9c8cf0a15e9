"""GB300-native implementation of the data-parallel hot path of CPDP
(Controlled Periodic Data Parallelism with SlowMo momentum).

- ``cpdp``: binding of the C ABI in include/cpdp.h (libcpdp.so, CUDA, sm_103a)
- ``state.CPDPState``: W replicas on one GPU driven through that library
- ``workloads``: seeded synthetic inputs shaped like the paper's models
- ``build``: compiles libcpdp.so in-tree
"""
from . import cpdp, workloads  # noqa: F401

__all__ = ["cpdp", "workloads"]
