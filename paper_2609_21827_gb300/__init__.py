"""RheoSampling draft-tree sampling and verification on one GB300 (sm_103a).

The compute lives in ``librheo.so`` (hand-written CUDA, C ABI in
``include/rheo.h``); ``rheo`` is its ctypes binding and ``synth`` the seeded
synthetic workloads.  Build the library with ``build.build()``.
"""
from .rheo import (Config, Pruned, RheoError, Tree, VerifyOut, Workspace, expand, library_path, prune, status,
                   verify)

__all__ = ["Config", "Tree", "Pruned", "VerifyOut", "Workspace", "expand", "prune", "verify", "status",
           "RheoError", "library_path"]
