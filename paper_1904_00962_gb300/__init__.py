"""GB300 (sm_103a) LAMB / LARS optimizer step behind a C ABI.

`binding` is the ctypes layer over liblamb.so (include/lamb.h), `state` holds
the PyTorch device buffers, `workloads` generates the seeded synthetic
parameter layouts, and `build` compiles the library in-tree.
"""
from . import binding  # noqa: F401

__all__ = ["binding", "build", "state", "workloads"]
