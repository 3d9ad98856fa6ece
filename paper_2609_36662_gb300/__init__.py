"""GB300-native outer synchronisation round of AutoLoCo (arxiv 2609.36662).

The product is the C-ABI library libaloco.so (include/aloco.h) built from
csrc/ for sm_103a; ``aloco`` is its ctypes binding and ``workloads`` draws
seeded synthetic inputs.  Importing the package does not load the library;
the first call into ``aloco`` does, and fails loudly if it is not built.
"""
from . import workloads  # noqa: F401

__all__ = ["aloco", "workloads", "build"]
