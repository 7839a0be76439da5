"""GB300-native contrastive-decoding (CD) verification step of Decoupled Contrastive Decoding.

The compute path is the C-ABI library ``libdcd.so`` (hand-written CUDA for sm_103a, declared in
``include/dcd.h``); ``paper_2608_12913_gb300.dcd`` is its thin ctypes binding with the same
entry-point names.  ``workloads`` holds the seeded synthetic input generators.
"""

import importlib

__all__ = ["dcd", "workloads"]


def __getattr__(name):
    if name in __all__:
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
