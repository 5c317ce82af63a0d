"""GB300-native marginal-cost routing simulator ("Calibrate, Then Route").

The compute path is the CUDA library ``libctr.so`` built from ``csrc/``; the
Python names below are thin ctypes marshalling over its C ABI
(``include/ctr.h``).  Importing the package does not load the library; the
first call of a ``ctr_*`` function does, and fails loudly if it is missing.
"""
__all__ = ["ctr_gen_trace", "ctr_score_batch", "ctr_simulate", "ctr_goodput", "ctr_workspace_bytes",
           "ctr_strerror", "CtrError"]


def __getattr__(name):
    if name in __all__:
        from . import ctr
        return getattr(ctr, name)
    raise AttributeError(name)
