"""GB300-native (sm_103a) AdaPLD draft-construction step.

The compute path is the CUDA library ``libadapld.so`` (built from ``csrc/``)
behind a C ABI (``include/adapld.h``); :mod:`.native` is its thin ctypes
binding.  Importing the package does not load the library: the binding loads
it on first use and raises if it is missing.
"""
__all__ = ["native", "synth"]
