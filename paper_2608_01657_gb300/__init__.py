"""GB300-native batched prefix-cache step of PrefixShield (arXiv 2608.01657).

The compute path is the CUDA library ``libprefixshield.so`` (C ABI declared in
``include/prefixshield.h``); ``binding`` is its thin ctypes layer.  Importing
this package does not load the library: ``binding.load()`` does, and it fails
loudly when the library has not been built.
"""
__all__ = ["binding", "workloads", "build"]
