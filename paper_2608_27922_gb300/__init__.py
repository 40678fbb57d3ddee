"""GB300-native DensityKV: per-head historical KV bank update and bank-reading attention.

The compute path is the CUDA library ``lib/libdkv.so`` (C ABI in ``include/dkv.h``);
``paper_2608_27922_gb300.dkv`` is its thin ctypes binding.  Importing this package
does not load the library; ``dkv.lib()`` does, and raises if it is missing.
"""
__all__ = ["dkv", "build"]
