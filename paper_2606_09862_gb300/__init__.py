"""GB300-native Blurry Window Attention (BLA): chunked prefill, decode and backward.

The compute path is the CUDA library ``libbla_gb300.so`` (C ABI declared in
include/bla.h); ``paper_2606_09862_gb300.bla`` is its thin ctypes binding.
Importing this package does not load the library; the binding loads it on
first use and raises if it is missing.
"""
