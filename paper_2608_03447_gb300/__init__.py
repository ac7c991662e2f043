"""GB300-native verifier of Approximate Speculative Decoding (arXiv 2608.03447).

The compute lives in ``libasd.so`` (CUDA for sm_103a, C ABI declared in
``include/asd.h``); ``paper_2608_03447_gb300.asd`` is the thin ctypes binding
with the same entry-point names. Importing this package loads nothing: the
library is opened on first use and a missing library is an error, never a
fallback.
"""
