"""GB300 (sm_103a) batched verification for DiP-SD edge servers (arXiv 2604.20919).

The compute lives in libdipsd.so (C ABI: include/dipsd.h); `dipsd` is its
Python binding.  Importing this package loads nothing; `dipsd.load()` does.
"""
__all__ = ["dipsd", "build"]
