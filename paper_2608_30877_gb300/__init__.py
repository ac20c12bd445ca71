"""GB300 (sm_103a) group-wise int4 weight-only (W4A16) linear layers.

The compute lives in libw4a16.so (C ABI, include/w4a16.h); `w4a16` is its
thin Python binding and `synthetic` draws the seeded workloads.  Importing
the package loads nothing: the library is opened on first use.
"""
