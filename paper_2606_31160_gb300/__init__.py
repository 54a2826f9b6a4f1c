"""GB300-native verify step of two-reasoner speculative decoding.

The compute lives in the C-ABI library libsd.so (sources in csrc/, header in
include/sd.h at the repository root); this package holds its ctypes binding
(`sd`), the in-tree build (`build`) and the seeded synthetic workloads
(`workloads`).
"""
