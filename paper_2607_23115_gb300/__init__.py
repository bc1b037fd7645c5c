"""GB300-native chunk-dedup hot path of Gleam's weight cache (paper Sec. 4.1.2).

The compute runs in libgleam.so (hand-written CUDA for sm_103a behind the C ABI
in include/gleam.h); this package is its thin ctypes binding plus the seeded
synthetic workload generators.  There is no CPU fallback: calling into the
binding without the built library raises.
"""
