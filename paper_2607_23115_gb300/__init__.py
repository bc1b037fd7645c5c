"""GB300-native chunk-dedup hot path of Gleam's weight cache (paper Sec. 4.1.2).

The compute runs in libgleam.so (hand-written CUDA for sm_103a behind the C ABI
in include/gleam.h); ``binding`` is its thin ctypes binding under the same
names, ``cache`` a convenience wrapper over it, and ``workloads`` the seeded
synthetic payload generators.  There is no CPU fallback: calling into the
binding without the built library raises.
"""
from . import binding  # noqa: F401  (loads nothing until first use)
