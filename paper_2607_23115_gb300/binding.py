"""ctypes binding of libgleam.so: the C ABI of include/gleam.h under the same
names, argument marshalling only.  Device buffers may be passed as torch
tensors (their data_ptr() is used) or as raw integer addresses; streams as
torch.cuda.Stream objects, raw handles or None (legacy default stream).

There is no fallback: if libgleam.so has not been built, every call raises.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libgleam.so")

GLEAM_OK = 0
GLEAM_ERR_INVALID_ARG = -1
GLEAM_ERR_NOT_DEVICE_PTR = -2
GLEAM_ERR_CUDA = -3
GLEAM_ERR_CAPACITY = -4
GLEAM_ERR_TIMEOUT = -5
GLEAM_ERR_NOMEM = -6
GLEAM_ERR_INTERNAL = -7

GLEAM_KEY16 = 0x1
GLEAM_DEBUG_CHECKS = 0x2
GLEAM_PAPER_IDS = 0x4
GLEAM_EVICT_LRU = 0x8
GLEAM_OVERLAP_CALLS = 0x10
GLEAM_DEBUG_WAIT_LIMIT_NS = 1
GLEAM_DEBUG_SKIP_ARRIVE = 2
GLEAM_DEBUG_CLOCK = 3
GLEAM_DEBUG_DROP_ENTRY = 4
GLEAM_DEBUG_SMALL_CALLS = 5
GLEAM_DEBUG_SPECULATE = 6

# Every symbol include/gleam.h declares (checked by the ABI test).
EXPORTS = (
    "gleam_cache_create", "gleam_cache_create_ex", "gleam_cache_destroy",
    "gleam_cache_reserve", "gleam_fingerprint", "gleam_dedup_copy",
    "gleam_dedup_copy_async", "gleam_dedup_copy_batch", "gleam_dedup_copy_noalloc",
    "gleam_dedup_copy_host_async", "gleam_dedup_copy_host_batch", "gleam_block_check",
    "gleam_cache_stats", "gleam_cache_export",
    "gleam_cache_read_slot", "gleam_cache_debug_insert", "gleam_cache_debug_set",
    "gleam_cache_snapshot", "gleam_cache_restore", "gleam_snapshot_destroy",
    "gleam_cache_profile", "gleam_cache_profile_read", "gleam_status_string",
)


class gleam_stats_t(ctypes.Structure):
    _fields_ = [(f, ctypes.c_uint64) for f in (
        "calls", "chunks", "hits_cache", "hits_intra", "misses", "inserts",
        "verify_rejects", "slots_used", "bytes_used", "capacity_bytes", "nslots",
        "chunk_bytes", "evictions", "spec_chunks")]


class gleam_payload_t(ctypes.Structure):
    _fields_ = [("d_buf", ctypes.c_void_p), ("n", ctypes.c_size_t),
                ("d_hit_mask", ctypes.c_void_p), ("d_miss_idx", ctypes.c_void_p),
                ("d_miss_bytes", ctypes.c_void_p), ("d_result", ctypes.c_void_p),
                ("d_chunk_slot", ctypes.c_void_p)]


RESULT_FIELDS = ("status", "n_miss", "n_hit_cache", "n_hit_intra", "verify_rejects",
                 "miss_bytes")
RESULT_WORDS = len(RESULT_FIELDS)  # gleam_result_t = 6 x 64-bit words


class GleamError(RuntimeError):
    def __init__(self, rc: int, what: str = ""):
        self.rc = rc
        super().__init__("%s: %s (%d)" % (what or "gleam", gleam_status_string(rc), rc))


_lib = None


def lib() -> ctypes.CDLL:
    """Loads libgleam.so (raises if it was not built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(
            "libgleam.so is not built (expected at %s); run __graft_entry__.build() or "
            "python paper_2607_23115_gb300/build.py -- there is no CPU fallback" % LIB_PATH)
    l = ctypes.CDLL(LIB_PATH)
    vp, sz, u64, i32 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_uint64, ctypes.c_int
    sig = {
        "gleam_cache_create": (i32, [sz, sz, ctypes.POINTER(vp)]),
        "gleam_cache_create_ex": (i32, [sz, sz, ctypes.c_uint32, ctypes.POINTER(vp)]),
        "gleam_cache_destroy": (None, [vp]),
        "gleam_cache_reserve": (i32, [vp, u64]),
        "gleam_fingerprint": (i32, [vp, sz, sz, vp, vp]),
        "gleam_dedup_copy": (ctypes.c_int64, [vp, vp, sz, vp, vp, vp]),
        "gleam_dedup_copy_async": (i32, [vp, vp, sz, vp, vp, vp, vp, vp]),
        "gleam_dedup_copy_batch": (i32, [vp, ctypes.POINTER(gleam_payload_t), sz, vp, vp]),
        "gleam_dedup_copy_noalloc": (i32, [vp, vp, sz, vp, vp, vp, vp, vp]),
        "gleam_dedup_copy_host_async": (i32, [vp, vp, sz, vp, vp, vp, vp, vp]),
        "gleam_dedup_copy_host_batch": (i32, [vp, ctypes.POINTER(gleam_payload_t), sz, vp, vp]),
        "gleam_block_check": (i32, [vp, vp, sz, vp, vp, sz, vp, vp, vp]),
        "gleam_cache_stats": (i32, [vp, ctypes.POINTER(gleam_stats_t)]),
        "gleam_cache_export": (i32, [vp, vp, vp, u64, ctypes.POINTER(u64)]),
        "gleam_cache_read_slot": (i32, [vp, u64, vp, u64, ctypes.POINTER(u64)]),
        "gleam_cache_debug_insert": (i32, [vp, u64, vp, sz]),
        "gleam_cache_debug_set": (i32, [vp, i32, ctypes.c_int64]),
        "gleam_cache_snapshot": (i32, [vp, ctypes.POINTER(vp)]),
        "gleam_cache_restore": (i32, [vp, vp]),
        "gleam_snapshot_destroy": (None, [vp]),
        "gleam_cache_profile": (i32, [vp, i32]),
        "gleam_cache_profile_read": (i32, [vp, vp, vp, i32]),
        "gleam_status_string": (ctypes.c_char_p, [i32]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(l, name)
        fn.restype = res
        fn.argtypes = args
    _lib = l
    return l


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):  # numpy array (host memory)
        return x.ctypes.data
    raise TypeError("expected a tensor, array or integer address, got %r" % type(x))


def _stream(s) -> int | None:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


# ---- the C ABI, same names ----------------------------------------------

def gleam_status_string(rc: int) -> str:
    return lib().gleam_status_string(rc).decode()


def gleam_cache_create(capacity_bytes: int, chunk_bytes: int):
    h = ctypes.c_void_p()
    rc = lib().gleam_cache_create(capacity_bytes, chunk_bytes, ctypes.byref(h))
    return rc, h.value


def gleam_cache_create_ex(capacity_bytes: int, chunk_bytes: int, flags: int):
    h = ctypes.c_void_p()
    rc = lib().gleam_cache_create_ex(capacity_bytes, chunk_bytes, flags, ctypes.byref(h))
    return rc, h.value


def gleam_cache_destroy(cache) -> None:
    lib().gleam_cache_destroy(cache)


def gleam_cache_reserve(cache, max_chunks: int) -> int:
    return lib().gleam_cache_reserve(cache, max_chunks)


def gleam_fingerprint(d_buf, n: int, chunk_bytes: int, d_out, stream=None) -> int:
    return lib().gleam_fingerprint(_ptr(d_buf), n, chunk_bytes, _ptr(d_out), _stream(stream))


def gleam_dedup_copy(cache, d_buf, n: int, d_hit_mask, d_miss_idx, d_miss_bytes) -> int:
    return lib().gleam_dedup_copy(cache, _ptr(d_buf), n, _ptr(d_hit_mask), _ptr(d_miss_idx),
                                  _ptr(d_miss_bytes))


def gleam_dedup_copy_async(cache, d_buf, n: int, d_hit_mask, d_miss_idx, d_miss_bytes,
                           d_result=None, stream=None) -> int:
    return lib().gleam_dedup_copy_async(cache, _ptr(d_buf), n, _ptr(d_hit_mask),
                                        _ptr(d_miss_idx), _ptr(d_miss_bytes), _ptr(d_result),
                                        _stream(stream))


GLEAM_NOALLOC_MAX_CHUNKS = 65536


def gleam_dedup_copy_noalloc(cache, d_buf, n: int, d_hit_mask, d_miss_idx, d_miss_bytes,
                             d_result=None, stream=None) -> int:
    """The dedup call for callers that cannot allocate: a fixed library-owned
    scratch array replaces the cache's workspace (at most
    GLEAM_NOALLOC_MAX_CHUNKS chunks per call)."""
    return lib().gleam_dedup_copy_noalloc(cache, _ptr(d_buf), n, _ptr(d_hit_mask),
                                          _ptr(d_miss_idx), _ptr(d_miss_bytes), _ptr(d_result),
                                          _stream(stream))


def payload_array(payloads):
    """ctypes gleam_payload_t[] from (d_buf, n, d_hit_mask, d_miss_idx,
    d_miss_bytes, d_result[, d_chunk_slot]) tuples; reusable across calls."""
    arr = (gleam_payload_t * max(1, len(payloads)))()
    for k, t in enumerate(payloads):
        buf, n, mask, idx, packed, res = t[:6]
        slots = t[6] if len(t) > 6 else None
        arr[k] = gleam_payload_t(_ptr(buf), n, _ptr(mask), _ptr(idx), _ptr(packed), _ptr(res),
                                 _ptr(slots))
    arr.count = len(payloads)
    return arr


def gleam_dedup_copy_batch(cache, payloads, d_total=None, stream=None) -> int:
    """payloads: a payload_array(), or a sequence of tuples for it."""
    arr = payloads if hasattr(payloads, "count") else payload_array(payloads)
    return lib().gleam_dedup_copy_batch(cache, arr, arr.count, _ptr(d_total), _stream(stream))


def gleam_dedup_copy_host_async(cache, h_buf, n: int, d_hit_mask, d_miss_idx, d_miss_bytes,
                                d_result=None, stream=None) -> int:
    return lib().gleam_dedup_copy_host_async(cache, _ptr(h_buf), n, _ptr(d_hit_mask),
                                             _ptr(d_miss_idx), _ptr(d_miss_bytes),
                                             _ptr(d_result), _stream(stream))


def gleam_dedup_copy_host_batch(cache, payloads, d_total=None, stream=None) -> int:
    """payloads: a payload_array() whose buffers are page-locked host memory."""
    arr = payloads if hasattr(payloads, "count") else payload_array(payloads)
    return lib().gleam_dedup_copy_host_batch(cache, arr, arr.count, _ptr(d_total),
                                             _stream(stream))


def gleam_block_check(cache, d_block, block_bytes: int, d_offsets, d_slots, nrec: int,
                      d_mismatch, d_count, stream=None) -> int:
    return lib().gleam_block_check(cache, _ptr(d_block), block_bytes, _ptr(d_offsets),
                                   _ptr(d_slots), nrec, _ptr(d_mismatch), _ptr(d_count),
                                   _stream(stream))


def gleam_cache_stats(cache):
    st = gleam_stats_t()
    rc = lib().gleam_cache_stats(cache, ctypes.byref(st))
    return rc, {f: int(getattr(st, f)) for f, _ in gleam_stats_t._fields_}


def gleam_cache_export(cache, h_keys, h_lens, max_entries: int):
    count = ctypes.c_uint64()
    rc = lib().gleam_cache_export(cache, _ptr(h_keys), _ptr(h_lens), max_entries,
                                  ctypes.byref(count))
    return rc, count.value


def gleam_cache_read_slot(cache, slot: int, h_out, max_bytes: int):
    ln = ctypes.c_uint64()
    rc = lib().gleam_cache_read_slot(cache, slot, _ptr(h_out), max_bytes, ctypes.byref(ln))
    return rc, ln.value


def gleam_cache_debug_insert(cache, key: int, d_bytes, n: int) -> int:
    return lib().gleam_cache_debug_insert(cache, key, _ptr(d_bytes), n)


def gleam_cache_debug_set(cache, what: int, value: int) -> int:
    return lib().gleam_cache_debug_set(cache, what, value)


def gleam_cache_snapshot(cache):
    h = ctypes.c_void_p()
    rc = lib().gleam_cache_snapshot(cache, ctypes.byref(h))
    return rc, h.value


def gleam_cache_restore(cache, snap) -> int:
    return lib().gleam_cache_restore(cache, snap)


def gleam_snapshot_destroy(snap) -> None:
    lib().gleam_snapshot_destroy(snap)


def gleam_cache_profile(cache, enable: bool) -> int:
    return lib().gleam_cache_profile(cache, 1 if enable else 0)


def gleam_cache_profile_read(cache, nkernels: int = 2):
    """Returns (rc, [ms per kernel], [launches per kernel])."""
    ms = (ctypes.c_double * nkernels)()
    n = (ctypes.c_uint64 * nkernels)()
    rc = lib().gleam_cache_profile_read(cache, ctypes.addressof(ms), ctypes.addressof(n), nkernels)
    return rc, list(ms), [int(x) for x in n]
