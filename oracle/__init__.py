"""Gleam chunk-dedup oracle -- TEST INFRASTRUCTURE ONLY.

A ctypes wrapper over ``gleam_oracle.cpp``: the plain, single-threaded CPU
statement of the dedup hot path (paper Sec. 4.1.2, "Hash-based Weight Chunk
Retrieval", and App. B.1, "Hash Cost and Collision"; XXH64 from the public
xxHash specification).  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import it.  The CUDA library never does,
and the two share no code.

Every function here is pinned by ``tests/test_oracle_*.py`` against values the
oracle does not produce itself: published XXH64 vectors, the installed
libxxhash, zstd frame checksums, a pure-Python brute-force dedup on tiny
inputs, and closed forms of the synthetic workloads.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gleam_oracle.cpp")
_LIB = os.path.join(_HERE, "liboracle.so")

OK = 0
ERR_INVALID_ARG = -1
ERR_CAPACITY = -4
KEY16 = 1
PAPER_IDS = 4
EVICT_LRU = 8
NO_SLOT = 0xFFFFFFFF

STAT_FIELDS = (
    "calls", "chunks", "hits_cache", "hits_intra", "misses", "inserts",
    "verify_rejects", "slots_used", "bytes_used", "capacity_bytes", "nslots",
    "chunk_bytes", "evictions",
)
RESULT_FIELDS = ("n_miss", "n_hit_cache", "n_hit_intra", "verify_rejects", "miss_bytes")


def build(force: bool = False) -> str:
    """Compile the oracle with the host C++ compiler (portable C++17)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp%d" % os.getpid()
        subprocess.check_call(
            ["g++", "-O2", "-std=c++17", "-shared", "-fPIC", "-o", tmp, _SRC])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = _bind(ctypes.CDLL(build()))
    return _lib


def _bind(l):
    """Declares the C signatures on a loaded oracle library."""
    if True:
        u64, sz, vp = ctypes.c_uint64, ctypes.c_size_t, ctypes.c_void_p
        l.oracle_xxh64.restype = u64
        l.oracle_xxh64.argtypes = [vp, sz, u64]
        l.oracle_md5.restype = None
        l.oracle_md5.argtypes = [vp, sz, vp]
        l.oracle_fingerprint.restype = ctypes.c_int
        l.oracle_fingerprint.argtypes = [vp, sz, sz, vp]
        l.oracle_cache_create.restype = vp
        l.oracle_cache_create.argtypes = [sz, sz, ctypes.c_uint32, ctypes.POINTER(ctypes.c_int)]
        l.oracle_cache_destroy.restype = None
        l.oracle_cache_destroy.argtypes = [vp]
        l.oracle_dedup.restype = ctypes.c_int64
        l.oracle_dedup.argtypes = [vp, vp, sz, vp, vp, vp, vp]
        l.oracle_dedup_batch.restype = ctypes.c_int64
        l.oracle_dedup_batch.argtypes = [vp, sz, vp, vp, vp, vp, vp, vp, vp]
        l.oracle_block_check.restype = ctypes.c_int64
        l.oracle_block_check.argtypes = [vp, vp, u64, vp, vp, u64, vp]
        l.oracle_debug_insert.restype = ctypes.c_int
        l.oracle_debug_insert.argtypes = [vp, u64, vp, sz]
        l.oracle_cache_stats.restype = None
        l.oracle_cache_stats.argtypes = [vp, vp]
        l.oracle_cache_entries.restype = u64
        l.oracle_cache_entries.argtypes = [vp, vp, vp, u64]
        l.oracle_slot_bytes.restype = ctypes.c_int64
        l.oracle_slot_bytes.argtypes = [vp, u64, vp, u64]
    return l


def _u8(buf) -> np.ndarray:
    a = np.frombuffer(buf, dtype=np.uint8) if isinstance(buf, (bytes, bytearray, memoryview)) \
        else np.ascontiguousarray(buf).view(np.uint8).reshape(-1)
    return a


def xxh64(data, seed: int = 0) -> int:
    a = _u8(data)
    return int(lib().oracle_xxh64(a.ctypes.data, a.size, seed))


def md5(data) -> bytes:
    a = _u8(data)
    out = np.zeros(16, dtype=np.uint8)
    lib().oracle_md5(a.ctypes.data, a.size, out.ctypes.data)
    return out.tobytes()


def paper_key(chunk) -> int:
    """The paper's identifier (App. B.1): MD5 of the first min(len, 128) bytes,
    first 8 digest bytes as a little-endian integer."""
    a = _u8(chunk)
    return int.from_bytes(md5(a[:128])[:8], "little")


def fingerprint(data, chunk_bytes: int) -> np.ndarray:
    """XXH64 (seed 0) of every chunk_bytes-byte chunk; chunk_bytes == 0: of the whole buffer."""
    a = _u8(data)
    n = a.size
    count = 1 if chunk_bytes == 0 else (n + chunk_bytes - 1) // chunk_bytes
    out = np.zeros(count, dtype=np.uint64)
    rc = lib().oracle_fingerprint(a.ctypes.data, n, chunk_bytes, out.ctypes.data)
    assert rc == OK
    return out


class OracleCache:
    """The sequential weight cache: index + stored chunk bytes + statistics."""

    def __init__(self, capacity_bytes: int, chunk_bytes: int, flags: int = 0):
        err = ctypes.c_int(0)
        self._h = lib().oracle_cache_create(capacity_bytes, chunk_bytes, flags, ctypes.byref(err))
        if not self._h:
            raise ValueError("oracle_cache_create rejected its arguments (%d)" % err.value)
        self.chunk_bytes = chunk_bytes
        self.flags = flags

    def close(self):
        if self._h:
            lib().oracle_cache_destroy(self._h)
            self._h = None

    def __del__(self):
        self.close()

    def dedup(self, data, chunk_slots: bool = False):
        """Returns (rc, hit_mask u32[], miss_idx u32[n_miss], packed u8[packed_bytes]),
        plus the slot holding every chunk's bytes (u32[N]) if chunk_slots."""
        a = _u8(data)
        n = a.size
        C = self.chunk_bytes
        nch = (n + C - 1) // C
        mask = np.zeros(max(1, (nch + 31) // 32), dtype=np.uint32)
        miss = np.zeros(max(1, nch), dtype=np.uint32)
        packed = np.zeros(max(1, n), dtype=np.uint8)
        slots = np.zeros(max(1, nch), dtype=np.uint32) if chunk_slots else None
        rc = int(lib().oracle_dedup(self._h, a.ctypes.data, n, mask.ctypes.data,
                                    miss.ctypes.data, packed.ctypes.data,
                                    slots.ctypes.data if chunk_slots else None))
        if chunk_slots:
            if rc < 0:
                return rc, None, None, None, None
            r = self._finish(rc, n, nch, mask, miss, packed)
            return r + (slots[:nch].copy(),)
        return self._finish(rc, n, nch, mask, miss, packed)

    def dedup_batch(self, datas, chunk_slots: bool = False):
        """One call over several payloads (a batch).  Returns (rc, outs, results):
        outs[k] = (hit_mask, miss_idx, packed[, chunk_slots]) of payload k and
        results[k] = dict of RESULT_FIELDS; (rc, None, None) on an error."""
        C = self.chunk_bytes
        arrs = [_u8(d) for d in datas]
        count = len(arrs)
        nch = [(a.size + C - 1) // C for a in arrs]
        masks = [np.zeros(max(1, (m + 31) // 32), dtype=np.uint32) for m in nch]
        misses = [np.zeros(max(1, m), dtype=np.uint32) for m in nch]
        packeds = [np.zeros(max(1, a.size), dtype=np.uint8) for a in arrs]
        slots = [np.zeros(max(1, m), dtype=np.uint32) for m in nch] if chunk_slots else None
        P = ctypes.c_void_p * max(1, count)
        bufs = P(*[a.ctypes.data for a in arrs])
        ns = (ctypes.c_size_t * max(1, count))(*[a.size for a in arrs])
        res = np.zeros(max(1, 5 * count), dtype=np.uint64)
        rc = int(lib().oracle_dedup_batch(
            self._h, count, bufs, ns, P(*[m.ctypes.data for m in masks]),
            P(*[m.ctypes.data for m in misses]), P(*[m.ctypes.data for m in packeds]),
            P(*[m.ctypes.data for m in slots]) if chunk_slots else None, res.ctypes.data))
        if rc < 0:
            return rc, None, None
        outs, results = [], []
        for k in range(count):
            r = {f: int(res[5 * k + j]) for j, f in enumerate(RESULT_FIELDS)}
            _, mk, mi, pk = self._finish(r["n_miss"], arrs[k].size, nch[k], masks[k], misses[k],
                                         packeds[k])
            outs.append((mk, mi, pk) + ((slots[k][:nch[k]].copy(),) if chunk_slots else ()))
            results.append(r)
        return rc, outs, results

    def _finish(self, rc, n, nch, mask, miss, packed):
        C = self.chunk_bytes
        if rc < 0:
            return rc, None, None, None
        miss = miss[:rc].copy()
        nbytes = 0
        if rc:
            last = int(miss[-1])
            tail = n - last * C if last == nch - 1 else C
            nbytes = (rc - 1) * C + min(C, tail)
        return rc, mask[: (nch + 31) // 32].copy(), miss, packed[:nbytes].copy()

    def block_check(self, block, offsets, slots):
        """(number of mismatching records, mismatch flags u8[nrec])."""
        b = _u8(block)
        offs = np.ascontiguousarray(offsets, dtype=np.uint64)
        sl = np.ascontiguousarray(slots, dtype=np.uint32)
        flags = np.zeros(max(1, offs.size), dtype=np.uint8)
        bad = int(lib().oracle_block_check(self._h, b.ctypes.data, b.size, offs.ctypes.data,
                                           sl.ctypes.data, offs.size, flags.ctypes.data))
        return bad, flags[: offs.size]

    def debug_insert(self, key: int, data) -> int:
        a = _u8(data)
        return int(lib().oracle_debug_insert(self._h, key, a.ctypes.data, a.size))

    def stats(self) -> dict:
        out = np.zeros(len(STAT_FIELDS), dtype=np.uint64)
        lib().oracle_cache_stats(self._h, out.ctypes.data)
        return {k: int(v) for k, v in zip(STAT_FIELDS, out)}

    def entries(self):
        """(keys u64[slots_used], lens u32[slots_used]) ordered by slot."""
        used = self.stats()["slots_used"]
        keys = np.zeros(max(1, used), dtype=np.uint64)
        lens = np.zeros(max(1, used), dtype=np.uint32)
        lib().oracle_cache_entries(self._h, keys.ctypes.data, lens.ctypes.data, used)
        return keys[:used], lens[:used]

    def slot_bytes(self, slot: int) -> bytes:
        out = np.zeros(self.chunk_bytes, dtype=np.uint8)
        ln = int(lib().oracle_slot_bytes(self._h, slot, out.ctypes.data, out.size))
        if ln < 0:
            raise IndexError(slot)
        return out[:ln].tobytes()
