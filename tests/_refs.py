"""Independent references that pin the oracle (no code shared with it).

* libxxhash: the xxHash project's own shared library, as installed on this
  machine, called through ctypes.
* zstd frames: RFC 8878 lets a frame carry a content checksum equal to the low
  32 bits of XXH64(content, seed 0).  We build a frame of raw blocks around the
  bytes with a claimed checksum and ask libzstd (through pyarrow) to decode
  it; libzstd refuses a frame whose checksum does not match.
* brute-force dedup: the sequential rule of the weight cache written with
  plain byte-string comparisons and no hashing at all (optionally with keys
  from libxxhash for counting verify rejects).
"""
from __future__ import annotations

import ctypes
import ctypes.util
import struct

import pytest

_xxh = None


def libxxhash():
    """ctypes handle of the installed libxxhash, or skip."""
    global _xxh
    if _xxh is None:
        for name in ("libxxhash.so.0", ctypes.util.find_library("xxhash")):
            if not name:
                continue
            try:
                l = ctypes.CDLL(name)
                l.XXH64.restype = ctypes.c_uint64
                l.XXH64.argtypes = [ctypes.c_char_p, ctypes.c_size_t, ctypes.c_uint64]
                _xxh = l
                break
            except OSError:
                continue
    if _xxh is None:
        pytest.skip("libxxhash not installed here")
    return _xxh


def xxh64_lib(data: bytes, seed: int = 0) -> int:
    return int(libxxhash().XXH64(bytes(data), len(data), seed))


def _zstd_frame(content: bytes, checksum32: int) -> bytes:
    # Frame header descriptor: content-size field 8 bytes (flag 3), single
    # segment (no window descriptor), content checksum present, no dictionary.
    out = bytearray(struct.pack("<I", 0xFD2FB528))
    out.append((3 << 6) | (1 << 5) | (1 << 2))
    out += struct.pack("<Q", len(content))
    blocks = [content[i:i + 131072] for i in range(0, len(content), 131072)] or [b""]
    for k, blk in enumerate(blocks):
        last = 1 if k == len(blocks) - 1 else 0
        header = last | (0 << 1) | (len(blk) << 3)  # raw block
        out += header.to_bytes(3, "little")
        out += blk
    out += struct.pack("<I", checksum32 & 0xFFFFFFFF)
    return bytes(out)


def zstd_accepts_checksum(content: bytes, checksum32: int) -> bool:
    """True iff libzstd decodes the frame, i.e. checksum32 == low32(XXH64(content))."""
    pa = pytest.importorskip("pyarrow")
    if not pa.Codec.is_available("zstd"):
        pytest.skip("pyarrow built without zstd")
    try:
        got = pa.decompress(_zstd_frame(bytes(content), checksum32),
                            decompressed_size=len(content), codec="zstd").to_pybytes()
    except Exception:
        return False
    assert got == bytes(content)
    return True


class BruteCache:
    """The weight cache by its definition: an ordered list of stored byte
    strings; a chunk is a hit iff byte-equal to a stored one of equal length."""

    def __init__(self, nslots: int, key_fn=None, paper_min: int = 0):
        self.nslots = nslots
        self.items = []       # (key, bytes) in slot order
        self.key_fn = key_fn  # bytes -> key, only for counting verify rejects
        self.paper_min = paper_min  # chunks shorter than this are never cached

    def insert(self, key, data: bytes):
        self.items.append((key, bytes(data)))

    def dedup(self, payload: bytes, C: int):
        n = len(payload)
        N = (n + C - 1) // C
        staged = list(self.items)
        slots0 = len(staged)
        mask, miss, packed, slots = [0] * ((N + 31) // 32), [], bytearray(), []
        hits_cache = hits_intra = rejects = 0
        for i in range(N):
            c = payload[i * C:(i + 1) * C]
            if len(c) < self.paper_min:  # recorded, never cached
                miss.append(i)
                slots.append(0xFFFFFFFF)
                packed += c
                continue
            found = None
            for s, (_, b) in enumerate(staged):
                if b == c:
                    found = s
                    break
            if found is not None:
                mask[i // 32] |= 1 << (i % 32)
                slots.append(found)
                if found < slots0:
                    hits_cache += 1
                else:
                    hits_intra += 1
                continue
            key = self.key_fn(c) if self.key_fn else None
            if self.key_fn and any(k == key and len(b) == len(c) for k, b in staged):
                rejects += 1
            if len(staged) >= self.nslots:
                return -4, None
            miss.append(i)
            slots.append(len(staged))
            packed += c
            staged.append((key, c))
        self.items = staged
        return len(miss), dict(mask=mask, miss=miss, packed=bytes(packed), hits_cache=hits_cache,
                               hits_intra=hits_intra, rejects=rejects, slots=slots)
