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

    def __init__(self, nslots: int, key_fn=None, paper_min: int = 0, lru: bool = False):
        self.nslots = nslots
        self.items = []       # (key, bytes) in slot order
        self.key_fn = key_fn  # bytes -> key, only for counting verify rejects
        self.paper_min = paper_min  # chunks shorter than this are never cached
        self.lru = lru        # evict least recently used slots instead of failing
        self.clock = 0
        self.last_use = []    # per slot: the clock value of the call that last used it
        self.evictions = 0

    def insert(self, key, data: bytes):
        self.items.append((key, bytes(data)))
        self.clock += 1
        self.last_use.append(self.clock)

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

    def dedup_batch(self, payloads, C: int):
        """One call over several payloads, by definition: each chunk, payload
        after payload, is a hit iff byte-equal to a stored chunk or to an
        earlier miss of the call.  Then the misses get slots: never-used ones,
        and (LRU) the least recently used slots the call did not hit, ties by
        lower slot, in ascending slot order.  Returns (rc, [per-payload dict])."""
        total = sum((len(p) + C - 1) // C for p in payloads)
        if total == 0:
            return 0, [None] * len(payloads)
        self.clock += 1
        now = self.clock
        slots0 = len(self.items)
        fresh = []   # (bytes, payload number, key) in miss order
        used = set()
        outs = []
        for k, payload in enumerate(payloads):
            n = len(payload)
            N = (n + C - 1) // C
            o = dict(mask=[0] * ((N + 31) // 32), miss=[], packed=bytearray(), slots=[],
                     hits_cache=0, hits_intra=0, rejects=0)
            for i in range(N):
                c = payload[i * C:(i + 1) * C]
                if len(c) < self.paper_min:
                    o["miss"].append(i)
                    o["slots"].append(("none",))
                    o["packed"] += c
                    continue
                found = None
                for s, (_, b) in enumerate(self.items):
                    if b == c:
                        found = ("cache", s)
                        break
                if found is None:
                    for r, (b, kk, _) in enumerate(fresh):
                        if b == c:
                            found = ("fresh", r)
                            break
                if found is not None:
                    o["mask"][i // 32] |= 1 << (i % 32)
                    o["slots"].append(found)
                    if found[0] == "cache":
                        used.add(found[1])
                        o["hits_cache"] += 1
                    elif fresh[found[1]][1] == k:
                        o["hits_intra"] += 1
                    else:
                        o["hits_cache"] += 1
                    continue
                key = self.key_fn(c) if self.key_fn else None
                if self.key_fn and (any(kk == key and len(b) == len(c) for kk, b in self.items) or
                                    any(kk == key and len(b) == len(c) for b, _, kk in fresh)):
                    o["rejects"] += 1
                o["miss"].append(i)
                o["slots"].append(("fresh", len(fresh)))
                o["packed"] += c
                fresh.append((c, k, key))
            outs.append(o)
        M = len(fresh)
        victims = []
        if M > self.nslots - slots0:
            if not self.lru:
                return -4, None
            need = M - (self.nslots - slots0)
            cands = sorted((s for s in range(slots0) if s not in used),
                           key=lambda s: (self.last_use[s], s))
            if len(cands) < need:
                return -4, None
            victims = sorted(cands[:need])
        slot_of = victims + list(range(slots0, slots0 + M - len(victims)))
        for r, (b, _, key) in enumerate(fresh):
            s = slot_of[r]
            if s < len(self.items):
                self.items[s] = (key, b)
                self.last_use[s] = now
            else:
                self.items.append((key, b))
                self.last_use.append(now)
        for s in used:
            self.last_use[s] = now
        self.evictions += len(victims)
        for o in outs:
            o["slots"] = [0xFFFFFFFF if t[0] == "none" else t[1] if t[0] == "cache"
                          else slot_of[t[1]] for t in o["slots"]]
            o["packed"] = bytes(o["packed"])
        return sum(len(o["miss"]) for o in outs), outs
