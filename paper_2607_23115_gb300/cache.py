"""Convenience layer over the binding: a Cache object that raises GleamError on
failure and allocates worst-case output buffers with torch on the payload's
device.  All work still happens in libgleam.so."""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import numpy as np
import torch

from . import binding as B


def _check(rc: int, what: str) -> int:
    if rc < 0:
        raise B.GleamError(rc, what)
    return rc


@dataclass
class DedupOutputs:
    """Worst-case sized outputs of one dedup call on a payload of n bytes."""
    hit_mask: torch.Tensor    # int32 view of u32[ceil(N/32)]
    miss_idx: torch.Tensor    # int32 view of u32[N]
    miss_bytes: torch.Tensor  # uint8[n]

    @staticmethod
    def alloc(n: int, chunk_bytes: int, device) -> "DedupOutputs":
        N = (n + chunk_bytes - 1) // chunk_bytes
        return DedupOutputs(
            torch.empty(max(1, (N + 31) // 32), dtype=torch.int32, device=device),
            torch.empty(max(1, N), dtype=torch.int32, device=device),
            torch.empty(max(1, n), dtype=torch.uint8, device=device))


def fingerprint(buf: torch.Tensor, chunk_bytes: int, out: Optional[torch.Tensor] = None,
                stream=None) -> torch.Tensor:
    """XXH64 of every chunk (int64 view of u64), or of the whole buffer when
    chunk_bytes == 0."""
    n = buf.numel() * buf.element_size()
    count = 1 if chunk_bytes == 0 else (n + chunk_bytes - 1) // chunk_bytes
    if out is None:
        out = torch.empty(max(1, count), dtype=torch.int64, device=buf.device)
    _check(B.gleam_fingerprint(buf, n, chunk_bytes, out, stream), "gleam_fingerprint")
    return out[:count]


class Cache:
    def __init__(self, capacity_bytes: int, chunk_bytes: int, flags: int = 0):
        rc, h = B.gleam_cache_create_ex(capacity_bytes, chunk_bytes, flags)
        _check(rc, "gleam_cache_create_ex")
        self.handle = h
        self.chunk_bytes = chunk_bytes
        self.flags = flags

    def close(self):
        if self.handle:
            B.gleam_cache_destroy(self.handle)
            self.handle = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def reserve(self, max_chunks: int):
        _check(B.gleam_cache_reserve(self.handle, max_chunks), "gleam_cache_reserve")

    def dedup(self, buf: torch.Tensor, out: Optional[DedupOutputs] = None):
        """Synchronous dedup; returns (n_miss, outputs)."""
        n = buf.numel() * buf.element_size()
        if out is None:
            out = DedupOutputs.alloc(n, self.chunk_bytes, buf.device)
        rc = B.gleam_dedup_copy(self.handle, buf, n, out.hit_mask, out.miss_idx, out.miss_bytes)
        return _check(rc, "gleam_dedup_copy"), out

    def dedup_async(self, buf: torch.Tensor, out: DedupOutputs,
                    result: Optional[torch.Tensor] = None, stream=None):
        n = buf.numel() * buf.element_size()
        _check(B.gleam_dedup_copy_async(self.handle, buf, n, out.hit_mask, out.miss_idx,
                                        out.miss_bytes, result, stream),
               "gleam_dedup_copy_async")

    @staticmethod
    def batch_items(bufs, outs, results=None, chunk_slots=None):
        """Payload array for dedup_batch (build once, reuse for repeated calls)."""
        items = []
        for k, (b, o) in enumerate(zip(bufs, outs)):
            n = b.numel() * b.element_size()
            r = results[k] if results is not None else None
            sl = chunk_slots[k] if chunk_slots is not None else None
            items.append((b, n, o.hit_mask, o.miss_idx, o.miss_bytes, r, sl))
        return B.payload_array(items)

    def block_check(self, block: torch.Tensor, offsets: torch.Tensor, slots: torch.Tensor,
                    mismatch: Optional[torch.Tensor] = None, count: Optional[torch.Tensor] = None,
                    stream=None) -> torch.Tensor:
        """Device int64[1] count of records whose bytes no longer match (async)."""
        if count is None:
            count = torch.zeros(1, dtype=torch.int64, device=block.device)
        _check(B.gleam_block_check(self.handle, block, block.numel() * block.element_size(),
                                   offsets, slots, offsets.numel(), mismatch, count, stream),
               "gleam_block_check")
        return count

    def dedup_batch(self, bufs, outs=None, results=None, total: Optional[torch.Tensor] = None,
                    stream=None, items=None):
        """One call over several payloads, equivalent to dedup_async on each in
        order.  results: per-payload int64[6] tensors (or None)."""
        if items is None:
            items = self.batch_items(bufs, outs, results)
        _check(B.gleam_dedup_copy_batch(self.handle, items, total, stream),
               "gleam_dedup_copy_batch")

    def dedup_host(self, hbuf: torch.Tensor, out: DedupOutputs, result=None, stream=None):
        """Async dedup of a payload in page-locked host memory (read in place)."""
        n = hbuf.numel() * hbuf.element_size()
        _check(B.gleam_dedup_copy_host_async(self.handle, hbuf, n, out.hit_mask, out.miss_idx,
                                             out.miss_bytes, result, stream),
               "gleam_dedup_copy_host_async")

    def dedup_host_batch(self, hbufs=None, outs=None, results=None, total=None, stream=None,
                         items=None):
        if items is None:
            items = self.batch_items(hbufs, outs, results)
        _check(B.gleam_dedup_copy_host_batch(self.handle, items, total, stream),
               "gleam_dedup_copy_host_batch")

    def stats(self) -> dict:
        rc, st = B.gleam_cache_stats(self.handle)
        _check(rc, "gleam_cache_stats")
        return st

    def export(self):
        used = self.stats()["slots_used"]
        keys = np.zeros(max(1, used), dtype=np.uint64)
        lens = np.zeros(max(1, used), dtype=np.uint32)
        rc, count = B.gleam_cache_export(self.handle, keys, lens, used)
        _check(rc, "gleam_cache_export")
        return keys[:used], lens[:used], count

    def read_slot(self, slot: int) -> bytes:
        out = np.zeros(self.chunk_bytes, dtype=np.uint8)
        rc, ln = B.gleam_cache_read_slot(self.handle, slot, out, out.size)
        _check(rc, "gleam_cache_read_slot")
        return out[:ln].tobytes()

    def debug_insert(self, key: int, data: torch.Tensor):
        n = data.numel() * data.element_size()
        _check(B.gleam_cache_debug_insert(self.handle, key & (2**64 - 1), data, n),
               "gleam_cache_debug_insert")

    def debug_set(self, what: int, value: int):
        _check(B.gleam_cache_debug_set(self.handle, what, value), "gleam_cache_debug_set")

    def snapshot(self) -> "Snapshot":
        rc, h = B.gleam_cache_snapshot(self.handle)
        _check(rc, "gleam_cache_snapshot")
        return Snapshot(h)

    def restore(self, snap: "Snapshot"):
        _check(B.gleam_cache_restore(self.handle, snap.handle), "gleam_cache_restore")


class Snapshot:
    def __init__(self, handle):
        self.handle = handle

    def close(self):
        if self.handle:
            B.gleam_snapshot_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def result_dict(result: torch.Tensor) -> dict:
    """Host view of a device gleam_result_t held in an int64[6] tensor."""
    v = result.cpu().tolist()
    return dict(zip(B.RESULT_FIELDS, v))
