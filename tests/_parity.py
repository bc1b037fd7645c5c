"""GPU-vs-oracle comparison helpers (element by element, bit-exact)."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300.cache import Cache, DedupOutputs

DEV = torch.device("cuda:0")
STAT_KEYS = ("calls", "chunks", "hits_cache", "hits_intra", "misses", "inserts",
             "verify_rejects", "slots_used", "bytes_used")


def to_device(host: torch.Tensor, offset: int = 0) -> torch.Tensor:
    """Copy of a CPU uint8 tensor on the GPU, starting `offset` bytes past a
    256-byte boundary."""
    if offset == 0:
        return host.to(DEV)
    big = torch.empty(host.numel() + offset, dtype=torch.uint8, device=DEV)
    v = big[offset:]
    v.copy_(host)
    return v


def dedup_both(gc: Cache, oc: oracle.OracleCache, host: torch.Tensor, *, offset: int = 0,
               packed_offset: int = 0):
    """One call on both sides; asserts identical outcome and outputs."""
    C = gc.chunk_bytes
    n = host.numel()
    rc_o, mask_o, miss_o, packed_o = oc.dedup(host.numpy())
    d = to_device(host, offset)
    out = DedupOutputs.alloc(n, C, DEV)
    if packed_offset:
        big = torch.empty(max(1, n) + packed_offset, dtype=torch.uint8, device=DEV)
        out.miss_bytes = big[packed_offset:]
    try:
        rc, out = gc.dedup(d, out)
    except B.GleamError as e:
        rc = e.rc
    assert rc == rc_o, (rc, rc_o)
    if rc < 0 or n == 0:
        return rc
    mask = out.hit_mask.cpu().numpy().view(np.uint32)[: len(mask_o)]
    miss = out.miss_idx.cpu().numpy().view(np.uint32)[:rc]
    packed = out.miss_bytes.cpu().numpy()[: len(packed_o)]
    assert np.array_equal(mask, mask_o), "hit mask differs"
    assert np.array_equal(miss, miss_o), "miss indices differ"
    assert np.array_equal(packed, packed_o), "packed miss bytes differ"
    return rc


def compare_cache(gc: Cache, oc: oracle.OracleCache, check_bytes: int = 64):
    """Counters equal; index as a set of (slot, key, len) equal; stored bytes
    equal for every slot (or `check_bytes` sampled slots when larger)."""
    st, so = gc.stats(), oc.stats()
    for k in STAT_KEYS:
        assert st[k] == so[k], (k, st[k], so[k])
    keys, lens, count = gc.export()
    okeys, olens = oc.entries()
    assert count == st["slots_used"]
    assert np.array_equal(keys, okeys), "index keys differ"
    assert np.array_equal(lens, olens), "index lengths differ"
    used = st["slots_used"]
    slots = range(used) if used <= check_bytes else \
        np.random.default_rng(0).choice(used, check_bytes, replace=False).tolist()
    for s in slots:
        assert gc.read_slot(int(s)) == oc.slot_bytes(int(s)), s
