"""KEY16 mode, many misses under one index key (chunks found by search,
tests/golden/key16_class.txt: 48 chunks of 32 bytes and 4 of 20 bytes whose
XXH64 share the low 16 bits).  Each miss of a (16-bit key, length) class
starts its index insert at its own place after the key's home position; the
calls below build that run, extend it past entries of earlier calls and of the
second class (the short last chunks) under the same key, and, with LRU
eviction, past the holes that evictions leave.  Every call's outputs and the
cache must equal the oracle's, and a call that sends every chunk again must
find each one (no entry cut off from the home position)."""
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from tests._parity import compare_cache, dedup_both

C = 32
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "key16_class.txt")


def _chunks():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            hexbytes, fp = line.split()
            rows.append((bytes.fromhex(hexbytes), int(fp, 16)))
    full = [r for r in rows if len(r[0]) == C]
    tails = [r for r in rows if len(r[0]) < C]
    return full, tails


def test_fixture_chunks_share_one_index_key():
    # distinct chunks, each with its recorded oracle fingerprint, all with the
    # same low 16 bits
    full, tails = _chunks()
    assert len(full) == 48 and len(tails) == 4
    assert len({c for c, _ in full + tails}) == 52
    for c, fp in full + tails:
        assert oracle.xxh64(np.frombuffer(c, dtype=np.uint8)) == fp
    assert len({fp & 0xFFFF for _, fp in full + tails}) == 1


def _payload(rng, full, ids, nfill, tail=None):
    """The class chunks `ids` at random places among nfill random chunks,
    then the short chunk `tail` (if any) as the payload's last chunk."""
    rows = [np.frombuffer(full[i][0], dtype=np.uint8) for i in ids]
    rows += [rng.integers(0, 256, C, dtype=np.uint8) for _ in range(nfill)]
    order = rng.permutation(len(rows))
    data = b"".join(rows[k].tobytes() for k in order)
    if tail is not None:
        data += tail
    return torch.frombuffer(bytearray(data), dtype=torch.uint8)


@pytest.mark.gpu
@pytest.mark.usefixtures("call_path")
@pytest.mark.parametrize("lru", [False, True])
@pytest.mark.parametrize("nfill", [0, 3000])
def test_many_misses_of_one_index_key(nfill, lru):
    from paper_2607_23115_gb300.cache import Cache
    full, tails = _chunks()
    rng = np.random.default_rng(11 + nfill + lru)
    if lru:  # the second call evicts most of the first call's slots
        nslots = nfill + 40
        flags, oflags = B.GLEAM_KEY16 | B.GLEAM_EVICT_LRU, oracle.KEY16 | oracle.EVICT_LRU
    else:
        nslots = 4 * (nfill + 60)
        flags, oflags = B.GLEAM_KEY16, oracle.KEY16
    gc = Cache(nslots * C, C, flags)
    oc = oracle.OracleCache(nslots * C, C, oflags)
    with gc:
        dedup_both(gc, oc, _payload(rng, full, range(0, 24), nfill, tails[0][0]))
        compare_cache(gc, oc)
        dedup_both(gc, oc, _payload(rng, full, range(12, 48), nfill, tails[1][0]))
        compare_cache(gc, oc)
        # the first call's chunks again (with LRU most were evicted), then every
        # class chunk, two of them twice in the call
        first, every = list(range(24)) + [5], list(range(48)) + [5, 40]
        dedup_both(gc, oc, _payload(rng, full, first, 0, tails[0][0]))
        compare_cache(gc, oc)
        dedup_both(gc, oc, _payload(rng, full, every, 0, tails[1][0]))
        compare_cache(gc, oc)
        if lru:  # (nfill 0: 49 distinct chunks do not fit the cache: that call failed)
            dedup_both(gc, oc, _payload(rng, full, first, 0, tails[0][0]))
            compare_cache(gc, oc)
        else:  # nothing evicted: every chunk is found
            assert dedup_both(gc, oc, _payload(rng, full, every, 0)) == 0
