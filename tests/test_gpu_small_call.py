"""The single-block kernel that runs a whole small call (hash, resolve and
rank, pack) against the oracle, at the edges of where the library chooses it
(64 chunks, 256 KiB) and with the limit raised so that one block hashes
several ranges of chunks in turn; every case is also run with that path off,
and both runs must give the same outputs and cache."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache
from tests._parity import compare_cache, dedup_both

pytestmark = pytest.mark.gpu
KiB, MiB = 1024, 1 << 20


def _alphabet_payload(rng, C, nch, alphabet, tail):
    parts = [alphabet[int(rng.integers(len(alphabet)))] for _ in range(nch)]
    if tail:
        parts.append(W.random_bytes(tail, seed=int(rng.integers(1 << 30))))
    return torch.cat(parts) if parts else torch.zeros(0, dtype=torch.uint8)


def _run(limit, C, flags, calls, seed):
    """The calls on a cache whose single-block limit is `limit` chunks (0: off),
    each checked against the oracle; returns the cache's export."""
    gc = Cache(4 * MiB, C, flags)
    oc = oracle.OracleCache(4 * MiB, C, flags)
    gc.debug_set(B.GLEAM_DEBUG_SMALL_CALLS, limit)
    rng = np.random.default_rng(seed)
    alphabet = [W.random_bytes(C, seed=500 + k) for k in range(24)] + \
        [torch.zeros(C, dtype=torch.uint8)]
    with gc:
        for nch, tail, offset in calls:
            dedup_both(gc, oc, _alphabet_payload(rng, C, nch, alphabet, tail), offset=offset)
        compare_cache(gc, oc)
        keys, lens, count = gc.export()
        st = gc.stats()
        st.pop("spec_chunks")  # a speed counter: how much was written ahead
        return sorted(zip(keys[:count].tolist(), lens[:count].tolist())), st


@pytest.mark.parametrize("key16", [False, True])
def test_edges_of_the_single_block_path(key16):
    C = 4 * KiB
    flags = B.GLEAM_KEY16 if key16 else 0
    # chunks and tail bytes around 64 chunks / 256 KiB; offset 4 is unaligned
    # (always the three-launch path)
    calls = [(1, 0, 0), (0, 100, 0), (63, 0, 0), (64, 0, 0), (63, 4095, 0), (64, 1, 0),
             (65, 0, 0), (2, 0, 4), (40, 17, 0), (64, 0, 0), (16, 0, 0)]
    on = _run(64, C, flags, calls, seed=1)
    off = _run(0, C, flags, calls, seed=1)
    assert on == off


@pytest.mark.parametrize("C", [32, 1 * KiB])
def test_one_block_hashing_several_ranges(C):
    # with the limit raised, a call of up to 1000 chunks runs in one block that
    # hashes 64 chunks at a time
    calls = [(1000, 0, 0), (700, 5, 0), (129, 0, 0), (256, C - 1, 0), (64, 0, 0), (65, 0, 0)]
    raised = _run(1000, C, 0, calls, seed=C)
    off = _run(0, C, 0, calls, seed=C)
    assert raised == off


def test_small_calls_near_a_full_lru_cache():
    # a full LRU cache evicts; the library then runs the three-launch path
    C = 1 * KiB
    nslots = 48
    gc = Cache(nslots * C, C, B.GLEAM_EVICT_LRU)
    oc = oracle.OracleCache(nslots * C, C, B.GLEAM_EVICT_LRU)
    rng = np.random.default_rng(7)
    alphabet = [W.random_bytes(C, seed=900 + k) for k in range(100)]
    with gc:
        for call in range(40):
            nch = int(rng.integers(1, 20))
            dedup_both(gc, oc, _alphabet_payload(rng, C, nch, alphabet, 0))
        compare_cache(gc, oc)
        assert gc.stats()["evictions"] == oc.stats()["evictions"] > 0


def test_the_library_takes_the_single_block_path():
    # a call that runs as one kernel has nothing in the profile's second phase
    # (its events are recorded back to back); with the path off, the resolve
    # and pack kernels take several microseconds per call there
    C = 4 * KiB
    payloads = [W.random_bytes(16 * C, seed=700 + k).to("cuda") for k in range(20)]
    phase1 = {}
    for limit in (64, 0):
        gc = Cache(4 * MiB, C)
        gc.debug_set(B.GLEAM_DEBUG_SMALL_CALLS, limit)
        with gc:
            B.gleam_cache_profile(gc.handle, True)
            for p in payloads:
                gc.dedup(p)
            rc, ms, n = B.gleam_cache_profile_read(gc.handle, 2)
            assert rc == 0 and n == [20, 20]
            phase1[limit] = ms[1] * 1e3 / 20  # us per call
    assert phase1[64] < 3.0, phase1
    assert phase1[0] > 5.0, phase1


@pytest.mark.parametrize("C", [1 * KiB, 4 * KiB, 64 * KiB])
def test_write_through_never_changes_outputs(C):
    # payloads of misses only (written ahead and used), then payloads mixing
    # hits, in-call duplicates and misses (written ahead where they land, copied
    # over elsewhere), under every write-through mode and both call paths
    rng = np.random.default_rng(C)
    fresh = iter(range(10_000, 20_000))
    alphabet = [W.random_bytes(C, seed=300 + k) for k in range(8)]
    calls = []
    for k in range(10):
        nch = int(rng.integers(1, 200))
        if k % 3 == 0:  # misses only
            parts = [W.random_bytes(C, seed=next(fresh)) for _ in range(nch)]
        else:
            parts = [alphabet[int(rng.integers(len(alphabet)))] if rng.random() < 0.5
                     else W.random_bytes(C, seed=next(fresh)) for _ in range(nch)]
        if rng.random() < 0.5:
            parts.append(W.random_bytes(int(rng.integers(1, C)), seed=next(fresh)))
        calls.append(torch.cat(parts))
    exports = []
    for mode in (0, 1, 2):
        for small in (64, 0):
            gc = Cache(4096 * C, C)
            oc = oracle.OracleCache(4096 * C, C)
            gc.debug_set(B.GLEAM_DEBUG_SPECULATE, mode)
            gc.debug_set(B.GLEAM_DEBUG_SMALL_CALLS, small)
            with gc:
                for payload in calls:
                    dedup_both(gc, oc, payload)
                compare_cache(gc, oc)
                st = gc.stats()
                if mode == 1:
                    assert st["spec_chunks"] > 0
                if mode == 2:
                    assert st["spec_chunks"] == 0
                keys, lens, count = gc.export()
                exports.append(sorted(zip(keys[:count].tolist(), lens[:count].tolist())))
    assert all(e == exports[0] for e in exports)
