"""Pins the oracle's LRU eviction (paper Sec. 4.1.3: shareable blocks are
evicted by last use) and its batch call against a hash-free brute force,
a worked example whose slots are fixed by hand, and invariants."""
import numpy as np
import pytest

import oracle
from tests._refs import BruteCache, xxh64_lib


def _bits(mask, N):
    return [(int(mask[i // 32]) >> (i % 32)) & 1 for i in range(N)]


def _check_batch(oc, bc, payloads, C):
    rc, outs, res = oc.dedup_batch(payloads, chunk_slots=True)
    brc, bouts = bc.dedup_batch(payloads, C)
    assert rc == brc
    if rc < 0:
        return rc
    for k, p in enumerate(payloads):
        if len(p) == 0:
            continue
        N = (len(p) + C - 1) // C
        mask, miss, packed, slots = outs[k]
        b = bouts[k]
        assert _bits(mask, N) == _bits(b["mask"], N)
        assert miss.tolist() == b["miss"]
        assert packed.tobytes() == b["packed"]
        assert slots.tolist() == b["slots"]
        assert res[k]["n_miss"] == len(b["miss"])
        assert res[k]["n_hit_cache"] == b["hits_cache"]
        assert res[k]["n_hit_intra"] == b["hits_intra"]
        assert res[k]["verify_rejects"] == b["rejects"]
        assert res[k]["miss_bytes"] == len(b["packed"])
    return rc


def _check_state(oc, bc):
    st = oc.stats()
    assert st["slots_used"] == len(bc.items)
    assert st["evictions"] == bc.evictions
    assert st["bytes_used"] == sum(len(b) for _, b in bc.items)
    keys, lens = oc.entries()
    for s, (key, b) in enumerate(bc.items):
        assert oc.slot_bytes(s) == b
        assert int(lens[s]) == len(b)
        if bc.key_fn:
            assert int(keys[s]) == key
    return st


@pytest.mark.parametrize("key16", [False, True])
@pytest.mark.parametrize("seed", range(8))
def test_lru_batches_match_brute_force(seed, key16):
    """Random batches over a small alphabet into a cache that fills up, so
    most calls evict: outputs, per-payload results, slots, stored bytes and
    counters equal the brute force."""
    rng = np.random.default_rng(100 + seed)
    C = 64
    alphabet = [rng.integers(0, 256, C, dtype=np.uint8).tobytes() for _ in range(24)]
    nslots = int(rng.integers(6, 14))
    flags = oracle.EVICT_LRU | (oracle.KEY16 if key16 else 0)
    oc = oracle.OracleCache(nslots * C, C, flags)
    kf = (lambda b: xxh64_lib(b) & 0xFFFF) if key16 else xxh64_lib
    bc = BruteCache(nslots, key_fn=kf, lru=True)
    evicted = capacity = 0
    for _ in range(30):
        payloads = []
        for _ in range(int(rng.integers(1, 4))):
            nch = int(rng.integers(0, 6))
            data = b"".join(alphabet[int(rng.integers(len(alphabet)))] for _ in range(nch))
            if rng.random() < 0.3:
                data += rng.integers(0, 256, int(rng.integers(1, C)), dtype=np.uint8).tobytes()
            payloads.append(data)
        before = oc.stats()
        rc = _check_batch(oc, bc, payloads, C)
        if rc < 0:
            assert rc == oracle.ERR_CAPACITY and oc.stats() == before
            capacity += 1
        st = _check_state(oc, bc)
        assert st["slots_used"] <= nslots
        assert st["inserts"] - st["evictions"] == st["slots_used"]
        evicted = st["evictions"]
    assert evicted > 0


def test_worked_example_slots_by_hand():
    """Four slots.  Call 1 stores A B C D (slots 0-3, last use 1).  Call 2 hits A
    (last use 2).  Call 3 stores E: the least recent slots are B C D (use 1),
    the lowest of them is B's, so E takes slot 1.  Call 4 brings B back: it
    misses and evicts C (slot 2).  Call 5 = [D, F] as one call: D is hit, so
    the victim is the oldest other slot, A (use 2), not D."""
    C = 32
    A, B_, Cc, D, E, F = (bytes([v]) * C for v in (1, 2, 3, 4, 5, 6))
    oc = oracle.OracleCache(4 * C, C, oracle.EVICT_LRU)
    assert oc.dedup(A + B_ + Cc + D, chunk_slots=True)[4].tolist() == [0, 1, 2, 3]
    assert oc.dedup(A, chunk_slots=True)[4].tolist() == [0]
    out = oc.dedup(E, chunk_slots=True)
    assert out[0] == 1 and out[4].tolist() == [1]
    out = oc.dedup(B_, chunk_slots=True)
    assert out[0] == 1 and out[4].tolist() == [2]
    out = oc.dedup(D + F, chunk_slots=True)
    assert out[0] == 1 and out[4].tolist() == [3, 0]
    assert [oc.slot_bytes(s) for s in range(4)] == [F, E, B_, D]
    assert oc.stats()["evictions"] == 3


def test_a_call_never_evicts_what_it_hits():
    """Every slot is hit by the call and one chunk is new: nothing may be
    evicted, so the call fails with CAPACITY and changes nothing."""
    C = 32
    chunks = [bytes([v]) * C for v in range(1, 5)]
    oc = oracle.OracleCache(4 * C, C, oracle.EVICT_LRU)
    assert oc.dedup(b"".join(chunks))[0] == 4
    st = oc.stats()
    assert oc.dedup(b"".join(chunks) + bytes([9]) * C)[0] == oracle.ERR_CAPACITY
    assert oc.stats() == st
    # without one of them the new chunk fits by evicting the unused one
    out = oc.dedup(b"".join(chunks[1:]) + bytes([9]) * C, chunk_slots=True)
    assert out[0] == 1 and out[4].tolist() == [1, 2, 3, 0]


def test_more_misses_than_slots_fail_even_with_lru():
    C = 32
    oc = oracle.OracleCache(3 * C, C, oracle.EVICT_LRU)
    four = b"".join(bytes([v]) * C for v in range(4))
    assert oc.dedup(four)[0] == oracle.ERR_CAPACITY
    assert oc.stats()["slots_used"] == 0


@pytest.mark.parametrize("seed", range(4))
def test_batch_without_eviction_equals_its_calls_in_order(seed):
    """R12: a batch gives the outputs and final cache of its calls made one
    after the other, when nothing has to be evicted."""
    rng = np.random.default_rng(200 + seed)
    C = 64
    alphabet = [rng.integers(0, 256, C, dtype=np.uint8).tobytes() for _ in range(10)]
    payloads = []
    for _ in range(5):
        nch = int(rng.integers(0, 8))
        payloads.append(b"".join(alphabet[int(rng.integers(10))] for _ in range(nch)) +
                        rng.integers(0, 256, int(rng.integers(0, 3)) * 17, dtype=np.uint8).tobytes())
    a = oracle.OracleCache(1000 * C, C)
    b = oracle.OracleCache(1000 * C, C)
    rc, outs, res = a.dedup_batch(payloads, chunk_slots=True)
    total = 0
    for k, p in enumerate(payloads):
        r = b.dedup(p, chunk_slots=True)
        if len(p) == 0:
            continue
        total += r[0]
        for x, y in zip(outs[k], r[1:]):
            assert np.array_equal(x, y)
        assert res[k]["n_miss"] == r[0]
    assert rc == total
    sa, sb = a.stats(), b.stats()
    for k in ("calls", "chunks", "hits_cache", "hits_intra", "misses", "inserts",
              "verify_rejects", "slots_used", "bytes_used"):
        assert sa[k] == sb[k], k
    ka, la = a.entries()
    kb, lb = b.entries()
    assert np.array_equal(ka, kb) and np.array_equal(la, lb)


def test_without_the_flag_a_full_cache_fails():
    C = 32
    oc = oracle.OracleCache(2 * C, C)
    assert oc.dedup(bytes([1]) * C + bytes([2]) * C)[0] == 2
    assert oc.dedup(bytes([3]) * C)[0] == oracle.ERR_CAPACITY
    assert oc.stats()["evictions"] == 0
