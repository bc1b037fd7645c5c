"""Pins of the oracle's paper-identifier mode (App. B.1): MD5 of a chunk's
first 1024 bits as the key, chunks under 1 KiB never cached; verify kept."""
import hashlib
import os

import numpy as np
import pytest

import oracle
from tests._refs import BruteCache
from tests.test_oracle_dedup import _mask_bits

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "md5_vectors.txt")


def _vectors():
    out = []
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip("\n"):
            continue
        text, digest = line.rstrip("\n").split("\t")
        out.append((text.encode("ascii"), digest))
    return out


@pytest.mark.parametrize("text,digest", _vectors())
def test_rfc1321_test_suite(text, digest):
    assert oracle.md5(text).hex() == digest


def test_every_length_0_to_300_vs_hashlib():
    data = np.random.default_rng(41).integers(0, 256, 300, dtype=np.uint8).tobytes()
    for n in range(301):
        assert oracle.md5(data[:n]) == hashlib.md5(data[:n]).digest(), n


def _hashlib_key(chunk: bytes) -> int:
    return int.from_bytes(hashlib.md5(chunk[:128]).digest()[:8], "little")


def test_paper_key_is_md5_of_the_first_128_bytes():
    data = np.random.default_rng(42).integers(0, 256, 5000, dtype=np.uint8).tobytes()
    for n in (1, 100, 127, 128, 129, 1024, 5000):
        assert oracle.paper_key(data[:n]) == _hashlib_key(data[:n])
    # only the prefix matters
    assert oracle.paper_key(data[:128] + bytes(1000)) == oracle.paper_key(data[:128])


@pytest.mark.parametrize("key16", [False, True])
@pytest.mark.parametrize("seed", range(4))
def test_paper_mode_matches_brute_force(seed, key16):
    rng = np.random.default_rng(200 + seed)
    C = 2048
    flags = oracle.PAPER_IDS | (oracle.KEY16 if key16 else 0)
    keyf = (lambda b: _hashlib_key(b) & 0xFFFF) if key16 else _hashlib_key
    oc = oracle.OracleCache(300 * C, C, flags)
    bc = BruteCache(300, key_fn=keyf, paper_min=1024)
    # chunks sharing a 128-byte prefix: same paper key, different bytes
    head = rng.integers(0, 256, 128, dtype=np.uint8).tobytes()
    alphabet = [head + rng.integers(0, 256, C - 128, dtype=np.uint8).tobytes() for _ in range(6)]
    alphabet += [rng.integers(0, 256, C, dtype=np.uint8).tobytes() for _ in range(6)]
    for call in range(8):
        parts = [alphabet[int(rng.integers(len(alphabet)))] for _ in range(int(rng.integers(0, 30)))]
        if rng.random() < 0.7:  # ragged tails, some under 1 KiB
            parts.append(rng.integers(0, 256, int(rng.choice([100, 700, 1023, 1024, 1500])),
                                      dtype=np.uint8).tobytes())
        payload = b"".join(parts)
        before = oc.stats()
        out = oc.dedup(payload, chunk_slots=True)
        brc, b = bc.dedup(payload, C)
        assert out[0] == brc
        if brc < 0:
            continue
        _, mask, miss, packed, slots = out
        N = (len(payload) + C - 1) // C
        assert _mask_bits(mask, N) == _mask_bits(b["mask"], N)
        assert miss.tolist() == b["miss"] and packed.tobytes() == b["packed"]
        assert slots.tolist() == b["slots"]
        after = oc.stats()
        assert after["verify_rejects"] - before["verify_rejects"] == b["rejects"]
    keys, lens = oc.entries()
    assert len(keys) == len(bc.items)
    for s, (k, data) in enumerate(bc.items):
        assert oc.slot_bytes(s) == data and int(keys[s]) == k


def test_same_prefix_chunks_are_separated_by_the_verify():
    """Without the byte check these would alias (the paper trusts the hash);
    with it, outputs equal the full-XXH64 mode whenever no chunk is < 1 KiB."""
    rng = np.random.default_rng(43)
    C = 4096
    head = rng.integers(0, 256, 128, dtype=np.uint8).tobytes()
    chunks = [head + rng.integers(0, 256, C - 128, dtype=np.uint8).tobytes() for _ in range(50)]
    payload = b"".join(chunks[int(i)] for i in rng.integers(0, 50, 400))
    a = oracle.OracleCache(1000 * C, C, oracle.PAPER_IDS)
    b = oracle.OracleCache(1000 * C, C)
    ra, ma, ia, pa = a.dedup(payload)
    rb, mb, ib, pb = b.dedup(payload)
    assert ra == rb == len(set(payload[i:i + C] for i in range(0, len(payload), C)))
    assert (ma == mb).all() and (ia == ib).all() and (pa == pb).all()
    assert a.stats()["verify_rejects"] == ra - 1  # every later distinct chunk collides


def test_small_chunks_are_never_cached():
    C = 4096
    oc = oracle.OracleCache(100 * C, C, oracle.PAPER_IDS)
    small = bytes(range(200)) * 3           # 600 bytes
    for _ in range(3):
        rc, mask, miss, packed, slots = oc.dedup(small, chunk_slots=True)
        assert rc == 1 and int(mask[0]) == 0 and slots.tolist() == [oracle.NO_SLOT]
    st = oc.stats()
    assert st["slots_used"] == 0 and st["inserts"] == 0 and st["misses"] == 3
