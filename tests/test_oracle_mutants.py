"""The pins bind: each plausible mistake planted in a copy of the oracle (a
dropped term, a wrong constant, shift or rotation, a wrong index, a missed
case of the dedup rule) makes at least one pin fail.  Mutants are built from
the oracle's source on the CPU; the real oracle is never modified."""
import ctypes
import os
import subprocess
import tempfile

import numpy as np
import pytest

import oracle
from tests import test_oracle_dedup as D
from tests import test_oracle_lru as L
from tests._refs import xxh64_lib

MUTANTS = [
    ("round rotate 31 -> 30", "acc = rotl64(acc, 31);", "acc = rotl64(acc, 30);"),
    ("convergence rotate 18 -> 17", "rotl64(v[3], 18)", "rotl64(v[3], 17)"),
    ("length term dropped", "h += static_cast<uint64_t>(len);", ""),
    ("4-byte tail uses P2", "h ^= static_cast<uint64_t>(read_le32(p + off)) * kP1;",
     "h ^= static_cast<uint64_t>(read_le32(p + off)) * kP2;"),
    ("avalanche shift 29 -> 28", "h ^= h >> 29;", "h ^= h >> 28;"),
    ("length not part of a candidate", "if (it->second.len != len) continue;", ""),
    ("earlier misses of the call not looked up", "look(fresh_index, fresh_bytes, true);", ""),
    ("reject counted without a candidate", "if (candidate) ++P.rejects;", "++P.rejects;"),
    ("capacity off by one", "if (stored > c->nslots - slots0)", "if (stored >= c->nslots - slots0)"),
    ("miss packed at its chunk offset", "std::memcpy(P.packed + rank * C, chunk, len);\n      Entry e",
     "std::memcpy(P.packed + i * C, chunk, len);\n      Entry e"),
    ("hit reports a fresh slot", "if (P.chunk_slot) P.chunk_slot[i] = static_cast<uint32_t>(hit_slot);",
     "if (P.chunk_slot) P.chunk_slot[i] = static_cast<uint32_t>(slots0 + stored);"),
    ("LRU evicts the most recently used",
     "return c->last_use[x] != c->last_use[y] ? c->last_use[x] < c->last_use[y] : x < y;",
     "return c->last_use[x] != c->last_use[y] ? c->last_use[x] > c->last_use[y] : x < y;"),
    ("LRU ties go to the higher slot",
     "return c->last_use[x] != c->last_use[y] ? c->last_use[x] < c->last_use[y] : x < y;",
     "return c->last_use[x] != c->last_use[y] ? c->last_use[x] < c->last_use[y] : x > y;"),
    ("a call may evict what it hits", "if (!used[s]) cand.push_back(s);", "cand.push_back(s);"),
    ("hits do not refresh the last use", "if (used[s]) c->last_use[s] = now;", ""),
    ("victims keep their index entries",
     "it = gone[it->second.slot] ? c->index.erase(it) : std::next(it);", "it = std::next(it);"),
    ("an earlier payload's miss counts as in-call",
     "if (fresh_payload[hit_slot] == k) ++P.hits_intra; else ++P.hits_cache;", "++P.hits_intra;"),
]


def _pins_hold() -> bool:
    """A quick battery of the pins in test_oracle_xxh64 / test_oracle_dedup."""
    try:
        for text, seed, digest in [(b"", 0, 0xEF46DB3751D8E999), (b"abc", 0, 0x44BC2CF5AD770999),
                                   (b"Nobody inspects the spammish repetition", 0,
                                    0xFBCEA83C8A378BF1)]:
            assert oracle.xxh64(text, seed) == digest
        data = np.random.default_rng(11).integers(0, 256, 300, dtype=np.uint8).tobytes()
        for n in range(0, 301, 7):
            assert oracle.xxh64(data[:n]) == xxh64_lib(data[:n])
        for seed in (0, 1, 3):
            for key16 in (False, True):
                D.test_random_sequences_match_brute_force(seed, key16)
        D.test_capacity_leaves_cache_unchanged()
        D.test_tail_length_is_part_of_equality()
        D.test_crafted_collisions_are_rejected()
        D.test_length_is_part_of_a_candidate()
        for seed in (0, 1):
            L.test_lru_batches_match_brute_force(seed, False)
        L.test_lru_batches_match_brute_force(2, True)
        L.test_worked_example_slots_by_hand()
        L.test_a_call_never_evicts_what_it_hits()
    except AssertionError:
        return False
    return True


@pytest.fixture(scope="module")
def src():
    with open(oracle._SRC) as f:
        return f.read()


def test_the_real_oracle_passes_the_battery():
    assert _pins_hold()


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_is_caught(src, name, old, new, monkeypatch, tmp_path):
    assert src.count(old) == 1, name
    cpp = tmp_path / "mutant.cpp"
    cpp.write_text(src.replace(old, new))
    so = tmp_path / "libmutant.so"
    subprocess.check_call(["g++", "-O1", "-std=c++17", "-shared", "-fPIC", "-o", str(so), str(cpp)])
    monkeypatch.setattr(oracle, "_lib", oracle._bind(ctypes.CDLL(str(so))))
    assert not _pins_hold(), "mutant survived: " + name
