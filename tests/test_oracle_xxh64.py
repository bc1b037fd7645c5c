"""Pins the oracle's XXH64 against values it does not compute itself.

Published vectors (tests/golden), the installed libxxhash over every length
0..300 and across the 32-byte-stripe, 8-, 4- and 1-byte tail paths, and zstd
frame checksums (low 32 bits, decoded by libzstd).
"""
import os

import numpy as np
import pytest

import oracle
from tests._refs import xxh64_lib, zstd_accepts_checksum

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "xxh64_vectors.txt")


def _vectors():
    out = []
    with open(GOLDEN) as f:
        for line in f:
            if line.startswith("#") or not line.strip("\n"):
                continue
            text, seed, digest = line.rstrip("\n").split("\t")
            out.append((text.encode("ascii"), int(seed), int(digest, 16)))
    return out


def test_golden_file_has_vectors():
    v = _vectors()
    assert len(v) >= 6
    assert any(len(t) >= 32 for t, _, _ in v), "need a vector on the 32-byte stripe path"
    assert any(len(t) == 0 for t, _, _ in v)


@pytest.mark.parametrize("text,seed,digest", _vectors())
def test_published_vectors(text, seed, digest):
    assert oracle.xxh64(text, seed) == digest


def test_every_length_0_to_300_vs_libxxhash():
    rng = np.random.default_rng(11)
    data = rng.integers(0, 256, 300, dtype=np.uint8).tobytes()
    for n in range(0, 301):
        for seed in (0, 1, 2654435761, 2**64 - 1):
            assert oracle.xxh64(data[:n], seed) == xxh64_lib(data[:n], seed), (n, seed)


def test_large_and_odd_lengths_vs_libxxhash():
    rng = np.random.default_rng(12)
    for n in (1023, 1024, 4096 + 7, 65536, 65536 + 31, (1 << 20) + 13):
        data = rng.integers(0, 256, n, dtype=np.uint8).tobytes()
        assert oracle.xxh64(data) == xxh64_lib(data), n


def test_lengths_vs_zstd_frame_checksum():
    rng = np.random.default_rng(13)
    data = rng.integers(0, 256, 300, dtype=np.uint8).tobytes()
    for n in list(range(0, 80)) + [95, 96, 127, 128, 255, 256, 299]:
        h = oracle.xxh64(data[:n], 0)
        assert zstd_accepts_checksum(data[:n], h & 0xFFFFFFFF), n
        # and the frame check is discriminating: a wrong checksum is refused
        assert not zstd_accepts_checksum(data[:n], (h ^ 1) & 0xFFFFFFFF), n


def test_large_vs_zstd_frame_checksum():
    rng = np.random.default_rng(14)
    for n in (4096, 65536, 300001):
        data = rng.integers(0, 256, n, dtype=np.uint8).tobytes()
        assert zstd_accepts_checksum(data, oracle.xxh64(data) & 0xFFFFFFFF)


def test_single_bit_flips_change_the_hash():
    rng = np.random.default_rng(15)
    data = bytearray(rng.integers(0, 256, 4096, dtype=np.uint8).tobytes())
    base = oracle.xxh64(bytes(data))
    seen = {base}
    for bit in rng.choice(4096 * 8, 64, replace=False):
        d = bytearray(data)
        d[bit // 8] ^= 1 << (bit % 8)
        h = oracle.xxh64(bytes(d))
        assert h not in seen
        seen.add(h)


def test_fingerprint_chunks_and_whole_buffer():
    rng = np.random.default_rng(16)
    data = rng.integers(0, 256, 10 * 1024 + 77, dtype=np.uint8)
    raw = data.tobytes()
    for C in (32, 96, 1024, 4096, 10 * 1024 + 77, 1 << 16):
        fps = oracle.fingerprint(data, C)
        N = (len(raw) + C - 1) // C
        assert fps.shape == (N,)
        for i in range(N):
            assert int(fps[i]) == xxh64_lib(raw[i * C:(i + 1) * C]), (C, i)
    assert int(oracle.fingerprint(data, 0)[0]) == xxh64_lib(raw)
    assert int(oracle.fingerprint(np.zeros(0, np.uint8), 0)[0]) == 0xEF46DB3751D8E999
    assert oracle.fingerprint(np.zeros(0, np.uint8), 64).shape == (0,)
