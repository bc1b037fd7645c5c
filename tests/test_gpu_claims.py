"""Group claims made by the hash kernel for a call resolved in one launch (one
payload of at most 16,384 chunks, more than one resolve block): two different
chunks whose claims meet in the per-call table with the same 32-bit tag (found
by search, tests/golden/claim_tag_collision.txt) make the call take its general
path, which claims the groups again by the whole fingerprint.  Outputs and the
cache must equal the oracle's, with and without in-call duplicates of either
chunk, and when the call is repeated."""
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import workloads as W
from tests._parity import compare_cache, dedup_both

C = 32
N = 300  # a 1,024-entry group table, two resolve blocks
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                      "claim_tag_collision.txt")


def _pair():
    vals = {}
    with open(GOLDEN) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            parts = line.split()
            vals[parts[0]] = parts[1:]
    a = np.frombuffer(bytes.fromhex(vals["chunk_a"][0]), dtype=np.uint8)
    b = np.frombuffer(bytes.fromhex(vals["chunk_b"][0]), dtype=np.uint8)
    return a, b, int(vals["xxh64_a"][0], 16), int(vals["xxh64_b"][0], 16)


def test_fixture_chunks_have_their_recorded_fingerprints():
    # the pair is two distinct chunks whose oracle fingerprints are the ones
    # written next to them
    a, b, ha, hb = _pair()
    assert len(a) == len(b) == C and not np.array_equal(a, b)
    assert oracle.xxh64(a) == ha and oracle.xxh64(b) == hb and ha != hb


def _payload(extra_dups: bool) -> torch.Tensor:
    a, b, _, _ = _pair()
    rows = W.random_bytes(N * C, seed=91).view(N, C).clone()
    rows[10] = torch.from_numpy(a.copy())
    rows[200] = torch.from_numpy(b.copy())
    if extra_dups:
        rows[250] = rows[10]
        rows[260] = rows[200]
        rows[299] = rows[10]
    return rows.reshape(-1).contiguous()


@pytest.mark.gpu
@pytest.mark.usefixtures("call_path")
@pytest.mark.parametrize("extra_dups", [False, True])
def test_tag_collision_takes_the_general_path_with_oracle_results(extra_dups):
    from paper_2607_23115_gb300.cache import Cache
    payload = _payload(extra_dups)
    gc = Cache(4 * N * C, C)
    oc = oracle.OracleCache(4 * N * C, C)
    with gc:
        dedup_both(gc, oc, payload)
        dedup_both(gc, oc, payload)  # every chunk now a cache hit
        compare_cache(gc, oc)
        st = gc.stats()
        assert st["hits_intra"] == (3 if extra_dups else 0)
