"""GLEAM_PAPER_IDS (App. B.1 identifiers: MD5 of the first 1024 bits, chunks
under 1 KiB never cached) vs the oracle, bit for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache
from tests._parity import compare_cache, dedup_both
from tests.test_gpu_batch import _batch_vs_oracle

pytestmark = pytest.mark.gpu
KiB, MiB = 1024, 1 << 20


def _pair(cap, C, key16=False):
    g = B.GLEAM_PAPER_IDS | (B.GLEAM_KEY16 if key16 else 0)
    o = oracle.PAPER_IDS | (oracle.KEY16 if key16 else 0)
    return Cache(cap, C, g), oracle.OracleCache(cap, C, o)


def _alphabet(rng, C, n_same_prefix=8, n_other=8):
    head = torch.from_numpy(rng.integers(0, 256, 128, dtype=np.uint8))
    same = [torch.cat([head, torch.from_numpy(rng.integers(0, 256, C - 128, dtype=np.uint8))])
            for _ in range(n_same_prefix)]
    other = [torch.from_numpy(rng.integers(0, 256, C, dtype=np.uint8)) for _ in range(n_other)]
    return same + other


@pytest.mark.parametrize("key16", [False, True])
@pytest.mark.parametrize("C", [1024, 4096])
def test_paper_ids_single_calls_match_oracle(C, key16):
    rng = np.random.default_rng(C + key16)
    gc, oc = _pair(4000 * C, C, key16)
    alphabet = _alphabet(rng, C)
    with gc:
        for call in range(10):
            parts = [alphabet[int(rng.integers(len(alphabet)))]
                     for _ in range(int(rng.integers(0, 300)))]
            if rng.random() < 0.7:
                tail = int(rng.choice([1, 100, 1023, 1024, 1025, C - 1]))
                parts.append(torch.from_numpy(rng.integers(0, 256, tail, dtype=np.uint8)))
            payload = torch.cat(parts) if parts else torch.zeros(0, dtype=torch.uint8)
            dedup_both(gc, oc, payload, offset=int(rng.choice([0, 0, 8, 3])))
        compare_cache(gc, oc)
        assert gc.stats()["verify_rejects"] > 0


def test_paper_ids_batches_match_sequential_oracle():
    rng = np.random.default_rng(5)
    C = 2048
    gc, oc = _pair(20000 * C, C)
    alphabet = _alphabet(rng, C)
    with gc:
        for _ in range(3):
            pays = []
            for _ in range(int(rng.integers(1, 40))):
                parts = [alphabet[int(rng.integers(len(alphabet)))]
                         for _ in range(int(rng.integers(0, 60)))]
                parts.append(torch.from_numpy(rng.integers(0, 256, int(rng.choice([500, 1500])),
                                                           dtype=np.uint8)))
                pays.append(torch.cat(parts))
            _batch_vs_oracle(gc, oc, pays)
        compare_cache(gc, oc)


def test_without_small_chunks_paper_ids_give_the_xxh64_outputs():
    C = 4096
    rng = np.random.default_rng(6)
    alphabet = _alphabet(rng, C, 20, 20)
    payload = torch.cat([alphabet[int(i)] for i in rng.integers(0, 40, 3000)])
    a, b = Cache(8000 * C, C, B.GLEAM_PAPER_IDS), Cache(8000 * C, C)
    with a, b:
        na, oa = a.dedup(payload.cuda())
        nb, ob = b.dedup(payload.cuda())
        assert na == nb
        assert torch.equal(oa.hit_mask, ob.hit_mask)
        assert torch.equal(oa.miss_idx[:na], ob.miss_idx[:nb])
        assert torch.equal(oa.miss_bytes[: na * C], ob.miss_bytes[: nb * C])
        assert a.stats()["verify_rejects"] > 0 == b.stats()["verify_rejects"]


def test_paper_ids_llama_shaped_bit_flips():
    C = 64 * KiB
    up = W.weight_upload(W.scaled_shapes(W.llama3_8b_shapes(), 8)[:40], torch.bfloat16)
    gc, oc = _pair(512 * MiB, C)
    with gc:
        pays = [up.payload(k).clone() for k in range(len(up.sizes))]
        _batch_vs_oracle(gc, oc, pays)
        chunks = up.chunks(C)
        ids = W.select_chunks(len(chunks), 0.10)
        W.flip_one_bit_per_chunk(up.buf, chunks, ids)
        pays = [up.payload(k).clone() for k in range(len(up.sizes))]
        tot = _batch_vs_oracle(gc, oc, pays)
        small = sum(1 for _, _, ln in chunks if ln < 1024)
        assert tot["n_miss"] == len(set(ids.tolist()) | {i for i, c in enumerate(chunks) if c[2] < 1024})
        compare_cache(gc, oc)
