"""Feature combinations against the oracle: LRU eviction with host-resident
payloads and host outputs, with the paper's identifiers, with KEY16 and the
debug checks — outputs, results, counters and stored bytes bit for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300.cache import Cache, result_dict
from tests._parity import DEV, compare_cache

pytestmark = [pytest.mark.gpu, pytest.mark.usefixtures("call_path")]


def _batch(gc, oc, payloads, host=False, host_out=False):
    C = gc.chunk_bytes
    rc_o, outs_o, res_o = oc.dedup_batch([p.numpy() for p in payloads], chunk_slots=True)
    bufs, masks, idxs, packeds, slots = [], [], [], [], []
    for p in payloads:
        n = p.numel()
        N = (n + C - 1) // C
        bufs.append(p.pin_memory() if host else p.to(DEV))
        masks.append(torch.zeros(max(1, (N + 31) // 32), dtype=torch.int32, device=DEV))
        mk = (lambda *a, **k: torch.empty(*a, **k).pin_memory()) if host_out else \
            (lambda *a, **k: torch.empty(*a, device=DEV, **k))
        idxs.append(mk(max(1, N), dtype=torch.int32))
        packeds.append(mk(max(1, n), dtype=torch.uint8))
        slots.append(mk(max(1, N), dtype=torch.int32))
    res = torch.zeros(len(payloads), B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    total = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    items = B.payload_array([(bufs[k], payloads[k].numel(), masks[k], idxs[k], packeds[k], res[k],
                              slots[k]) for k in range(len(payloads))])
    call = B.gleam_dedup_copy_host_batch if host else B.gleam_dedup_copy_batch
    assert call(gc.handle, items, total, None) == 0
    torch.cuda.synchronize()
    tot = result_dict(total)
    if rc_o < 0:
        assert tot["status"] == rc_o
        return rc_o
    assert tot["status"] == 0 and tot["n_miss"] == rc_o, (tot, rc_o)
    for k, p in enumerate(payloads):
        if p.numel() == 0:
            continue
        mask_o, miss_o, packed_o, slots_o = outs_o[k]
        r = result_dict(res[k])
        for f, v in res_o[k].items():
            assert r[f] == v, (k, f)
        N = (p.numel() + C - 1) // C
        assert np.array_equal(masks[k].cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o)
        assert np.array_equal(idxs[k].cpu().numpy().view(np.uint32)[: len(miss_o)], miss_o)
        assert np.array_equal(packeds[k].cpu().numpy()[: len(packed_o)], packed_o)
        assert np.array_equal(slots[k].cpu().numpy().view(np.uint32)[:N], slots_o)
    return rc_o


def _rand_batches(seed, C, alphabet_n, steps, max_chunks):
    rng = np.random.default_rng(seed)
    alphabet = [rng.integers(0, 256, C, dtype=np.uint8).tobytes() for _ in range(alphabet_n)]
    for _ in range(steps):
        pays = []
        for _ in range(int(rng.integers(1, 4))):
            data = b"".join(alphabet[int(rng.integers(alphabet_n))]
                            for _ in range(int(rng.integers(0, max_chunks))))
            if rng.random() < 0.3:
                data += rng.integers(0, 256, int(rng.integers(1, C)), dtype=np.uint8).tobytes()
            pays.append(torch.frombuffer(bytearray(data), dtype=torch.uint8) if data
                        else torch.empty(0, dtype=torch.uint8))
        yield pays


@pytest.mark.parametrize("host_out", [False, True])
def test_lru_with_host_payloads(host_out):
    C, nslots = 1024, 48
    gc = Cache(nslots * C, C, B.GLEAM_EVICT_LRU)
    oc = oracle.OracleCache(nslots * C, C, oracle.EVICT_LRU)
    with gc:
        for pays in _rand_batches(1, C, 100, 30, 16):
            _batch(gc, oc, pays, host=True, host_out=host_out)
            compare_cache(gc, oc)
        assert oc.stats()["evictions"] > 50 and gc.stats()["evictions"] == oc.stats()["evictions"]


def test_paper_ids_with_lru_and_debug_checks():
    C, nslots = 2048, 40
    gc = Cache(nslots * C, C, B.GLEAM_EVICT_LRU | B.GLEAM_PAPER_IDS | B.GLEAM_DEBUG_CHECKS)
    oc = oracle.OracleCache(nslots * C, C, oracle.EVICT_LRU | oracle.PAPER_IDS)
    with gc:
        for pays in _rand_batches(2, C, 90, 30, 14):
            _batch(gc, oc, pays)
            compare_cache(gc, oc)
        assert gc.stats()["evictions"] == oc.stats()["evictions"] > 0


def test_key16_lru_debug_checks():
    C, nslots = 256, 64
    gc = Cache(nslots * C, C, B.GLEAM_EVICT_LRU | B.GLEAM_KEY16 | B.GLEAM_DEBUG_CHECKS)
    oc = oracle.OracleCache(nslots * C, C, oracle.EVICT_LRU | oracle.KEY16)
    with gc:
        for pays in _rand_batches(3, C, 200, 30, 20):
            _batch(gc, oc, pays)
            compare_cache(gc, oc)
        assert gc.stats()["evictions"] == oc.stats()["evictions"] > 0
