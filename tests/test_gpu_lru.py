"""GLEAM_EVICT_LRU (paper Sec. 4.1.3, reading R16) on the GPU against the
oracle: single calls and batches that keep a small cache full, so that most
calls evict; per-payload outputs, chunk slots, results, counters, the index
by slot and the stored bytes, bit for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300.cache import Cache, DedupOutputs, result_dict
from tests._parity import DEV, STAT_KEYS, compare_cache, to_device

pytestmark = [pytest.mark.gpu, pytest.mark.usefixtures("call_path")]
KiB = 1024


def _compare_all(gc, oc, check_bytes=64):
    compare_cache(gc, oc, check_bytes)
    assert gc.stats()["evictions"] == oc.stats()["evictions"]


def _batch_both(gc, oc, payloads):
    """One batch call on both sides; returns the status."""
    C = gc.chunk_bytes
    rc_o, outs_o, res_o = oc.dedup_batch([p.numpy() for p in payloads], chunk_slots=True)
    bufs = [to_device(p) for p in payloads]
    outs = [DedupOutputs.alloc(p.numel(), C, DEV) for p in payloads]
    res = torch.zeros(len(bufs), B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    total = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    slots = [torch.full((max(1, (p.numel() + C - 1) // C),), -1, dtype=torch.int32, device=DEV)
             for p in payloads]
    items = gc.batch_items(bufs, outs, [res[k] for k in range(len(bufs))], slots)
    gc.dedup_batch(None, items=items, total=total)
    torch.cuda.synchronize()
    tot = result_dict(total)
    if rc_o < 0:
        assert tot["status"] == rc_o, (tot, rc_o)
        return rc_o
    assert tot["status"] == 0 and tot["n_miss"] == rc_o, (tot, rc_o)
    for k, p in enumerate(payloads):
        if p.numel() == 0:
            continue
        mask_o, miss_o, packed_o, slots_o = outs_o[k]
        r = result_dict(res[k])
        for f, v in res_o[k].items():
            assert r[f] == v, (k, f, r[f], v)
        o = outs[k]
        nch = (p.numel() + C - 1) // C
        assert np.array_equal(o.hit_mask.cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o), k
        assert np.array_equal(o.miss_idx.cpu().numpy().view(np.uint32)[: len(miss_o)], miss_o), k
        assert np.array_equal(o.miss_bytes.cpu().numpy()[: len(packed_o)], packed_o), k
        assert np.array_equal(slots[k].cpu().numpy().view(np.uint32)[:nch], slots_o), k
    return rc_o


def _alphabet_payload(rng, alphabet, nch, C, tail):
    data = b"".join(alphabet[int(rng.integers(len(alphabet)))] for _ in range(nch))
    if tail:
        data += rng.integers(0, 256, tail, dtype=np.uint8).tobytes()
    return torch.frombuffer(bytearray(data), dtype=torch.uint8) if data else \
        torch.empty(0, dtype=torch.uint8)


@pytest.mark.parametrize("key16", [False, True])
@pytest.mark.parametrize("C", [64, 4 * KiB])
def test_lru_random_batches_match_oracle(C, key16):
    rng = np.random.default_rng(7 + C + key16)
    alphabet = [rng.integers(0, 256, C, dtype=np.uint8).tobytes() for _ in range(96)]
    nslots = 40
    flags = B.GLEAM_EVICT_LRU | (B.GLEAM_KEY16 if key16 else 0)
    gc = Cache(nslots * C, C, flags)
    oc = oracle.OracleCache(nslots * C, C, oracle.EVICT_LRU | (oracle.KEY16 if key16 else 0))
    capacity = 0
    for step in range(40):
        payloads = [_alphabet_payload(rng, alphabet, int(rng.integers(0, 12)), C,
                                      int(rng.integers(1, C)) if rng.random() < 0.3 else 0)
                    for _ in range(int(rng.integers(1, 4)))]
        rc = _batch_both(gc, oc, payloads)
        capacity += rc == oracle.ERR_CAPACITY
        _compare_all(gc, oc)
    assert oc.stats()["evictions"] > 50


@pytest.mark.parametrize("start_clock", [0, 0xFFF0, 0xFFFE0000])
def test_lru_many_slots_and_ties_across_blocks(start_clock):
    """A 20,000-slot cache filled by one call (one clock value: every slot
    ties), then calls that each need thousands of victims: the ties are broken
    by slot number across all blocks of the grid, and the 16-bit radix bins are
    crossed when the clock starts near a multiple of 2^16."""
    C = 256
    nslots = 20000
    gc = Cache(nslots * C, C, B.GLEAM_EVICT_LRU)
    gc.debug_set(B.GLEAM_DEBUG_CLOCK, start_clock)
    oc = oracle.OracleCache(nslots * C, C, oracle.EVICT_LRU)
    g = torch.Generator().manual_seed(5)
    base = torch.randint(0, 256, (nslots * C,), dtype=torch.uint8, generator=g)
    _batch_both(gc, oc, [base])
    for step in range(6):
        # a few old chunks are touched again, the rest is new
        pick = torch.randint(0, nslots, (500,), generator=g)
        old = base.view(nslots, C)[pick].reshape(-1)
        new = torch.randint(0, 256, ((3000 + 1000 * step) * C,), dtype=torch.uint8, generator=g)
        _batch_both(gc, oc, [old, new])
        _compare_all(gc, oc, check_bytes=256)
    assert oc.stats()["evictions"] > 10000


def test_failed_call_gives_the_stamps_back():
    """A call that hits the oldest slot and brings more new chunks than the
    other slots can take fails with CAPACITY; its hit must not count as a use,
    so the next call evicts that oldest slot, as the oracle (which never saw
    the failed call) does."""
    C = 64
    chunks = [bytes([v]) * C for v in range(1, 9)]
    gc = Cache(8 * C, C, B.GLEAM_EVICT_LRU)
    oc = oracle.OracleCache(8 * C, C, oracle.EVICT_LRU)
    t = lambda b: torch.frombuffer(bytearray(b), dtype=torch.uint8)
    for ch in chunks:  # slot k gets last use k + 1
        _batch_both(gc, oc, [t(ch)])
    failing = chunks[0] + b"".join(bytes([50 + v]) * C for v in range(8))
    assert _batch_both(gc, oc, [t(failing)]) == oracle.ERR_CAPACITY
    _compare_all(gc, oc)
    assert _batch_both(gc, oc, [t(bytes([100]) * C)]) == 1
    _compare_all(gc, oc)
    assert gc.read_slot(0) == bytes([100]) * C


def test_timeout_in_an_lru_call_leaves_the_order_unchanged():
    C = 4 * KiB
    nslots = 64
    gc = Cache(nslots * C, C, B.GLEAM_EVICT_LRU)
    oc = oracle.OracleCache(nslots * C, C, oracle.EVICT_LRU)
    g = torch.Generator().manual_seed(3)
    first = torch.randint(0, 256, (nslots * C,), dtype=torch.uint8, generator=g)
    _batch_both(gc, oc, [first])
    # the failing call hits half of the slots and brings 8 new chunks
    again = first.view(nslots, C)[::2].reshape(-1)
    fresh = torch.randint(0, 256, (8 * C,), dtype=torch.uint8, generator=g)
    gc.debug_set(B.GLEAM_DEBUG_WAIT_LIMIT_NS, 200_000_000)
    gc.debug_set(B.GLEAM_DEBUG_SKIP_ARRIVE, 0)
    bufs = [to_device(again), to_device(fresh)]
    outs = [DedupOutputs.alloc(b.numel(), C, DEV) for b in bufs]
    total = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    gc.dedup_batch(bufs, outs, total=total)
    torch.cuda.synchronize()
    assert result_dict(total)["status"] == B.GLEAM_ERR_TIMEOUT
    gc.debug_set(B.GLEAM_DEBUG_WAIT_LIMIT_NS, 4_000_000_000)
    _compare_all(gc, oc)
    # the oracle never saw the failed call: the next call must evict the same slots
    assert _batch_both(gc, oc, [fresh]) == 8
    _compare_all(gc, oc)


def test_single_calls_and_noalloc_with_eviction():
    """gleam_dedup_copy and the allocation-free call evict like the oracle."""
    C = 1 * KiB
    nslots = 100
    gc = Cache(nslots * C, C, B.GLEAM_EVICT_LRU)
    oc = oracle.OracleCache(nslots * C, C, oracle.EVICT_LRU)
    g = torch.Generator().manual_seed(11)
    pool = torch.randint(0, 256, (300, C), dtype=torch.uint8, generator=g)
    for step in range(30):
        pick = torch.randint(0, 300, (int(torch.randint(1, 60, (1,), generator=g)),), generator=g)
        host = pool[pick].reshape(-1).contiguous()
        rc_o, mask_o, miss_o, packed_o, slots_o = oc.dedup(host.numpy(), chunk_slots=True)
        d = to_device(host)
        out = DedupOutputs.alloc(host.numel(), C, DEV)
        if step % 2:
            res = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
            rc = B.gleam_dedup_copy_noalloc(gc.handle, d, host.numel(), out.hit_mask,
                                            out.miss_idx, out.miss_bytes, res, None)
            assert rc == 0
            torch.cuda.synchronize()
            r = result_dict(res)
            rc = r["status"] if r["status"] else r["n_miss"]
        else:
            try:
                rc, out = gc.dedup(d, out)
            except B.GleamError as e:
                rc = e.rc
        assert rc == rc_o, (step, rc, rc_o)
        if rc >= 0:
            assert np.array_equal(out.hit_mask.cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o)
            assert np.array_equal(out.miss_idx.cpu().numpy().view(np.uint32)[:rc], miss_o)
            assert np.array_equal(out.miss_bytes.cpu().numpy()[: len(packed_o)], packed_o)
        _compare_all(gc, oc)
    assert oc.stats()["evictions"] > 100


def test_without_the_flag_nothing_is_evicted():
    C = 64
    gc = Cache(4 * C, C)
    d = torch.randint(0, 256, (5 * C,), dtype=torch.uint8,
                      generator=torch.Generator().manual_seed(1)).to(DEV)  # 5 distinct chunks
    with pytest.raises(B.GleamError) as e:
        gc.dedup(d)
    assert e.value.rc == B.GLEAM_ERR_CAPACITY
    assert gc.stats()["evictions"] == 0
