"""gleam_dedup_copy_batch vs the oracle making the same calls one at a time:
per-payload outputs and results, counters and final cache, bit for bit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache, DedupOutputs, result_dict
from tests._parity import DEV, compare_cache, to_device

pytestmark = [pytest.mark.gpu, pytest.mark.usefixtures("call_path")]
KiB, MiB = 1024, 1 << 20


def _batch_vs_oracle(gc, oc, payloads_host, offsets=None, expect_rc=None):
    C = gc.chunk_bytes
    bufs = [to_device(h, (offsets[k] if offsets else 0)) for k, h in enumerate(payloads_host)]
    outs = [DedupOutputs.alloc(h.numel(), C, DEV) for h in payloads_host]
    res = torch.zeros(len(bufs), B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    total = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    slots = [torch.full((max(1, (h.numel() + C - 1) // C),), -1, dtype=torch.int32, device=DEV)
             for h in payloads_host]
    items = gc.batch_items(bufs, outs, [res[k] for k in range(len(bufs))], slots)
    gc.dedup_batch(None, items=items, total=total)
    torch.cuda.synchronize()
    tot = result_dict(total)
    if expect_rc is not None:
        assert tot["status"] == expect_rc
        return tot
    assert tot["status"] == 0, tot
    sums = dict(n_miss=0, n_hit_cache=0, n_hit_intra=0, verify_rejects=0, miss_bytes=0)
    for k, h in enumerate(payloads_host):
        before = oc.stats()
        out_o = oc.dedup(h.numpy(), chunk_slots=True)
        rc, mask_o, miss_o, packed_o, slots_o = out_o
        after = oc.stats()
        r = result_dict(res[k])
        assert r["status"] == 0 and r["n_miss"] == rc, (k, r, rc)
        assert r["miss_bytes"] == len(packed_o)
        assert r["n_hit_cache"] == after["hits_cache"] - before["hits_cache"], k
        assert r["n_hit_intra"] == after["hits_intra"] - before["hits_intra"], k
        assert r["verify_rejects"] == after["verify_rejects"] - before["verify_rejects"], k
        for f in sums:
            sums[f] += r[f]
        if h.numel() == 0:
            continue
        o = outs[k]
        assert np.array_equal(o.hit_mask.cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o), k
        assert np.array_equal(o.miss_idx.cpu().numpy().view(np.uint32)[:rc], miss_o), k
        assert np.array_equal(o.miss_bytes.cpu().numpy()[: len(packed_o)], packed_o), k
        nch = (h.numel() + C - 1) // C
        assert np.array_equal(slots[k].cpu().numpy().view(np.uint32)[:nch], slots_o), k
    for f in sums:
        assert tot[f] == sums[f], f
    return tot


def test_llama_shaped_batch_with_bit_flips():
    C = 64 * KiB
    up = W.weight_upload(W.scaled_shapes(W.llama3_8b_shapes(), 8)[:80], torch.bfloat16)
    gc, oc = Cache(512 * MiB, C), oracle.OracleCache(512 * MiB, C)
    with gc:
        pays = [up.payload(k).clone() for k in range(len(up.sizes))]
        _batch_vs_oracle(gc, oc, pays)
        chunks = up.chunks(C)
        ids = W.select_chunks(len(chunks), 0.10)
        W.flip_one_bit_per_chunk(up.buf, chunks, ids)
        pays = [up.payload(k).clone() for k in range(len(up.sizes))]
        tot = _batch_vs_oracle(gc, oc, pays)
        assert tot["n_miss"] == len(ids)
        compare_cache(gc, oc)


def test_cross_payload_duplicates_tails_and_empty_payloads():
    C = 4 * KiB
    a = W.random_bytes(10 * C + 100, seed=1)
    b = W.random_bytes(3 * C, seed=2)
    tail = a[10 * C:].clone()               # 100 bytes, equal to a's tail chunk
    empty = torch.zeros(0, dtype=torch.uint8)
    pays = [a, empty, b, a.clone(), tail, torch.cat([b, tail]), empty, b[:C].clone()]
    gc, oc = Cache(64 * MiB, C), oracle.OracleCache(64 * MiB, C)
    with gc:
        _batch_vs_oracle(gc, oc, pays, offsets=[0, 0, 16, 0, 1, 0, 0, 4])
        compare_cache(gc, oc)


@pytest.mark.parametrize("key16", [False, True])
def test_random_batches_match_sequential_calls(key16):
    rng = np.random.default_rng(77 + key16)
    C = 1 * KiB
    flags = B.GLEAM_KEY16 if key16 else 0
    gc, oc = Cache(40000 * C, C, flags), oracle.OracleCache(40000 * C, C, flags)
    alphabet = [W.random_bytes(C, seed=500 + k) for k in range(300)]
    tails = [W.random_bytes(int(rng.integers(1, C)), seed=900 + k) for k in range(5)]
    with gc:
        for batch in range(4):
            pays = []
            for _ in range(int(rng.integers(1, 60))):
                parts = [alphabet[int(rng.integers(len(alphabet)))]
                         for _ in range(int(rng.integers(0, 80)))]
                if rng.random() < 0.5:
                    parts.append(tails[int(rng.integers(len(tails)))])
                pays.append(torch.cat(parts) if parts else torch.zeros(0, dtype=torch.uint8))
            _batch_vs_oracle(gc, oc, pays,
                             offsets=[int(rng.choice([0, 0, 0, 8, 3])) for _ in pays])
        compare_cache(gc, oc)


def test_key16_batch_with_crafted_collisions():
    C = 4 * KiB
    adv = W.adversarial_payload(8 * MiB, C)
    gc = Cache(64 * MiB, C, B.GLEAM_KEY16)
    oc = oracle.OracleCache(64 * MiB, C, oracle.KEY16)
    with gc:
        pick, rows = W.crafted_collisions(adv, C, count=64)
        host_rows = adv.buf.view(-1, C)[pick].numpy()
        for i, r in enumerate(rows):
            key = oracle.xxh64(host_rows[i])
            assert oc.debug_insert(key, r.numpy()) == 0
            gc.debug_insert(key, r.to(DEV))
        pays = [p.clone() for p in adv.buf.split(100 * C)]   # chunk-aligned payloads
        tot = _batch_vs_oracle(gc, oc, pays)
        assert tot["verify_rejects"] >= 64
        compare_cache(gc, oc)


def test_batch_capacity_is_all_or_nothing():
    C = 1 * KiB
    gc, oc = Cache(100 * C, C), oracle.OracleCache(100 * C, C)
    with gc:
        _batch_vs_oracle(gc, oc, [W.random_bytes(30 * C, seed=1), W.random_bytes(30 * C, seed=2)])
        before = gc.stats()
        tot = _batch_vs_oracle(gc, oc, [W.random_bytes(30 * C, seed=3),
                                        W.random_bytes(30 * C, seed=4)],
                               expect_rc=B.GLEAM_ERR_CAPACITY)
        assert tot["n_miss"] == 0
        assert gc.stats() == before
        _batch_vs_oracle(gc, oc, [W.random_bytes(30 * C, seed=3)])
        compare_cache(gc, oc)


def test_batch_then_single_calls_interleave():
    C = 4 * KiB
    up = W.weight_upload(W.scaled_shapes(W.gpt2_small_shapes(), 8), torch.float32)
    gc, oc = Cache(128 * MiB, C), oracle.OracleCache(128 * MiB, C)
    s = torch.cuda.Stream()
    with gc:
        pays = [up.payload(k).clone() for k in range(len(up.sizes))]
        _batch_vs_oracle(gc, oc, pays[: len(pays) // 2])
        from tests._parity import dedup_both
        for p in pays[len(pays) // 2:]:
            dedup_both(gc, oc, p)
        _batch_vs_oracle(gc, oc, pays)
        compare_cache(gc, oc)
