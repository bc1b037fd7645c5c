"""Calls that overlap on the GPU (GLEAM_OVERLAP_CALLS): gleam_dedup_copy_async
calls enqueued back to back on one stream, each fingerprinting its payload
while the calls before it may still be running and waiting for them only
before it reads the index, against the oracle making the same calls one after
another: outputs, per-call results and the final cache, bit for bit.  Later
calls repeat chunks that earlier calls insert, so a call's hits include
chunks inserted by a call that was still running when it started."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache, DedupOutputs, result_dict
from tests._parity import DEV, compare_cache

pytestmark = [pytest.mark.gpu, pytest.mark.usefixtures("call_path")]
KiB, MiB = 1024, 1 << 20


def _calls_vs_oracle(gc, oc, payloads_host, streams=None):
    """Every payload as one async call, all enqueued before any result is read
    (on `streams[k]` if given, else the legacy default stream); then each
    call's outputs against the oracle's same call."""
    C = gc.chunk_bytes
    bufs = [h.to(DEV) for h in payloads_host]
    outs = [DedupOutputs.alloc(h.numel(), C, DEV) for h in payloads_host]
    res = torch.zeros(len(bufs), B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    torch.cuda.synchronize()
    for k in range(len(bufs)):
        gc.dedup_async(bufs[k], outs[k], res[k], stream=streams[k] if streams else None)
    torch.cuda.synchronize()
    totals = dict(n_miss=0, n_hit_cache=0, n_hit_intra=0, verify_rejects=0)
    for k, h in enumerate(payloads_host):
        before = oc.stats()
        rc, mask_o, miss_o, packed_o = oc.dedup(h.numpy())
        after = oc.stats()
        if h.numel() == 0:
            continue
        r = result_dict(res[k])
        assert r["status"] == 0 and r["n_miss"] == rc, (k, r, rc)
        assert r["miss_bytes"] == len(packed_o), k
        assert r["n_hit_cache"] == after["hits_cache"] - before["hits_cache"], k
        assert r["n_hit_intra"] == after["hits_intra"] - before["hits_intra"], k
        assert r["verify_rejects"] == after["verify_rejects"] - before["verify_rejects"], k
        o = outs[k]
        assert np.array_equal(o.hit_mask.cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o), k
        assert np.array_equal(o.miss_idx.cpu().numpy().view(np.uint32)[:rc], miss_o), k
        assert np.array_equal(o.miss_bytes.cpu().numpy()[: len(packed_o)], packed_o), k
        for f in totals:
            totals[f] += r[f]
    return totals


def _repeating_calls(C, seed):
    """Calls whose chunks repeat chunks of the calls just before them: a large
    first call (slow to fingerprint), then calls re-sending part of it, chunks
    repeated within a call, equal ragged tails, and fresh chunks."""
    base = W.random_bytes(700 * C, seed=seed).view(-1, C)
    rng = np.random.default_rng(seed)
    tail = W.random_bytes(C // 3, seed=seed + 1)
    calls = [base[0:250].reshape(-1),
             base[120:300].reshape(-1),                                     # half repeats call 0
             torch.cat([base[torch.from_numpy(rng.integers(0, 300, 40))].reshape(-1), tail]),
             tail.clone(),                                                  # call 2's tail alone
             base[torch.from_numpy(rng.integers(250, 700, 600))].reshape(-1),  # in-call repeats
             torch.zeros(0, dtype=torch.uint8),
             torch.cat([base[690:700].reshape(-1), base[0:3].reshape(-1)]),
             W.random_bytes(5 * C + 17, seed=seed + 2)]
    return [c.contiguous() for c in calls]


@pytest.mark.parametrize("C", [4 * KiB, 64 * KiB])
def test_calls_hit_chunks_that_still_running_calls_insert(C):
    calls = _repeating_calls(C, 71)
    gc = Cache(4096 * C, C, B.GLEAM_OVERLAP_CALLS)
    oc = oracle.OracleCache(4096 * C, C)
    with gc:
        t = _calls_vs_oracle(gc, oc, calls)
        assert t["n_hit_cache"] > 0 and t["n_hit_intra"] > 0
        # the same calls again: every chunk is now a cache hit
        t = _calls_vs_oracle(gc, oc, calls)
        assert t["n_miss"] == 0
        compare_cache(gc, oc)


def test_weight_upload_then_fine_tuned_variant_call_per_tensor():
    # one call per tensor: the base upload (all misses), then the variant with
    # one flipped bit in a tenth of the chunks (the misses), then the base again
    # (the flipped chunks' originals are still cached: all hits)
    C = 64 * KiB
    up = W.weight_upload(W.scaled_shapes(W.llama3_8b_shapes(), 8)[:60], torch.bfloat16)
    base = [up.payload(k).clone() for k in range(len(up.sizes))]
    chunks = up.chunks(C)
    ids = W.select_chunks(len(chunks), 0.10)
    W.flip_one_bit_per_chunk(up.buf, chunks, ids)
    variant = [up.payload(k).clone() for k in range(len(up.sizes))]
    gc = Cache(1024 * MiB, C, B.GLEAM_OVERLAP_CALLS)
    oc = oracle.OracleCache(1024 * MiB, C)
    with gc:
        _calls_vs_oracle(gc, oc, base)
        t = _calls_vs_oracle(gc, oc, variant)
        assert t["n_miss"] == len(ids)
        t = _calls_vs_oracle(gc, oc, base)
        assert t["n_miss"] == 0
        compare_cache(gc, oc)


def test_key16_collisions_across_overlapping_calls():
    # 16-bit keys: chunks of different calls share keys, crafted entries share
    # the keys of chunks to come; every candidate must be compared
    C = 4 * KiB
    adv = W.adversarial_payload(2048 * C, C)
    pick, rows = W.crafted_collisions(adv, C, count=32)
    gc = Cache(8192 * C, C, B.GLEAM_KEY16 | B.GLEAM_OVERLAP_CALLS)
    oc = oracle.OracleCache(8192 * C, C, oracle.KEY16)
    buf = adv.buf.view(-1, C)
    with gc:
        for i in range(32):
            key = oracle.xxh64(buf[int(pick[i])].numpy())
            gc.debug_insert(key, rows[i].to(DEV))
            oc.debug_insert(key, rows[i].numpy())
        calls = [buf[a:b].reshape(-1).contiguous() for a, b in
                 ((0, 600), (300, 900), (900, 1000), (0, 1200), (1200, 2048), (100, 2000))]
        t = _calls_vs_oracle(gc, oc, calls)
        assert t["verify_rejects"] > 0 and t["n_hit_cache"] > 0
        compare_cache(gc, oc)


def test_overlap_flag_with_a_stream_switch_paper_ids_and_eviction():
    # calls alternating between two streams are still ordered by the library;
    # paper identifiers and evicting caches take the waiting path: same results
    C = 4 * KiB
    calls = _repeating_calls(C, 72)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    streams = [s1 if k % 3 else s2 for k in range(len(calls))]
    for flags, oflags, cap in ((0, 0, 4096), (B.GLEAM_PAPER_IDS, oracle.PAPER_IDS, 4096),
                               (B.GLEAM_EVICT_LRU, oracle.EVICT_LRU, 400)):
        gc = Cache(cap * C, C, flags | B.GLEAM_OVERLAP_CALLS)
        oc = oracle.OracleCache(cap * C, C, oflags)
        with gc:
            _calls_vs_oracle(gc, oc, calls, streams)
            _calls_vs_oracle(gc, oc, calls[::-1], streams)
            if flags == B.GLEAM_EVICT_LRU:
                assert gc.stats()["evictions"] > 0
            compare_cache(gc, oc)
