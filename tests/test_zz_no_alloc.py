"""gleam_dedup_copy_noalloc: the dedup call for callers that cannot allocate
device memory while they run (for instance code inside an intercepted CUDA
call, where a cudaMalloc would re-enter the interception).  It must give
exactly the outputs, results and cache state of gleam_dedup_copy_async.

This file sorts last so that a run stopping at its first failure has run
every other test before it; it also passes when run alone."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache, DedupOutputs, result_dict
from tests._parity import compare_cache

pytestmark = [pytest.mark.gpu, pytest.mark.usefixtures("call_path")]
DEV = torch.device("cuda:0")
C = 4096


def _call(fn, cache, buf, out, res):
    n = buf.numel()
    rc = fn(cache.handle, buf, n, out.hit_mask, out.miss_idx, out.miss_bytes, res, None)
    assert rc == B.GLEAM_OK, B.gleam_status_string(rc)


def _same_outputs(oa, ob, ra, rb):
    a, b = result_dict(ra), result_dict(rb)
    assert a == b and a["status"] == 0
    nm, mb = a["n_miss"], a["miss_bytes"]
    assert torch.equal(oa.hit_mask, ob.hit_mask)
    assert torch.equal(oa.miss_idx[:nm], ob.miss_idx[:nm])
    assert torch.equal(oa.miss_bytes[:mb], ob.miss_bytes[:mb])
    return a


def test_noalloc_matches_the_allocating_call_on_two_calls_in_a_row():
    # call 1: fresh chunks with in-call duplicates; call 2: hits on call 1's
    # inserts, new misses and a ragged tail
    base = W.random_bytes(300 * C, seed=61).view(-1, C)
    idx1 = torch.from_numpy(np.random.default_rng(1).integers(0, 200, 500))
    idx2 = torch.from_numpy(np.random.default_rng(2).integers(100, 300, 700))
    p1 = base[idx1].reshape(-1).contiguous().to(DEV)
    p2 = torch.cat([base[idx2].reshape(-1), W.random_bytes(1234, seed=62)]).to(DEV)

    ca, cb = Cache(4096 * C, C), Cache(4096 * C, C)
    outs = [DedupOutputs.alloc(p.numel(), C, DEV) for p in (p1, p2, p1, p2)]
    res = torch.zeros(4, B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    try:
        _call(B.gleam_dedup_copy_async, ca, p1, outs[0], res[0])
        _call(B.gleam_dedup_copy_noalloc, cb, p1, outs[2], res[2])
        torch.cuda.synchronize()
        r1 = _same_outputs(outs[0], outs[2], res[0], res[2])
        assert r1["n_hit_intra"] > 0

        free_before = torch.cuda.mem_get_info()[0]
        _call(B.gleam_dedup_copy_async, ca, p2, outs[1], res[1])
        _call(B.gleam_dedup_copy_noalloc, cb, p2, outs[3], res[3])
        torch.cuda.synchronize()
        r2 = _same_outputs(outs[1], outs[3], res[1], res[3])
        assert r2["n_hit_cache"] > 0 and r2["n_miss"] > 0
        assert torch.cuda.mem_get_info()[0] == free_before  # no device allocation

        sa, sb = ca.stats(), cb.stats()
        # spec_chunks is a speed counter of the write-through, not cache state
        sa.pop("spec_chunks")
        sb.pop("spec_chunks")
        assert sa == sb
        ka, la, na = ca.export()
        kb, lb, nb = cb.export()
        assert na == nb and np.array_equal(ka, kb) and np.array_equal(la, lb)
        for s in range(0, sa["slots_used"], 37):
            assert ca.read_slot(s) == cb.read_slot(s)
    finally:
        ca.close()
        cb.close()


def test_noalloc_rejects_payloads_beyond_its_scratch():
    cb = Cache(1 << 30, 1024)
    try:
        n = (B.GLEAM_NOALLOC_MAX_CHUNKS + 1) * 1024
        buf = torch.zeros(n, dtype=torch.uint8, device=DEV)
        out = DedupOutputs.alloc(n, 1024, DEV)
        rc = B.gleam_dedup_copy_noalloc(cb.handle, buf, n, out.hit_mask, out.miss_idx,
                                        out.miss_bytes, None, None)
        assert rc == B.GLEAM_ERR_INVALID_ARG
        assert cb.stats()["calls"] == 0
    finally:
        cb.close()


def _noalloc_vs_oracle(gc, oc, host, out, res):
    """One allocation-free call against the oracle's call on the same bytes."""
    d = host.to(DEV)
    _call(B.gleam_dedup_copy_noalloc, gc, d, out, res)
    torch.cuda.synchronize()
    rc_o, mask_o, miss_o, packed_o = oc.dedup(host.numpy())
    r = result_dict(res)
    assert r["status"] == 0 and r["n_miss"] == rc_o
    assert np.array_equal(out.hit_mask.cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o)
    assert np.array_equal(out.miss_idx.cpu().numpy().view(np.uint32)[:rc_o], miss_o)
    assert np.array_equal(out.miss_bytes.cpu().numpy()[: len(packed_o)], packed_o)
    return r


def test_noalloc_first_call_on_a_fresh_cache_allocates_nothing():
    # the scratch array and the kernels are set up when the cache is created,
    # so not even the first call on a new cache may take device memory
    host = torch.cat([W.random_bytes(40 * C, seed=63), W.random_bytes(40 * C, seed=63)])
    d = host.to(DEV)
    out = DedupOutputs.alloc(d.numel(), C, DEV)
    res = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    gc = Cache(1024 * C, C)
    oc = oracle.OracleCache(1024 * C, C)
    try:
        torch.cuda.synchronize()
        free_before = torch.cuda.mem_get_info()[0]
        _call(B.gleam_dedup_copy_noalloc, gc, d, out, res)
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free_before
        rc_o, mask_o, miss_o, packed_o = oc.dedup(host.numpy())
        assert result_dict(res)["n_miss"] == rc_o == 40
        assert np.array_equal(out.miss_idx.cpu().numpy().view(np.uint32)[:rc_o], miss_o)
        compare_cache(gc, oc)
    finally:
        gc.close()
        oc.close()


@pytest.mark.parametrize("flags", [B.GLEAM_KEY16, B.GLEAM_PAPER_IDS],
                         ids=["key16", "paper-ids"])
def test_noalloc_key_modes_match_the_allocating_call_and_the_oracle(flags):
    # KEY16: 16-bit keys, so unrelated chunks share keys and the verify must
    # separate them; paper identifiers: MD5 of the first 128 bytes, chunks
    # under 1 KiB never cached (the ragged tail and the 600-byte payload)
    Cs = 2048
    base = W.random_bytes(900 * Cs, seed=64).view(-1, Cs)
    rng = np.random.default_rng(5)
    p1 = torch.cat([base[torch.from_numpy(rng.integers(0, 700, 1500))].reshape(-1),
                    W.random_bytes(700, seed=65)])
    p2 = torch.cat([base[torch.from_numpy(rng.integers(300, 900, 1800))].reshape(-1),
                    W.random_bytes(1500, seed=66)])
    p3 = W.random_bytes(600, seed=67)
    ga, gb = Cache(8192 * Cs, Cs, flags), Cache(8192 * Cs, Cs, flags)
    oc = oracle.OracleCache(8192 * Cs, Cs, oracle.KEY16 if flags == B.GLEAM_KEY16
                            else oracle.PAPER_IDS)
    try:
        for k, host in enumerate((p1, p2, p3)):
            oa, ob = (DedupOutputs.alloc(host.numel(), Cs, DEV) for _ in range(2))
            ra, rb = (torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV) for _ in range(2))
            _call(B.gleam_dedup_copy_async, ga, host.to(DEV), oa, ra)
            r = _noalloc_vs_oracle(gb, oc, host, ob, rb)
            _same_outputs(oa, ob, ra, rb)
            if k == 1:
                assert r["n_hit_cache"] > 0
                if flags == B.GLEAM_KEY16:
                    assert r["verify_rejects"] > 0
        compare_cache(gb, oc)
        sa, sb = ga.stats(), gb.stats()
        sa.pop("spec_chunks")
        sb.pop("spec_chunks")
        assert sa == sb
    finally:
        ga.close()
        gb.close()
        oc.close()


def test_noalloc_at_its_maximum_size():
    # exactly GLEAM_NOALLOC_MAX_CHUNKS chunks: the group table fills to its
    # limit; a quarter of the chunks repeat earlier ones
    Cs = 1024
    n_ch = B.GLEAM_NOALLOC_MAX_CHUNKS
    uniq = W.random_bytes((n_ch * 3 // 4) * Cs, seed=68).view(-1, Cs)
    rep = uniq[torch.from_numpy(np.random.default_rng(6).integers(0, len(uniq), n_ch - len(uniq)))]
    host = torch.cat([uniq, rep]).reshape(-1)
    assert host.numel() == n_ch * Cs
    ga, gb = Cache(2 * n_ch * Cs, Cs), Cache(2 * n_ch * Cs, Cs)
    oc = oracle.OracleCache(2 * n_ch * Cs, Cs)
    try:
        oa, ob = (DedupOutputs.alloc(host.numel(), Cs, DEV) for _ in range(2))
        ra, rb = (torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV) for _ in range(2))
        _call(B.gleam_dedup_copy_async, ga, host.to(DEV), oa, ra)
        r = _noalloc_vs_oracle(gb, oc, host, ob, rb)
        _same_outputs(oa, ob, ra, rb)
        assert r["n_miss"] == len(uniq) and r["n_hit_intra"] == n_ch - len(uniq)
        compare_cache(gb, oc)
    finally:
        ga.close()
        gb.close()
        oc.close()


def test_noalloc_after_a_timed_out_call():
    # a call whose grid barrier runs out (one block leaves without arriving)
    # leaves the cache unchanged; the next call, which reuses the same scratch
    # array, must start from a clean state
    Cs = 1024
    gc = Cache(64 << 20, Cs)
    oc = oracle.OracleCache(64 << 20, Cs)
    try:
        first = W.random_bytes(3000 * Cs, seed=69)
        out = DedupOutputs.alloc(first.numel(), Cs, DEV)
        res = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
        _noalloc_vs_oracle(gc, oc, first, out, res)
        before = gc.stats()
        gc.debug_set(B.GLEAM_DEBUG_WAIT_LIMIT_NS, 50_000_000)  # 50 ms
        gc.debug_set(B.GLEAM_DEBUG_SKIP_ARRIVE, 1)
        second = torch.cat([W.random_bytes(4000 * Cs, seed=70), first[: 1000 * Cs]])
        d = second.to(DEV)
        out2 = DedupOutputs.alloc(d.numel(), Cs, DEV)
        res2 = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
        _call(B.gleam_dedup_copy_noalloc, gc, d, out2, res2)
        torch.cuda.synchronize()
        assert result_dict(res2)["status"] == B.GLEAM_ERR_TIMEOUT
        assert gc.stats() == before
        gc.debug_set(B.GLEAM_DEBUG_WAIT_LIMIT_NS, 4_000_000_000)
        r = _noalloc_vs_oracle(gc, oc, second, out2, res2)
        assert r["n_hit_cache"] == 1000 and r["n_miss"] == 4000
        compare_cache(gc, oc)
    finally:
        gc.close()
        oc.close()
