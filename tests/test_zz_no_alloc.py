"""gleam_dedup_copy_noalloc: the dedup call for callers that cannot allocate
device memory while they run (for instance code inside an intercepted CUDA
call, where a cudaMalloc would re-enter the interception).  It must give
exactly the outputs, results and cache state of gleam_dedup_copy_async.

This file sorts last so that a run stopping at its first failure has run
every other test before it; it also passes when run alone."""
import numpy as np
import pytest
import torch

from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache, DedupOutputs, result_dict

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
