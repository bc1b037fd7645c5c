"""Argument errors, device-pointer checks and the bounded device wait."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache, DedupOutputs
from tests._parity import DEV, compare_cache, dedup_both

pytestmark = [pytest.mark.gpu, pytest.mark.usefixtures("call_path")]


def test_host_pointers_are_rejected():
    C = 1024
    with Cache(1 << 20, C) as gc:
        host = torch.zeros(4 * C, dtype=torch.uint8)
        out = DedupOutputs.alloc(4 * C, C, DEV)
        rc = B.gleam_dedup_copy(gc.handle, host, host.numel(), out.hit_mask, out.miss_idx,
                                out.miss_bytes)
        assert rc == B.GLEAM_ERR_NOT_DEVICE_PTR
        pinned = torch.zeros(4 * C, dtype=torch.uint8).pin_memory()
        rc = B.gleam_dedup_copy(gc.handle, pinned, pinned.numel(), out.hit_mask, out.miss_idx,
                                out.miss_bytes)
        assert rc == B.GLEAM_ERR_NOT_DEVICE_PTR
        d = host.to(DEV)
        rc = B.gleam_dedup_copy(gc.handle, d, d.numel(), out.hit_mask, None, out.miss_bytes)
        assert rc == B.GLEAM_ERR_INVALID_ARG
        assert gc.stats()["calls"] == 0


def test_bounded_wait_times_out_and_cache_stays_usable():
    C = 1024
    gc = Cache(64 << 20, C)
    oc = oracle.OracleCache(64 << 20, C)
    with gc:
        dedup_both(gc, oc, W.random_bytes(3000 * C, seed=1))
        before = gc.stats()
        gc.debug_set(B.GLEAM_DEBUG_WAIT_LIMIT_NS, 50_000_000)   # 50 ms
        gc.debug_set(B.GLEAM_DEBUG_SKIP_ARRIVE, 1)
        d = W.random_bytes(5000 * C, seed=2).to(DEV)
        with pytest.raises(B.GleamError) as e:
            gc.dedup(d)
        assert e.value.rc == B.GLEAM_ERR_TIMEOUT
        assert gc.stats() == before
        gc.debug_set(B.GLEAM_DEBUG_WAIT_LIMIT_NS, 4_000_000_000)
        dedup_both(gc, oc, W.random_bytes(5000 * C, seed=2))
        compare_cache(gc, oc)
