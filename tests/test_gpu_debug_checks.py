"""GLEAM_DEBUG_CHECKS: the after-call index check passes on every healthy
cache state (plain, LRU with evictions, paper identifiers) and reports a
cache whose index has been damaged on purpose."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache
from tests._parity import DEV, compare_cache, dedup_both

pytestmark = [pytest.mark.gpu, pytest.mark.usefixtures("call_path")]
KiB, MiB = 1024, 1 << 20


@pytest.mark.parametrize("extra,oflags", [(0, 0), (B.GLEAM_EVICT_LRU, oracle.EVICT_LRU),
                                          (B.GLEAM_PAPER_IDS, oracle.PAPER_IDS)])
def test_checks_pass_on_healthy_caches(extra, oflags):
    C = 4 * KiB
    cap = 96 * C
    gc = Cache(cap, C, B.GLEAM_DEBUG_CHECKS | extra)
    oc = oracle.OracleCache(cap, C, oflags)
    rng = np.random.default_rng(4)
    pool = [W.random_bytes(C, seed=100 + k) for k in range(160)]
    with gc:
        for step in range(25):
            parts = [pool[int(i)] for i in rng.integers(0, 160, int(rng.integers(1, 40)))]
            if rng.random() < 0.3:
                parts.append(W.random_bytes(int(rng.integers(1, C)), seed=step))
            rc = dedup_both(gc, oc, torch.cat(parts))
            assert rc >= 0 or (rc == B.GLEAM_ERR_CAPACITY and not extra & B.GLEAM_EVICT_LRU)
        compare_cache(gc, oc)


def test_a_damaged_index_is_reported():
    C = 4 * KiB
    gc = Cache(1 * MiB, C, B.GLEAM_DEBUG_CHECKS)
    with gc:
        d = W.random_bytes(32 * C, seed=1).to(DEV)
        n_miss, _ = gc.dedup(d)
        assert n_miss == 32
        gc.debug_set(B.GLEAM_DEBUG_DROP_ENTRY, 5)   # slot 5 loses its index entry
        with pytest.raises(B.GleamError) as e:
            gc.dedup(W.random_bytes(C, seed=2).to(DEV))
        assert e.value.rc == B.GLEAM_ERR_INTERNAL
