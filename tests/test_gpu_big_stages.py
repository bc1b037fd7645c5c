"""Calls of large chunks that fit one wave of the hash kernel's 2 KiB-stage
variant (C = 64 KiB, a few hundred KiB to a few MiB per call, calls not
overlapping): the prefix hint is the fold after the first 512 bytes, taken in
the middle of stage 0, and the speculative verify compares all of stage 0.
Payloads with ragged tails around the stage and prefix sizes, uploaded, sent
again (hinted hits), then sent with one bit flipped at positions on both sides
of those boundaries (misses found at different stages), each call against the
oracle."""
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import workloads as W
from tests._parity import compare_cache, dedup_both

pytestmark = [pytest.mark.gpu, pytest.mark.usefixtures("call_path")]
KiB = 1024
C = 64 * KiB
FLIPS = (0, 511, 512, 513, 1000, 2047, 2048, 2049, 4095, 4096, 40000, C - 1)


@pytest.mark.parametrize("tail", [0, 600, 1000, 2047, 2048, 2049, 40000])
def test_upload_resend_and_flips_around_stage_boundaries(tail):
    from paper_2607_23115_gb300.cache import Cache
    nfull = len(FLIPS)
    base = W.random_bytes(nfull * C + tail, seed=4000 + tail)
    gc = Cache(64 * C, C)
    oc = oracle.OracleCache(64 * C, C)
    with gc:
        dedup_both(gc, oc, base)
        dedup_both(gc, oc, base)  # hinted hits, stage 0 compared whole
        flipped = base.clone()
        for k, pos in enumerate(FLIPS):  # chunk k differs at byte pos
            flipped[k * C + pos] ^= 1 << (k % 8)
        if tail:
            flipped[nfull * C + tail // 2] ^= 0x40  # and the tail chunk, mid-way
        rc = dedup_both(gc, oc, flipped)
        assert rc == nfull + (1 if tail else 0)
        dedup_both(gc, oc, base)  # the originals are still cached
        compare_cache(gc, oc)
