"""gleam_fingerprint vs the oracle: every length path, chunk size, alignment."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import fingerprint

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _on_device(host, offset=0):
    big = torch.empty(host.numel() + offset + 1, dtype=torch.uint8, device=DEV)
    v = big[offset: offset + host.numel()]
    v.copy_(host)
    return v


def test_whole_buffer_every_length_0_to_300():
    host = W.random_bytes(300, seed=21)
    for offset in (0, 3):
        for n in range(0, 301):
            d = _on_device(host[:n], offset)
            got = fingerprint(d, 0).cpu().numpy().view(np.uint64)[0]
            assert got == oracle.xxh64(host[:n].numpy()), (n, offset)


@pytest.mark.parametrize("C", [32, 96, 1000, 1024, 4096, 65536, 1 << 20])
@pytest.mark.parametrize("offset", [0, 8, 5])
def test_chunked_with_ragged_tail(C, offset):
    host = W.random_bytes(3 * (1 << 20) + 777, seed=22)
    d = _on_device(host, offset)
    got = fingerprint(d, C).cpu().numpy().view(np.uint64)
    assert np.array_equal(got, oracle.fingerprint(host.numpy(), C))


def test_many_chunks_spanning_many_blocks():
    host = W.fp16_payload(32 << 20, seed=0)
    got = fingerprint(host.to(DEV), 4096).cpu().numpy().view(np.uint64)
    assert np.array_equal(got, oracle.fingerprint(host.numpy(), 4096))


def test_empty_payload_chunked_writes_nothing():
    out = torch.full((4,), 7, dtype=torch.int64, device=DEV)
    d = torch.empty(16, dtype=torch.uint8, device=DEV)[:0]
    r = fingerprint(d, 64, out=out)
    assert r.numel() == 0 and (out.cpu() == 7).all()
