"""Host-resident payloads: the kernels read page-locked host memory in place and
only the misses are written to the device.  Same outputs as the oracle."""
import ctypes

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


def _pinned(host: torch.Tensor, offset: int = 0) -> torch.Tensor:
    big = torch.empty(host.numel() + offset, dtype=torch.uint8).pin_memory()
    v = big[offset:]
    v.copy_(host)
    return v


def _host_call(gc, oc, host, offset=0):
    C = gc.chunk_bytes
    hb = _pinned(host, offset)
    out = DedupOutputs.alloc(host.numel(), C, DEV)
    res = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    gc.dedup_host(hb, out, res)
    torch.cuda.synchronize()
    r = result_dict(res)
    rc, mask_o, miss_o, packed_o = oc.dedup(host.numpy())
    assert r["status"] == 0 and r["n_miss"] == rc and r["miss_bytes"] == len(packed_o)
    assert np.array_equal(out.hit_mask.cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o)
    assert np.array_equal(out.miss_idx.cpu().numpy().view(np.uint32)[:rc], miss_o)
    assert np.array_equal(out.miss_bytes.cpu().numpy()[: len(packed_o)], packed_o)
    return rc


@pytest.mark.parametrize("key16", [False, True])
def test_host_payload_calls_match_oracle(key16):
    C = 4 * KiB
    flags = B.GLEAM_KEY16 if key16 else 0
    gc, oc = Cache(64 * MiB, C, flags), oracle.OracleCache(64 * MiB, C, flags)
    host = W.fp16_payload(4 * MiB, seed=0)
    with gc:
        _host_call(gc, oc, host[: 2 * MiB])
        _host_call(gc, oc, torch.cat([host, host[:1000]]))
        _host_call(gc, oc, host[: 3 * MiB + 77], offset=5)   # unaligned host view
        _host_call(gc, oc, W.random_bytes(100, seed=3))      # one short chunk
        compare_cache(gc, oc)


def test_host_batch_matches_sequential_oracle():
    C = 64 * KiB
    up = W.weight_upload(W.scaled_shapes(W.llama3_8b_shapes(), 8)[:40], torch.bfloat16)
    gc, oc = Cache(256 * MiB, C), oracle.OracleCache(256 * MiB, C)
    pinned = up.buf.pin_memory()
    with gc:
        for rep in range(2):
            if rep == 1:
                chunks = up.chunks(C)
                ids = W.select_chunks(len(chunks), 0.10)
                W.flip_one_bit_per_chunk(up.buf, chunks, ids)
                pinned.copy_(up.buf)
            nt = len(up.sizes)
            hbufs = [pinned[up.offsets[k]: up.offsets[k] + up.sizes[k]] for k in range(nt)]
            outs = [DedupOutputs.alloc(s, C, DEV) for s in up.sizes]
            res = torch.zeros(nt, B.RESULT_WORDS, dtype=torch.int64, device=DEV)
            gc.dedup_host_batch(hbufs, outs, [res[k] for k in range(nt)])
            torch.cuda.synchronize()
            rr = res.cpu().numpy()
            for k in range(nt):
                rc, mask_o, miss_o, packed_o = oc.dedup(up.payload(k).numpy())
                assert rr[k, 0] == 0 and rr[k, 1] == rc
                o = outs[k]
                assert np.array_equal(o.hit_mask.cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o)
                assert np.array_equal(o.miss_idx.cpu().numpy().view(np.uint32)[:rc], miss_o)
                assert np.array_equal(o.miss_bytes.cpu().numpy()[: len(packed_o)], packed_o)
        compare_cache(gc, oc)


def test_registered_numpy_memory_is_accepted():
    C = 4 * KiB
    arr = np.random.default_rng(4).integers(0, 256, 3 * MiB, dtype=np.uint8)
    rt = torch.cuda.cudart()
    assert int(rt.cudaHostRegister(arr.ctypes.data, arr.nbytes, 0)) == 0
    try:
        gc, oc = Cache(16 * MiB, C), oracle.OracleCache(16 * MiB, C)
        with gc:
            out = DedupOutputs.alloc(arr.nbytes, C, DEV)
            rc = B.gleam_dedup_copy_host_async(gc.handle, arr.ctypes.data, arr.nbytes,
                                               out.hit_mask, out.miss_idx, out.miss_bytes)
            assert rc == B.GLEAM_OK
            torch.cuda.synchronize()
            ro, mask_o, miss_o, packed_o = oc.dedup(arr)
            assert np.array_equal(out.miss_bytes.cpu().numpy()[: len(packed_o)], packed_o)
            compare_cache(gc, oc)
    finally:
        rt.cudaHostUnregister(arr.ctypes.data)


def test_pageable_and_device_memory_are_rejected_by_the_host_entry():
    C = 4 * KiB
    with Cache(16 * MiB, C) as gc:
        out = DedupOutputs.alloc(8 * C, C, DEV)
        pageable = np.zeros(8 * C, dtype=np.uint8)
        rc = B.gleam_dedup_copy_host_async(gc.handle, pageable.ctypes.data, pageable.nbytes,
                                           out.hit_mask, out.miss_idx, out.miss_bytes)
        assert rc == B.GLEAM_ERR_NOT_DEVICE_PTR
        d = torch.zeros(8 * C, dtype=torch.uint8, device=DEV)
        rc = B.gleam_dedup_copy_host_async(gc.handle, d, d.numel(), out.hit_mask, out.miss_idx,
                                           out.miss_bytes)
        assert rc == B.GLEAM_ERR_NOT_DEVICE_PTR
        assert gc.stats()["calls"] == 0


@pytest.mark.parametrize("offset", [0, 3])
def test_indices_packed_bytes_and_slots_written_to_pinned_host_memory(offset):
    """The host entries may put the miss indices, packed miss bytes and chunk
    slots in page-locked host memory; the kernels write them over the link."""
    C = 4 * KiB
    gc, oc = Cache(64 * MiB, C), oracle.OracleCache(64 * MiB, C)
    host = W.fp16_payload(4 * MiB, seed=1)
    with gc:
        for payload in (host[: 2 * MiB], torch.cat([host, host[:1000]]), host[: 3 * MiB + 77]):
            n = payload.numel()
            N = (n + C - 1) // C
            hb = _pinned(payload, offset)
            mask = torch.zeros((N + 31) // 32, dtype=torch.int32, device=DEV)
            idx = torch.full((N,), -1, dtype=torch.int32).pin_memory()
            packed = _pinned(torch.zeros(n, dtype=torch.uint8), offset)
            slots = torch.full((N,), -1, dtype=torch.int32).pin_memory()
            res = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
            items = B.payload_array([(hb, n, mask, idx, packed, res, slots)])
            rc = B.gleam_dedup_copy_host_batch(gc.handle, items, None, None)
            assert rc == 0, rc
            torch.cuda.synchronize()
            r = result_dict(res)
            rc_o, mask_o, miss_o, packed_o, slots_o = oc.dedup(payload.numpy(), chunk_slots=True)
            assert r["status"] == 0 and r["n_miss"] == rc_o
            assert np.array_equal(mask.cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o)
            assert np.array_equal(idx.numpy().view(np.uint32)[:rc_o], miss_o)
            assert np.array_equal(packed.numpy()[: len(packed_o)], packed_o)
            assert np.array_equal(slots.numpy().view(np.uint32), slots_o)
        compare_cache(gc, oc)
