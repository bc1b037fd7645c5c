"""gleam_block_check (paper Sec. 4.1.1, weight-block identification at cudaFree
time) vs the oracle, on records taken from the dedup calls' chunk slots."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache, DedupOutputs

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
KiB, MiB = 1024, 1 << 20


def _upload_records(gc, oc, up, C):
    """One batch call over the upload; records (offset in the flat buffer, slot)
    for every chunk, from the GPU's chunk slots, checked against the oracle's."""
    nt = len(up.sizes)
    dbuf = up.buf.to(DEV)
    bufs = [dbuf[up.offsets[k]: up.offsets[k] + up.sizes[k]] for k in range(nt)]
    outs = [DedupOutputs.alloc(s, C, DEV) for s in up.sizes]
    slots = [torch.zeros((s + C - 1) // C, dtype=torch.int32, device=DEV) for s in up.sizes]
    gc.dedup_batch(None, items=gc.batch_items(bufs, outs, None, slots))
    torch.cuda.synchronize()
    offs, sl = [], []
    for k in range(nt):
        so = oc.dedup(up.payload(k).numpy(), chunk_slots=True)[4]
        g = slots[k].cpu().numpy().view(np.uint32)
        assert np.array_equal(g, so), k
        offs += [up.offsets[k] + i * C for i in range(len(g))]
        sl += g.tolist()
    return dbuf, np.array(offs, dtype=np.uint64), np.array(sl, dtype=np.uint32)


def _check_both(gc, oc, dblock, offs, sl):
    d_off = torch.from_numpy(offs.view(np.int64)).to(DEV)
    d_sl = torch.from_numpy(sl.view(np.int32)).to(DEV)
    flags = torch.full((max(1, len(offs)),), 7, dtype=torch.uint8, device=DEV)
    cnt = gc.block_check(dblock, d_off, d_sl, flags)
    torch.cuda.synchronize()
    bad_o, flags_o = oc.block_check(dblock.cpu().numpy(), offs, sl)
    assert int(cnt.item()) == bad_o
    assert np.array_equal(flags.cpu().numpy()[: len(offs)], flags_o)
    return bad_o


@pytest.mark.parametrize("C", [4 * KiB, 64 * KiB])
def test_unchanged_block_passes_and_edits_are_found(C):
    up = W.weight_upload(W.scaled_shapes(W.llama3_8b_shapes(), 8)[:40], torch.bfloat16)
    gc, oc = Cache(512 * MiB, C), oracle.OracleCache(512 * MiB, C)
    with gc:
        dblock, offs, sl = _upload_records(gc, oc, up, C)
        # a second upload of the same weights hits everywhere: same slots
        dblock2, offs2, sl2 = _upload_records(gc, oc, up, C)
        assert np.array_equal(sl, sl2)
        assert _check_both(gc, oc, dblock, offs, sl) == 0
        # in-place edits (an activation written into the block): exactly the
        # records covering them mismatch
        rng = np.random.default_rng(3)
        for pos in rng.integers(0, up.total_bytes, 9).tolist():
            dblock[pos] ^= 0x5A
        assert _check_both(gc, oc, dblock, offs, sl) > 0


def test_records_out_of_range_or_naming_unused_slots_mismatch():
    C = 4 * KiB
    gc, oc = Cache(64 * MiB, C), oracle.OracleCache(64 * MiB, C)
    with gc:
        host = W.random_bytes(16 * C + 100, seed=8)
        d = host.to(DEV)
        out = DedupOutputs.alloc(d.numel(), C, DEV)
        slots = torch.zeros(17, dtype=torch.int32, device=DEV)
        gc.dedup_batch(None, items=gc.batch_items([d], [out], None, [slots]))
        oc.dedup(host.numpy())
        sl = slots.cpu().numpy().view(np.uint32).copy()
        offs = np.arange(17, dtype=np.uint64) * C
        assert _check_both(gc, oc, d, offs, sl) == 0
        offs2 = offs.copy()
        offs2[3] = d.numel() - 10           # runs past the end of the block
        sl2 = sl.copy()
        sl2[5] = 10**6                       # no such slot
        sl2[6] = sl[7]                       # another chunk's bytes
        assert _check_both(gc, oc, d, offs2, sl2) == 3
        # an empty record list passes
        cnt = gc.block_check(d, torch.zeros(0, dtype=torch.int64, device=DEV),
                             torch.zeros(0, dtype=torch.int32, device=DEV))
        torch.cuda.synchronize()
        assert int(cnt.item()) == 0
