"""Parity at the full sizes of the benchmark configurations, in the launch
configuration bench.py times (one gleam_dedup_copy_batch call per upload).

Where the oracle finishes in seconds (64 MiB fp16 payload, the 498 MB GPT-2
upload, the 1 GiB adversarial payload at every chunk size and key mode) every
output is compared element by element.  For the 16 GB Llama-3-8B upload and
the 100,000-call stream the checks are closed forms of the generators plus
sampled outputs the oracle computes one by one."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import binding as B
from paper_2607_23115_gb300 import workloads as W
from paper_2607_23115_gb300.cache import Cache, DedupOutputs, fingerprint, result_dict

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
KiB, MiB, GiB = 1 << 10, 1 << 20, 1 << 30


def _batch(cache, bufs, C):
    outs = [DedupOutputs.alloc(b.numel(), C, DEV) for b in bufs]
    res = torch.zeros(len(bufs), B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    total = torch.zeros(B.RESULT_WORDS, dtype=torch.int64, device=DEV)
    cache.dedup_batch(bufs, outs, [res[k] for k in range(len(bufs))], total)
    torch.cuda.synchronize()
    t = result_dict(total)
    assert t["status"] == 0, t
    return outs, res.cpu().numpy(), t


def _compare_payload(out, r, host, oc):
    rc, mask_o, miss_o, packed_o = oc.dedup(host)
    assert int(r[1]) == rc and int(r[5]) == len(packed_o)
    assert np.array_equal(out.hit_mask.cpu().numpy().view(np.uint32)[: len(mask_o)], mask_o)
    assert np.array_equal(out.miss_idx.cpu().numpy().view(np.uint32)[:rc], miss_o)
    assert np.array_equal(out.miss_bytes[: len(packed_o)].cpu().numpy(), packed_o)


def test_fp16_64mib_half_prefilled_full_parity():
    C = 4 * KiB
    buf = W.fp16_payload(64 * MiB, seed=0, device=DEV)
    host = buf.cpu().numpy()
    N = buf.numel() // C
    sel = W.select_chunks(N, 0.5)
    pre = W.gather_chunks(buf, C, sel)
    oc = oracle.OracleCache(128 * MiB, C)
    with Cache(128 * MiB, C) as gc:
        outs, r, _ = _batch(gc, [pre], C)
        _compare_payload(outs[0], r[0], pre.cpu().numpy(), oc)
        outs, r, t = _batch(gc, [buf], C)
        _compare_payload(outs[0], r[0], host, oc)
        assert t["n_miss"] == N - len(sel) == 8192
        fps = fingerprint(buf, C).cpu().numpy().view(np.uint64)
        assert np.array_equal(fps, oracle.fingerprint(host, C))


def test_gpt2_upload_two_passes_full_parity():
    C = 4 * KiB
    up = W.weight_upload(W.gpt2_small_shapes(), torch.float32, device=DEV)
    bufs = [up.payload(k) for k in range(len(up.sizes))]
    hosts = [b.cpu().numpy() for b in bufs]
    nchunks = len(up.chunks(C))
    assert nchunks == 121551
    oc = oracle.OracleCache(1 * GiB, C)
    with Cache(1 * GiB, C) as gc:
        for rep in range(2):
            outs, r, t = _batch(gc, bufs, C)
            for k in range(len(bufs)):
                _compare_payload(outs[k], r[k], hosts[k], oc)
            assert t["n_miss"] == (nchunks if rep == 0 else 0)
        st = gc.stats()
        so = oc.stats()
        for f in ("chunks", "hits_cache", "hits_intra", "misses", "slots_used", "bytes_used"):
            assert st[f] == so[f], f


def test_llama3_8b_upload_closed_form_and_samples():
    C = 64 * KiB
    up = W.weight_upload(W.llama3_8b_shapes(), torch.bfloat16, device=DEV)
    nt = len(up.sizes)
    bufs = [up.payload(k) for k in range(nt)]
    chunks = up.chunks(C)
    assert len(chunks) == 245121
    rng = np.random.default_rng(5)
    sample_t = sorted(set(rng.choice(np.arange(1, nt - 1), 3, replace=False).tolist()) | {1})
    base_host = {k: bufs[k].cpu().numpy().copy() for k in sample_t}
    with Cache(24 * GiB, C) as gc:
        _, _, t0 = _batch(gc, bufs, C)
        assert t0["n_miss"] == len(chunks)
        ids = W.select_chunks(len(chunks), 0.10)
        W.flip_one_bit_per_chunk(up.buf, chunks, ids)
        outs, r, t = _batch(gc, bufs, C)
        # closed form: the misses are exactly the bit-flipped chunks
        assert t["n_miss"] == len(ids) and t["n_hit_cache"] == len(chunks) - len(ids)
        first = np.cumsum([0] + [(s + C - 1) // C for s in up.sizes])
        got = set()
        for k in range(nt):
            nm = int(r[k, 1])
            idx = outs[k].miss_idx[:nm].cpu().numpy().view(np.uint32).astype(np.int64)
            assert np.all(np.diff(idx) > 0)
            got.update((first[k] + idx).tolist())
        assert got == set(ids.tolist())
        # sampled tensors: the oracle on (base tensor, perturbed tensor) alone gives the
        # same outputs, since random tensors share no chunk with each other
        for k in sample_t:
            oc = oracle.OracleCache(2 * GiB, C)
            oc.dedup(base_host[k])
            _compare_payload(outs[k], r[k], bufs[k].cpu().numpy(), oc)
        # sampled slots of the cache hold the bytes of the chunk inserted there
        st = gc.stats()
        assert st["slots_used"] == len(chunks) + len(ids)
        flipped = set(ids.tolist())
        for s in rng.choice(len(chunks), 24, replace=False).tolist():
            _, off, ln = chunks[s]
            now = up.buf[off:off + ln].cpu().numpy()
            stored = np.frombuffer(gc.read_slot(int(s)), dtype=np.uint8)
            if s in flipped:  # slot s holds the base bytes: one bit away from the payload
                assert sum(bin(x).count("1") for x in (stored ^ now).tolist()) == 1
            else:
                assert np.array_equal(stored, now)
        order = sorted(flipped)  # the second pass inserted the flipped chunks in order
        for j in rng.choice(len(order), 8, replace=False).tolist():
            _, off, ln = chunks[order[j]]
            assert gc.read_slot(len(chunks) + j) == up.buf[off:off + ln].cpu().numpy().tobytes()


def test_small_call_stream_full_size():
    C = 4 * KiB
    up = W.small_call_upload(100000, device=DEV)
    sizes = up.sizes
    nchunks = sum((s + C - 1) // C for s in sizes)
    with Cache(32 * GiB, C) as gc:
        pre = W.random_bytes(2 * 10**9 // C * C, seed=W.SEED_PREFILL, device=DEV)
        _batch(gc, [pre], C)
        slots0 = gc.stats()["slots_used"]
        rng = np.random.default_rng(9)
        done = 0
        for lo in range(0, len(sizes), 25000):
            ks = list(range(lo, min(len(sizes), lo + 25000)))
            bufs = [up.payload(k) for k in ks]
            outs, r, t = _batch(gc, bufs, C)
            nb = sum((sizes[k] + C - 1) // C for k in ks)
            assert t["n_miss"] == nb and t["n_hit_cache"] == 0  # random bytes: all misses
            for j in rng.choice(len(ks), 8, replace=False).tolist():
                oc = oracle.OracleCache(2 * MiB, C)
                _compare_payload(outs[j], r[j], bufs[j].cpu().numpy(), oc)
            done += nb
        assert done == nchunks
        assert gc.stats()["slots_used"] == slots0 + nchunks


@pytest.mark.parametrize("C", [1 * KiB, 4 * KiB, 16 * KiB, 64 * KiB])
@pytest.mark.parametrize("key16", [False, True])
def test_adversarial_1gib_full_parity(C, key16):
    adv = W.adversarial_payload(1 * GiB, C, device=DEV)
    host = adv.buf.cpu().numpy()
    flags = B.GLEAM_KEY16 if key16 else 0
    oc = oracle.OracleCache(2 * GiB, C, flags)
    with Cache(2 * GiB, C, flags) as gc:
        if key16:
            pick, rows = W.crafted_collisions(adv, C, count=64)
            hrows = host.reshape(-1, C)[pick.numpy()]
            for i in range(64):
                key = oracle.xxh64(hrows[i])
                assert oc.debug_insert(key, rows[i].cpu().numpy()) == 0
                gc.debug_insert(key, rows[i])
        outs, r, t = _batch(gc, [adv.buf], C)
        _compare_payload(outs[0], r[0], host, oc)
        rnd = int((adv.kind == 2).sum())
        npat = len(set(adv.pattern_id[adv.kind == 1].tolist()))
        assert t["n_miss"] == 1 + npat + rnd
        st, so = gc.stats(), oc.stats()
        for f in ("hits_cache", "hits_intra", "misses", "verify_rejects", "slots_used"):
            assert st[f] == so[f], f
        if key16:
            assert st["verify_rejects"] >= 64
