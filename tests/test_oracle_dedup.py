"""Pins the oracle's sequential dedup (paper Sec. 4.1.2) against brute force,
invariants, mode equivalence and the closed forms of the synthetic workloads."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_23115_gb300 import workloads as W
from tests._refs import BruteCache, xxh64_lib


def _mask_bits(mask, N):
    return [(int(mask[i // 32]) >> (i % 32)) & 1 for i in range(N)]


def _payload_from_alphabet(rng, alphabet, nchunks, C, tail):
    parts = [alphabet[rng.integers(len(alphabet))] for _ in range(nchunks)]
    data = b"".join(parts)
    if tail:
        data += rng.integers(0, 256, tail, dtype=np.uint8).tobytes()
    return data


def _check_against_brute(oc: oracle.OracleCache, bc: BruteCache, payload: bytes, C: int):
    out = oc.dedup(payload, chunk_slots=True)
    rc = out[0]
    brc, b = bc.dedup(payload, C)
    assert rc == brc
    if rc < 0:
        return rc
    _, mask, miss, packed, slots = out
    N = (len(payload) + C - 1) // C
    assert _mask_bits(mask, N) == _mask_bits(b["mask"], N)
    assert miss.tolist() == b["miss"]
    assert packed.tobytes() == b["packed"]
    assert slots.tolist() == b["slots"]
    return rc, b


@pytest.mark.parametrize("key16", [False, True])
@pytest.mark.parametrize("seed", range(6))
def test_random_sequences_match_brute_force(seed, key16):
    rng = np.random.default_rng(100 + seed)
    C = int(rng.choice([32, 64, 96, 128]))
    nslots = int(rng.integers(40, 200))
    flags = oracle.KEY16 if key16 else 0
    keyf = (lambda b: xxh64_lib(b) & 0xFFFF) if key16 else xxh64_lib
    oc = oracle.OracleCache(nslots * C, C, flags)
    bc = BruteCache(nslots, key_fn=keyf)
    alphabet = [rng.integers(0, 256, C, dtype=np.uint8).tobytes() for _ in range(12)]
    alphabet.append(bytes(C))
    total_rejects = 0
    for call in range(8):
        payload = _payload_from_alphabet(rng, alphabet, int(rng.integers(0, 40)), C,
                                         int(rng.integers(0, C)) if rng.random() < 0.6 else 0)
        before = oc.stats()
        out = _check_against_brute(oc, bc, payload, C)
        if out == oracle.ERR_CAPACITY:
            assert oc.stats() == before  # unchanged on CAPACITY
            continue
        rc, b = out
        after = oc.stats()
        N = (len(payload) + C - 1) // C
        if N == 0:
            assert after == before
            continue
        assert after["hits_cache"] - before["hits_cache"] == b["hits_cache"]
        assert after["hits_intra"] - before["hits_intra"] == b["hits_intra"]
        assert after["verify_rejects"] - before["verify_rejects"] == b["rejects"]
        total_rejects += b["rejects"]
        # invariants
        assert after["chunks"] - before["chunks"] == N
        assert (after["hits_cache"] + after["hits_intra"] + after["misses"]
                - before["hits_cache"] - before["hits_intra"] - before["misses"]) == N
        assert after["inserts"] - before["inserts"] == rc
        assert after["slots_used"] - before["slots_used"] == rc
    # final cache contents equal the brute-force store, slot by slot
    keys, lens = oc.entries()
    assert len(keys) == len(bc.items)
    for s, (k, data) in enumerate(bc.items):
        assert oc.slot_bytes(s) == data
        assert int(lens[s]) == len(data)
        assert int(keys[s]) == k


def test_key16_and_64bit_modes_give_identical_outputs():
    rng = np.random.default_rng(7)
    C = 64
    a = oracle.OracleCache(4096 * C, C, 0)
    b = oracle.OracleCache(4096 * C, C, oracle.KEY16)
    alphabet = [rng.integers(0, 256, C, dtype=np.uint8).tobytes() for _ in range(300)]
    for _ in range(5):
        p = _payload_from_alphabet(rng, alphabet, 400, C, 17)
        ra, ma, ia, pa = a.dedup(p)
        rb, mb, ib, pb = b.dedup(p)
        assert ra == rb and (ma == mb).all() and (ia == ib).all() and (pa == pb).all()
    # with 300 distinct chunks in 65536 buckets a few 16-bit keys collide
    assert b.stats()["verify_rejects"] >= a.stats()["verify_rejects"] == 0


def test_crafted_collisions_are_rejected():
    """Entries whose 16-bit key matches a payload chunk but whose bytes differ by
    one bit: every such chunk must be a miss counted as a verify reject."""
    rng = np.random.default_rng(8)
    C = 128
    chunks = [rng.integers(0, 256, C, dtype=np.uint8).tobytes() for _ in range(64)]
    oc = oracle.OracleCache(1024 * C, C, oracle.KEY16)
    for c in chunks:
        flipped = bytearray(c)
        flipped[int(rng.integers(C))] ^= 1 << int(rng.integers(8))
        assert oc.debug_insert(xxh64_lib(c), bytes(flipped)) == 0
    rc, mask, miss, packed = oc.dedup(b"".join(chunks))
    assert rc == 64 and int(mask[0]) == 0 and int(mask[1]) == 0
    st = oc.stats()
    assert st["verify_rejects"] >= 64
    # the planted entries are still the only ones for those keys: a second
    # identical call hits every chunk (on the entries the first call inserted)
    rc2, mask2, _, _ = oc.dedup(b"".join(chunks))
    assert rc2 == 0 and int(mask2[0]) == 0xFFFFFFFF and int(mask2[1]) == 0xFFFFFFFF


def test_capacity_leaves_cache_unchanged():
    C = 64
    oc = oracle.OracleCache(10 * C, C)
    rng = np.random.default_rng(9)
    p1 = rng.integers(0, 256, 6 * C, dtype=np.uint8).tobytes()
    assert oc.dedup(p1)[0] == 6
    s = oc.stats()
    p2 = rng.integers(0, 256, 5 * C, dtype=np.uint8).tobytes()
    assert oc.dedup(p2)[0] == oracle.ERR_CAPACITY
    assert oc.stats() == s
    assert oc.dedup(p2[: 4 * C])[0] == 4
    assert oc.stats()["slots_used"] == 10


def test_zero_length_and_bad_arguments():
    oc = oracle.OracleCache(1 << 20, 1024)
    assert oc.dedup(b"")[0] == 0
    assert oc.stats()["calls"] == 0
    for bad in ((1 << 20, 0), (1 << 20, 33), (1 << 20, 16), (100, 1024), (1 << 20, 32 << 20)):
        with pytest.raises(ValueError):
            oracle.OracleCache(*bad)


def test_tail_length_is_part_of_equality():
    C = 64
    oc = oracle.OracleCache(100 * C, C)
    z = bytes(C)
    rc, mask, miss, packed = oc.dedup(z + z[:10])
    assert rc == 2 and miss.tolist() == [0, 1] and len(packed) == C + 10
    rc, mask, miss, packed = oc.dedup(z[:10] + b"")   # a 10-byte payload = one tail chunk
    assert rc == 0 and int(mask[0]) == 1
    rc, mask, miss, packed = oc.dedup(z[:11])
    assert rc == 1


# ---- closed forms of the workload generators (small versions) -------------

def test_prefilled_half_misses_exactly_the_complement():
    C = 1024
    buf = W.fp16_payload(256 * C, seed=0).numpy()
    N = 256
    sel = W.select_chunks(N, 0.5)
    oc = oracle.OracleCache(512 * C, C)
    pre = W.gather_chunks(torch.from_numpy(buf), C, sel).numpy()
    assert oc.dedup(pre)[0] == 128
    rc, mask, miss, packed = oc.dedup(buf)
    expect = sorted(set(range(N)) - set(sel.tolist()))
    assert rc == 128 and miss.tolist() == expect
    st = oc.stats()
    assert st["hits_cache"] == 128 and st["hits_intra"] == 0


def test_weight_upload_second_pass_all_hits():
    C = 1024
    up = W.weight_upload(W.scaled_shapes(W.gpt2_small_shapes(), 16), torch.float32)
    oc = oracle.OracleCache(64 << 20, C)
    total_chunks = len(up.chunks(C))
    misses = sum(oc.dedup(up.payload(k).numpy())[0] for k in range(len(up.sizes)))
    assert misses == total_chunks
    s1 = oc.stats()
    for k in range(len(up.sizes)):
        rc, mask, miss, packed = oc.dedup(up.payload(k).numpy())
        assert rc == 0
    s2 = oc.stats()
    assert s2["slots_used"] == s1["slots_used"] and s2["hits_cache"] == total_chunks


def test_bit_flipped_chunks_are_exactly_the_misses():
    C = 1024
    up = W.weight_upload(W.scaled_shapes(W.llama3_8b_shapes(), 64)[:40], torch.bfloat16)
    oc = oracle.OracleCache(64 << 20, C)
    for k in range(len(up.sizes)):
        oc.dedup(up.payload(k).numpy())
    chunks = up.chunks(C)
    ids = W.select_chunks(len(chunks), 0.10, seed=W.SEED_SELECT)
    W.flip_one_bit_per_chunk(up.buf, chunks, ids)
    flipped = set(ids.tolist())
    got = []
    g = 0
    for k in range(len(up.sizes)):
        rc, mask, miss, packed = oc.dedup(up.payload(k).numpy())
        got += [g + int(i) for i in miss]
        g += (up.sizes[k] + C - 1) // C
    assert sorted(got) == sorted(flipped)


def test_adversarial_miss_count_closed_form():
    C = 1024
    adv = W.adversarial_payload(512 * C, C)
    buf = adv.buf.numpy()
    # random-class chunks must be pairwise distinct for the closed form
    rows = buf.reshape(-1, C)
    rnd = (adv.kind == 2).nonzero().flatten().tolist()
    assert len({rows[i].tobytes() for i in rnd}) == len(rnd)
    oc = oracle.OracleCache(4096 * C, C)
    rc, mask, miss, packed = oc.dedup(buf)
    n_pat = len(set(adv.pattern_id[adv.kind == 1].tolist()))
    assert rc == 1 + n_pat + len(rnd)
    oc16 = oracle.OracleCache(4096 * C, C, oracle.KEY16)
    pick, rows_f = W.crafted_collisions(adv, C, count=64)
    for i, r in zip(pick.tolist(), rows_f.numpy()):
        assert oc16.debug_insert(xxh64_lib(rows[i].tobytes()), r) == 0
    rc16, mask16, miss16, packed16 = oc16.dedup(buf)
    assert rc16 == rc and (miss16 == miss).all() and (packed16 == packed).all()
    assert oc16.stats()["verify_rejects"] >= 64


def test_block_check_matches_brute_force():
    """Weight-block identification (paper Sec. 4.1.1): a block still holds
    weights iff every chunk recorded from its host-to-device writes matches."""
    rng = np.random.default_rng(21)
    C = 64
    oc = oracle.OracleCache(1000 * C, C)
    block = bytearray(rng.integers(0, 256, 40 * C + 17, dtype=np.uint8).tobytes())
    # two "HtoD writes" into the block at offsets 0 and 20*C (+ ragged tail)
    offs, slots = [], []
    for base, length in ((0, 20 * C), (20 * C, 20 * C + 17)):
        _, _, _, _, sl = oc.dedup(bytes(block[base:base + length]), chunk_slots=True)
        offs += [base + i * C for i in range(len(sl))]
        slots += sl.tolist()
    bad, flags = oc.block_check(bytes(block), offs, slots)
    assert bad == 0 and not flags.any()
    # change one byte in record 7 and one in the tail record: exactly those differ
    block[7 * C + 5] ^= 0x10
    block[40 * C + 3] ^= 0x01
    bad, flags = oc.block_check(bytes(block), offs, slots)
    expect = [0] * len(offs)
    expect[7] = 1
    expect[len(offs) - 1] = 1
    assert bad == 2 and flags.tolist() == expect
    # brute force over the same records: compare stored bytes with the block
    for r, (o, s_) in enumerate(zip(offs, slots)):
        stored = oc.slot_bytes(s_)
        assert (bytes(block[o:o + len(stored)]) != stored) == bool(flags[r])
    # a record past the block's end, or naming no stored slot, mismatches
    bad, flags = oc.block_check(bytes(block[: 10 * C]), [9 * C + 1, 0], [0, 10**6])
    assert bad == 2


def test_length_is_part_of_a_candidate():
    """An entry with the chunk's key but another length is not a candidate: the
    chunk is a miss without a verify reject (R6: rejects need key + length)."""
    rng = np.random.default_rng(31)
    C = 256
    chunk = rng.integers(0, 256, C, dtype=np.uint8).tobytes()
    for key16 in (False, True):
        oc = oracle.OracleCache(64 * C, C, oracle.KEY16 if key16 else 0)
        assert oc.debug_insert(xxh64_lib(chunk), chunk[:-1]) == 0   # same key, shorter
        rc, mask, miss, packed = oc.dedup(chunk)
        assert rc == 1 and oc.stats()["verify_rejects"] == 0
        assert oc.debug_insert(xxh64_lib(chunk), bytes(C)) == 0     # same key and length
        rc, mask, miss, packed = oc.dedup(chunk + chunk[:100])
        # the first chunk now hits the entry the previous call inserted
        assert rc == 1 and int(mask[0]) == 1 and oc.stats()["verify_rejects"] == 0
        other = bytearray(chunk)
        other[5] ^= 1
        assert oc.debug_insert(xxh64_lib(bytes(other)), bytes(other)[:-1]) == 0
        oc2 = oracle.OracleCache(64 * C, C, oracle.KEY16 if key16 else 0)
        assert oc2.debug_insert(xxh64_lib(bytes(other)), bytes(C)) == 0  # key match, bytes differ
        rc, _, _, _ = oc2.dedup(bytes(other))
        assert rc == 1 and oc2.stats()["verify_rejects"] == 1
