"""Writes claim_tag_collision.txt: two 32-byte chunks with different XXH64
fingerprints whose claims in the per-call group table of a one-payload call
collide in both the 32-bit tag and the home position of a 1,024-entry table.

The library's staged hash kernel claims a miss's group entry with a 64-bit
compare-and-swap that stores a 32-bit tag of the chunk's (fingerprint, length)
pair; a second chunk that meets an entry with its own tag sends the call down
the general path, where the groups are claimed again by the whole fingerprint.
Distinct pairs share a tag only by chance, so the test that uses these chunks
needs them found by search.  Position and tag are the low bits and the high
32 bits of the MurmurHash3 64-bit finaliser (Appleby) of fingerprint XOR
(length << 40), restated below; the fingerprints come from the oracle.

Run from the repository root: python tests/golden/make_claim_tag_collision.py
"""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)
import oracle  # noqa: E402

C = 32
TABLE = 1024           # a call of 300 chunks: next power of two of 2 x 300
CANDIDATES = 1 << 23   # 8 Mi chunks: about seven colliding pairs expected
SEED = 20260731


def mix64(k: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        k = k ^ (k >> np.uint64(33))
        k = k * np.uint64(0xFF51AFD7ED558CCD)
        k = k ^ (k >> np.uint64(33))
        k = k * np.uint64(0xC4CEB9FE1A85EC53)
        k = k ^ (k >> np.uint64(33))
    return k


def main():
    rng = np.random.default_rng(SEED)
    data = rng.integers(0, 256, size=CANDIDATES * C, dtype=np.uint8)
    fp = oracle.fingerprint(data, C).astype(np.uint64)
    mixed = mix64(fp ^ np.uint64(C << 40))
    tag = mixed >> np.uint64(32)
    pos = mixed & np.uint64(TABLE - 1)
    key = (tag << np.uint64(10)) | pos
    order = np.argsort(key, kind="stable")
    ks = key[order]
    same = np.nonzero(ks[1:] == ks[:-1])[0]
    for i in same:
        a, b = int(order[i]), int(order[i + 1])
        if fp[a] != fp[b]:
            break
    else:
        raise SystemExit("no colliding pair among the candidates")
    ca = data[a * C:(a + 1) * C].tobytes()
    cb = data[b * C:(b + 1) * C].tobytes()
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "claim_tag_collision.txt")
    with open(out, "w") as f:
        f.write("# two 32-byte chunks, distinct XXH64 (seed 0), same claim tag and home\n"
                "# position in a 1,024-entry group table; written by "
                "make_claim_tag_collision.py\n")
        f.write("chunk_a %s\nchunk_b %s\n" % (ca.hex(), cb.hex()))
        f.write("xxh64_a %016x\nxxh64_b %016x\n" % (int(fp[a]), int(fp[b])))
        f.write("tag %08x position %d\n" % (int(tag[a]), int(pos[a])))
    print(out)


if __name__ == "__main__":
    main()
