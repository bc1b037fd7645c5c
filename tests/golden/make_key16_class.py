"""Writes key16_class.txt: 48 distinct 32-byte chunks whose XXH64
fingerprints (seed 0) share their low 16 bits, so that in KEY16 mode (index
key = the low 16 bits of the fingerprint) they all have one index key, and
with one length one (16-bit key, length) class; and 4 chunks of 20 bytes with
the same low 16 bits (a second class under the same index key, as a payload's
short last chunk).

A call that sends many of them makes many misses of one class: in the cache
index all of them start their linear probe at one home position.  Such chunks
occur by chance once in 65,536, so the test that uses them needs them found by
search; the fingerprints come from the oracle.

Run from the repository root: python tests/golden/make_key16_class.py
"""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)
import oracle  # noqa: E402

C = 32
COUNT = 48
TAIL = 20
TAIL_COUNT = 4
BATCH = 1 << 22   # candidate chunks per search step (128 MiB)
SEED = 20261202


def search(rng, size, count, target):
    """count distinct size-byte chunks whose XXH64 has the low 16 bits target
    (None: those of the first candidate); returns (target, [(chunk, xxh64)])."""
    found, seen = [], set()
    while len(found) < count:
        data = rng.integers(0, 256, size=BATCH * size, dtype=np.uint8)
        fp = oracle.fingerprint(data, size)
        if target is None:
            target = int(fp[0]) & 0xFFFF
        for i in np.nonzero((fp & np.uint64(0xFFFF)) == np.uint64(target))[0]:
            chunk = data[i * size:(i + 1) * size].tobytes()
            if chunk not in seen and len(found) < count:
                seen.add(chunk)
                found.append((chunk, int(fp[i])))
    return target, found


def main():
    rng = np.random.default_rng(SEED)
    target, found = search(rng, C, COUNT, None)
    _, tails = search(rng, TAIL, TAIL_COUNT, target)
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "key16_class.txt")
    with open(out, "w") as f:
        f.write("# %d distinct %d-byte chunks, then %d of %d bytes, whose XXH64 (seed 0) has\n"
                "# the low 16 bits %04x; chunk, then its XXH64; written by make_key16_class.py\n"
                % (COUNT, C, TAIL_COUNT, TAIL, target))
        for chunk, h in found + tails:
            f.write("%s %016x\n" % (chunk.hex(), h))
    print(out)


if __name__ == "__main__":
    main()
