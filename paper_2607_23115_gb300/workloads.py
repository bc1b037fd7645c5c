"""Seeded synthetic payloads with the shapes of the dedup workloads.

Input generation only: nothing here hashes, compares or decides anything, so
the CUDA path and the CPU oracle can both be fed from it without sharing any
of the method's arithmetic.  Every generator is deterministic in its seed and
runs on any torch device; bytes generated on a GPU are copied to the host
for the oracle, so both sides always see identical bytes.

Seeds follow one convention: 0 payload values, 1 chunk selection, 2
perturbation, 3 crafted collision entries, 4 unrelated prefill data.

Workloads (model weights stand in for the paper's llama/llava/sd uploads,
Tab. 2 and Tab. 8; no checkpoint is needed, values are ~N(0, 0.02)):
  * fp16 payload: one 64 MiB buffer of fp16 values, half of its 4 KiB chunks
    pre-cached.
  * GPT-2-small weight upload: 148 fp32 tensors, one call per tensor.
  * Llama-3-8B weight upload: 291 bf16 tensors, 10% of 64 KiB chunks carry one
    flipped bit relative to the cached base (a fine-tuned variant).
  * small-call stream: log-uniform 4 KiB..1 MiB payloads of random bytes.
  * adversarial: 25% all-zero chunks, 25% copies of 16 patterns, 50% random.
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import List, Sequence, Tuple

import torch

SEED_VALUES = 0
SEED_SELECT = 1
SEED_PERTURB = 2
SEED_CRAFTED = 3
SEED_PREFILL = 4

ALIGN = 256  # tensor start alignment inside a flat upload buffer (allocator-like)

KiB = 1024
MiB = 1024 * KiB
GiB = 1024 * MiB


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=torch.device(device))
    g.manual_seed(seed)
    return g


# ---------------------------------------------------------------------------
# tensor inventories
# ---------------------------------------------------------------------------

def gpt2_small_shapes() -> List[Tuple[str, Tuple[int, ...]]]:
    """GPT-2 small: 12 layers, d=768, ffn=3072, vocab 50257, ctx 1024 (148 tensors)."""
    d, f, v, ctx = 768, 3072, 50257, 1024
    out = [("wte", (v, d)), ("wpe", (ctx, d))]
    for l in range(12):
        p = "h.%d." % l
        out += [
            (p + "ln_1.weight", (d,)), (p + "ln_1.bias", (d,)),
            (p + "attn.c_attn.weight", (d, 3 * d)), (p + "attn.c_attn.bias", (3 * d,)),
            (p + "attn.c_proj.weight", (d, d)), (p + "attn.c_proj.bias", (d,)),
            (p + "ln_2.weight", (d,)), (p + "ln_2.bias", (d,)),
            (p + "mlp.c_fc.weight", (d, f)), (p + "mlp.c_fc.bias", (f,)),
            (p + "mlp.c_proj.weight", (f, d)), (p + "mlp.c_proj.bias", (d,)),
        ]
    out += [("ln_f.weight", (d,)), ("ln_f.bias", (d,))]
    return out


def llama3_8b_shapes() -> List[Tuple[str, Tuple[int, ...]]]:
    """Llama-3-8B: 32 layers, hidden 4096, 32 q / 8 kv heads of 128, ffn 14336,
    vocab 128256 (291 tensors)."""
    h, kv, f, v = 4096, 1024, 14336, 128256
    out = [("embed_tokens", (v, h))]
    for l in range(32):
        p = "layers.%d." % l
        out += [
            (p + "input_layernorm", (h,)),
            (p + "q_proj", (h, h)), (p + "k_proj", (kv, h)),
            (p + "v_proj", (kv, h)), (p + "o_proj", (h, h)),
            (p + "post_attention_layernorm", (h,)),
            (p + "gate_proj", (f, h)), (p + "up_proj", (f, h)), (p + "down_proj", (h, f)),
        ]
    out += [("norm", (h,)), ("lm_head", (v, h))]
    return out


def scaled_shapes(shapes, div: int) -> List[Tuple[str, Tuple[int, ...]]]:
    """Same tensor list with every dimension divided by `div` (small test cases)."""
    return [(n, tuple(max(1, s // div) for s in shp)) for n, shp in shapes]


# ---------------------------------------------------------------------------
# flat uploads: one buffer, one cudaMemcpy payload per tensor
# ---------------------------------------------------------------------------

@dataclass
class Upload:
    """A set of payloads laid out in one flat uint8 buffer."""
    buf: torch.Tensor          # uint8, on `device`
    offsets: List[int]         # byte offset of each payload (ALIGN-aligned)
    sizes: List[int]           # byte length of each payload

    def payload(self, k: int) -> torch.Tensor:
        return self.buf[self.offsets[k]: self.offsets[k] + self.sizes[k]]

    @property
    def total_bytes(self) -> int:
        return sum(self.sizes)

    def chunks(self, chunk_bytes: int) -> List[Tuple[int, int, int]]:
        """(payload k, byte offset in buf, length) of every chunk, in call order."""
        out = []
        for k, (o, s) in enumerate(zip(self.offsets, self.sizes)):
            for i in range((s + chunk_bytes - 1) // chunk_bytes):
                out.append((k, o + i * chunk_bytes, min(chunk_bytes, s - i * chunk_bytes)))
        return out


def layout(sizes: Sequence[int], align: int = ALIGN) -> Tuple[List[int], int]:
    offs, pos = [], 0
    for s in sizes:
        offs.append(pos)
        pos += (s + align - 1) // align * align
    return offs, max(pos, align)


def weight_upload(shapes, dtype: torch.dtype, std: float = 0.02, seed: int = SEED_VALUES,
                  device="cpu") -> Upload:
    """Tensors ~N(0, std) in `dtype`, drawn in list order from one generator."""
    itemsize = torch.empty((), dtype=dtype).element_size()
    sizes = [math.prod(s) * itemsize for _, s in shapes]
    offs, total = layout(sizes)
    buf = torch.zeros(total, dtype=torch.uint8, device=device)
    g = _gen(seed, device)
    for (name, shp), o, s in zip(shapes, offs, sizes):
        t = torch.randn(math.prod(shp), dtype=torch.float32, generator=g, device=device)
        t = t.mul_(std).to(dtype)
        buf[o:o + s].copy_(t.view(torch.uint8))
        del t
    return Upload(buf, offs, sizes)


def fp16_payload(nbytes: int = 64 * MiB, std: float = 0.02, seed: int = SEED_VALUES,
                 device="cpu") -> torch.Tensor:
    """One payload of fp16 values ~N(0, std), as uint8."""
    g = _gen(seed, device)
    t = torch.randn(nbytes // 2, dtype=torch.float32, generator=g, device=device)
    return t.mul_(std).to(torch.float16).view(torch.uint8)


def random_bytes(n: int, seed: int, device="cpu") -> torch.Tensor:
    g = _gen(seed, device)
    return torch.randint(0, 256, (n,), dtype=torch.uint8, generator=g, device=device)


def select_chunks(nchunks: int, frac: float, seed: int = SEED_SELECT) -> torch.Tensor:
    """A seeded random subset of round(frac * nchunks) chunk ids (CPU int64, in
    draw order)."""
    g = _gen(seed, "cpu")
    k = int(round(frac * nchunks))
    return torch.randperm(nchunks, generator=g)[:k]


def gather_chunks(buf: torch.Tensor, chunk_bytes: int, ids: torch.Tensor) -> torch.Tensor:
    """Concatenation of the listed full chunks of `buf` (all ids must be full chunks)."""
    n = buf.numel()
    full = n // chunk_bytes
    assert bool((ids < full).all()), "gather_chunks takes full chunks only"
    view = buf[: full * chunk_bytes].view(full, chunk_bytes)
    return view[ids.to(buf.device)].reshape(-1).contiguous()


def flip_one_bit_per_chunk(buf: torch.Tensor, chunk_list, ids: torch.Tensor,
                           seed: int = SEED_PERTURB) -> torch.Tensor:
    """Flips one seeded bit inside each chunk listed by `ids` (indices into
    chunk_list = [(payload, offset, length), ...]).  In place; returns the byte
    offsets that were changed (CPU int64)."""
    g = _gen(seed, "cpu")
    ids = ids.cpu()
    offs = torch.tensor([chunk_list[i][1] for i in ids.tolist()], dtype=torch.int64)
    lens = torch.tensor([chunk_list[i][2] for i in ids.tolist()], dtype=torch.int64)
    r = torch.rand(len(ids), generator=g, dtype=torch.float64)
    bit = (r * (lens * 8).to(torch.float64)).to(torch.int64).clamp_max(lens * 8 - 1)
    byte_pos = offs + bit // 8
    mask = (torch.ones_like(bit) << (bit % 8)).to(torch.uint8)
    pos_dev = byte_pos.to(buf.device)
    buf[pos_dev] = buf[pos_dev] ^ mask.to(buf.device)
    return byte_pos


def loguniform_sizes(count: int, lo: int = 4 * KiB, hi: int = MiB,
                     seed: int = SEED_SELECT) -> List[int]:
    """floor(exp(U(ln lo, ln hi))) bytes, seeded."""
    g = _gen(seed, "cpu")
    u = torch.rand(count, generator=g, dtype=torch.float64)
    s = torch.exp(math.log(lo) + u * (math.log(hi) - math.log(lo))).floor().to(torch.int64)
    return [int(x) for x in s.clamp(lo, hi).tolist()]


def small_call_upload(count: int, seed: int = SEED_VALUES, device="cpu", lo: int = 4 * KiB,
                      hi: int = MiB) -> Upload:
    """`count` payloads of uniform random bytes with log-uniform sizes."""
    sizes = loguniform_sizes(count, lo, hi)
    offs, total = layout(sizes)
    buf = random_bytes(total, seed, device)
    return Upload(buf, offs, sizes)


@dataclass
class Adversarial:
    buf: torch.Tensor        # uint8 payload
    kind: torch.Tensor       # per chunk: 0 zero, 1 pattern, 2 random (CPU int8)
    pattern_id: torch.Tensor # per chunk: pattern 0..15 for kind 1, else -1 (CPU)


def adversarial_payload(nbytes: int, chunk_bytes: int, n_patterns: int = 16,
                        device="cpu") -> Adversarial:
    """25% all-zero chunks, 25% copies of `n_patterns` random patterns, 50%
    random bytes, placed by a seeded permutation.  nbytes % chunk_bytes == 0."""
    assert nbytes % chunk_bytes == 0
    n = nbytes // chunk_bytes
    perm = torch.randperm(n, generator=_gen(SEED_SELECT, "cpu"))
    kind = torch.full((n,), 2, dtype=torch.int8)
    q = n // 4
    kind[perm[:q]] = 0
    kind[perm[q:2 * q]] = 1
    pid = torch.full((n,), -1, dtype=torch.int64)
    pid[perm[q:2 * q]] = torch.randint(0, n_patterns, (q,), generator=_gen(SEED_PERTURB, "cpu"))
    buf = random_bytes(nbytes, SEED_VALUES, device).view(n, chunk_bytes)
    patterns = random_bytes(n_patterns * chunk_bytes, SEED_CRAFTED, device).view(n_patterns, chunk_bytes)
    zero_ids = (kind == 0).nonzero().flatten().to(buf.device)
    buf[zero_ids] = 0
    pat_ids = (kind == 1).nonzero().flatten()
    buf[pat_ids.to(buf.device)] = patterns[pid[pat_ids].to(buf.device)]
    return Adversarial(buf.reshape(-1), kind, pid)


def crafted_collisions(adv: Adversarial, chunk_bytes: int, count: int = 64,
                       seed: int = SEED_CRAFTED):
    """Picks `count` random-class chunks and returns (chunk ids, bytes with one
    flipped bit each as a [count, C] uint8 tensor).  The caller keys each
    entry by the fingerprint of the ORIGINAL chunk, so the index holds an
    entry whose key matches but whose bytes do not."""
    rnd = (adv.kind == 2).nonzero().flatten()
    g = _gen(seed, "cpu")
    pick = rnd[torch.randperm(rnd.numel(), generator=g)[:count]].sort().values
    rows = adv.buf.view(-1, chunk_bytes)[pick.to(adv.buf.device)].clone()
    bit = torch.randint(0, chunk_bytes * 8, (count,), generator=g)
    rows_cpu = rows.cpu()
    for r in range(count):
        b = int(bit[r])
        rows_cpu[r, b // 8] ^= (1 << (b % 8))
    return pick, rows_cpu.to(adv.buf.device)
