// First-occurrence resolution, stream compaction, packing and insertion for
// one dedup call over one or more payloads (paper Sec. 4.1.2: a chunk that is
// not resident travels in full and becomes reusable).
//
// The result must equal deciding the chunks one at a time, payload after
// payload, in ascending order.  Given the probe/verify outcome against the
// cache as it was when the call started (kHit0 or not), that rule reduces to:
//   * any other chunk is a hit iff an earlier chunk of the call has the same
//     length and bytes; its leader is the first such chunk;
//   * the misses are the leaders, inserted in ascending order at
//     slot = slots_used + rank;
//   * a hit on a leader from an earlier payload is, for its own payload, a hit
//     on the cache (that payload's call would have found the insert);
//   * a leader counts as a verify reject iff the cache had a key+length
//     candidate for it, or an earlier leader of the call has its key+length.
//
// Two launches follow the hash kernel.  k_dedup, cooperative, with phases
// separated by bounded grid barriers:
//   A  outputs are cleared; every non-resident chunk claims the entry of its
//      (key, length) in a per-call table and posts its number as the group
//      minimum;
//   B  each unresolved chunk compares itself (whole warp, 16-byte loads) with
//      its group's minimum: equal -> duplicate, number == minimum -> leader
//      of this round, else it stays for the next round (different bytes under
//      one key: a true 64-bit collision, or KEY16 test mode);
//   C  group minima of the remaining chunks are reset and re-posted (A);
//   D  leaders are counted per contiguous block range; the exclusive rank of
//      every chunk (and of every stored miss) follows from the block totals
//      plus warp ballots.
// k_pack, a regular launch of one wave, then writes hit masks, miss indices,
// chunk slots and per-payload counters, copies every miss by rank to the
// packed output and its arena slot and inserts it into the index; its last
// block publishes the counters and results and leaves the per-call state
// zeroed for the next call.
//
// A call with few chunks runs instead as one single-block kernel,
// k_small_call: the staged hash, then k_dedup's and k_pack's steps with a
// grid of one block (every grid barrier a block barrier), so that the call
// costs one launch and no kernel boundary.
#include "gleam_internal.cuh"
#include "staged_hash.cuh"

namespace gleam {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
#ifndef GLEAM_COPY_STREAMING_STORES
#define GLEAM_COPY_STREAMING_STORES 1
#endif
#ifndef GLEAM_COPY_VEC
#define GLEAM_COPY_VEC 8
#endif
#ifndef GLEAM_DEDUP_BLOCKS_PER_SM
#define GLEAM_DEDUP_BLOCKS_PER_SM 3
#endif
#ifndef GLEAM_DEDUP_CHUNKS_PER_BLOCK
#define GLEAM_DEDUP_CHUNKS_PER_BLOCK 1024
#endif
#ifndef GLEAM_CHAIN_PREFETCH
#define GLEAM_CHAIN_PREFETCH 1
#endif
#ifndef GLEAM_PACK_MINBLOCKS
#define GLEAM_PACK_MINBLOCKS 3
#endif
#if GLEAM_PACK_MINBLOCKS > 1
#define GLEAM_PACK_BOUNDS __launch_bounds__(kThreads, GLEAM_PACK_MINBLOCKS)
#else
#define GLEAM_PACK_BOUNDS __launch_bounds__(kThreads)
#endif
constexpr int kCopyVec = GLEAM_COPY_VEC;  // 16-byte vectors per lane in flight while copying
// In-call duplicates of at most this many bytes are compared kSmallCmpWays at a time.
#ifndef GLEAM_SMALL_CMP_WAYS
#define GLEAM_SMALL_CMP_WAYS 2
#endif
constexpr uint32_t kSmallCmpBytes = 1024;
constexpr uint32_t kSmallCmpWays = GLEAM_SMALL_CMP_WAYS;

__device__ __forceinline__ uint32_t ldcg_u32(const uint32_t* p) { return __ldcg(p); }

// Whole-warp byte equality of two full chunks of the payload.
__device__ bool warp_equal(const uint8_t* x, const uint8_t* y, uint32_t len, bool vec) {
  const uint32_t lane = threadIdx.x & 31;
  bool diff = false;
  uint32_t done = 0;
  if (vec) {
    const uint32_t nv = len >> 4;
    const uint4* xv = reinterpret_cast<const uint4*>(x);
    const uint4* yv = reinterpret_cast<const uint4*>(y);
    for (uint32_t k0 = 0; k0 < nv; k0 += 128) {
      uint4 u[4], w[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const uint32_t k = k0 + r * 32 + lane;
        if (k < nv) {
          u[r] = __ldcs(xv + k);
          w[r] = __ldcs(yv + k);
        } else {
          u[r] = make_uint4(0, 0, 0, 0);
          w[r] = u[r];
        }
      }
#pragma unroll
      for (int r = 0; r < 4; ++r)
        diff |= (u[r].x != w[r].x) | (u[r].y != w[r].y) | (u[r].z != w[r].z) | (u[r].w != w[r].w);
      if (__any_sync(0xffffffffu, diff)) return false;
    }
    done = nv << 4;
  }
  for (uint32_t k = done + lane; k < len; k += 32) diff |= (x[k] != y[k]);
  return !__any_sync(0xffffffffu, diff);
}

// Whole-warp copy of one chunk to the packed output and to its arena slot
// (d2 == nullptr: to the packed output only).  The path of copies that cannot
// be bulk copies (host or managed memory, unaligned addresses): out of line,
// away from the code that every call runs.
__device__ __noinline__ void warp_copy2(uint8_t* d1, uint8_t* d2, const uint8_t* s, uint32_t len, bool vec) {
  const uint32_t lane = threadIdx.x & 31;
  uint32_t done = 0;
  if (vec) {
    const uint32_t nv = len >> 4;
    const uint4* sv = reinterpret_cast<const uint4*>(s);
    uint4* d1v = reinterpret_cast<uint4*>(d1);
    uint4* d2v = reinterpret_cast<uint4*>(d2);
    for (uint32_t k0 = 0; k0 < nv; k0 += 32 * kCopyVec) {
      uint4 u[kCopyVec];
#pragma unroll
      for (int r = 0; r < kCopyVec; ++r) {
        const uint32_t k = k0 + r * 32 + lane;
        if (k < nv) u[r] = __ldg(sv + k);
      }
#pragma unroll
      for (int r = 0; r < kCopyVec; ++r) {
        const uint32_t k = k0 + r * 32 + lane;
        if (k < nv) {
#if GLEAM_COPY_STREAMING_STORES
          __stcs(d1v + k, u[r]);
          if (d2) __stcs(d2v + k, u[r]);
#else
          d1v[k] = u[r];
          if (d2) d2v[k] = u[r];
#endif
        }
      }
    }
    done = nv << 4;
  }
  for (uint32_t k = done + lane; k < len; k += 32) {
    const uint8_t b = s[k];
    d1[k] = b;
    if (d2) d2[k] = b;
  }
}

// ---- bulk asynchronous copies (k_pack's miss copies) -------------------------
//
// Lane 0 of a warp moves the warp's misses through kPackBufs shared-memory
// buffers of kPackPiece bytes: a bulk copy (the TMA engine, no registers)
// brings a piece in and signals an mbarrier with its byte count, then two bulk
// copies write it to the packed output and the arena slot.  Up to kPackBufs
// pieces are in flight per warp across chunk boundaries.  Needs 16-byte
// aligned addresses; a chunk's last len % 16 bytes are copied by its lane.
#ifndef GLEAM_PACK_GRAB
#define GLEAM_PACK_GRAB 1
#endif
#ifndef GLEAM_PACK_BULK
#define GLEAM_PACK_BULK 1
#endif
constexpr uint32_t kPackPiece = 2048;
constexpr uint32_t kPackBufs = 4;
struct PackMeta {
  unsigned long long src, d1, d2;
  uint32_t len, pad;
};
// per warp: the buffers, then the mbarriers (64 B), then the batch's metadata;
// a multiple of 128 bytes so that every warp's buffers start 128-byte aligned
constexpr uint32_t kPackWarpBytes =
    (kPackBufs * kPackPiece + 64 + 32 * (uint32_t)sizeof(PackMeta) + 127) & ~127u;
constexpr uint32_t kPackSmem = GLEAM_PACK_BULK ? kWarps * kPackWarpBytes : 0;

__device__ __forceinline__ void mbar_init(uint32_t bar) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(done)
      : "r"(bar), "r"(parity)
      : "memory");
  return done != 0;
}
// Waits for the mbarrier's phase of this parity, for at most limit_ns.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity,
                                         unsigned long long limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer_ns() - t0 > limit_ns) return false;
  return true;
}
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void bulk_store(void* dst, uint32_t src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(src),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
template <int N>
__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group %0;" ::"n"(N) : "memory");
}
// Until at most n (0..3; more waits for 3) newest bulk store groups still read
// shared memory.
__device__ __forceinline__ void bulk_wait_read_n(uint32_t n) {
  if (n == 0) bulk_wait_read<0>();
  else if (n == 1) bulk_wait_read<1>();
  else if (n == 2) bulk_wait_read<2>();
  else bulk_wait_read<3>();
}
static_assert(kPackBufs == 4, "bulk_wait_read_n covers up to kPackBufs - 1 pending groups");

// Ring state of one warp's lane 0, kept across its batches of 32 misses.
struct PackRing {
  uint32_t issued, consumed, phase;
};

// Lane 0: the whole-16-byte part of chunks 0..m-1 of `meta`; false if a
// piece did not arrive within limit_ns (the pieces still in flight have then
// been waited for, again with the limit).
__device__ bool bulk_copy_batch(const PackMeta* meta, uint32_t m, uint32_t bufs, uint32_t bars,
                                PackRing& ring, unsigned long long limit_ns) {
  auto nbytes = [&](uint32_t j) { return meta[j].len & ~15u; };
  uint32_t ij = 0, ioff = 0, cj = 0, coff = 0;  // issue and consume cursors
  while (ij < m && nbytes(ij) == 0) ++ij;
  cj = ij;
  while (cj < m) {
    while (ring.issued - ring.consumed < kPackBufs && ij < m) {
      const uint32_t b = ring.issued % kPackBufs;
      // the store that last read buffer b (piece issued - kPackBufs) must be done reading
      if (ring.issued >= kPackBufs) bulk_wait_read_n(kPackBufs - 1 - (ring.issued - ring.consumed));
      const uint32_t nb = nbytes(ij);
      const uint32_t bytes = min(kPackPiece, nb - ioff);
      mbar_expect_tx(bars + 8 * b, bytes);
      bulk_load(bufs + b * kPackPiece, reinterpret_cast<const uint8_t*>(meta[ij].src) + ioff, bytes,
                bars + 8 * b);
      ++ring.issued;
      ioff += bytes;
      if (ioff == nb) {
        ioff = 0;
        do ++ij;
        while (ij < m && nbytes(ij) == 0);
      }
    }
    const uint32_t b = ring.consumed % kPackBufs;
    if (!mbar_wait(bars + 8 * b, (ring.phase >> b) & 1u, limit_ns)) {
      for (uint32_t k = ring.consumed; k < ring.issued; ++k) {  // let the loads land
        const uint32_t bb = k % kPackBufs;
        mbar_wait(bars + 8 * bb, (ring.phase >> bb) & 1u, limit_ns);
        ring.phase ^= 1u << bb;
      }
      ring.consumed = ring.issued;
      return false;
    }
    ring.phase ^= 1u << b;
    const uint32_t nb = nbytes(cj);
    const uint32_t bytes = min(kPackPiece, nb - coff);
    bulk_store(reinterpret_cast<uint8_t*>(meta[cj].d1) + coff, bufs + b * kPackPiece, bytes);
    if (meta[cj].d2) bulk_store(reinterpret_cast<uint8_t*>(meta[cj].d2) + coff, bufs + b * kPackPiece, bytes);
    bulk_commit();
    ++ring.consumed;
    coff += bytes;
    if (coff == nb) {
      coff = 0;
      do ++cj;
      while (cj < m && nbytes(cj) == 0);
    }
  }
  return true;
}

__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// The rest of an insert's linear probe in KEY16 mode, from `pos` (the probe's
// `probe`-th position): all chunks of one 16-bit key share a home position,
// so an insert walks the cluster of the key's earlier entries.  The slot words
// of the next kScanEntries entries are read at once and the first that was
// free is claimed: one round trip per kScanEntries entries instead of one per
// entry.  While a call inserts, entries only go from free to used (evictions
// finish before), so an entry read as used stays used and is passed over
// safely; a claim that loses the race moves on to the next entry.  (With full
// 64-bit keys the entry after a used home is mostly free, and claiming it
// directly is one round trip fewer.)  False if the table is full.
constexpr uint32_t kScanEntries = 8;
__device__ __noinline__ bool index_insert_scan(IndexEntry* index, uint64_t mask,
                                               unsigned long long key, uint32_t slot,
                                               uint32_t len, uint64_t pos, uint64_t probe) {
  while (probe <= mask) {
    uint32_t free_bits = 0;
#pragma unroll
    for (uint32_t k = 0; k < kScanEntries; ++k)
      free_bits |= (ldcg_u32(&index[(pos + k) & mask].slot) == kEmptySlot ? 1u : 0u) << k;
    if (free_bits == 0) {
      pos = (pos + kScanEntries) & mask;
      probe += kScanEntries;
      continue;
    }
    const uint32_t k = __ffs(free_bits) - 1;
    probe += k;
    if (probe > mask) break;
    pos = (pos + k) & mask;
    if (atomicCAS(&index[pos].slot, kEmptySlot, slot) == kEmptySlot) {
      index[pos].key = key;
      index[pos].len = len;
      return true;
    }
    pos = (pos + 1) & mask;
    ++probe;
  }
  return false;
}

// Claims a free index entry for (key, slot, len); false if the table is full.
// scan: the rest of the probe by index_insert_scan (KEY16 index keys).
// place: the probe starts that many entries after the key's home position.
// With KEY16 classes the misses of a call that share an index key (and
// length) have the places 0 .. n-1, so each starts at its own entry instead
// of walking past the others; an entry stays reachable from the home
// position: a free entry left between the home position and a miss's entry
// (at place q) would have been taken by the miss whose place is q.
__device__ bool index_insert(IndexEntry* index, uint64_t mask, unsigned long long key,
                             uint32_t slot, uint32_t len, bool scan = false,
                             uint32_t place = 0) {
  uint64_t pos = (mix64(key) + place) & mask;
  for (uint64_t probe = 0; probe <= mask; ++probe) {
    const uint32_t old = atomicCAS(&index[pos].slot, kEmptySlot, slot);
    if (old == kEmptySlot) {
      index[pos].key = key;
      index[pos].len = len;
      return true;
    }
    pos = (pos + 1) & mask;
    if (scan) return index_insert_scan(index, mask, key, slot, len, pos, probe + 1);
  }
  return false;
}

// index_insert in two halves: the first claim attempt at the key's home
// position (issued early; its result is not waited for until it is needed),
// then, given that attempt's result, the entry's fields or the rest of the
// probe.  Together they do what index_insert does.
struct PendingInsert {
  uint64_t pos;
  uint32_t old;
};
__device__ __forceinline__ PendingInsert index_insert_begin(IndexEntry* index, uint64_t mask,
                                                            unsigned long long key, uint32_t slot) {
  const uint64_t pos = mix64(key) & mask;
  return PendingInsert{pos, atomicCAS(&index[pos].slot, kEmptySlot, slot)};
}
__device__ bool index_insert_end(IndexEntry* index, uint64_t mask, unsigned long long key,
                                 uint32_t slot, uint32_t len, PendingInsert p, bool scan = false) {
  uint64_t pos = p.pos;
  uint32_t old = p.old;
  for (uint64_t probe = 0;;) {
    if (old == kEmptySlot) {
      index[pos].key = key;
      index[pos].len = len;
      return true;
    }
    if (++probe > mask) return false;
    pos = (pos + 1) & mask;
    if (scan) return index_insert_scan(index, mask, key, slot, len, pos, probe);
    old = atomicCAS(&index[pos].slot, kEmptySlot, slot);
  }
}

// Finds or claims the per-call group entry of (key, len) for chunk g;
// *claimed tells whether g claimed it (else another chunk of the group did).
// cas_first: claim without reading the entry first (one round trip fewer
// where entries are mostly free; the read spares a contended entry the
// atomics of every chunk of a large group).
__device__ uint32_t group_entry(const DedupArgs& a, uint32_t g, unsigned long long k,
                                uint32_t len, bool* claimed = nullptr, bool cas_first = false) {
  uint64_t pos = mix64(k ^ ((unsigned long long)len << 40)) & a.tbl_mask;
  for (uint64_t probe = 0; probe <= a.tbl_mask; ++probe) {
    uint32_t o = cas_first && probe == 0 ? 0u : ldcg_u32(&a.tbl[pos].owner);
    if (o == 0) {
      o = atomicCAS(&a.tbl[pos].owner, 0u, g + 1);
      if (o == 0) {
        if (claimed) *claimed = true;
        return (uint32_t)pos;
      }
    }
    if (a.ch.key[o - 1] == k && a.ch.len[o - 1] == len) {
      if (claimed) *claimed = false;
      return (uint32_t)pos;
    }
    pos = (pos + 1) & a.tbl_mask;
  }
  return 0xFFFFFFFFu;  // cannot happen: the table has >= 2 Ntot entries
}

// KEY16 with XXH64 keys: finds or claims chunk g's entry in the per-call table
// of (16-bit index key, length) classes.
__device__ uint32_t class_entry(const DedupArgs& a, uint32_t g, unsigned long long k16,
                                uint32_t len) {
  uint64_t pos = mix64(k16 ^ ((unsigned long long)len << 40)) & a.tbl_mask;
  for (uint64_t probe = 0; probe <= a.tbl_mask; ++probe) {
    uint32_t o = ldcg_u32(&a.cls_tbl[pos].owner);
    if (o == 0) {
      o = atomicCAS(&a.cls_tbl[pos].owner, 0u, g + 1);
      if (o == 0) return (uint32_t)pos;
    }
    if ((a.ch.key[o - 1] & 0xFFFFull) == k16 && a.ch.len[o - 1] == len) return (uint32_t)pos;
    pos = (pos + 1) & a.tbl_mask;
  }
  return 0xFFFFFFFFu;  // cannot happen: the table has >= 2 Ntot entries
}

// The index key of a group key (KEY16 mode: its low 16 bits).
__device__ __forceinline__ unsigned long long index_key(const DedupArgs& a,
                                                        unsigned long long k) {
  return a.key16 ? (k & 0xFFFFull) : k;
}

__device__ __forceinline__ const PayloadDesc& desc(const DedupArgs& a, uint32_t p) {
  return a.count > 1 ? a.table[p] : a.one;
}

template <typename T>
__device__ __forceinline__ T block_sum(T v, T* red) {
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  T t = 0;
#pragma unroll
  for (int k = 0; k < kWarps; ++k) t += red[k];
  return t;
}

// Sum of v over the lanes of `peers`, added to *dst by the one lane of the
// group whose dst is not null.
__device__ __forceinline__ void add_in_group(unsigned long long* dst, unsigned peers, uint32_t v) {
  const uint32_t sum = __reduce_add_sync(peers, v);
  if (dst && sum) atomicAdd(dst, sum);
}

// ---- LRU eviction (paper Sec. 4.1.3; reading R16) ---------------------------
//
// The K slots to evict are the K smallest (last use, slot number) among the
// used slots whose last use is before this call (the call's own hits were
// stamped with its clock value in phase A).  The cut-off stamp is found by a
// two-pass radix select on its high and low 16 bits; the victims are then the
// slots older than the cut-off plus the lowest-numbered slots at it.  Their
// index and hint-table entries are removed without tombstones surviving the
// call: each is first replaced by a tombstone, then every cluster (maximal
// run of occupied entries) that holds one is rebuilt by its single owner
// thread, moving each live entry, in cluster order, to the first hole between
// its home position and itself, and finally the remaining tombstones become
// empty.  Clusters shrink but never merge, so owners never meet.

// Rebuilds the cluster that starts at `start` (its predecessor is empty).
__device__ void compact_cluster(IndexEntry* t, unsigned long long mask, unsigned long long start) {
  unsigned long long len = 0;
  bool any = false;
  for (unsigned long long q = start; len <= mask; q = (q + 1) & mask, ++len) {
    const uint32_t sl = t[q].slot;
    if (sl == kEmptySlot) break;
    any |= sl == kTombSlot;
  }
  if (!any) return;
  for (unsigned long long k = 0; k < len; ++k) {
    const unsigned long long q = (start + k) & mask;
    const IndexEntry e = t[q];
    if (e.slot == kTombSlot) continue;
    for (unsigned long long j = mix64(e.key) & mask; j != q; j = (j + 1) & mask) {
      if (t[j].slot == kTombSlot) {
        t[j] = e;
        t[q].slot = kTombSlot;
        break;
      }
    }
  }
}

// Exclusive block-wide prefix of per-thread flags, in thread order, for one
// 256-slot step; returns the thread's offset and adds the step's total to
// *running (shared arrays: kWarps counts + offsets).
__device__ __forceinline__ uint32_t block_rank(bool f, uint32_t* cnt, uint32_t* off,
                                               unsigned long long* running_total) {
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t b = __ballot_sync(0xffffffffu, f);
  if (lane == 0) cnt[w] = __popc(b);
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t acc = 0;
    for (int k = 0; k < kWarps; ++k) {
      off[k] = acc;
      acc += cnt[k];
    }
    cnt[0] = acc;
  }
  __syncthreads();
  const uint32_t r = off[w] + __popc(b & ((1u << lane) - 1u));
  const uint32_t step = cnt[0];
  __syncthreads();
  *running_total += step;
  return r;
}

// Selects and removes the K victims; false if a grid barrier failed.
__device__ bool lru_evict(const DedupArgs& a, uint32_t G, uint32_t bid,
                          unsigned long long slots0, unsigned long long K,
                          unsigned long long* sred, uint32_t* cnt, uint32_t* off,
                          unsigned long long* red64) {
  static_assert(kLruBins == kThreads * kThreads, "one part of kThreads bins per thread");
  const uint32_t lane = threadIdx.x & 31;
  const unsigned long long tid = (unsigned long long)bid * kThreads + threadIdx.x;
  const unsigned long long nth = (unsigned long long)G * kThreads;
  const uint32_t now = a.epoch;

  // cut-off stamp: radix select on the high, then the low 16 bits
  uint32_t hi_bin = 0;
  unsigned long long below = 0;
  for (int pass = 0; pass < 2; ++pass) {
    for (unsigned long long base = tid - lane; base < slots0; base += nth) {
      const unsigned long long sl = base + lane;
      uint32_t key = 0xFFFFFFFFu;
      if (sl < slots0) {
        const uint32_t u = __ldcg(&a.last_use[sl]);
        if (u != now && (pass == 0 || (u >> 16) == hi_bin)) key = pass == 0 ? (u >> 16) : (u & 0xFFFFu);
      }
      const unsigned peers = __match_any_sync(0xffffffffu, key);
      if (key != 0xFFFFFFFFu && lane == (uint32_t)(__ffs(peers) - 1))
        atomicAdd(&a.bins[key], (uint32_t)__popc(peers));
    }
    if (!grid_barrier(a.ctl, G, a.wait_ns, false)) return false;
    if (bid == 0) {
      // the bin holding the K-th candidate: partial sums of 256 bins per
      // thread (16-byte loads), the part holding it, then that part's bins
      constexpr uint32_t kPer = kLruBins / kThreads;
      const uint4* b4 = reinterpret_cast<const uint4*>(a.bins + threadIdx.x * kPer);
      unsigned long long part = 0;
#pragma unroll 16
      for (uint32_t j = 0; j < kPer / 4; ++j) {
        const uint4 v = __ldcg(b4 + j);
        part += (unsigned long long)v.x + v.y + v.z + v.w;
      }
      sred[threadIdx.x] = part;
      __syncthreads();
      const unsigned long long target = K - below;  // >= 1 candidates in this range
      if (threadIdx.x == 0) {
        unsigned long long acc = 0;
        uint32_t pi = 0;
        while (pi + 1 < (uint32_t)kThreads && acc + sred[pi] < target) acc += sred[pi++];
        off[0] = pi;
        sred[kThreads - 1] = acc;  // candidates before part pi (its own sum is no longer needed)
      }
      __syncthreads();
      const uint32_t pi = off[0];
      const unsigned long long acc0 = sred[kThreads - 1];
      __syncthreads();
      sred[threadIdx.x] = __ldcg(&a.bins[pi * kPer + threadIdx.x]);
      __syncthreads();
      if (threadIdx.x == 0) {
        unsigned long long acc = acc0;
        uint32_t j = 0;
        while (j + 1 < kPer && acc + sred[j] < target) acc += sred[j++];
        const uint32_t bin = pi * kPer + j;
        if (pass == 0) {
          a.ctl->lru_hi = bin;
          a.ctl->lru_below = acc;
        } else {
          a.ctl->lru_cut = (hi_bin << 16) | bin;
          a.ctl->lru_below = below + acc;
          a.ctl->lru_ties = target - acc;
        }
      }
      __syncthreads();
      uint4* z4 = reinterpret_cast<uint4*>(a.bins);
      for (uint32_t j = threadIdx.x; j < kLruBins / 4; j += kThreads) z4[j] = make_uint4(0, 0, 0, 0);
    }
    if (!grid_barrier(a.ctl, G, a.wait_ns, false)) return false;
    hi_bin = __ldcg(&a.ctl->lru_hi);
    below = __ldcg(&a.ctl->lru_below);
  }
  const uint32_t cut = __ldcg(&a.ctl->lru_cut);
  const unsigned long long ties = __ldcg(&a.ctl->lru_ties);

  // per contiguous slot range: candidates older than the cut-off, and at it
  const unsigned long long per = ((slots0 + G - 1) / G + 31) & ~31ull;
  const unsigned long long lo = min(slots0, bid * per);
  const unsigned long long hi = min(slots0, lo + per);
  {
    uint32_t nlt = 0, ntie = 0;
    for (unsigned long long sl = lo + threadIdx.x; sl < hi; sl += kThreads) {
      const uint32_t u = __ldcg(&a.last_use[sl]);
      if (u != now) {
        nlt += u < cut;
        ntie += u == cut;
      }
    }
    const unsigned long long t_lt = block_sum<unsigned long long>(nlt, red64);
    const unsigned long long t_tie = block_sum<unsigned long long>(ntie, red64);
    if (threadIdx.x == 0) {
      a.bcount[bid] = (uint32_t)t_tie;
      a.bcount[G + bid] = (uint32_t)t_lt;
    }
  }
  if (!grid_barrier(a.ctl, G, a.wait_ns, false)) return false;
  {
    unsigned long long tie_before = 0, lt_before = 0;
    for (uint32_t j = threadIdx.x; j < bid; j += kThreads) {
      tie_before += __ldcg(&a.bcount[j]);
      lt_before += __ldcg(&a.bcount[G + j]);
    }
    tie_before = block_sum<unsigned long long>(tie_before, red64);
    lt_before = block_sum<unsigned long long>(lt_before, red64);
    unsigned long long vrun = lt_before + min(ties, tie_before), trun = tie_before;
    unsigned long long vbytes = 0;
    for (unsigned long long t0 = lo; t0 < hi; t0 += kThreads) {
      const unsigned long long sl = t0 + threadIdx.x;
      const uint32_t u = sl < hi ? __ldcg(&a.last_use[sl]) : now;
      const bool tie = u != now && u == cut;
      const unsigned long long tb = trun;
      const uint32_t tr = block_rank(tie, cnt, off, &trun);
      const bool victim = (u != now && u < cut) || (tie && tb + tr < ties);
      const unsigned long long vb = vrun;
      const uint32_t vr = block_rank(victim, cnt, off, &vrun);
      if (victim && vb + vr < K) {  // always: the counts above add up to K
        a.victims[vb + vr] = (uint32_t)sl;
        a.vflag[sl] = 1;
        vbytes += a.slot_len[sl];
      }
    }
    vbytes = block_sum<unsigned long long>(vbytes, red64);
    if (threadIdx.x == 0 && vbytes) atomicAdd(&a.ctl->acc_victim_bytes, vbytes);
  }
  if (!grid_barrier(a.ctl, G, a.wait_ns, false)) return false;

  // the victims' entries leave the index and the hint table
  const unsigned long long tsize = a.index_mask + 1;
  for (unsigned long long q = tid; q < tsize; q += nth) {
    const uint32_t s1 = a.index[q].slot;
    if (s1 < slots0 && a.vflag[s1]) a.index[q].slot = kTombSlot;
    const uint32_t s2 = a.hints[q].slot;
    if (s2 < slots0 && a.vflag[s2]) a.hints[q].slot = kTombSlot;
  }
  if (!grid_barrier(a.ctl, G, a.wait_ns, false)) return false;
  for (unsigned long long q = tid; q < tsize; q += nth) {
    const unsigned long long prev = (q + tsize - 1) & a.index_mask;
    if (a.index[q].slot != kEmptySlot && a.index[prev].slot == kEmptySlot)
      compact_cluster(a.index, a.index_mask, q);
    if (a.hints[q].slot != kEmptySlot && a.hints[prev].slot == kEmptySlot)
      compact_cluster(a.hints, a.index_mask, q);
  }
  if (!grid_barrier(a.ctl, G, a.wait_ns, false)) return false;
  for (unsigned long long q = tid; q < tsize; q += nth) {
    if (a.index[q].slot == kTombSlot) a.index[q].slot = kEmptySlot;
    if (a.hints[q].slot == kTombSlot) a.hints[q].slot = kEmptySlot;
  }
  for (unsigned long long r = tid; r < K; r += nth) a.vflag[a.victims[r]] = 0;
  return true;
}

// Posts ~g as a candidate minimum of group entry `e` (0xFFFFFFFF: none), one
// atomic per group of lanes that share the entry.  Called by the whole warp.
template <typename Entry>
__device__ __forceinline__ void post_minimum(Entry* tbl, uint32_t e, uint32_t g,
                                             unsigned peers) {
  const uint32_t m = __reduce_max_sync(peers, e != 0xFFFFFFFFu ? ~g : 0u);
  // a group of many chunks (all-zero chunks, say) would queue its atomics on
  // one address: skip the atomic when a smaller number is already posted
  if (e != 0xFFFFFFFFu && (threadIdx.x & 31) == (uint32_t)(__ffs(peers) - 1) &&
      ldcg_u32(&tbl[e].minv) < m)
    atomicMax(&tbl[e].minv, m);
}
__device__ __forceinline__ void post_minimum(CallEntry* tbl, uint32_t e, uint32_t g) {
  post_minimum(tbl, e, g, __match_any_sync(0xffffffffu, e));
}

// KEY16 classes: posts ~g as a candidate minimum of class entry `e`
// (0xFFFFFFFF: none) and returns the lane's place among the misses of the
// class (counted in the entry), one atomic of each kind per group of lanes
// that share the entry.  Called by the whole warp.
__device__ __forceinline__ uint32_t post_class(ClassEntry* tbl, uint32_t e, uint32_t g) {
  const uint32_t lane = threadIdx.x & 31;
  const unsigned peers = __match_any_sync(0xffffffffu, e);
  post_minimum(tbl, e, g, peers);
  const int first = __ffs(peers) - 1;
  uint32_t base = 0;
  if (e != 0xFFFFFFFFu && lane == (uint32_t)first)
    base = atomicAdd(&tbl[e].count, (uint32_t)__popc(peers));
  return __shfl_sync(0xffffffffu, base, first) + __popc(peers & ((1u << lane) - 1u));
}
__device__ __forceinline__ void post_minimum(const DedupArgs& a, uint32_t e, uint32_t g) {
  post_minimum(a.tbl, e, g);
}

// The first-occurrence resolution and miss ranks of a call, run by block
// `bid` of a grid of G co-resident blocks.  claimed: the caller has done
// phase A (claims and minima posted, outputs cleared) and passed a grid
// barrier since, with outcome `ok0`.
__device__ __forceinline__ void resolve_rank(const DedupArgs& a, uint32_t G, uint32_t bid,
                                             bool claimed = false, bool ok0 = true) {
  __shared__ unsigned long long red64[kWarps];
  __shared__ uint32_t warp_cnt[kWarps];
  __shared__ uint32_t warp_off[kWarps];
  __shared__ uint32_t swarp_cnt[kWarps];
  __shared__ uint32_t swarp_off[kWarps];
  __shared__ unsigned long long s_slots0;
  __shared__ unsigned long long sred[kThreads];
  __shared__ int s_err1;

  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t tid = bid * kThreads + threadIdx.x;
  const uint32_t nth = G * kThreads;
  const uint32_t N = (uint32_t)a.Ntot;
  const bool skip = (int)bid == a.skip_block;
  const ChunkArrays& ch = a.ch;

  // thread 0's read of the slot count completes while phase A runs
  const unsigned long long my_slots0 =
      threadIdx.x == 0 ? *(volatile const unsigned long long*)&a.dstats[ST_SLOTS_USED] : 0ull;

  // ---- A: clear outputs, round-1 claims; LRU: stamp the slots hit ----------
  if (!claimed) {
    unsigned long long distinct = 0;
    for (uint32_t p = tid; p < a.count; p += nth) {
      gleam_result_t* r = desc(a, p).result;
      if (r) {
        r->n_miss = 0;
        r->n_hit_cache = 0;
        r->n_hit_intra = 0;
        r->verify_rejects = 0;
        r->miss_bytes = 0;
      }
    }
    // warp-uniform steps, so that chunks of one group in a warp post their
    // minimum with one atomic (all-zero chunks, say, share a group)
    for (uint32_t base = tid - lane; base < N; base += nth) {
      const uint32_t g = base + lane;
      uint32_t post = 0xFFFFFFFFu;  // group entry that gets this chunk's number
      if (g < N) {
        // every operand at once: the claim below then waits for none of them
        const uint8_t st = ch.status[g];
        const unsigned long long key = ch.key[g];
        const uint32_t len = ch.len[g];
        const PayloadDesc& P = desc(a, ch.pidx[g]);
        const unsigned long long i = g - P.chunk_base;
        if ((i & 31) == 0) P.mask[i >> 5] = 0;
        if (st == kHit0) {
          ch.res[g] = kResHit0;
          if (a.lru) {  // the first chunk to stamp a slot keeps its old value
            const uint32_t old = atomicExch(&a.last_use[ch.ent[g]], a.epoch);
            ch.old[g] = old;
            distinct += old != a.epoch;
          }
        } else if (st == kUncached) {  // never cached: a miss of its own, in no group
          ch.ent[g] = 0xFFFFFFFFu;
          ch.res[g] = kResLeader | kResNoSlot | 1u;
        } else {
          const uint32_t e = group_entry(a, g, key, len);
          if (e == 0xFFFFFFFFu) {
            atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
            ch.ent[g] = 0xFFFFFFFFu;
            ch.res[g] = kResLeader | 1u;
          } else {
            ch.ent[g] = e;
            ch.res[g] = kResUnresolved;
            post = e;
          }
        }
      }
      post_minimum(a, post, g);
    }
    if (a.lru) {
      distinct = block_sum<unsigned long long>(distinct, red64);
      if (threadIdx.x == 0 && distinct) atomicAdd(&a.ctl->acc_distinct, distinct);
    }
  }
  bool ok = claimed ? ok0 : grid_barrier(a.ctl, G, a.wait_ns, skip);

  // ---- B/C: rounds until every chunk is a hit, duplicate or leader ---------
  uint32_t round = 1;
  while (ok) {
    bool stay = false;  // one of this thread's chunks is left for the next round
    if (tid == 0) atomicExch(&a.ctl->unres[(round + 1) % 3], 0u);
    // W chunks per warp step: 32, or fewer when there are too few chunks to
    // give every warp a step (large chunks), so the compares spread over the grid
    const uint32_t nwarps = nth / 32;
    uint32_t W = 32;
    while (W > 1 && (unsigned long long)N < (unsigned long long)nwarps * W) W >>= 1;
    for (uint32_t base = (tid / 32) * W; base < N; base += nwarps * W) {
      const uint32_t g = base + lane;
      bool need = false, lead = false;
      uint32_t m = 0;
      if (lane < W && g < N && ldcg_u32(&ch.res[g]) == kResUnresolved) {
        m = ~ldcg_u32(&a.tbl[ch.ent[g]].minv);
        if (m == g) {
          ch.res[g] = kResLeader | round;
          lead = true;
        } else if (m > g) {  // the group minimum can only be below g: table damaged
          atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
          ch.res[g] = kResLeader | round;
          lead = true;
        } else if (ch.hint[g] != ch.hint[m]) {
          // different first 512 bytes (the prefix hints differ), so different
          // chunks: no byte compare, the chunk waits for a later round
          atomicAdd(&a.ctl->unres[round % 3], 1u);
          stay = true;
        } else {
          need = true;
        }
      }
      if (a.classes) {
        // KEY16: a new leader (a miss) claims the class of its 16-bit index
        // key and length, posts its number there and takes its place among
        // the class's misses (where its index insert starts); after the last
        // round a class minimum below a leader's number is an earlier miss of
        // its index key and length (a reject).  Groups are whole fingerprints, so
        // nearly all leaders are found in the first round, while the other warps
        // compare their duplicates.
        uint32_t cpost = 0xFFFFFFFFu;
        if (lead) {
          cpost = class_entry(a, g, ch.key[g] & 0xFFFFull, ch.len[g]);
          if (cpost == 0xFFFFFFFFu) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
        }
        const uint32_t place = post_class(a.cls_tbl, cpost, g);
        if (lead) ch.cls[g] = cpost | ((unsigned long long)place << 32);
      }
      uint32_t todo = __ballot_sync(0xffffffffu, need);
      // every lane fetches its own chunk's operands at once, so that each
      // compare below waits for its bytes only, not for their addresses first
      unsigned long long xs = 0, ys = 0;
      uint32_t ln = 0;
      if (need) {
        xs = ch.src[g];
        ys = ch.src[m];
        ln = ch.len[g];
      }
      // duplicates of at most kSmallCmpBytes (whole 16-byte pieces, aligned
      // operands) are compared up to kSmallCmpWays at a time, every lane loading
      // its pieces of all of them before any result is needed; the others one
      // by one
      unsigned small = __ballot_sync(0xffffffffu, need && ln <= kSmallCmpBytes && (ln & 15) == 0 &&
                                                      ((xs | ys) & 15) == 0);
      auto settle = [&](int j, bool eq) {
        if (lane == (uint32_t)j) {
          if (eq) {
            ch.ent[g] = m;  // the leader, for the hit's classification
            ch.res[g] = kResDup;
          } else {
            atomicAdd(&a.ctl->unres[round % 3], 1u);
            stay = true;
          }
        }
      };
      while (kSmallCmpWays > 1 && __popc(small) >= 2) {
        int js[kSmallCmpWays];
        uint32_t cnt = 0;
        while (cnt < kSmallCmpWays && small) {
          js[cnt++] = __ffs(small) - 1;
          small &= small - 1;
        }
        uint4 u[kSmallCmpWays][kSmallCmpBytes / 512], v[kSmallCmpWays][kSmallCmpBytes / 512];
#pragma unroll
        for (uint32_t c = 0; c < kSmallCmpWays; ++c) {
          if (c < cnt) {
            const uint4* x = reinterpret_cast<const uint4*>(__shfl_sync(0xffffffffu, xs, js[c]));
            const uint4* y = reinterpret_cast<const uint4*>(__shfl_sync(0xffffffffu, ys, js[c]));
            const uint32_t np = __shfl_sync(0xffffffffu, ln, js[c]) >> 4;
#pragma unroll
            for (uint32_t r = 0; r < kSmallCmpBytes / 512; ++r) {
              const uint32_t k = r * 32 + lane;
              u[c][r] = k < np ? __ldcs(x + k) : make_uint4(0, 0, 0, 0);
              v[c][r] = k < np ? __ldcs(y + k) : make_uint4(0, 0, 0, 0);
            }
          }
        }
#pragma unroll
        for (uint32_t c = 0; c < kSmallCmpWays; ++c) {
          if (c < cnt) {
            bool diff = false;
#pragma unroll
            for (uint32_t r = 0; r < kSmallCmpBytes / 512; ++r)
              diff |= (u[c][r].x != v[c][r].x) | (u[c][r].y != v[c][r].y) |
                      (u[c][r].z != v[c][r].z) | (u[c][r].w != v[c][r].w);
            settle(js[c], !__any_sync(0xffffffffu, diff));
            todo &= ~(1u << js[c]);
          }
        }
      }
      while (todo) {
        const int j = __ffs(todo) - 1;
        todo &= todo - 1;
        const uint8_t* x = reinterpret_cast<const uint8_t*>(__shfl_sync(0xffffffffu, xs, j));
        const uint8_t* y = reinterpret_cast<const uint8_t*>(__shfl_sync(0xffffffffu, ys, j));
        const uint32_t len = __shfl_sync(0xffffffffu, ln, j);
        const bool vec = (((uintptr_t)x | (uintptr_t)y) & 15) == 0;
        settle(j, warp_equal(x, y, len, vec));
      }
    }
    if (G == 1) {  // the block's own count, without the round trip to the counter
      if (!__syncthreads_or(stay)) break;
    } else {
      ok = grid_barrier(a.ctl, G, a.wait_ns, false);
      if (!ok) break;
      if (ldcg_u32(&a.ctl->unres[round % 3]) == 0) break;
    }
    for (uint32_t g = tid; g < N; g += nth)
      if (ldcg_u32(&ch.res[g]) == kResUnresolved) a.tbl[ch.ent[g]].minv = 0;
    ok = grid_barrier(a.ctl, G, a.wait_ns, false);
    if (!ok) break;
    for (uint32_t base = tid - lane; base < N; base += nth) {
      const uint32_t g = base + lane;
      post_minimum(a, g < N && ldcg_u32(&ch.res[g]) == kResUnresolved ? ch.ent[g] : 0xFFFFFFFFu, g);
    }
    ok = grid_barrier(a.ctl, G, a.wait_ns, false);
    ++round;
  }

  // ---- D1: misses per contiguous block range --------------------------------
  const uint64_t per = (((uint64_t)N + G - 1) / G + 31) & ~31ull;
  const uint32_t lo = (uint32_t)min((uint64_t)N, bid * per);
  const uint32_t hi = (uint32_t)min((uint64_t)N, lo + per);
  unsigned long long before = 0, total = 0, sbefore = 0, stotal = 0, evict = 0;
  if (ok) {
    uint32_t cnt = 0, scnt = 0;
    for (uint32_t g = lo + threadIdx.x; g < hi; g += kThreads) {
      const uint32_t r = ldcg_u32(&ch.res[g]);
      if (r & kResLeader) {
        ++cnt;
        if (!(r & kResNoSlot)) ++scnt;
        // a verify reject: the cache had a key+length candidate, or an
        // earlier miss of the call has this key and length (another leader
        // of a later round; with classes, an earlier leader of the class)
        bool earlier;
        if (a.classes) {
          const uint32_t cl = (uint32_t)ch.cls[g];  // in range unless the call failed
          earlier = cl <= a.tbl_mask && ~ldcg_u32(&a.cls_tbl[cl].minv) < g;
        } else {
          earlier = (r & kResRoundMask) > 1;
        }
        const bool rej = !(r & kResNoSlot) && (ch.status[g] == kMissCand || earlier);
        if (rej) ch.res[g] = r | kResReject;
        // leave the group table zeroed for the next call: every claimed entry
        // belongs to a group with at least one leader
        const uint32_t e = ch.ent[g];
        if (e != 0xFFFFFFFFu) {
          a.tbl[e].owner = 0u;
          a.tbl[e].minv = 0u;
        }
      }
    }
    const unsigned long long c = block_sum<unsigned long long>(cnt, red64);
    const unsigned long long sc = block_sum<unsigned long long>(scnt, red64);
    if (G == 1) {
      total = c;
      stotal = sc;
    } else {
      if (threadIdx.x == 0) {
        a.bcount[bid] = (uint32_t)c;
        a.bcount[G + bid] = (uint32_t)sc;
      }
      ok = grid_barrier(a.ctl, G, a.wait_ns, false);
    }
  }
  if (threadIdx.x == 0) s_slots0 = my_slots0;
  __syncthreads();
  const unsigned long long slots0 = s_slots0;
  // ---- D2: exclusive miss rank of every chunk; per-payload start ranks ------
  if (ok && G > 1) {
    for (uint32_t j = threadIdx.x; j < G; j += kThreads) {
      const uint32_t v = ldcg_u32(&a.bcount[j]);
      const uint32_t sv = ldcg_u32(&a.bcount[G + j]);
      total += v;
      stotal += sv;
      if (j < bid) {
        before += v;
        sbefore += sv;
      }
    }
    before = block_sum<unsigned long long>(before, red64);
    total = block_sum<unsigned long long>(total, red64);
    sbefore = block_sum<unsigned long long>(sbefore, red64);
    stotal = block_sum<unsigned long long>(stotal, red64);
  }
  if (ok) {
    if (stotal > a.nslots - slots0) {
      // LRU: evict the missing slots among those this call did not hit
      evict = stotal - (a.nslots - slots0);
      if (!a.lru || evict > slots0 - __ldcg(&a.ctl->acc_distinct)) {
        if (threadIdx.x == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_CAPACITY);
        ok = false;
      }
    }
  }
  if (ok && a.classes) {
    // every read of the class table happened before the last barrier: the
    // grid clears the call's whole table with plain 16-byte stores (a
    // clear per chunk would first load the chunk's class entry)
    uint4* t4 = reinterpret_cast<uint4*>(a.cls_tbl);
    const unsigned long long n4 = a.tbl_mask + 1;  // one 16-byte store per entry
    for (unsigned long long e = tid; e < n4; e += nth) t4[e] = make_uint4(0u, 0u, 0u, 0u);
  }
  if (ok) {
    unsigned long long running = before, srunning = sbefore;
    for (uint32_t t = lo; t < hi; t += kThreads) {
      const uint32_t g = t + threadIdx.x;
      const bool valid = g < hi;
      const uint32_t rv = valid ? ldcg_u32(&ch.res[g]) : 0u;
      const bool miss = valid && (rv & kResLeader);
      const bool stored = miss && !(rv & kResNoSlot);
      const uint32_t mb = __ballot_sync(0xffffffffu, miss);
      const uint32_t sb = __ballot_sync(0xffffffffu, stored);
      if (lane == 0) {
        warp_cnt[w] = __popc(mb);
        swarp_cnt[w] = __popc(sb);
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        uint32_t acc = 0, sacc = 0;
        for (int k = 0; k < kWarps; ++k) {
          warp_off[k] = acc;
          acc += warp_cnt[k];
          swarp_off[k] = sacc;
          sacc += swarp_cnt[k];
        }
        warp_cnt[0] = acc;
        swarp_cnt[0] = sacc;
      }
      __syncthreads();
      const uint32_t below = (1u << lane) - 1u;
      if (valid) {
        const uint32_t r = (uint32_t)(running + warp_off[w] + __popc(mb & below));
        ch.rank[g] = r;
        if (miss) ch.order[r] = g;
        if (stored) ch.srank[g] = (uint32_t)(srunning + swarp_off[w] + __popc(sb & below));
        const uint32_t p = ch.pidx[g];
        if (g == desc(a, p).chunk_base) a.pstart[p] = r;
      }
      running += warp_cnt[0];
      srunning += swarp_cnt[0];
      __syncthreads();
    }
    ok = grid_barrier(a.ctl, G, a.wait_ns, false);
  }
  if (ok && evict && G == 1) {  // its barriers did not read the error word
    if (threadIdx.x == 0) s_err1 = ld_volatile_s32(&a.ctl->err);
    __syncthreads();
    ok = s_err1 == 0;
  }
  if (ok && evict) ok = lru_evict(a, G, bid, slots0, evict, sred, warp_cnt, warp_off, red64);
  // totals for k_pack (the capacity check above left them unpublished on error)
  if (ok && bid == 0 && threadIdx.x == 0) {
    a.ctl->acc_misses = total;
    a.ctl->acc_stored = stotal;
    a.ctl->evict_k = evict;
  }
}

// The end of a call, run by every block: the last block to get here
// publishes the counters and results and leaves the per-call state (group
// table, control block) as the next call expects it.  total/stored/evict/
// vbytes: the call's misses, stored misses, evicted slots and their bytes;
// s_sum: a grid of one block's sums (hits, intra hits, rejects, miss bytes,
// stored bytes, chunks written ahead, of them used), else the control block's.
// After an error that may have stopped the leaders before they cleared their
// entries: the whole group table (and class table), and an eviction's
// histogram and flags.  Out of line: rare, and kept out of the code that
// every call runs.
__device__ __noinline__ void clear_after_error(const DedupArgs& a) {
  for (unsigned long long e = threadIdx.x; e <= a.tbl_mask; e += kThreads) {
    a.tbl[e].owner = 0u;
    a.tbl[e].minv = 0u;
    if (a.classes) a.cls_tbl[e] = ClassEntry{0u, 0u, 0u, 0u};
  }
  if (a.lru) {  // an eviction that stopped half-way may have left these set
    for (uint32_t j = threadIdx.x; j < kLruBins; j += kThreads) a.bins[j] = 0u;
    for (unsigned long long j = threadIdx.x; j < a.nslots; j += kThreads) a.vflag[j] = 0;
  }
}

__device__ __forceinline__ void finish_call(const DedupArgs& a, uint32_t G,
                                            unsigned long long slots0,
                                            unsigned long long total,
                                            unsigned long long s_stored,
                                            unsigned long long evict,
                                            unsigned long long s_vbytes,
                                            const unsigned long long* s_sum) {
  const uint32_t N = (uint32_t)a.Ntot;
  __shared__ int s_last;
  __syncthreads();
  if (threadIdx.x == 0) {
    if (G == 1) {  // the block barrier already orders the block's own writes
      s_last = 1;
    } else {
      __threadfence();
      s_last = atomicAdd(&a.ctl->done, 1u) == G - 1;
    }
  }
  __syncthreads();
  if (!s_last) return;
  if (G > 1) __threadfence();
  const int err = ld_volatile_s32(&a.ctl->err);
  if (threadIdx.x == 0) {
    const bool one = G == 1;
    const unsigned long long misses = total;
    const unsigned long long hc = one ? s_sum[0] : __ldcg(&a.ctl->acc_hits_cache);
    const unsigned long long hi2 = one ? s_sum[1] : __ldcg(&a.ctl->acc_hits_intra);
    const unsigned long long rej = one ? s_sum[2] : __ldcg(&a.ctl->acc_rejects);
    const unsigned long long mbytes = one ? s_sum[3] : __ldcg(&a.ctl->acc_miss_bytes);
    const unsigned long long sbytes = one ? s_sum[4] : __ldcg(&a.ctl->acc_stored_bytes);
    const unsigned long long stored = s_stored;
    const unsigned long long vbytes = s_vbytes;
    const unsigned long long spec = one ? s_sum[5] : __ldcg(&a.ctl->spec_tried);
    const unsigned long long spec_used = one ? s_sum[6] : __ldcg(&a.ctl->spec_used);
    if (err == 0 && a.spec_state) {
      // automatic write-through: stays on while at least half of the chunks
      // written ahead were used; once off, tried again after 256 calls
      uint32_t* st = a.spec_state;
      if (spec) {
        st[0] = 2 * spec_used >= spec ? 1u : 0u;
        st[1] = 0;
      } else if (st[0] == 0 && ++st[1] >= 256) {
        st[0] = 1;
        st[1] = 0;
      }
      *a.spec_mirror = st[0];
    }
    if (err == 0) {  // no reads: the counters change by atomic adds
      atomicAdd(&a.dstats[ST_CALLS], a.ncalls);
      atomicAdd(&a.dstats[ST_CHUNKS], (unsigned long long)N);
      atomicAdd(&a.dstats[ST_HITS_CACHE], hc);
      atomicAdd(&a.dstats[ST_HITS_INTRA], hi2);
      atomicAdd(&a.dstats[ST_MISSES], misses);
      atomicAdd(&a.dstats[ST_INSERTS], stored);
      atomicAdd(&a.dstats[ST_REJECTS], rej);
      a.dstats[ST_SLOTS_USED] = slots0 + stored - evict;
      atomicAdd(&a.dstats[ST_BYTES_USED], sbytes - vbytes);
      atomicAdd(&a.dstats[ST_EVICTIONS], evict);
      if (spec) atomicAdd(&a.dstats[ST_SPEC_CHUNKS], spec);
    }
    gleam_result_t* t = a.total;
    t->status = err;
    t->n_miss = err ? 0 : misses;
    t->n_hit_cache = err ? 0 : hc;
    t->n_hit_intra = err ? 0 : hi2;
    t->verify_rejects = err ? 0 : rej;
    t->miss_bytes = err ? 0 : mbytes;
  }
  for (uint32_t p = threadIdx.x; p < a.count; p += kThreads) {
    gleam_result_t* r = desc(a, p).result;
    if (!r) continue;
    r->status = err;
    if (err) {
      r->n_miss = 0;
      r->n_hit_cache = 0;
      r->n_hit_intra = 0;
      r->verify_rejects = 0;
      r->miss_bytes = 0;
    }
  }
  // Leave the per-call state as the next call expects it: the group table
  // (cleared entry by entry by the leaders, or here in full after an error
  // that may have stopped them) and the control block.
  if (err) clear_after_error(a);
  __syncthreads();
  if (threadIdx.x == 0) {
    DevCtl* c = a.ctl;
    c->bar_count = 0;
    c->copy_next = 0;
    c->err = 0;
    c->unres[0] = c->unres[1] = c->unres[2] = 0;
    c->shared_groups = 0;
    c->acc_hits_cache = c->acc_hits_intra = c->acc_rejects = 0;
    c->acc_misses = c->acc_miss_bytes = 0;
    c->acc_stored = c->acc_stored_bytes = 0;
    c->acc_distinct = c->evict_k = c->lru_below = c->lru_ties = c->acc_victim_bytes = 0;
    c->lru_hi = c->lru_cut = 0;
    c->spec_tried = c->spec_used = 0;
    c->done = 0;
  }
  __threadfence();
}


// Second kernel of the call (a regular launch sized for the copies): hit
// masks, miss indices, chunk slots, per-payload counters, then every miss by
// rank copied by whole warps to the packed output and its arena slot and
// inserted into the index; the last block publishes the counters and results
// and leaves the per-call state zeroed.  Nothing is written after an error.
__device__ __forceinline__ void pack_publish(const DedupArgs& a, uint32_t G, uint32_t bid,
                                             uint8_t* pack_smem) {
  __shared__ unsigned long long red64[kWarps];
  __shared__ unsigned long long s_slots0, s_total, s_evict;
  // a grid of one block keeps its totals here instead of in the control block
  __shared__ unsigned long long s_stored, s_vbytes, s_sum[7];
  __shared__ int s_err;
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t N = (uint32_t)a.Ntot;
  const ChunkArrays& ch = a.ch;
  if (threadIdx.x == 0) {
    s_slots0 = *(volatile const unsigned long long*)&a.dstats[ST_SLOTS_USED];
    s_err = ld_volatile_s32(&a.ctl->err);
    s_total = __ldcg(&a.ctl->acc_misses);
    s_evict = __ldcg(&a.ctl->evict_k);
    s_stored = __ldcg(&a.ctl->acc_stored);
    s_vbytes = __ldcg(&a.ctl->acc_victim_bytes);
    for (int k = 0; k < 7; ++k) s_sum[k] = 0;
  }
  __syncthreads();
  const unsigned long long slots0 = s_slots0;
  const unsigned long long total = s_total;
  const unsigned long long evict = s_evict;
  const bool ok = s_err == 0;
#if GLEAM_PACK_BULK
  const uint32_t wbase = (uint32_t)__cvta_generic_to_shared(pack_smem) + w * kPackWarpBytes;
  const uint32_t bufs = wbase, bars = wbase + kPackBufs * kPackPiece;
  PackMeta* meta = reinterpret_cast<PackMeta*>(pack_smem + w * kPackWarpBytes +
                                               kPackBufs * kPackPiece + 64);
  PackRing ring{0u, 0u, 0u};
  if (lane == 0) {
    for (uint32_t b = 0; b < kPackBufs; ++b) mbar_init(bars + 8 * b);
    mbar_fence_init();
  }
  __syncwarp();
  bool bulk_failed = false;
#endif
  // slot of the stored miss of stored rank sr: the evicted slots in ascending
  // order, then never-used slots
  auto slot_of = [&](uint32_t sr) -> unsigned long long {
    return sr < evict ? (unsigned long long)__ldcg(&a.victims[sr]) : slots0 + (sr - evict);
  };

  // ---- after an error: give the hit slots their last use back (LRU) ---------
  if (!ok && a.lru) {
    for (unsigned long long g = (unsigned long long)bid * kThreads + threadIdx.x; g < N;
         g += (unsigned long long)G * kThreads)
      if (ch.status[g] == kHit0 && ch.old[g] != a.epoch) a.last_use[ch.ent[g]] = ch.old[g];
  }

  // ---- hit masks, miss indices, chunk slots, counters ------------------------
  if (ok) {
    unsigned long long n_hc = 0, n_hi = 0, n_rej = 0, n_bytes = 0, n_sbytes = 0;
    uint32_t n_spec = 0, n_spec_used = 0;  // write-through: chunks written ahead, used
    // Each warp classifies a contiguous range of chunks (whole 32-chunk
    // steps), so that its steps mostly fall in one payload: the counters of a
    // payload are summed in the warp over its steps and added once where the
    // warp leaves the payload, instead of once per step by every warp on the
    // same few addresses (a one-payload call of a million chunks would queue
    // ~10^5 atomics on one result).
    const unsigned long long nsteps = ((unsigned long long)N + 31) / 32;
    const unsigned long long cw_n = (unsigned long long)G * kWarps;
    const unsigned long long cw = (unsigned long long)bid * kWarps + w;
    const unsigned long long c_lo = nsteps * cw / cw_n * 32;
    const unsigned long long c_hi = min((unsigned long long)N, nsteps * (cw + 1) / cw_n * 32);
    gleam_result_t* acc_res = nullptr;  // the payload whose counters the warp holds
    unsigned long long acc_hc = 0, acc_hi = 0, acc_miss = 0, acc_rej = 0, acc_len = 0;
    auto flush = [&]() {
      if (acc_res && lane == 0) {
        if (acc_hc) atomicAdd((unsigned long long*)&acc_res->n_hit_cache, acc_hc);
        if (acc_hi) atomicAdd((unsigned long long*)&acc_res->n_hit_intra, acc_hi);
        if (acc_miss) atomicAdd((unsigned long long*)&acc_res->n_miss, acc_miss);
        if (acc_rej) atomicAdd((unsigned long long*)&acc_res->verify_rejects, acc_rej);
        if (acc_len) atomicAdd((unsigned long long*)&acc_res->miss_bytes, acc_len);
      }
      acc_res = nullptr;
      acc_hc = acc_hi = acc_miss = acc_rej = acc_len = 0;
    };
    for (unsigned long long t = c_lo; t < c_hi; t += 32) {
      const uint32_t g = (uint32_t)(t + lane);
      const bool valid = t + lane < c_hi;
      const uint32_t r = valid ? ldcg_u32(&ch.res[g]) : 0u;
      const uint32_t p = valid ? ch.pidx[g] : 0xFFFFFFFFu;
      const bool miss = valid && (r & kResLeader);
      bool hc = false, hi2 = false, rej = false;
      uint32_t len = 0, bit = 0;
      unsigned long long mw = 0;  // address of the chunk's hit-mask word, if a hit
      gleam_result_t* res = nullptr;
      if (valid) {
        const PayloadDesc& P = desc(a, p);
        const unsigned long long i = g - P.chunk_base;
        res = P.result;
        if (r & kResHit0) hc = true;
        if (r & kResDup) {
          if (ch.pidx[ch.ent[g]] == p) hi2 = true;  // leader in the same payload
          else hc = true;                           // inserted by an earlier payload
        }
        if (hc || hi2) {
          mw = (unsigned long long)(P.mask + (i >> 5));
          bit = 1u << (i & 31);
        }
        if (P.chunk_slot) {
          uint32_t sl;
          if (r & kResHit0) sl = ch.ent[g];                                      // matched slot
          else if (r & kResDup) sl = (uint32_t)slot_of(__ldcg(&ch.srank[ch.ent[g]]));  // leader's
          else if (r & kResNoSlot) sl = kEmptySlot;                              // never cached
          else sl = (uint32_t)slot_of(ch.srank[g]);                              // its new slot
          P.chunk_slot[i] = sl;
        }
        if (miss) {
          len = ch.len[g];
          P.miss_idx[ch.rank[g] - __ldcg(&a.pstart[p])] = (uint32_t)i;
          rej = (r & kResReject) != 0;
        }
      }
      n_spec += a.spec_active && valid && ch.spec[g];
      n_hc += hc;
      n_hi += hi2;
      n_rej += rej;
      n_bytes += len;
      if (!(r & kResNoSlot)) n_sbytes += len;
      // hit-mask words and per-payload result counters: one atomic per group
      // of lanes that share the word or the payload
      const unsigned mpeers = __match_any_sync(0xffffffffu, mw);
      const uint32_t bits = __reduce_or_sync(mpeers, bit);
      if (mw && lane == (uint32_t)(__ffs(mpeers) - 1)) atomicOr((uint32_t*)mw, bits);
      const unsigned peers = __match_any_sync(0xffffffffu, res ? p : 0xFFFFFFFFu);
      if (peers == 0xffffffffu && res) {  // the whole step in one payload that has a result
        if (res != acc_res) {
          flush();
          acc_res = res;
        }
        acc_hc += __reduce_add_sync(0xffffffffu, (uint32_t)hc);
        acc_hi += __reduce_add_sync(0xffffffffu, (uint32_t)hi2);
        acc_miss += __reduce_add_sync(0xffffffffu, (uint32_t)miss);
        acc_rej += __reduce_add_sync(0xffffffffu, (uint32_t)rej);
        acc_len += __reduce_add_sync(0xffffffffu, len);
      } else {  // payload boundaries: one atomic per group of lanes per counter
        const bool lead = res && lane == (uint32_t)(__ffs(peers) - 1);
        add_in_group((unsigned long long*)(lead ? &res->n_hit_cache : nullptr), peers, hc);
        add_in_group((unsigned long long*)(lead ? &res->n_hit_intra : nullptr), peers, hi2);
        add_in_group((unsigned long long*)(lead ? &res->n_miss : nullptr), peers, miss);
        add_in_group((unsigned long long*)(lead ? &res->verify_rejects : nullptr), peers, rej);
        add_in_group((unsigned long long*)(lead ? &res->miss_bytes : nullptr), peers, len);
      }
    }
    flush();
    // Every miss's bytes, in pieces of kPackPiece bytes: piece k of the miss
    // of rank r is number r * ppc + k (ppc = pieces of a whole chunk; a
    // shorter miss has fewer), and warp gw owns the contiguous numbers
    // [plo, phi), so that a call with few misses still spreads its copies over
    // every warp (one 64 KiB miss is 32 pieces) and a call with many streams
    // whole runs of chunks per warp.  The lanes fetch the metadata of 32
    // pieces at once (mostly one chunk's: the same addresses), then the pieces
    // go to the packed output and the miss's arena slot, all but those of
    // misses the hash kernel already wrote there.
    const unsigned long long nw = (unsigned long long)G * kWarps;
    const unsigned long long gw = (unsigned long long)bid * kWarps + w;
    const unsigned long long ppc = (a.C + kPackPiece - 1) / kPackPiece;
    const unsigned long long npieces = total * ppc;
    const unsigned long long plo = npieces * gw / nw, phi = npieces * (gw + 1) / nw;
    // written ahead by the hash kernel exactly where it belongs: with no
    // eviction, stored rank g means every earlier chunk of the call is a
    // stored miss, so the chunk's packed offset is i*C and its slot
    // slots_used + g, the places it was written to
    auto written_ahead = [&](uint32_t gg, uint32_t sr) {
      return a.spec_active && evict == 0 && sr == gg && ch.spec[gg];
    };
#if GLEAM_PACK_GRAB
    // With GLEAM_PACK_GRAB the warps take their steps of 32 pieces from a
    // counter of the call instead (each asks for its next step before it
    // copies the current one), so that warps on SMs that copy faster take
    // more.  The static ranges remain where the hash kernel wrote likely
    // misses ahead (the steps then copy little, and the counter's round trip
    // would be most of a step) and for counts the 32-bit counter cannot hold.
    const bool grab = !a.spec_active && npieces < (1ull << 31);
#else
    const bool grab = false;
#endif
    unsigned long long step = plo, step_end = phi;
    if (grab) {
      uint32_t b0 = 0;
      if (lane == 0) b0 = atomicAdd(&a.ctl->copy_next, 32u);
      step = __shfl_sync(0xffffffffu, b0, 0);
      step_end = npieces;
    }
    while (step < step_end) {
      uint32_t next = 0;
      if (grab && lane == 0) next = atomicAdd(&a.ctl->copy_next, 32u);
      const unsigned long long shi = min(step_end, step + 32);
      const unsigned long long pc = step + lane;
      uint32_t bytes = 0;
      bool copy = false;
      unsigned long long src = 0, d1 = 0, d2 = 0;
      if (pc < shi) {
        const unsigned long long r = pc / ppc;
        const uint32_t off = (uint32_t)(pc - r * ppc) * kPackPiece;
        const uint32_t gg = ch.order[r];
        const uint32_t ln = ch.len[gg];
        if (off < ln) {
          const uint32_t pp = ch.pidx[gg];
          const PayloadDesc& P = desc(a, pp);
          bytes = min(kPackPiece, ln - off);
          src = ch.src[gg] + off;
          d1 = (unsigned long long)(P.packed + (r - a.pstart[pp]) * a.C + off);
          uint32_t sr = 0xFFFFFFFFu;
          if (!(ch.res[gg] & kResNoSlot)) {  // else sent, never cached
            sr = ch.srank[gg];
            d2 = (unsigned long long)(a.arena + slot_of(sr) * a.C + off);
          }
          copy = !written_ahead(gg, sr);
        }
      }
      const unsigned cmask = __ballot_sync(0xffffffffu, copy);  // lanes whose piece is copied
      const uint32_t m = __popc(cmask);
#if GLEAM_PACK_BULK
      const bool bulk =
          !a.plain_copy && __all_sync(0xffffffffu, !copy || ((src | d1 | d2) & 15) == 0);
      if (bulk) {
        if (copy) meta[__popc(cmask & ((1u << lane) - 1u))] = PackMeta{src, d1, d2, bytes, 0u};
        __syncwarp();
        if (lane == 0 && m && !bulk_failed &&
            !bulk_copy_batch(meta, m, bufs, bars, ring, a.wait_ns)) {
          bulk_failed = true;
          atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_TIMEOUT);
        }
        if (copy) {  // the piece's last bytes % 16 (only a miss's last piece has any)
          const uint8_t* sp = reinterpret_cast<const uint8_t*>(src);
          uint8_t* x = reinterpret_cast<uint8_t*>(d1);
          uint8_t* y = reinterpret_cast<uint8_t*>(d2);
          for (uint32_t k = bytes & ~15u; k < bytes; ++k) {
            x[k] = sp[k];
            if (y) y[k] = sp[k];
          }
        }
        __syncwarp();
      } else
#endif
      for (unsigned todo = cmask; todo; todo &= todo - 1) {
        const int j = __ffs(todo) - 1;
        const unsigned long long sj = __shfl_sync(0xffffffffu, src, j);
        const unsigned long long xj = __shfl_sync(0xffffffffu, d1, j);
        const unsigned long long yj = __shfl_sync(0xffffffffu, d2, j);
        const uint32_t lj = __shfl_sync(0xffffffffu, bytes, j);
        warp_copy2(reinterpret_cast<uint8_t*>(xj), reinterpret_cast<uint8_t*>(yj),
                   reinterpret_cast<const uint8_t*>(sj), lj, ((sj | xj | yj) & 15) == 0);
      }
      if (grab) step = __shfl_sync(0xffffffffu, next, 0);
      else step += 32;
    }
    // Every miss's index and hint-table entries, by rank: warp gw owns the
    // contiguous ranks [lo, hi), each lane inserting its own chunk (32
    // independent probes at a time).
    const unsigned long long lo = total * gw / nw, hi = total * (gw + 1) / nw;
    for (unsigned long long base = lo; base < hi; base += 32) {
      const unsigned long long r = base + lane;
      if (r >= hi) continue;
      const uint32_t gg = ch.order[r];
      if (ch.res[gg] & kResNoSlot) continue;  // sent, never cached
      const uint32_t ln = ch.len[gg];
      const uint32_t sr = ch.srank[gg];
      const unsigned long long slot = slot_of(sr);
      n_spec_used += written_ahead(gg, sr);
      a.slot_len[slot] = ln;
      a.slot_key[slot] = ch.key[gg];
      if (a.lru) a.last_use[slot] = a.epoch;
      if (!index_insert(a.index, a.index_mask, index_key(a, ch.key[gg]), (uint32_t)slot, ln,
                        a.key16, a.classes ? (uint32_t)(ch.cls[gg] >> 32) : 0u))
        atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
      if (!a.paper && ln >= kPrefixBytes &&
          !index_insert(a.hints, a.index_mask, ch.hint[gg], (uint32_t)slot, ln))
        atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
    }
#if GLEAM_PACK_BULK
    if (lane == 0) bulk_wait_all<0>();  // every piece written before the block ends
#endif
    n_hc = block_sum<unsigned long long>(n_hc, red64);
    n_hi = block_sum<unsigned long long>(n_hi, red64);
    n_rej = block_sum<unsigned long long>(n_rej, red64);
    n_bytes = block_sum<unsigned long long>(n_bytes, red64);
    n_sbytes = block_sum<unsigned long long>(n_sbytes, red64);
    const unsigned long long b_spec = block_sum<unsigned long long>(n_spec, red64);
    const unsigned long long b_spec_used = block_sum<unsigned long long>(n_spec_used, red64);
    if (threadIdx.x == 0 && G == 1) {
      s_sum[0] = n_hc;
      s_sum[1] = n_hi;
      s_sum[2] = n_rej;
      s_sum[3] = n_bytes;
      s_sum[4] = n_sbytes;
      s_sum[5] = b_spec;
      s_sum[6] = b_spec_used;
    } else if (threadIdx.x == 0) {
      atomicAdd(&a.ctl->acc_hits_cache, n_hc);
      atomicAdd(&a.ctl->acc_hits_intra, n_hi);
      atomicAdd(&a.ctl->acc_rejects, n_rej);
      atomicAdd(&a.ctl->acc_miss_bytes, n_bytes);
      atomicAdd(&a.ctl->acc_stored_bytes, n_sbytes);
      if (b_spec) atomicAdd(&a.ctl->spec_tried, b_spec);
      if (b_spec_used) atomicAdd(&a.ctl->spec_used, b_spec_used);
    }
  }

  finish_call(a, G, slots0, total, s_stored, evict, s_vbytes, s_sum);
}

// ---- one-launch resolve + pack of a one-payload call --------------------------
//
// A call of one payload that is launched chained (few enough chunks to leave
// most of the GPU idle) runs its resolution, ranks, packing and publishing in
// one launch.  Block b owns the contiguous chunks [b * per, (b + 1) * per),
// at most one per thread.  Phase 1 classifies them and claims their (key,
// length) groups without posting minima.  If no chunk of the call found its
// group claimed by another (no in-call duplicate and no key collision: the
// common case), every chunk that is not a cache hit is a miss of round one
// (its own group's first chunk), so after one grid barrier each block knows
// its misses' ranks from the blocks' counts, writes the outputs and inserts
// its misses; after a second barrier every warp of the grid copies its share
// of all misses' bytes (a block's own misses would leave the blocks that hold
// the most of them as the call's tail).  Otherwise the general algorithm
// takes over: the minima are posted and resolve_rank and pack_publish run on
// the same grid.
constexpr uint32_t kResolvePackSmem = kPackSmem;


// Bit k of the result: byte k of w (k < 4) is not kHit0.
__device__ __forceinline__ uint32_t not_hit_bits(uint32_t w) {
  const uint32_t x = w ^ (0x01010101u * kHit0);
  const uint32_t t = (((x & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | x) & 0x80808080u;  // bit 8k+7: byte k != 0
  return ((t >> 7) & 1u) | ((t >> 14) & 2u) | ((t >> 21) & 4u) | ((t >> 28) & 8u);
}

// This thread's share of the call's chunks that are not cache hits: among
// chunks [0, lim) (*below) and among all N (*all); the block's threads
// together cover every chunk once.
__device__ __forceinline__ void count_not_hit(const uint8_t* status, uint32_t N, uint32_t lim,
                                              uint32_t* below, uint32_t* all) {
  uint32_t b = 0, t = 0;
  const bool vec = ((uintptr_t)status & 15) == 0;
  for (uint32_t v = threadIdx.x; v * 16 < N; v += blockDim.x) {
    const uint32_t b0 = v * 16;
    uint32_t m = 0;
    if (vec && b0 + 16 <= N) {
      const uint4 q = __ldcg(reinterpret_cast<const uint4*>(status) + v);
      m = not_hit_bits(q.x) | not_hit_bits(q.y) << 4 | not_hit_bits(q.z) << 8 |
          not_hit_bits(q.w) << 12;
    } else {
      for (uint32_t k = 0; k < 16 && b0 + k < N; ++k)
        m |= (uint32_t)(__ldcg(status + b0 + k) != kHit0) << k;
    }
    t += __popc(m);
    const uint32_t nb = lim <= b0 ? 0u : min(lim - b0, 16u);
    b += __popc(m & ((1u << nb) - 1u));
  }
  *below = b;
  *all = t;
}

// The general algorithm on the one-launch kernel's grid, for a call with a
// shared group: if the hash kernel claimed the groups (pre), their entries are
// cleared and claimed again by the whole group key and length (a shared tag
// may be two different pairs'); then the group minima are posted, and the
// rounds, ranks and copies of k_dedup and k_pack run.  Out of line, so that
// the common path's code stays compact (the kernel runs once per call, on SMs
// whose instruction caches are cold).  Every thread of every block calls it;
// mine: this thread holds a chunk of a group (entry e, group key and length).
__device__ __noinline__ void resolve_pack_general(const DedupArgs& a, uint32_t G, uint32_t bid,
                                                  uint8_t* smem, bool ok, bool pre, bool mine,
                                                  uint32_t e, unsigned long long key,
                                                  uint32_t len, uint32_t g) {
  if (pre) {
    if (mine && e != 0xFFFFFFFFu)
      *reinterpret_cast<volatile unsigned long long*>(&a.tbl[e]) = 0ull;
    ok = grid_barrier(a.ctl, G, a.wait_ns, false) && ok;
    if (ok && mine) {
      bool claimed = true;
      e = group_entry(a, g, key, len, &claimed, true);
      if (e == 0xFFFFFFFFu) {
        atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
        a.ch.res[g] = kResLeader | 1u;
      }
      a.ch.ent[g] = e;
    }
  }
  if (ok) post_minimum(a, mine && e != 0xFFFFFFFFu ? e : 0xFFFFFFFFu, g);  // one chunk per thread
  ok = grid_barrier(a.ctl, G, a.wait_ns, false);
  resolve_rank(a, G, bid, true, ok);
  grid_barrier(a.ctl, G, a.wait_ns, false);
  pack_publish(a, G, bid, smem);
}

__device__ __forceinline__ void resolve_pack_fast(const DedupArgs& a, uint32_t G, uint32_t bid,
                                                  uint8_t* smem) {
  __shared__ unsigned long long red64[kWarps];
  __shared__ uint32_t wcnt[kWarps], swcnt[kWarps];
  __shared__ unsigned long long s_slots0, s_sum[7];
  __shared__ int s_shared, s_err;
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const ChunkArrays& ch = a.ch;
  const PayloadDesc& P = a.one;
  const uint32_t N = (uint32_t)a.Ntot;
  const uint32_t per = (N + G - 1) / G;  // <= kThreads (the host sizes the grid)
  const uint32_t g = bid * per + threadIdx.x;
  const bool valid = threadIdx.x < per && g < N;
  if (per > kThreads && threadIdx.x == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
  const unsigned long long my_slots0 =
      threadIdx.x == 0 ? *(volatile const unsigned long long*)&a.dstats[ST_SLOTS_USED] : 0ull;
  if (threadIdx.x == 0) s_shared = 0;

  // ---- 1: classify, clear the outputs, claim the groups ----------------------
  if (bid == 0 && threadIdx.x == 0 && P.result) {
    gleam_result_t* r = P.result;
    r->n_miss = r->n_hit_cache = r->n_hit_intra = r->verify_rejects = r->miss_bytes = 0;
  }
  uint8_t st = kMissNoCand;
  uint32_t len = 0, e = 0xFFFFFFFFu;
  unsigned long long key = 0, hint = 0;
  bool lead = false, stored = false, shared = false;
  // the hash kernel claimed the groups: every miss is stored (the staged
  // kernel marks no chunk uncached) and was given its entry there
  const bool pre = a.pre_claimed != 0;
  if (valid) {
    // the chunk's record at once (one round trip, whatever its status)
    st = ch.status[g];
    const unsigned long long key0 = ch.key[g];
    const uint32_t len0 = ch.len[g];
    const uint32_t ent0 = pre ? ch.ent[g] : 0u;
    hint = a.paper ? 0ull : ch.hint[g];
    if ((g & 31) == 0) P.mask[g >> 5] = 0;
    if (st == kHit0) {
      ch.res[g] = kResHit0;
    } else if (st == kUncached) {  // never cached: a miss of its own, in no group
      ch.ent[g] = 0xFFFFFFFFu;
      ch.res[g] = kResLeader | kResNoSlot | 1u;
      lead = true;
      len = len0;
    } else {
      key = key0;
      len = len0;
      bool claimed = true;
      e = pre ? ent0 : group_entry(a, g, key, len, &claimed, true);
      if (e == 0xFFFFFFFFu) {
        atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
        ch.res[g] = kResLeader | 1u;
      } else if (!pre) {
        ch.res[g] = kResUnresolved;
      }
      if (!pre) ch.ent[g] = e;
      shared = !claimed;
      lead = stored = true;
    }
  }
  const uint32_t c_b = __syncthreads_count(lead);
  const uint32_t s_b = __syncthreads_count(stored);
  if (__syncthreads_or(shared) && threadIdx.x == 0) {
    s_shared = 1;
    if (G > 1) atomicOr(&a.ctl->shared_groups, 1u);
  }
  bool ok = true;
  unsigned long long pre_before = 0, pre_total = 0;
  if (pre) {
    // no barrier: every block counts the misses before its chunks, and in
    // all, from the statuses the hash kernel wrote (at most 16 KiB of them)
    uint32_t mb = 0, mt = 0;
    count_not_hit(ch.status, N, bid * per, &mb, &mt);
    pre_before = block_sum<unsigned long long>(mb, red64);
    pre_total = block_sum<unsigned long long>(mt, red64);
    if (threadIdx.x == 0) {
      s_shared = (int)ldcg_u32(&a.ctl->shared_groups);
      s_slots0 = my_slots0;
      s_err = ld_volatile_s32(&a.ctl->err);
    }
    __syncthreads();
    ok = s_err == 0;
  } else {
    if (G > 1 && threadIdx.x == 0) {
      a.bcount[bid] = c_b;
      a.bcount[G + bid] = s_b;
    }
    ok = grid_barrier(a.ctl, G, a.wait_ns, false);
    if (threadIdx.x == 0) {
      if (G > 1) s_shared = (int)ldcg_u32(&a.ctl->shared_groups);
      s_slots0 = my_slots0;
      s_err = G == 1 ? ld_volatile_s32(&a.ctl->err) : 0;
    }
    __syncthreads();
    if (G == 1) ok = s_err == 0;  // a grid of one did not read the error word
  }

  if (s_shared) {
    resolve_pack_general(a, G, bid, smem, ok, pre, valid && st != kHit0 && st != kUncached, e,
                         key, len, g);
    return;
  }

  // ---- 2: the fast path: ranks, outputs, inserts; then copies ----------------
  const unsigned long long slots0 = s_slots0;
  unsigned long long before = 0, total = c_b, sbefore = 0, stotal = s_b;
  if (pre) {
    before = sbefore = pre_before;
    total = stotal = pre_total;
  } else if (G > 1) {
    unsigned long long b0 = 0, t0 = 0, sb0 = 0, st0 = 0;
    for (uint32_t j = threadIdx.x; j < G; j += kThreads) {
      const uint32_t v = ldcg_u32(&a.bcount[j]), sv = ldcg_u32(&a.bcount[G + j]);
      t0 += v;
      st0 += sv;
      if (j < bid) {
        b0 += v;
        sb0 += sv;
      }
    }
    before = block_sum<unsigned long long>(b0, red64);
    total = block_sum<unsigned long long>(t0, red64);
    sbefore = block_sum<unsigned long long>(sb0, red64);
    stotal = block_sum<unsigned long long>(st0, red64);
  }
  if (ok && stotal > a.nslots - slots0) {  // every block decides the same
    if (threadIdx.x == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_CAPACITY);
    ok = false;
  }
  unsigned long long n_hc = 0, n_rej = 0, n_bytes = 0, n_sbytes = 0;
  uint32_t n_spec = 0, n_spec_used = 0;
  unsigned long long ins_slot = ~0ull;  // the slot this thread's stored miss takes
  if (ok) {
    // ranks within the block, in chunk order
    const uint32_t mb = __ballot_sync(0xffffffffu, lead);
    const uint32_t sb = __ballot_sync(0xffffffffu, stored);
    if (lane == 0) {
      wcnt[w] = __popc(mb);
      swcnt[w] = __popc(sb);
    }
    __syncthreads();
    uint32_t woff = 0, swoff = 0;
    for (uint32_t k2 = 0; k2 < w; ++k2) {
      woff += wcnt[k2];
      swoff += swcnt[k2];
    }
    const uint32_t below = (1u << lane) - 1u;
    const unsigned long long r = before + woff + __popc(mb & below);
    const unsigned long long sr = sbefore + swoff + __popc(sb & below);
    const unsigned long long slot = slots0 + sr;
    const bool spec = a.spec_active && valid && ch.spec[g];
    n_spec += spec;
    n_spec_used += spec && stored && sr == g;
    if (lead) {
      P.miss_idx[r] = g;
      ch.order[r] = g;  // for the copies, spread over the grid below
      ch.srank[g] = stored ? (uint32_t)sr : kEmptySlot;
      n_rej += st == kMissCand;
      n_bytes += len;
      if (stored) n_sbytes += len;
    }
    // hit-mask words: one atomic per group of lanes that share a word
    const bool hit = valid && st == kHit0;
    n_hc += hit;
    const unsigned long long mw = hit ? (unsigned long long)(P.mask + (g >> 5)) : 0ull;
    const unsigned mpeers = __match_any_sync(0xffffffffu, mw);
    const uint32_t bits = __reduce_or_sync(mpeers, hit ? 1u << (g & 31) : 0u);
    if (mw && lane == (uint32_t)(__ffs(mpeers) - 1)) atomicOr((uint32_t*)mw, bits);
    if (P.chunk_slot && valid)
      P.chunk_slot[g] = hit ? ch.ent[g] : stored ? (uint32_t)slot : kEmptySlot;
    ins_slot = stored ? slot : ~0ull;
  }
  ok = grid_barrier(a.ctl, G, a.wait_ns, false) && ok;
  if (ok) {
    // each stored miss records its slot and starts its index inserts (the
    // first claim attempts), which complete after the copies below
    const bool ins = ins_slot != ~0ull;
    const bool ins_hint = ins && !a.paper && len >= kPrefixBytes;
    PendingInsert pi{0ull, 0u}, ph{0ull, 0u};
    if (ins) {
      a.slot_len[ins_slot] = len;
      a.slot_key[ins_slot] = key;
      pi = index_insert_begin(a.index, a.index_mask, index_key(a, key), (uint32_t)ins_slot);
      if (ins_hint) ph = index_insert_begin(a.hints, a.index_mask, hint, (uint32_t)ins_slot);
    }
    // every miss's bytes, in pieces of kPackPiece bytes spread over all the
    // grid's warps (piece k of the miss of rank r is number r * ppc + k), all
    // but those of misses the hash kernel already wrote where they belong
    // (stored rank g means every earlier chunk is a stored miss: no eviction
    // here)
    const unsigned long long nw = (unsigned long long)G * kWarps;
    const unsigned long long gw = (unsigned long long)bid * kWarps + w;
    const unsigned long long ppc = (a.C + kPackPiece - 1) / kPackPiece;
    const unsigned long long npieces = total * ppc;
    const unsigned long long plo = npieces * gw / nw, phi = npieces * (gw + 1) / nw;
#if GLEAM_PACK_BULK
    const uint32_t wbase = (uint32_t)__cvta_generic_to_shared(smem) + w * kPackWarpBytes;
    const uint32_t bufs = wbase, bars = wbase + kPackBufs * kPackPiece;
    PackMeta* meta = reinterpret_cast<PackMeta*>(smem + w * kPackWarpBytes + kPackBufs * kPackPiece + 64);
    PackRing ring{0u, 0u, 0u};
    bool bulk_failed = false;
    if (lane == 0) {
      for (uint32_t b = 0; b < kPackBufs; ++b) mbar_init(bars + 8 * b);
      mbar_fence_init();
    }
    __syncwarp();
#endif
    // pieces [lo, hi) of the call, 32 at a time
    auto copy_range = [&](unsigned long long lo, unsigned long long hi) {
      for (unsigned long long base = lo; base < hi; base += 32) {
        const unsigned long long pc = base + lane;
        uint32_t bytes = 0;
        bool copy = false;
        unsigned long long src = 0, d1 = 0, d2 = 0;
        if (pc < hi) {
          const unsigned long long rr = pc / ppc;
          const uint32_t off = (uint32_t)(pc - rr * ppc) * kPackPiece;
          const uint32_t gg = __ldcg(&ch.order[rr]);
          const uint32_t ln = (uint32_t)min(a.C, P.n - (unsigned long long)gg * a.C);
          if (off < ln) {
            const uint32_t srr = __ldcg(&ch.srank[gg]);
            const bool ahead = a.spec_active && srr == gg && ch.spec[gg];
            if (!ahead) {
              bytes = min(kPackPiece, ln - off);
              src = (unsigned long long)(P.buf + (unsigned long long)gg * a.C + off);
              d1 = (unsigned long long)(P.packed + rr * a.C + off);
              d2 = srr != kEmptySlot ? (unsigned long long)(a.arena + (slots0 + srr) * a.C + off)
                                     : 0ull;
              copy = true;
            }
          }
        }
        const unsigned cmask = __ballot_sync(0xffffffffu, copy);
#if GLEAM_PACK_BULK
        const bool bulk =
            !a.plain_copy && __all_sync(0xffffffffu, !copy || ((src | d1 | d2) & 15) == 0);
        if (bulk) {
          if (copy) meta[__popc(cmask & ((1u << lane) - 1u))] = PackMeta{src, d1, d2, bytes, 0u};
          __syncwarp();
          if (lane == 0 && cmask && !bulk_failed &&
              !bulk_copy_batch(meta, __popc(cmask), bufs, bars, ring, a.wait_ns)) {
            bulk_failed = true;
            atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_TIMEOUT);
          }
          if (copy) {  // the piece's last bytes % 16
            const uint8_t* sp = reinterpret_cast<const uint8_t*>(src);
            uint8_t* x = reinterpret_cast<uint8_t*>(d1);
            uint8_t* y = reinterpret_cast<uint8_t*>(d2);
            for (uint32_t k2 = bytes & ~15u; k2 < bytes; ++k2) {
              x[k2] = sp[k2];
              if (y) y[k2] = sp[k2];
            }
          }
          __syncwarp();
        } else
#endif
        for (unsigned todo = cmask; todo; todo &= todo - 1) {
          const int j = __ffs(todo) - 1;
          const unsigned long long sj = __shfl_sync(0xffffffffu, src, j);
          const unsigned long long xj = __shfl_sync(0xffffffffu, d1, j);
          const unsigned long long yj = __shfl_sync(0xffffffffu, d2, j);
          const uint32_t lj = __shfl_sync(0xffffffffu, bytes, j);
          warp_copy2(reinterpret_cast<uint8_t*>(xj), reinterpret_cast<uint8_t*>(yj),
                     reinterpret_cast<const uint8_t*>(sj), lj, ((sj | xj | yj) & 15) == 0);
        }
      }
    };
    if (a.copy_grab) {
      // the pieces taken copy_grab at a time from a counter of the call, the
      // warp's next grab requested before its current one is copied: warps
      // on SMs that copy faster take more
      const uint32_t grab = a.copy_grab;
      uint32_t nxt = 0;
      if (lane == 0) nxt = atomicAdd(&a.ctl->copy_next, grab);
      nxt = __shfl_sync(0xffffffffu, nxt, 0);
      while (nxt < npieces) {
        uint32_t nn = 0;
        if (lane == 0) nn = atomicAdd(&a.ctl->copy_next, grab);
        copy_range(nxt, min(npieces, (unsigned long long)nxt + grab));
        nxt = __shfl_sync(0xffffffffu, nn, 0);
      }
    } else {
#if GLEAM_CHAIN_PREFETCH
      // the warp's source pieces start their way into L2 at once (up to 32),
      // so that the copies below wait for L2 rather than HBM
      if (plo + lane < phi && !a.plain_copy) {
        const unsigned long long pc = plo + lane, rr = pc / ppc;
        const uint32_t off = (uint32_t)(pc - rr * ppc) * kPackPiece;
        const uint32_t gg = __ldcg(&ch.order[rr]);
        const uint32_t ln = (uint32_t)min(a.C, P.n - (unsigned long long)gg * a.C);
        const uint8_t* src = P.buf + (unsigned long long)gg * a.C + off;
        if (off < ln && ((uintptr_t)src & 15) == 0) {  // the prefetch wants 16-byte alignment
          const uint32_t pb = min(kPackPiece, ln - off) & ~15u;
          if (pb) prefetch_l2(src, pb);
        }
      }
#endif
      copy_range(plo, phi);
    }
    // each stored miss completes its inserts and frees the group entry it
    // claimed, while the last pieces' stores are still in flight
    if (ins) {
      if (!index_insert_end(a.index, a.index_mask, index_key(a, key), (uint32_t)ins_slot, len, pi,
                            a.key16))
        atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
      if (ins_hint &&
          !index_insert_end(a.hints, a.index_mask, hint, (uint32_t)ins_slot, len, ph))
        atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
      if (e != 0xFFFFFFFFu) a.tbl[e] = CallEntry{0u, 0u};  // owner and the claim's tag
    }
#if GLEAM_PACK_BULK
    if (lane == 0) bulk_wait_all<0>();  // every piece written before the block ends
#endif
  }
  n_hc = block_sum<unsigned long long>(n_hc, red64);
  n_rej = block_sum<unsigned long long>(n_rej, red64);
  n_bytes = block_sum<unsigned long long>(n_bytes, red64);
  n_sbytes = block_sum<unsigned long long>(n_sbytes, red64);
  const unsigned long long b_spec = block_sum<unsigned long long>(n_spec, red64);
  const unsigned long long b_spec_used = block_sum<unsigned long long>(n_spec_used, red64);
  if (threadIdx.x == 0 && P.result) {  // the payload's own counters (cleared in phase 1)
    gleam_result_t* res = P.result;
    if (n_hc) atomicAdd((unsigned long long*)&res->n_hit_cache, n_hc);
    if (c_b) atomicAdd((unsigned long long*)&res->n_miss, (unsigned long long)c_b);
    if (n_rej) atomicAdd((unsigned long long*)&res->verify_rejects, n_rej);
    if (n_bytes) atomicAdd((unsigned long long*)&res->miss_bytes, n_bytes);
  }
  if (threadIdx.x == 0) {
    if (G == 1) {
      s_sum[0] = n_hc;
      s_sum[1] = 0;  // no in-call duplicate on this path
      s_sum[2] = n_rej;
      s_sum[3] = n_bytes;
      s_sum[4] = n_sbytes;
      s_sum[5] = b_spec;
      s_sum[6] = b_spec_used;
    } else {
      if (n_hc) atomicAdd(&a.ctl->acc_hits_cache, n_hc);
      if (n_rej) atomicAdd(&a.ctl->acc_rejects, n_rej);
      if (n_bytes) atomicAdd(&a.ctl->acc_miss_bytes, n_bytes);
      if (n_sbytes) atomicAdd(&a.ctl->acc_stored_bytes, n_sbytes);
      if (b_spec) atomicAdd(&a.ctl->spec_tried, b_spec);
      if (b_spec_used) atomicAdd(&a.ctl->spec_used, b_spec_used);
    }
  }
  finish_call(a, G, slots0, total, stotal, 0ull, 0ull, s_sum);
}

__global__ void __launch_bounds__(kThreads) k_resolve_pack(DedupArgs a) {
  extern __shared__ __align__(128) uint8_t rp_smem[];
  pdl_trigger();
  pdl_wait();
  resolve_pack_fast(a, gridDim.x, blockIdx.x, rp_smem);
}

#ifndef GLEAM_DEDUP_MINBLOCKS
#define GLEAM_DEDUP_MINBLOCKS 3
#endif
// three co-resident blocks per SM (at most 85 registers): the resolve kernel's
// phases are chains of round trips that want every thread of the grid
__global__ void __launch_bounds__(kThreads, GLEAM_DEDUP_MINBLOCKS) k_dedup(DedupArgs a) {
  pdl_trigger();
  pdl_wait();
  resolve_rank(a, gridDim.x, blockIdx.x);
}

__global__ void GLEAM_PACK_BOUNDS k_pack(DedupArgs a) {
  extern __shared__ __align__(128) uint8_t pack_smem[];
  pdl_trigger();
  pdl_wait();
  pack_publish(a, gridDim.x, blockIdx.x, pack_smem);
}

// A whole small call in one block: the staged hash of its chunks (kThreads / 4
// at a time), then the resolution and ranks, then the copies, inserts and
// publish, separated by block barriers instead of kernel boundaries and grid
// barriers.  The pack reuses the shared memory of the hash stages.
constexpr uint32_t kSmallGroups = kThreads / 4;
constexpr uint32_t kSmallHashSmem = kSmallGroups * (uint32_t)kGroupBytes;
constexpr uint32_t kSmallSmem = kSmallHashSmem > kPackSmem ? kSmallHashSmem : kPackSmem;


// k_dedup's and k_pack's steps on a grid of one block (several payloads, LRU,
// a class table, or more chunks than threads): out of line, so that the small
// kernel's common path stays compact.
__device__ __noinline__ void small_call_general(const DedupArgs& a, uint8_t* smem) {
  resolve_rank(a, 1, 0);
  __syncthreads();
  pack_publish(a, 1, 0, smem);
}

template <bool kAhead, bool kPrefixAsync>
__global__ void __launch_bounds__(kThreads) k_small_call(HashArgs h, DedupArgs a) {
  extern __shared__ __align__(128) uint8_t small_smem[];
  pdl_trigger();
  if (!h.wait_late) pdl_wait();  // else in staged_range, before the first probe
  // Device-resident payloads (16-byte aligned here) are prefetched into L2 at
  // once, lane p taking payload p in 16 KiB pieces, so that the hash stages
  // wait for L2 rather than HBM.
  constexpr uint32_t kPiece = 16u << 10;
  if (!a.plain_copy && a.count <= 32 && threadIdx.x < a.count) {
    const PayloadDesc& P = desc(a, threadIdx.x);
    const unsigned long long nb = P.n & ~15ull;
    for (unsigned long long off = 0; off < nb; off += kPiece)
      prefetch_l2(P.buf + off, (uint32_t)min((unsigned long long)kPiece, nb - off));
  }
  const unsigned long long nvb = (h.Ntot * 4 + kThreads - 1) / kThreads;
  for (unsigned long long vb = 0; vb < nvb; ++vb) {
    __syncthreads();  // the previous range's groups are done with the shared memory
    staged_range<true, kAhead, true, kPrefixAsync>(h, vb, small_smem);
  }
  __syncthreads();  // every chunk's probe outcome written (and its stage copies landed)
  if (a.count == 1 && !a.lru && !a.classes && a.Ntot <= (unsigned long long)kThreads) {
    // one payload of at most one chunk per thread: the one-launch path's
    // steps, which for a call without duplicates rank the misses by a block
    // scan (no LRU: they stamp no last use)
    resolve_pack_fast(a, 1, 0, small_smem);
  } else {
    small_call_general(a, small_smem);
  }
}

// One warp per record: does the block still hold the recorded chunk's bytes?
__global__ void __launch_bounds__(kThreads) k_block_check(BlockCheckArgs a) {
  const uint32_t lane = threadIdx.x & 31;
  const unsigned long long warp = ((unsigned long long)blockIdx.x * kThreads + threadIdx.x) >> 5;
  const unsigned long long nwarps = ((unsigned long long)gridDim.x * kThreads) >> 5;
  const unsigned long long used = a.dstats[ST_SLOTS_USED];
  uint32_t bad = 0;
  for (unsigned long long r = warp; r < a.nrec; r += nwarps) {
    const unsigned long long off = a.offsets[r];
    const uint32_t slot = a.slots[r];
    bool differs = true;
    if (slot < used) {
      const uint32_t len = a.slot_len[slot];
      if (off <= a.block_bytes && len <= a.block_bytes - off) {
        const uint8_t* x = a.block + off;
        const uint8_t* y = a.arena + (unsigned long long)slot * a.C;
        const bool vec = (((uintptr_t)x | (uintptr_t)y) & 15) == 0;
        differs = !warp_equal(x, y, len, vec);
      }
    }
    if (lane == 0) {
      if (a.mismatch) a.mismatch[r] = differs ? 1 : 0;
      bad += differs;
    }
  }
  if (lane == 0 && bad) atomicAdd(a.count, (unsigned long long)bad);
}

__global__ void k_debug_insert(IndexEntry* index, uint64_t index_mask, uint32_t* slot_len,
                               unsigned long long* slot_key, unsigned long long* dstats,
                               unsigned long long key, uint32_t slot, uint32_t len, DevCtl* ctl,
                               uint32_t* last_use, uint32_t epoch) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  if (!index_insert(index, index_mask, key, slot, len)) {
    ctl->err = GLEAM_ERR_INTERNAL;
    return;
  }
  slot_len[slot] = len;
  slot_key[slot] = key;
  if (last_use) last_use[slot] = epoch;
  dstats[ST_SLOTS_USED] = (unsigned long long)slot + 1;
  dstats[ST_INSERTS] += 1;
  dstats[ST_BYTES_USED] += len;
}

// ---- GLEAM_DEBUG_CHECKS --------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_check_entries(IndexCheckArgs a) {
  const unsigned long long used = a.dstats[ST_SLOTS_USED];
  const unsigned long long n = a.index_mask + 1;
  bool bad = false;
  for (unsigned long long q = (unsigned long long)blockIdx.x * kThreads + threadIdx.x; q < n;
       q += (unsigned long long)gridDim.x * kThreads) {
    const IndexEntry e = a.index[q];
    if (e.slot != kEmptySlot) {
      if (e.slot >= used || e.len != a.slot_len[e.slot]) bad = true;
      else atomicAdd(&a.count[e.slot], 1u);
    }
    const IndexEntry h = a.hints[q];
    if (h.slot != kEmptySlot && (h.slot >= used || h.len != a.slot_len[h.slot])) bad = true;
  }
  if (bad) atomicExch(a.flag, 1u);
}

__global__ void __launch_bounds__(kThreads) k_check_slots(IndexCheckArgs a) {
  const unsigned long long used = a.dstats[ST_SLOTS_USED];
  bool bad = false;
  for (unsigned long long sl = (unsigned long long)blockIdx.x * kThreads + threadIdx.x; sl < used;
       sl += (unsigned long long)gridDim.x * kThreads) {
    bad |= a.count[sl] != 1u;
    a.count[sl] = 0u;
  }
  if (bad) atomicExch(a.flag, 1u);
}

__global__ void k_check_publish(IndexCheckArgs a) {
  if (*(volatile uint32_t*)a.flag == 0u) return;
  for (uint32_t p = threadIdx.x; p < a.npayloads; p += blockDim.x) {
    gleam_result_t* r = a.npayloads > 1 ? a.table[p].result : a.one.result;
    if (r) r->status = GLEAM_ERR_INTERNAL;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    a.total->status = GLEAM_ERR_INTERNAL;
    *a.flag = 0u;
  }
}

}  // namespace

cudaError_t launch_index_check(const IndexCheckArgs& a, cudaStream_t s) {
  const unsigned grid = 1024;
  k_check_entries<<<grid, kThreads, 0, s>>>(a);
  k_check_slots<<<grid, kThreads, 0, s>>>(a);
  k_check_publish<<<1, kThreads, 0, s>>>(a);
  return cudaGetLastError();
}

int dedup_threads() { return kThreads; }

int dedup_chunks_per_block() { return GLEAM_DEDUP_CHUNKS_PER_BLOCK; }

// Co-resident blocks per SM of the pack kernel.
int pack_blocks_per_sm() {
  int nb = 0;
  if (kPackSmem > 48 * 1024 &&
      cudaFuncSetAttribute((const void*)k_pack, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           kPackSmem) != cudaSuccess)
    return 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k_pack, kThreads, kPackSmem) !=
      cudaSuccess)
    return 0;
  return nb;
}

// Co-resident blocks per SM of the one-launch resolve + pack kernel (its grid
// barriers need every block of the grid resident at once).
int resolve_pack_blocks_per_sm() {
  int nb = 0;
  if (cudaFuncSetAttribute((const void*)k_resolve_pack, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           kResolvePackSmem) != cudaSuccess)
    return 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k_resolve_pack, kThreads,
                                                    kResolvePackSmem) != cudaSuccess)
    return 0;
  return nb;
}

// Co-resident blocks per SM for the cooperative launch (capped).
int dedup_blocks_per_sm() {
  int nb = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k_dedup, kThreads, 0) != cudaSuccess)
    return 0;
  return nb < GLEAM_DEDUP_BLOCKS_PER_SM ? nb : GLEAM_DEDUP_BLOCKS_PER_SM;
}

cudaError_t launch_dedup(const DedupArgs& a, int grid, int pack_grid, cudaStream_t s, bool pdl) {
  cudaError_t e;
  if (pdl) {
    e = launch_kernel(k_dedup, dim3(grid), dim3(kThreads), 0, s, true, a);
  } else {
    DedupArgs copy = a;
    void* args[] = {&copy};
    e = cudaLaunchCooperativeKernel((void*)k_dedup, dim3(grid), dim3(kThreads), args, 0, s);
  }
  if (e != cudaSuccess) return e;
  if (kPackSmem > 48 * 1024)
    cudaFuncSetAttribute((const void*)k_pack, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         kPackSmem);
  return launch_kernel(k_pack, dim3(pack_grid), dim3(kThreads), kPackSmem, s, pdl, a);
}

cudaError_t launch_resolve_pack(const DedupArgs& a, int grid, cudaStream_t s) {
  cudaFuncSetAttribute((const void*)k_resolve_pack, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       kResolvePackSmem);
  return launch_kernel(k_resolve_pack, dim3(grid), dim3(kThreads), kResolvePackSmem, s, true, a);
}

uint32_t small_call_groups() { return kSmallGroups; }

template <bool kAhead, bool kPrefixAsync>
cudaError_t launch_small(const HashArgs& h, const DedupArgs& a, cudaStream_t s, bool pdl) {
  cudaFuncSetAttribute((const void*)k_small_call<kAhead, kPrefixAsync>,
                       cudaFuncAttributeMaxDynamicSharedMemorySize, kSmallSmem);
  return launch_kernel(k_small_call<kAhead, kPrefixAsync>, dim3(1), dim3(kThreads), kSmallSmem, s,
                       pdl, h, a);
}

cudaError_t launch_small_call(const HashArgs& h, const DedupArgs& a, cudaStream_t s, bool pdl) {
  if (h.C <= kPrefixAsyncMaxChunk)
    return h.spec_mode ? launch_small<true, true>(h, a, s, pdl)
                       : launch_small<false, true>(h, a, s, pdl);
  return h.spec_mode ? launch_small<true, false>(h, a, s, pdl)
                     : launch_small<false, false>(h, a, s, pdl);
}

cudaError_t launch_block_check(const BlockCheckArgs& a, cudaStream_t s) {
  if (a.nrec == 0) return cudaSuccess;
  const unsigned long long warps = a.nrec < (1ull << 20) ? a.nrec : (1ull << 20);
  const unsigned grid = (unsigned)((warps * 32 + kThreads - 1) / kThreads);
  k_block_check<<<grid, kThreads, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_debug_insert(IndexEntry* index, uint64_t index_mask, uint32_t* slot_len,
                                unsigned long long* slot_key, unsigned long long* dstats,
                                unsigned long long key, uint32_t slot, uint32_t len, DevCtl* ctl,
                                uint32_t* last_use, uint32_t epoch, cudaStream_t s) {
  k_debug_insert<<<1, 32, 0, s>>>(index, index_mask, slot_len, slot_key, dstats, key, slot, len,
                                  ctl, last_use, epoch);
  return cudaGetLastError();
}

}  // namespace gleam
