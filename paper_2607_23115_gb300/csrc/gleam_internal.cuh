// Internal types and device helpers of libgleam (not part of the C ABI).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "gleam.h"

namespace gleam {

// ---------------------------------------------------------------------------
// Device data layout
// ---------------------------------------------------------------------------

constexpr uint32_t kEmptySlot = 0xFFFFFFFFu;
// A removed entry while an eviction rebuilds its cluster; no table holds one
// between calls.
constexpr uint32_t kTombSlot = 0xFFFFFFFEu;

// One entry of the cache index: open addressing, linear probing, load <= 1/2.
// An entry is free iff slot == kEmptySlot; key/len are valid once the insert
// kernel that claimed it has finished.
struct __align__(16) IndexEntry {
  unsigned long long key;  // XXH64 of the stored chunk (low 16 bits in KEY16 mode)
  uint32_t slot;           // arena slot holding the bytes
  uint32_t len;            // true length of the stored chunk
};

// One entry of the per-call group table used to find the first occurrence of
// each distinct chunk inside a call.  owner = 1 + index of the chunk that
// claimed the entry (0 = free); minv = ~(smallest unresolved chunk index of
// the group) so that a zero-filled table means "no minimum yet".
struct __align__(8) CallEntry {
  uint32_t owner;
  uint32_t minv;
};

// One entry of the per-call table of (16-bit index key, length) classes
// (KEY16 with XXH64 keys), over the call's misses: owner and minv as in
// CallEntry; count = misses of the class so far, so that each miss gets its
// own place (0, 1, ...) in the run of index entries that the class's misses
// occupy from the key's home position on.
struct __align__(16) ClassEntry {
  uint32_t owner;
  uint32_t minv;
  uint32_t count;
  uint32_t pad;
};

// Per-chunk outcome of the probe/verify kernel.
enum : uint8_t { kMissNoCand = 0, kMissCand = 1, kHit0 = 2, kUncached = 3 };

// Per-chunk resolution word of the dedup kernel.
constexpr uint32_t kResUnresolved = 0;
constexpr uint32_t kResHit0 = 0x20000000u;     // byte-equal to a cached chunk
constexpr uint32_t kResDup = 0x40000000u;      // byte-equal to an earlier miss
constexpr uint32_t kResLeader = 0x80000000u;   // | round in which it was resolved
constexpr uint32_t kResNoSlot = 0x10000000u;   // a miss that is never cached
constexpr uint32_t kResReject = 0x08000000u;   // a miss that had a key+length candidate
constexpr uint32_t kResRoundMask = 0x07FFFFFFu;

// Device counters of one cache, in gleam_stats_t order (the fields that
// change; capacity, slot count and chunk size are host constants).
enum StatIdx {
  ST_CALLS = 0, ST_CHUNKS, ST_HITS_CACHE, ST_HITS_INTRA, ST_MISSES, ST_INSERTS,
  ST_REJECTS, ST_SLOTS_USED, ST_BYTES_USED, ST_EVICTIONS, ST_SPEC_CHUNKS, ST_COUNT
};

// Per-call control block; starts zeroed and every dedup kernel leaves it zeroed.
struct DevCtl {
  unsigned int bar_count;  // grid-barrier arrivals of the call (nblocks per barrier)
  unsigned int copy_next;  // next piece to hand out (one-launch resolve + pack copies)
  int err;
  unsigned int done;
  unsigned int unres[3];
  unsigned int shared_groups;  // a chunk found its (key, length) group claimed by another
  unsigned long long acc_hits_cache;
  unsigned long long acc_hits_intra;
  unsigned long long acc_rejects;
  unsigned long long acc_misses;
  unsigned long long acc_miss_bytes;
  unsigned long long acc_stored;
  unsigned long long acc_stored_bytes;
  // LRU eviction (caches created with GLEAM_EVICT_LRU)
  unsigned long long acc_distinct;      // distinct cached slots hit by the call
  unsigned long long evict_k;           // slots the call evicts
  unsigned long long lru_below;         // candidates older than the cut-off bin / stamp
  unsigned long long lru_ties;          // candidates at the cut-off stamp to evict
  unsigned long long acc_victim_bytes;  // stored bytes of the evicted slots
  unsigned int lru_hi;                  // high 16 bits of the cut-off stamp
  unsigned int lru_cut;                 // the cut-off stamp
  // write-through of likely misses (HashArgs::spec_mode)
  unsigned long long spec_tried;        // chunks the hash kernel wrote ahead
  unsigned long long spec_used;         // misses whose copies that made unnecessary
};

// Position of a key in a power-of-two table: the 64-bit finaliser of
// MurmurHash3 (Appleby), so that 16-bit test keys spread as well as full ones.
__host__ __device__ __forceinline__ unsigned long long mix64(unsigned long long k) {
  k ^= k >> 33;
  k *= 0xff51afd7ed558ccdULL;
  k ^= k >> 33;
  k *= 0xc4ceb9fe1a85ec53ULL;
  k ^= k >> 33;
  return k;
}

// ---------------------------------------------------------------------------
// Kernel argument blocks and launchers (defined in the kernel TUs)
// ---------------------------------------------------------------------------

// One payload of a call (a batch of calls has one per payload), as the
// device sees it.  Chunks of all payloads are numbered consecutively:
// payload p owns global chunks [chunk_base, chunk_base + nchunks).
struct __align__(16) PayloadDesc {
  const uint8_t* buf;
  unsigned long long n;
  unsigned long long chunk_base;
  unsigned long long nchunks;
  uint32_t* mask;
  uint32_t* miss_idx;
  uint8_t* packed;
  gleam_result_t* result;  // may be null
  uint32_t* chunk_slot;    // may be null: slot holding each chunk's bytes
};

// Per-chunk workspace, indexed by global chunk number.
struct ChunkArrays {
  uint8_t* status;           // kHit0 / kMissCand / kMissNoCand
  unsigned long long* key;   // group key: the whole XXH64 (also in KEY16 mode, whose
                             // index key is its low 16 bits), or the paper's key
  uint32_t* len;             // true length
  unsigned long long* src;   // device address of the chunk's first byte
  uint32_t* pidx;            // payload number
  uint32_t* res;             // resolution word (kRes*)
  uint32_t* ent;             // cache hit: matched slot; else group-table entry, and
                             // the leader's number once a duplicate
  uint32_t* rank;            // exclusive count of misses before the chunk
  unsigned long long* hint;  // prefix hint (chunks of at least kPrefixBytes)
  uint32_t* order;           // order[r] = chunk number of the miss of rank r
  uint32_t* srank;           // exclusive count of stored (cached) misses before the chunk
  uint32_t* old;             // LRU: last use of a hit's slot before this call stamped it
  uint8_t* spec;             // 1: the hash kernel wrote the chunk to packed offset
                             // i*C of its payload and to arena slot slots_used + g
  unsigned long long* cls;   // KEY16, a miss: its entry in the per-call class table (low
                             // 32 bits) and its place among the class's misses (high 32)
};

// Speculative verify.  After the first kPrefixBytes of a chunk the four XXH64
// lane accumulators are folded into a 64-bit prefix hint; a second table
// (same layout as the index, key = hint) maps it to the slot of a cached chunk
// that began with the same bytes.  The rest of the chunk is then hashed and
// compared against that slot in the same pass, so a hit reads the payload
// once.  The hint only chooses what to compare against: a chunk is a hit only
// if the index (keyed by the full XXH64) lists the slot, and every other
// key+length candidate is still compared byte for byte.
constexpr uint32_t kPrefixBytes = 512;

struct HashArgs {
  const PayloadDesc* table;  // count > 1
  PayloadDesc one;           // count == 1
  uint32_t count;
  unsigned long long Ntot;   // chunks of all payloads
  unsigned long long C;      // chunk length (bytes)
  unsigned long long* fp_out;  // optional: XXH64 per chunk
  // probe + verify (index == nullptr: fingerprint only)
  const IndexEntry* index;
  unsigned long long index_mask;
  const IndexEntry* hints;   // prefix-hint table (same size as the index)
  const uint8_t* arena;
  const unsigned long long* slot_key;  // per slot: the stored chunk's whole fingerprint
  const unsigned long long* dstats;
  uint32_t key16;
  uint32_t paper;            // GLEAM_PAPER_IDS: MD5-prefix keys, small chunks uncached
  ChunkArrays ch;
  DevCtl* ctl;
  // write-through of likely misses (the host launches the variant of the
  // staged hash that does it when spec_mode is 1): a chunk of at least
  // kPrefixBytes with no prefix-hint match is written to its packed offset and
  // to arena slot slots_used + g as it streams by
  uint32_t spec_mode;
  uint8_t* arena_w;                // the arena, for those writes
  // the host knows the cache holds no chunk, or (chunks of at most
  // kHintedMaxChunk) so few against the call's chunks (fewer than one per
  // kHintedMinRatio) that the prefix-hinted verify would rarely find a copy to
  // stream: the kernel variant without it (and without its stage buffers, so
  // twice the groups per SM) runs, and every key+length candidate is compared
  // after the probe, which costs a larger chunk two more reads of its bytes
  // (KEY16 adversarial payloads with 64 cached entries: 1 KiB chunks +13%,
  // 64 KiB chunks -7% when they too took this variant)
  uint32_t no_hints;
  unsigned long long nslots;
  // Calls that overlap (GLEAM_OVERLAP_CALLS): the kernel was launched while the
  // cache's previous call may still be running, and waits for it only before
  // it probes the index.  Until then it reads the payload and, for the
  // speculative verify, the hint table and arena bytes of the slots counted as
  // used when it started, which no later call changes (no eviction).
  uint32_t wait_late;
  // Calls resolved by the one-launch kernel on more than one block (one
  // payload): the staged hash kernel claims each miss's entry in the per-call
  // group table as it records the chunk (ent and res as the resolve kernel
  // would set them; the entry's minv holds a tag of the chunk's (group key,
  // length) until the resolve kernel frees it; shared_groups if an entry with
  // the same tag was found), so that the resolve kernel needs no claims and
  // no barrier before its ranks.  Null: no claims here.
  CallEntry* claim_tbl;
  unsigned long long claim_mask;
};

struct DedupArgs {
  const PayloadDesc* table;
  PayloadDesc one;
  uint32_t count;
  unsigned long long Ntot;
  unsigned long long C;
  uint8_t* arena;
  IndexEntry* index;
  unsigned long long index_mask;
  IndexEntry* hints;
  unsigned long long nslots;
  uint32_t* slot_len;
  unsigned long long* slot_key;  // per slot: the group key of the stored chunk
  unsigned long long* dstats;
  ChunkArrays ch;
  uint32_t* pstart;          // per payload: misses before its first chunk
  CallEntry* tbl;
  unsigned long long tbl_mask;
  uint32_t* bcount;
  DevCtl* ctl;
  gleam_result_t* total;     // result of the whole call (never null)
  unsigned long long ncalls; // payloads with n > 0
  unsigned long long wait_ns;
  int skip_block;
  uint32_t paper;            // no prefix hints are kept in GLEAM_PAPER_IDS mode
  uint32_t key16;            // GLEAM_KEY16: index key = low 16 bits of the group key
  // KEY16 with XXH64 keys: chunks are grouped by their whole fingerprint, so a
  // miss's verify rejects inside the call (an earlier miss with the same
  // 16-bit key and length) come from this second per-call table of (16-bit
  // key, length) classes, each holding its smallest miss and its miss count
  uint32_t classes;
  ClassEntry* cls_tbl;       // KEY16 classes: as many entries as tbl
  uint32_t plain_copy;       // copy misses with loads and stores, not bulk copies
                             // (payloads or outputs in host or managed memory)
  // LRU eviction (GLEAM_EVICT_LRU; lru == 0: the other fields are unused)
  uint32_t lru;
  uint32_t epoch;            // this call's clock value
  uint32_t* last_use;        // per slot: clock value of its last use
  uint8_t* vflag;            // per slot: evicted by this call (zero between calls)
  uint32_t* victims;         // evicted slots in ascending order
  uint32_t* bins;            // 65536-bin histogram (zero between calls)
  // write-through: spec_active = the hash kernel of this call did it (ch.spec
  // is valid); feedback of the automatic mode: spec_state[0] = on, [1] = calls
  // since it went off (null: no feedback), and a copy of [0] in page-locked
  // host memory that the host reads when it launches the next call
  uint32_t spec_active;
  uint32_t* spec_state;
  uint32_t* spec_mirror;
  // the hash kernel claimed the misses' groups (HashArgs::claim_tbl)
  uint32_t pre_claimed;
  // one-launch resolve + pack: pieces of misses a warp takes at a time from a
  // counter of the call (1..32), or 0 for an equal share per warp
  uint32_t copy_grab;
};

constexpr uint32_t kLruBins = 65536;

// Paper-identifier mode (App. B.1): chunks shorter than this get no entry.
constexpr uint32_t kPaperMinCached = 1024;

// pdl: launched with programmatic stream serialization (the kernel waits on the
// GPU for the one before it; see pdl_trigger/pdl_wait).
constexpr unsigned long long kHintedMinRatio = 16;
constexpr unsigned long long kHintedMaxChunk = 4096;
cudaError_t launch_hash(const HashArgs& a, bool aligned, cudaStream_t s, bool pdl = false);
// Whether launch_hash runs the staged XXH64 kernel for these arguments (the
// one that can claim groups, HashArgs::claim_tbl).
bool hash_is_staged(const HashArgs& a, bool aligned);
// Loads the hash kernels' device code on the current GPU (cache creation does
// it, so that no later call loads code, which allocates device memory).
cudaError_t load_hash_kernels();
// The cooperative resolve/rank kernel on `grid` blocks, then the pack kernel
// (masks, indices, copies, inserts, publish) on `pack_grid` blocks.  pdl: both
// launched with programmatic stream serialization, the resolve kernel then as
// a regular launch (a cooperative one is never launched early); its grid must
// fit the GPU at once, and every block of it is resident before anything
// later on the stream can start, so its grid barriers still complete.
cudaError_t launch_dedup(const DedupArgs& a, int grid, int pack_grid, cudaStream_t s,
                         bool pdl = false);
// Resolve, rank, pack and publish of a one-payload call in one launch on
// `grid` blocks (see k_resolve_pack), with programmatic stream serialization.
cudaError_t launch_resolve_pack(const DedupArgs& a, int grid, cudaStream_t s);
// A whole call (hash, resolve and rank, pack) as one single-block kernel, for
// calls with few chunks whose payloads suit the staged hash (16-byte aligned)
// outside GLEAM_PAPER_IDS mode; the block hashes small_call_groups() chunks at
// a time.
cudaError_t launch_small_call(const HashArgs& h, const DedupArgs& a, cudaStream_t s,
                              bool pdl = false);
uint32_t small_call_groups();
cudaError_t launch_debug_insert(IndexEntry* index, uint64_t index_mask, uint32_t* slot_len,
                                unsigned long long* slot_key, unsigned long long* dstats,
                                unsigned long long key, uint32_t slot, uint32_t len, DevCtl* ctl,
                                uint32_t* last_use, uint32_t epoch, cudaStream_t s);
struct BlockCheckArgs {
  const uint8_t* block;
  unsigned long long block_bytes;
  const unsigned long long* offsets;
  const uint32_t* slots;
  unsigned long long nrec;
  uint8_t* mismatch;             // may be null
  unsigned long long* count;
  const uint8_t* arena;
  const uint32_t* slot_len;
  const unsigned long long* dstats;
  unsigned long long C;
};

cudaError_t launch_block_check(const BlockCheckArgs& a, cudaStream_t s);

// GLEAM_DEBUG_CHECKS: after a call, every index entry must name a used slot
// with its recorded length, every used slot must be named by exactly one
// index entry, and every hint entry must name a used slot of its length; a
// violation turns the call's statuses into GLEAM_ERR_INTERNAL.
struct IndexCheckArgs {
  const IndexEntry* index;
  const IndexEntry* hints;
  unsigned long long index_mask;
  const uint32_t* slot_len;
  const unsigned long long* dstats;
  uint32_t* count;           // per slot, zero between checks
  uint32_t* flag;            // zero between checks
  const PayloadDesc* table;  // the call's payloads (count > 1), or `one`
  PayloadDesc one;
  uint32_t npayloads;
  gleam_result_t* total;
};
cudaError_t launch_index_check(const IndexCheckArgs& a, cudaStream_t s);
int dedup_threads();
int dedup_chunks_per_block();
int dedup_blocks_per_sm();
int pack_blocks_per_sm();
int resolve_pack_blocks_per_sm();

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------

#ifdef __CUDACC__

__device__ __forceinline__ unsigned long long globaltimer_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ unsigned int ld_acquire_u32(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ int ld_volatile_s32(const int* p) {
  return *reinterpret_cast<const volatile int*>(p);
}

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// Programmatic dependent launch.  Every hot kernel lets the next kernel of its
// stream be launched as soon as all of its blocks have started (the next
// kernel's blocks then wait on the GPU instead of behind a launch), and waits
// for the kernel before it to finish, with its memory visible, before it
// touches anything that kernel may write.  Both are no-ops for a kernel
// launched without the attribute (or one whose predecessor is not a kernel).
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Grid-wide barrier for a cooperative launch.  Every wait is bounded by
// `wait_ns`: a block that gives up records GLEAM_ERR_TIMEOUT and every block
// then leaves through its epilogue.  `skip` makes the calling block leave
// without arriving (test hook for the bounded wait).  Returns true if the
// whole grid arrived and no error is recorded.  A grid of one block has no
// one to wait for: the block barrier orders its memory accesses, and it
// returns !skip without reading the error word (a caller about to make a
// change that an error must prevent reads it itself).
__device__ __forceinline__ bool grid_barrier(DevCtl* ctl, unsigned int nblocks,
                                             unsigned long long wait_ns, bool skip) {
  __shared__ int s_ok;  // the block's verdict, so that every thread agrees
  __syncthreads();
  if (nblocks == 1) return !skip;
  if (threadIdx.x == 0 && !skip) {
    // arrivals only grow during a call: this barrier is passed once the
    // count reaches the next multiple of nblocks (no reset, no second flag)
    __threadfence();
    const unsigned int arrived = atomicAdd(&ctl->bar_count, 1u);
    const unsigned int target = (arrived / nblocks + 1) * nblocks;
    if (arrived + 1 != target) {
      const unsigned long long t0 = globaltimer_ns();
      while (ld_acquire_u32(&ctl->bar_count) < target) {
        if (ld_volatile_s32(&ctl->err) != 0) break;
        if (globaltimer_ns() - t0 > wait_ns) {
          atomicCAS(&ctl->err, 0, (int)GLEAM_ERR_TIMEOUT);
          break;
        }
        __nanosleep(32);
      }
    }
    __threadfence();
  }
  if (threadIdx.x == 0) s_ok = (!skip && ld_volatile_s32(&ctl->err) == 0) ? 1 : 0;
  __syncthreads();
  return s_ok != 0;
}

// Payload owning global chunk g: the last p with chunk_base <= g (empty
// payloads share their base with the next one and are never chosen).
__device__ __forceinline__ uint32_t find_payload(const PayloadDesc* table, uint32_t count,
                                                 unsigned long long g) {
  uint32_t lo = 0, hi = count;
  while (hi - lo > 1) {
    const uint32_t mid = (lo + hi) >> 1;
    if (__ldg(&table[mid].chunk_base) <= g) lo = mid;
    else hi = mid;
  }
  return lo;
}

// The last p in [lo, hi) with chunk_base <= g, given table[lo].chunk_base <= g.
__device__ __forceinline__ uint32_t find_payload_in(const PayloadDesc* table, uint32_t lo,
                                                    uint32_t hi, unsigned long long g) {
  while (hi - lo > 1) {
    const uint32_t mid = (lo + hi) >> 1;
    if (__ldg(&table[mid].chunk_base) <= g) lo = mid;
    else hi = mid;
  }
  return lo;
}

// Payload owning chunk g, for a block whose threads handle consecutive chunks
// starting at g0 (g >= g0).  Warp 0 finds g0's payload with a 32-way search
// (32 independent loads per step, about log32(count) steps instead of
// log2(count) dependent ones) and stages the chunk bases of the 32 payloads
// from there in shared memory, where every thread then finds its own; a chunk
// past them falls back to bisection.  Every thread of the block must call it.
// scratch: 33 words of shared memory, free again when the call returns.
__device__ __forceinline__ uint32_t block_find_payload(const PayloadDesc* table, uint32_t count,
                                                       unsigned long long g0,
                                                       unsigned long long g,
                                                       unsigned long long* scratch) {
  unsigned long long* s_base = scratch;
  unsigned long long* s_p0 = scratch + 32;
  if (threadIdx.x < 32) {
    const uint32_t lane = threadIdx.x;
    // table[lo].chunk_base <= g0; hi == count or its base > g0.  Narrowed
    // until the 32-entry window at lo holds g0's payload (one round for up
    // to 1,024 payloads), not to one entry: the window load settles the rest.
    uint32_t lo = 0, hi = count;
    while (hi - lo > 32) {
      const uint32_t span = hi - lo;
      const uint32_t q = lo + 1 + (uint32_t)(((unsigned long long)(span - 1) * lane) >> 5);
      const unsigned m = __ballot_sync(0xffffffffu, __ldg(&table[q].chunk_base) <= g0);
      if (m == 0) {
        hi = lo + 1;
      } else {
        const int L = 31 - __clz(m);  // pivots grow with the lane, so m is a prefix
        const uint32_t qL = __shfl_sync(0xffffffffu, q, L);
        const uint32_t qN = __shfl_sync(0xffffffffu, q, L < 31 ? L + 1 : 31);
        lo = qL;
        if (L < 31) hi = qN;
      }
    }
    s_base[lane] = lo + lane < count ? __ldg(&table[lo + lane].chunk_base) : ~0ull;
    if (lane == 0) *s_p0 = lo;
  }
  __syncthreads();
  uint32_t lo = 0, hi = 32;
  while (hi - lo > 1) {
    const uint32_t mid = (lo + hi) >> 1;
    if (s_base[mid] <= g) lo = mid;
    else hi = mid;
  }
  const uint32_t p0 = (uint32_t)*s_p0;
  __syncthreads();  // the scratch may be reused from here on
  if (lo == 31 && p0 + 32 < count && __ldg(&table[p0 + 32].chunk_base) <= g)
    return find_payload_in(table, p0 + 32, count, g);
  return p0 + lo;
}

// Launches kern<<<grid, block, smem, s>>>(args...), with programmatic stream
// serialization when pdl is set.
template <typename... Params, typename... Args>
cudaError_t launch_kernel(void (*kern)(Params...), dim3 grid, dim3 block, size_t smem,
                          cudaStream_t s, bool pdl, Args&&... args) {
  if (!pdl) {
    kern<<<grid, block, smem, s>>>(static_cast<Args&&>(args)...);
    return cudaGetLastError();
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

#endif  // __CUDACC__

}  // namespace gleam
