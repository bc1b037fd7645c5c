/*
 * gleam.h -- C ABI of libgleam.so, the GB300 (sm_103a) chunk-dedup library.
 *
 * The operation (paper Sec. 4.1.2, "Hash-based Weight Chunk Retrieval"): before
 * a host-to-device cudaMemcpy payload crosses the network, the payload is
 * identified by hash against the set of chunks already resident on the
 * server; a resident chunk is replaced by (hash, size) metadata and only the
 * others travel in full, after which they are resident too.  App. B.1 ("Hash
 * Cost and Collision") describes the paper's own identifier (MD5 of a 128-byte
 * prefix, no byte check).  This library generalises it: every fixed C-byte
 * chunk is identified by XXH64 (seed 0) over its whole length, looked up in a
 * device-resident open-addressing index, and every key match is confirmed
 * byte for byte against the cached copy, so a hash collision can never make
 * two different chunks alias.
 *
 * Conventions shared by every call:
 *  - Plain C types only.  A "device pointer" is memory the calling process
 *    allocated on the cache's GPU (cudaMalloc, cudaMallocAsync or managed
 *    memory); host pointers are rejected with GLEAM_ERR_NOT_DEVICE_PTR.
 *  - The caller owns every buffer it passes.  The library owns the cache's
 *    arena, index and per-call workspace, allocated on the GPU that was
 *    current when the cache was created.
 *  - Errors are negative return values (enum gleam_status).  A call that
 *    returns an error other than GLEAM_ERR_CUDA leaves the cache unchanged.
 *  - Chunk i of an n-byte payload covers bytes [i*C, min(n, (i+1)*C)); the last
 *    chunk keeps its true length, and length is part of chunk equality.
 */
#ifndef GLEAM_H
#define GLEAM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A CUDA stream handle (ABI-identical to cudaStream_t).  NULL means the legacy
 * default stream, which orders against every blocking stream like cudaMemcpy. */
typedef struct CUstream_st* gleam_stream_t;

/* Opaque weight cache: device arena of fixed C-byte slots, device index, stats. */
typedef struct gleam_cache gleam_cache_t;

/* Opaque device-side copy of a cache's index and counters (test/bench helper). */
typedef struct gleam_snapshot gleam_snapshot_t;

enum gleam_status {
  GLEAM_OK = 0,
  GLEAM_ERR_INVALID_ARG = -1,   /* NULL handle/pointer, bad sizes, bad flags   */
  GLEAM_ERR_NOT_DEVICE_PTR = -2,/* a buffer is not device memory of this GPU  */
  GLEAM_ERR_CUDA = -3,          /* a CUDA runtime call failed                 */
  GLEAM_ERR_CAPACITY = -4,      /* misses do not fit the free (or, with
                                   GLEAM_EVICT_LRU, the evictable) slots      */
  GLEAM_ERR_TIMEOUT = -5,       /* a bounded device-side wait ran out         */
  GLEAM_ERR_NOMEM = -6,         /* device allocation failed                   */
  GLEAM_ERR_INTERNAL = -7       /* a device-side consistency check failed     */
};

/* Flags for gleam_cache_create_ex. */
#define GLEAM_KEY16 0x1u        /* test mode: index key = low 16 bits of XXH64,
                                   so unrelated chunks collide and every hit
                                   must be separated from them by the verify */
#define GLEAM_DEBUG_CHECKS 0x2u /* after every dedup call, check on the device
                                   that each index entry names a used slot of
                                   its recorded length, that each used slot has
                                   exactly one index entry, and that each hint
                                   entry names a used slot of its length; a
                                   violation makes the call's statuses (and the
                                   synchronous return) GLEAM_ERR_INTERNAL.  Costs
                                   a pass over the index and 4 bytes per slot. */
#define GLEAM_PAPER_IDS 0x4u    /* the paper's own identifier (App. B.1): the
                                   index key is MD5 of a chunk's first
                                   min(len, 128) bytes (first 8 digest bytes,
                                   little-endian) instead of XXH64 of the whole
                                   chunk, and chunks under 1024 bytes are
                                   recorded but never cached: always misses,
                                   given no slot, never deduplicated.  Every
                                   key match is still verified byte for byte. */
#define GLEAM_EVICT_LRU 0x8u    /* paper Sec. 4.1.3: when a call's misses do not
                                   fit the never-used slots, evict the least
                                   recently used slots that the call did not
                                   hit (last use = the latest call that hit or
                                   filled the slot; ties: lower slot first),
                                   instead of failing with GLEAM_ERR_CAPACITY.
                                   A batch is one call for this.  Costs 9 bytes
                                   of device memory per slot. */
#define GLEAM_OVERLAP_CALLS 0x10u /* consecutive calls of the cache on one
                                   stream may overlap on the GPU: a call of up
                                   to 8192 chunks fingerprints its payload
                                   while the calls before it are still running
                                   and waits for them (on the GPU, by
                                   programmatic dependent launch) only before
                                   it reads the cache's index; outputs and
                                   cache state are those of calls run one after
                                   another.  The caller promises that each
                                   payload is complete when its call is
                                   enqueued, or is written by work that the
                                   call already waits for without it: a copy,
                                   memset or event wait on the stream between
                                   the writer and the call, or a kernel that
                                   does not trigger its dependents early.  Not
                                   applied to GLEAM_EVICT_LRU caches (an
                                   eviction rewrites slots) nor with
                                   GLEAM_PAPER_IDS (the key is known after one
                                   stage); both stay correct. */

/* Cumulative counters of one cache (successful calls only). */
typedef struct gleam_stats {
  uint64_t calls;          /* gleam_dedup_copy* calls with n > 0             */
  uint64_t chunks;         /* chunks examined                                */
  uint64_t hits_cache;     /* chunks found byte-equal in the cache as it was
                              when their call started                        */
  uint64_t hits_intra;     /* chunks equal to an earlier miss of their call  */
  uint64_t misses;         /* chunks returned as misses (and inserted)       */
  uint64_t inserts;        /* entries added (misses + debug inserts)         */
  uint64_t verify_rejects; /* misses that had a key+length candidate whose
                              bytes differed (collisions caught by verify)   */
  uint64_t slots_used;     /* arena slots in use                             */
  uint64_t bytes_used;     /* sum of the stored chunks' true lengths         */
  uint64_t capacity_bytes; /* as passed to create                            */
  uint64_t nslots;         /* capacity_bytes / chunk_bytes                   */
  uint64_t chunk_bytes;    /* C                                              */
  uint64_t evictions;      /* slots reused by GLEAM_EVICT_LRU                */
  uint64_t spec_chunks;    /* chunks the hash kernel also wrote ahead to their
                              likely packed offset and arena slot
                              (write-through, GLEAM_DEBUG_SPECULATE); a
                              speed counter that outputs never depend on     */
} gleam_stats_t;

/* Written by the device when an asynchronous dedup call completes. */
typedef struct gleam_result {
  int64_t status;          /* GLEAM_OK or a negative gleam_status            */
  uint64_t n_miss;         /* misses = entries of miss_idx written           */
  uint64_t n_hit_cache;
  uint64_t n_hit_intra;
  uint64_t verify_rejects;
  uint64_t miss_bytes;     /* bytes written to the packed miss buffer        */
} gleam_result_t;

/* One payload of gleam_dedup_copy_batch: the arguments of one
 * gleam_dedup_copy_async call.  d_result may be NULL. */
typedef struct gleam_payload {
  const void* d_buf;
  size_t n;
  uint32_t* d_hit_mask;
  uint32_t* d_miss_idx;
  void* d_miss_bytes;
  gleam_result_t* d_result;
  /* optional (may be NULL), device u32[N]: the arena slot that holds chunk i's
   * bytes after the call -- the byte-equal cached chunk for a hit, the new
   * slot for a miss, 0xFFFFFFFF for a chunk that is never cached
   * (GLEAM_PAPER_IDS).  Records for gleam_block_check come from here. */
  uint32_t* d_chunk_slot;
} gleam_payload_t;

/* ---- cache lifetime ---------------------------------------------------- */

/* Creates a cache on the current GPU with floor(capacity_bytes/chunk_bytes)
 * slots of chunk_bytes each and an empty index (paper Sec. 4.1.3: the
 * server-side shareable pool; Sec. 4.1.2: the set of resident identifiers).
 * chunk_bytes: multiple of 32, 32..16 MiB.  The slot count must be 1..2^32-2.
 * flags: 0 or a combination of GLEAM_KEY16, GLEAM_DEBUG_CHECKS, GLEAM_PAPER_IDS,
 * GLEAM_EVICT_LRU and GLEAM_OVERLAP_CALLS.
 * On success *out owns about capacity_bytes + 32 B * slots of device memory.
 * Returns GLEAM_OK, GLEAM_ERR_INVALID_ARG, GLEAM_ERR_NOMEM or GLEAM_ERR_CUDA. */
int gleam_cache_create(size_t capacity_bytes, size_t chunk_bytes, gleam_cache_t** out);
int gleam_cache_create_ex(size_t capacity_bytes, size_t chunk_bytes, uint32_t flags,
                          gleam_cache_t** out);

/* Frees the arena, index and workspace after the cache's work has finished.
 * NULL is accepted.  The handle is invalid afterwards. */
void gleam_cache_destroy(gleam_cache_t* cache);

/* Pre-sizes the per-call workspace for payloads of up to max_chunks chunks,
 * so that later calls of that size allocate nothing.  Synchronous. */
int gleam_cache_reserve(gleam_cache_t* cache, uint64_t max_chunks);

/* ---- the hot path ------------------------------------------------------ */

/* Fingerprints (paper Sec. 4.1.2's per-payload hash; App. B.1):
 * d_out[i] = XXH64(seed 0) of chunk i of the n-byte device buffer d_buf, for
 * i < ceil(n/chunk_bytes).  chunk_bytes == 0 hashes the whole buffer into
 * d_out[0] (also for n == 0).  d_out: device array of u64, caller-owned.
 * Asynchronous on `stream`; any alignment of d_buf is accepted. */
int gleam_fingerprint(const void* d_buf, size_t n, size_t chunk_bytes, uint64_t* d_out,
                      gleam_stream_t stream);

/* Dedups one host-to-device payload already copied to the device (paper
 * Sec. 4.1.2).  Chunks are decided in ascending order, as if one at a time:
 * chunk i is a hit iff its bytes equal a cached chunk of the same length, or
 * an earlier miss of this same call; otherwise it is a miss, is appended to
 * the outputs and is inserted into the cache.
 * Outputs (device memory, caller-owned, sized for the worst case):
 *   d_hit_mask   u32[ceil(N/32)]: bit i%32 of word i/32 = chunk i is a hit,
 *                bits past N are 0;
 *   d_miss_idx   u32[N]: ascending indices of the misses;
 *   d_miss_bytes u8[n]: the r-th miss's bytes at offset r*C (true length for
 *                the last chunk) -- the bytes that must cross the network;
 *                bytes past the last miss are unspecified (the call may
 *                write there).
 * Synchronous like cudaMemcpy (runs on the legacy default stream).
 * Returns the number of misses (>= 0) or a negative gleam_status; on
 * GLEAM_ERR_CAPACITY and GLEAM_ERR_TIMEOUT the cache is unchanged and the
 * outputs are unspecified.  n == 0 returns 0 and touches nothing.
 * With GLEAM_EVICT_LRU, misses that do not fit the never-used slots take the
 * slots of least recently used chunks that this call did not hit. */
int64_t gleam_dedup_copy(gleam_cache_t* cache, const void* d_buf, size_t n,
                         uint32_t* d_hit_mask, uint32_t* d_miss_idx, void* d_miss_bytes);

/* Same as gleam_dedup_copy, enqueued on `stream` without a host sync.  The
 * outcome is written to the device struct *d_result (may be NULL) when the
 * call's work completes.  Calls on one cache must be ordered (one stream, or
 * explicit events): they share the cache's workspace.  Returns GLEAM_OK once
 * enqueued, or an argument/launch error.  The first call that needs a larger
 * workspace than any before it synchronises the stream to grow it (see
 * gleam_cache_reserve). */
int gleam_dedup_copy_async(gleam_cache_t* cache, const void* d_buf, size_t n,
                           uint32_t* d_hit_mask, uint32_t* d_miss_idx, void* d_miss_bytes,
                           gleam_result_t* d_result, gleam_stream_t stream);

/* Dedups `count` payloads in one call: the outputs, per-payload results and
 * final cache state are exactly those of `count` gleam_dedup_copy_async calls
 * made in array order (paper Sec. 4.1.2 applied to each intercepted
 * host-to-device copy in turn; a chunk equal to an earlier payload's miss is
 * a hit on the cache, as that payload's call would have inserted it).  All
 * chunks of all payloads are processed together, so per-call latency is paid
 * once.  Exceptions: if the misses of the whole batch do not fit the free
 * slots, the batch returns GLEAM_ERR_CAPACITY as a unit and the cache is
 * unchanged; with GLEAM_EVICT_LRU the batch is one call for eviction (one
 * clock value, victims chosen once, among the slots no payload of the batch
 * hit).  payloads: host array, read before the call returns (each
 * entry's buffers as for gleam_dedup_copy).  d_total (device, may be NULL)
 * receives the sums over the batch.  Asynchronous on `stream`; ordered after
 * the cache's previous call whatever its stream. */
int gleam_dedup_copy_batch(gleam_cache_t* cache, const gleam_payload_t* payloads, size_t count,
                           gleam_result_t* d_total, gleam_stream_t stream);

/* Host-resident payloads (paper Sec. 4.1.2 in its own order: the sender
 * decides what to send before anything is copied).  The payload stays in
 * page-locked host memory (cudaHostAlloc, or cudaHostRegister of existing
 * memory); the kernels read it in place over the CPU-GPU link, so the whole
 * payload is never written to device memory: only the misses are, to the
 * packed output and the arena.  h_buf / payload d_buf fields: page-locked
 * host memory (other host memory and device memory are rejected with
 * GLEAM_ERR_NOT_DEVICE_PTR).  Outputs: device memory; the miss indices, the
 * packed miss bytes and the chunk slots may also be page-locked host memory,
 * which the kernels then write over the link directly, so the bytes that must
 * cross the network land on the host without a separate copy (hit masks and
 * results stay in device memory: they are updated with atomics).  Semantics,
 * results and ordering are those of gleam_dedup_copy_async /
 * gleam_dedup_copy_batch. */
int gleam_dedup_copy_host_async(gleam_cache_t* cache, const void* h_buf, size_t n,
                                uint32_t* d_hit_mask, uint32_t* d_miss_idx, void* d_miss_bytes,
                                gleam_result_t* d_result, gleam_stream_t stream);
int gleam_dedup_copy_host_batch(gleam_cache_t* cache, const gleam_payload_t* payloads,
                                size_t count, gleam_result_t* d_total, gleam_stream_t stream);

/* ---- dedup without allocation -------------------------------------------
 * No counterpart in the paper: an addition for callers that cannot allocate
 * device memory while they run, e.g. code executing inside an intercepted CUDA
 * call (the server side of an API-remoting layer handling a host-to-device
 * copy), where a cudaMalloc would re-enter the interception or disturb the
 * memory map it keeps for the application.
 *
 * Same operation, outputs and cache update as gleam_dedup_copy_async, but the
 * per-call workspace is one fixed array of about 7.2 MiB in the library's
 * device image instead of memory allocated by the cache; the call itself only
 * enqueues memsets and kernels and allocates nothing.  Every GPU that loads
 * the library holds that array until the process exits.
 *  - Payloads of more than GLEAM_NOALLOC_MAX_CHUNKS chunks (ceil(n / C)) are
 *    rejected with GLEAM_ERR_INVALID_ARG; use gleam_dedup_copy_async for them.
 *  - gleam_cache_create[_ex] looks the array's device address up, on the
 *    cache's GPU, while it allocates the cache (the lookup may load the
 *    library's device code on that GPU, which is when the array is
 *    allocated), so that no call does any set-up.
 *  - Test hooks of gleam_cache_debug_set apply as to the other calls; kernel
 *    timing (gleam_cache_profile) does not cover this call: it records no
 *    events, so that it creates nothing.
 *  - All calls on a GPU, from every cache, share the one array and it keeps
 *    the last call's contents (the call clears what must start at zero).
 *    Calls that overlap on the GPU race and give wrong results: order them
 *    (one stream, or events).  Calls on one cache are ordered automatically.
 *  - d_result (device, may be NULL) receives the outcome, as for
 *    gleam_dedup_copy_async; n == 0 returns GLEAM_OK and does nothing. */
#define GLEAM_NOALLOC_MAX_CHUNKS 65536
int gleam_dedup_copy_noalloc(gleam_cache_t* cache, const void* d_buf, size_t n,
                             uint32_t* d_hit_mask, uint32_t* d_miss_idx, void* d_miss_bytes,
                             gleam_result_t* d_result, gleam_stream_t stream);

/* Weight-block identification at cudaFree time (paper Sec. 4.1.1): a block
 * (one cudaMalloc) is kept as weights only if every chunk written into it by
 * host-to-device copies is unchanged when it is freed.  Record r says that the
 * block's bytes at d_offsets[r] were written with the chunk now stored in
 * cache slot d_slots[r] (from d_chunk_slot of the dedup call that handled the
 * copy; for segments written more than once, keep the first write's records).
 * Each record is compared byte for byte with the block's current bytes.
 *   d_block: device memory of block_bytes bytes; d_offsets u64[nrec] and
 *   d_slots u32[nrec]: device arrays; d_mismatch: device u8[nrec] or NULL,
 *   receives 1 for a record whose bytes differ, that does not fit in the
 *   block, or that names an unused slot, else 0; d_count: device u64, receives
 *   the number of such records (0 = the block still holds its weights).
 * Asynchronous on `stream`, ordered after the cache's previous call; reads
 * the cache, changes nothing. */
int gleam_block_check(const gleam_cache_t* cache, const void* d_block, size_t block_bytes,
                      const uint64_t* d_offsets, const uint32_t* d_slots, size_t nrec,
                      uint8_t* d_mismatch, uint64_t* d_count, gleam_stream_t stream);

/* Copies the cache's counters to *out (host struct).  Waits for the cache's
 * outstanding work on the device. */
int gleam_cache_stats(const gleam_cache_t* cache, gleam_stats_t* out);

/* ---- inspection and test helpers (not on the hot path) ------------------ */

/* Index contents ordered by slot: h_keys[s], h_lens[s] for s < min(max,
 * slots_used) (host arrays).  *count receives the number of index entries. */
int gleam_cache_export(const gleam_cache_t* cache, uint64_t* h_keys, uint32_t* h_lens,
                       uint64_t max, uint64_t* count);

/* Copies the stored bytes of `slot` to host memory h_out (at most max bytes);
 * *len receives the stored length. */
int gleam_cache_read_slot(const gleam_cache_t* cache, uint64_t slot, void* h_out,
                          uint64_t max, uint64_t* len);

/* Stores len bytes from device memory d_bytes under an arbitrary key (masked
 * to 16 bits in GLEAM_KEY16 mode) in the next free slot.  Used to plant
 * colliding entries that the verify must reject.  Synchronous. */
int gleam_cache_debug_insert(gleam_cache_t* cache, uint64_t key, const void* d_bytes,
                             size_t len);

/* Test hooks.  what = GLEAM_DEBUG_WAIT_LIMIT_NS: limit of every device-side
 * wait in nanoseconds (default 4e9); what = GLEAM_DEBUG_SKIP_ARRIVE: the block
 * with this index (-1 = none) leaves the next call's first grid barrier
 * without arriving, so the other blocks' bounded waits run out and the call
 * returns GLEAM_ERR_TIMEOUT with the cache unchanged. */
#define GLEAM_DEBUG_WAIT_LIMIT_NS 1
#define GLEAM_DEBUG_SKIP_ARRIVE 2
/* what = GLEAM_DEBUG_CLOCK: sets the GLEAM_EVICT_LRU clock (the value of the
 * latest call, 0 .. 2^32-2; the next call takes value + 1), so that tests can
 * reach clock values of any size.  The clock is 32 bits: a cache that has
 * served 2^32 - 1 calls no longer orders its slots exactly. */
#define GLEAM_DEBUG_CLOCK 3
/* what = GLEAM_DEBUG_DROP_ENTRY: removes the index entry of slot `value`
 * (damages the cache on purpose, to test GLEAM_DEBUG_CHECKS).  Synchronous. */
#define GLEAM_DEBUG_DROP_ENTRY 4
/* what = GLEAM_DEBUG_SMALL_CALLS: the largest call, in chunks, that may run as
 * one single-block kernel instead of three launches (default 64; 0 turns that
 * path off).  Only the speed changes: every output is the same either way. */
#define GLEAM_DEBUG_SMALL_CALLS 5
/* what = GLEAM_DEBUG_SPECULATE: the write-through of likely misses.  A chunk
 * that no cached chunk begins like (no prefix-hint match) is written by the
 * hash kernel, as it streams by, to packed offset i*C of its payload and to
 * arena slot slots_used + g (g = its number in the call); the pack step then
 * skips the copies of every miss whose rank puts it exactly there (a payload,
 * or a run of payloads, of misses only) and copies the others over (for
 * payloads in host memory this also spares the second read over the link).
 * It needs 16-byte-aligned payloads and packed buffers, chunks of at least
 * 512 bytes and 64-bit or KEY16 keys (not GLEAM_PAPER_IDS).  0 = automatic
 * (default: on while at least half of the chunks written ahead are used,
 * retried every 256 calls once off), 1 = always, 2 = never.  Only the speed
 * changes: every output is the same either way. */
#define GLEAM_DEBUG_SPECULATE 6
int gleam_cache_debug_set(gleam_cache_t* cache, int what, int64_t value);

/* Device-side copy of the index, slot count and counters (and, for a
 * GLEAM_EVICT_LRU cache, the slot lengths and last uses), for restoring the
 * cache between timed repetitions.  Arena bytes are not copied: those past
 * the saved slot count are never read, and a slot that an eviction reused
 * after the snapshot keeps its new bytes, so its restored entry no longer
 * matches them and its chunk misses (every hit is verified).  The
 * write-through's automatic state (GLEAM_DEBUG_SPECULATE) is not part of a
 * snapshot: it follows the calls made. */
int gleam_cache_snapshot(gleam_cache_t* cache, gleam_snapshot_t** out);
int gleam_cache_restore(gleam_cache_t* cache, const gleam_snapshot_t* snap);
void gleam_snapshot_destroy(gleam_snapshot_t* snap);

/* Kernel timing for benchmarks.  While enabled, every dedup call (except
 * gleam_dedup_copy_noalloc) records CUDA events on its own stream around its
 * two phases: phase 0 is the kernel that
 * fingerprints, probes and verifies; phase 1 is the two kernels that resolve
 * duplicates and rank the misses, then compact, pack and insert; a small
 * call that runs as one single-block kernel (GLEAM_DEBUG_SMALL_CALLS) counts
 * all of its time in phase 0.
 * gleam_cache_profile_read waits for the recorded calls, writes the summed
 * device time (ms) and count of calls of phase k to h_ms[k] and
 * h_launches[k] for k < nkernels (host arrays), and starts a new tally. */
int gleam_cache_profile(gleam_cache_t* cache, int enable);
int gleam_cache_profile_read(gleam_cache_t* cache, double* h_ms, uint64_t* h_launches,
                             int nkernels);

/* Short English name of a gleam_status value. */
const char* gleam_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* GLEAM_H */
