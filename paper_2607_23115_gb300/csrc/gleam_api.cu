// Host side of the C ABI declared in include/gleam.h: argument checks, the
// cache object (arena, index, counters, per-call workspace) and the launch
// sequence of one dedup call.  Every step of the path runs in the kernels of
// hash_probe.cu and dedup_compact.cu; nothing here touches payload bytes.
#include <cuda.h>

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "gleam_internal.cuh"

using namespace gleam;

struct gleam_cache {
  int device = 0;
  size_t capacity_bytes = 0;
  uint64_t C = 0;
  uint64_t nslots = 0;
  uint32_t flags = 0;

  uint8_t* arena = nullptr;
  IndexEntry* index = nullptr;
  IndexEntry* hints = nullptr;  // prefix-hint table, index_cap entries
  uint64_t index_cap = 0;  // power of two >= 2 * nslots
  uint32_t* slot_len = nullptr;
  unsigned long long* slot_key = nullptr;  // per slot: the stored chunk's group key
  unsigned long long* dstats = nullptr;

  // LRU eviction (GLEAM_EVICT_LRU)
  uint32_t* last_use = nullptr;  // per slot
  uint8_t* vflag = nullptr;      // per slot
  uint32_t* victims = nullptr;   // per slot
  uint32_t* bins = nullptr;      // kLruBins
  uint32_t epoch = 0;            // clock value of the latest call

  // GLEAM_DEBUG_CHECKS
  uint32_t* dbg_count = nullptr;  // per slot
  uint32_t* dbg_flag = nullptr;

  // per-call workspace (per chunk, by global chunk number)
  uint64_t ws_chunks = 0;
  void* ws = nullptr;
  ChunkArrays ch{};
  CallEntry* tbl = nullptr;
  ClassEntry* cls_tbl = nullptr;  // KEY16: (16-bit key, length) classes, tbl_cap entries
  uint64_t tbl_cap = 0;

  // payload tables of multi-payload calls
  uint64_t tab_cap = 0;
  PayloadDesc* d_table = nullptr;
  PayloadDesc* h_table = nullptr;  // pinned staging for the table copy
  uint32_t* d_pstart = nullptr;
  cudaEvent_t table_copied = nullptr;

  DevCtl* ctl = nullptr;
  uint32_t* bcount = nullptr;
  gleam_result_t* d_result = nullptr;
  gleam_result_t* h_result = nullptr;      // page-locked, mapped: gleam_dedup_copy's result
  gleam_result_t* h_result_dev = nullptr;  // its device address
  int coop_max_blocks = 0;
  int pack_max_blocks = 0;  // pack kernel: all co-resident blocks
  int rp_max_blocks = 0;    // one-launch resolve + pack: all co-resident blocks
  cudaEvent_t done = nullptr;

  // single-block calls: the largest call (in chunks) that runs as one kernel,
  // and an upper bound of the slots in use (no device read needed), which
  // tells when a call of an LRU cache cannot need an eviction
  uint64_t small_max_chunks = 0;
  uint64_t slots_bound = 0;

  // write-through of likely misses (HashArgs::spec_mode)
  uint32_t* spec_state = nullptr;   // device: [0] on, [1] calls since it went off
  uint32_t* spec_mirror = nullptr;  // page-locked, mapped: [0] as of the last finished call
  int spec_hook = 0;                // GLEAM_DEBUG_SPECULATE: 0 auto, 1 always, 2 never

  unsigned long long wait_ns = 4000000000ULL;
  int skip_block = -1;

  // id (cudaStreamGetId) of the stream `done` was last recorded on: a call on
  // that same stream is ordered after it without an event wait
  unsigned long long done_stream = ~0ull;

  // device address of the allocation-free call's scratch array on this GPU,
  // looked up when the cache is created
  uint8_t* na_scratch = nullptr;

  // kernel timing (gleam_cache_profile)
  bool profile = false;
  std::vector<cudaEvent_t> ev_pool;  // 3 events per recorded call
  size_t ev_used = 0;

  std::mutex mu;
};

struct gleam_snapshot {
  int device = 0;
  const gleam_cache* owner = nullptr;
  IndexEntry* index = nullptr;
  IndexEntry* hints = nullptr;
  uint64_t index_cap = 0;
  unsigned long long* dstats = nullptr;
  uint32_t* slot_len = nullptr;  // LRU caches: slot lengths, keys and last uses too
  unsigned long long* slot_key = nullptr;
  uint32_t* last_use = nullptr;
  uint64_t nslots = 0;
  uint64_t slots_bound = 0;  // the cache's host-side bound of its used slots
};

namespace {

constexpr uint64_t kMinChunk = 32;
constexpr uint64_t kMaxChunk = 16ull << 20;
constexpr uint64_t kMaxChunks = 0xFFFFFFFEull;  // chunk numbers are 32-bit

class DeviceGuard {
 public:
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev_) != cudaSuccess) prev_ = -1;
    if (prev_ != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev_ >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev_) cudaSetDevice(prev_);
  }

 private:
  int prev_ = -1;
};

uint64_t next_pow2(uint64_t x) {
  uint64_t p = 1;
  while (p < x) p <<= 1;
  return p;
}

uint64_t align256(uint64_t x) { return (x + 255) & ~255ull; }

int cuda_err(cudaError_t e) {
  if (e == cudaSuccess) return GLEAM_OK;
  cudaGetLastError();  // clear the non-sticky error state for later calls
  return e == cudaErrorMemoryAllocation ? GLEAM_ERR_NOMEM : GLEAM_ERR_CUDA;
}

// ---- device pointer checks -------------------------------------------------
//
// A pointer is accepted iff the runtime reports device memory of the cache's
// GPU (or managed memory).  When the driver reports the allocation's address
// range, the accessed span must lie inside it; the range is then remembered
// for the rest of the same call, so that payloads and outputs carved from one
// buffer are checked with a single query.
typedef CUresult (*PtrAttrsFn)(unsigned int, CUpointer_attribute*, void**, CUdeviceptr);

PtrAttrsFn driver_ptr_attrs() {
  static PtrAttrsFn fn = []() -> PtrAttrsFn {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuPointerGetAttributes", &f, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    return reinterpret_cast<PtrAttrsFn>(f);
  }();
  return fn;
}

class PtrChecker {
 public:
  explicit PtrChecker(int device) : device_(device) {}

  // Whether any pointer checked so far was managed memory.
  bool saw_managed() const { return managed_; }

  // GLEAM_OK iff [p, p + bytes) is page-locked host memory (cudaHostAlloc or
  // cudaHostRegister) that the device can read; *dev receives the address to
  // use in device code.
  int check_host(const void* p, uint64_t bytes, const void** dev) {
    if (p == nullptr) return GLEAM_ERR_INVALID_ARG;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
      cudaGetLastError();
      return GLEAM_ERR_NOT_DEVICE_PTR;
    }
    if (at.type != cudaMemoryTypeHost || at.devicePointer == nullptr)
      return GLEAM_ERR_NOT_DEVICE_PTR;
    *dev = at.devicePointer;
    if (PtrAttrsFn fn = driver_ptr_attrs()) {
      CUpointer_attribute attrs[2] = {CU_POINTER_ATTRIBUTE_RANGE_START_ADDR,
                                      CU_POINTER_ATTRIBUTE_RANGE_SIZE};
      CUdeviceptr start = 0;
      size_t size = 0;
      void* data[2] = {&start, &size};
      const uintptr_t a = reinterpret_cast<uintptr_t>(*dev);
      if (fn(2, attrs, data, (CUdeviceptr)a) == CUDA_SUCCESS && size > 0 &&
          (a < start || a + bytes > start + size))
        return GLEAM_ERR_INVALID_ARG;  // span overruns the registration
    }
    return GLEAM_OK;
  }

  // GLEAM_OK iff [p, p + bytes) is device memory of the device.
  int check(const void* p, uint64_t bytes) {
    if (p == nullptr) return GLEAM_ERR_INVALID_ARG;
    const uintptr_t a = reinterpret_cast<uintptr_t>(p);
    const uintptr_t b = a + bytes;
    for (int k = 0; k < kRanges; ++k)
      if (hi_[k] > lo_[k] && a >= lo_[k] && b <= hi_[k]) return GLEAM_OK;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
      cudaGetLastError();
      return GLEAM_ERR_NOT_DEVICE_PTR;
    }
    const bool ok = at.type == cudaMemoryTypeManaged ||
                    (at.type == cudaMemoryTypeDevice && at.device == device_);
    if (!ok) return GLEAM_ERR_NOT_DEVICE_PTR;
    managed_ = managed_ || at.type == cudaMemoryTypeManaged;
    if (PtrAttrsFn fn = driver_ptr_attrs()) {
      CUpointer_attribute attrs[2] = {CU_POINTER_ATTRIBUTE_RANGE_START_ADDR,
                                      CU_POINTER_ATTRIBUTE_RANGE_SIZE};
      CUdeviceptr start = 0;
      size_t size = 0;
      void* data[2] = {&start, &size};
      if (fn(2, attrs, data, (CUdeviceptr)a) == CUDA_SUCCESS && size > 0) {
        if (a < start || b > start + size) return GLEAM_ERR_INVALID_ARG;  // span overruns
        lo_[next_] = start;
        hi_[next_] = start + size;
        next_ = (next_ + 1) % kRanges;
      }
    }
    return GLEAM_OK;
  }

 private:
  static constexpr int kRanges = 8;
  int device_;
  uintptr_t lo_[kRanges] = {};
  uintptr_t hi_[kRanges] = {};
  int next_ = 0;
  bool managed_ = false;
};

void free_ws(gleam_cache* c) {
  if (c->ws) cudaFree(c->ws);
  c->ws = nullptr;
  c->ws_chunks = 0;
  c->tbl_cap = 0;
  c->ch = ChunkArrays{};
  c->tbl = nullptr;
  c->cls_tbl = nullptr;
}

// Grows the per-chunk workspace to hold `nchunks` chunks.  Waits for the
// cache's previous work first (it may still be using the old workspace).
int ensure_ws(gleam_cache* c, uint64_t nchunks) {
  if (nchunks <= c->ws_chunks) return GLEAM_OK;
  uint64_t cap = std::max<uint64_t>({nchunks, 2 * c->ws_chunks, 4096});
  cap = std::min<uint64_t>(cap, kMaxChunks);
  if (cap < nchunks) cap = nchunks;
  const uint64_t tcap = next_pow2(2 * cap);
  const uint64_t sz[16] = {align256(cap),     align256(cap * 8), align256(cap * 4),
                           align256(cap * 8), align256(cap * 4), align256(cap * 4),
                           align256(cap * 4), align256(cap * 4), align256(cap * 8),
                           align256(cap * 4), align256(cap * 4), align256(cap * 4),
                           align256(cap),     align256(tcap * sizeof(CallEntry)),
                           align256(cap * 8), align256(tcap * sizeof(ClassEntry))};
  uint64_t total = 0;
  for (uint64_t x : sz) total += x;
  int rc = cuda_err(cudaEventSynchronize(c->done));
  if (rc != GLEAM_OK) return rc;
  free_ws(c);
  void* p = nullptr;
  if ((rc = cuda_err(cudaMalloc(&p, total))) != GLEAM_OK) return rc;
  if ((rc = cuda_err(cudaMemset(p, 0, total))) != GLEAM_OK) {
    cudaFree(p);
    return rc;
  }
  uint8_t* b = static_cast<uint8_t*>(p);
  c->ws = p;
  c->ch.status = b;
  b += sz[0];
  c->ch.key = reinterpret_cast<unsigned long long*>(b);
  b += sz[1];
  c->ch.len = reinterpret_cast<uint32_t*>(b);
  b += sz[2];
  c->ch.src = reinterpret_cast<unsigned long long*>(b);
  b += sz[3];
  c->ch.pidx = reinterpret_cast<uint32_t*>(b);
  b += sz[4];
  c->ch.res = reinterpret_cast<uint32_t*>(b);
  b += sz[5];
  c->ch.ent = reinterpret_cast<uint32_t*>(b);
  b += sz[6];
  c->ch.rank = reinterpret_cast<uint32_t*>(b);
  b += sz[7];
  c->ch.hint = reinterpret_cast<unsigned long long*>(b);
  b += sz[8];
  c->ch.order = reinterpret_cast<uint32_t*>(b);
  b += sz[9];
  c->ch.srank = reinterpret_cast<uint32_t*>(b);
  b += sz[10];
  c->ch.old = reinterpret_cast<uint32_t*>(b);
  b += sz[11];
  c->ch.spec = b;
  b += sz[12];
  c->tbl = reinterpret_cast<CallEntry*>(b);
  b += sz[13];
  c->ch.cls = reinterpret_cast<unsigned long long*>(b);
  b += sz[14];
  c->cls_tbl = reinterpret_cast<ClassEntry*>(b);
  c->tbl_cap = tcap;
  c->ws_chunks = cap;
  return GLEAM_OK;
}

// Grows the payload tables to `count` payloads.
int ensure_tables(gleam_cache* c, uint64_t count) {
  if (count <= c->tab_cap) return GLEAM_OK;
  const uint64_t cap = std::max<uint64_t>({count, 2 * c->tab_cap, 64});
  int rc = cuda_err(cudaEventSynchronize(c->done));
  if (rc != GLEAM_OK) return rc;
  if (c->d_table) cudaFree(c->d_table);
  if (c->h_table) cudaFreeHost(c->h_table);
  if (c->d_pstart) cudaFree(c->d_pstart);
  c->d_table = nullptr;
  c->h_table = nullptr;
  c->d_pstart = nullptr;
  c->tab_cap = 0;
  if ((rc = cuda_err(cudaMalloc(&c->d_table, cap * sizeof(PayloadDesc)))) != GLEAM_OK) return rc;
  if ((rc = cuda_err(cudaMallocHost(&c->h_table, cap * sizeof(PayloadDesc)))) != GLEAM_OK) return rc;
  if ((rc = cuda_err(cudaMalloc(&c->d_pstart, cap * sizeof(uint32_t)))) != GLEAM_OK) return rc;
  c->tab_cap = cap;
  return GLEAM_OK;
}

void destroy_cache(gleam_cache* c) {
  if (!c) return;
  {
    DeviceGuard g(c->device);
    cudaDeviceSynchronize();
    free_ws(c);
    if (c->arena) cudaFree(c->arena);
    if (c->index) cudaFree(c->index);
    if (c->hints) cudaFree(c->hints);
    if (c->slot_len) cudaFree(c->slot_len);
    if (c->slot_key) cudaFree(c->slot_key);
    if (c->dstats) cudaFree(c->dstats);
    if (c->last_use) cudaFree(c->last_use);
    if (c->vflag) cudaFree(c->vflag);
    if (c->victims) cudaFree(c->victims);
    if (c->bins) cudaFree(c->bins);
    if (c->dbg_count) cudaFree(c->dbg_count);
    if (c->dbg_flag) cudaFree(c->dbg_flag);
    if (c->ctl) cudaFree(c->ctl);
    if (c->spec_state) cudaFree(c->spec_state);
    if (c->spec_mirror) cudaFreeHost(c->spec_mirror);
    if (c->bcount) cudaFree(c->bcount);
    if (c->d_result) cudaFree(c->d_result);
    if (c->h_result) cudaFreeHost(c->h_result);
    if (c->d_table) cudaFree(c->d_table);
    if (c->h_table) cudaFreeHost(c->h_table);
    if (c->d_pstart) cudaFree(c->d_pstart);
    if (c->table_copied) cudaEventDestroy(c->table_copied);
    if (c->done) cudaEventDestroy(c->done);
    for (cudaEvent_t e : c->ev_pool) cudaEventDestroy(e);
    cudaGetLastError();
  }
  delete c;
}

int wait_done(const gleam_cache* c) { return cuda_err(cudaEventSynchronize(c->done)); }

// Validates one payload and fills its device descriptor (chunk_base left 0).
int describe(gleam_cache* c, PtrChecker& chk, const gleam_payload_t& p, PayloadDesc* d,
             bool host_payload = false) {
  const uint64_t N = (p.n + c->C - 1) / c->C;
  if (N > kMaxChunks) return GLEAM_ERR_INVALID_ARG;
  d->buf = static_cast<const uint8_t*>(p.d_buf);
  d->n = p.n;
  d->chunk_base = 0;
  d->nchunks = N;
  d->mask = p.d_hit_mask;
  d->miss_idx = p.d_miss_idx;
  d->packed = static_cast<uint8_t*>(p.d_miss_bytes);
  d->result = p.d_result;
  d->chunk_slot = p.d_chunk_slot;
  int rc;
  // An output that the kernels only store to (no atomics) may, for the host
  // entries, also be page-locked host memory: *out receives the address the
  // kernels use.
  auto check_out = [&](void* ptr, uint64_t bytes, void** out) -> int {
    int r = chk.check(ptr, bytes);
    if (r != GLEAM_ERR_NOT_DEVICE_PTR || !host_payload) return r;
    const void* dev = nullptr;
    if ((r = chk.check_host(ptr, bytes, &dev)) != GLEAM_OK) return r;
    *out = const_cast<void*>(dev);
    return GLEAM_OK;
  };
  if (p.d_result && (rc = chk.check(p.d_result, sizeof(gleam_result_t))) != GLEAM_OK) return rc;
  if (p.d_chunk_slot && N &&
      (rc = check_out(p.d_chunk_slot, N * 4, reinterpret_cast<void**>(&d->chunk_slot))) != GLEAM_OK)
    return rc;
  if (p.n == 0) return GLEAM_OK;
  if (host_payload) {
    const void* dev = nullptr;
    if ((rc = chk.check_host(p.d_buf, p.n, &dev)) != GLEAM_OK) return rc;
    d->buf = static_cast<const uint8_t*>(dev);
  } else if ((rc = chk.check(p.d_buf, p.n)) != GLEAM_OK) {
    return rc;
  }
  if ((rc = chk.check(p.d_hit_mask, ((N + 31) / 32) * 4)) != GLEAM_OK) return rc;
  if ((rc = check_out(p.d_miss_idx, N * 4, reinterpret_cast<void**>(&d->miss_idx))) != GLEAM_OK)
    return rc;
  if ((rc = check_out(p.d_miss_bytes, p.n, reinterpret_cast<void**>(&d->packed))) != GLEAM_OK)
    return rc;
  return GLEAM_OK;
}

// Blocks of the cooperative dedup launch: enough for its per-chunk phases
// (chunks / dedup_chunks_per_block) and for its miss copies (one block per
// kBytesPerDedupBlock of payload), at most the co-resident maximum.
constexpr uint64_t kBytesPerDedupBlock = 256ull << 10;

int dedup_grid(const gleam_cache* c, uint64_t nchunks, uint64_t nbytes) {
  const uint64_t per_block = dedup_chunks_per_block();
  const uint64_t want = std::max<uint64_t>((nchunks + per_block - 1) / per_block,
                                           (nbytes + kBytesPerDedupBlock - 1) / kBytesPerDedupBlock);
  return (int)std::max<uint64_t>(1, std::min<uint64_t>(c->coop_max_blocks, want));
}

// Blocks of the pack kernel: one per 256 chunks or per kBytesPerPackBlock of
// payload, up to one full wave of co-resident blocks.
#ifndef GLEAM_PACK_BYTES_PER_BLOCK
#define GLEAM_PACK_BYTES_PER_BLOCK (32ull << 10)
#endif
constexpr uint64_t kBytesPerPackBlock = GLEAM_PACK_BYTES_PER_BLOCK;

int pack_grid(const gleam_cache* c, uint64_t nchunks, uint64_t nbytes) {
  const uint64_t want = std::max<uint64_t>((nchunks + 255) / 256,
                                           (nbytes + kBytesPerPackBlock - 1) / kBytesPerPackBlock);
  return (int)std::max<uint64_t>(1, std::min<uint64_t>(c->pack_max_blocks, want));
}

// The LRU fields of a call's kernel arguments; takes the call's clock value.
void set_lru(gleam_cache* c, DedupArgs* d, uint64_t nchunks) {
  if (!(c->flags & GLEAM_EVICT_LRU)) return;
  if (nchunks) ++c->epoch;
  d->lru = 1u;
  d->epoch = c->epoch;
  d->last_use = c->last_use;
  d->vflag = c->vflag;
  d->victims = c->victims;
  d->bins = c->bins;
}

// A call of at most this many payload bytes may run as the single-block kernel.
constexpr uint64_t kSmallMaxBytes = 256ull << 10;

// Whether a call runs as one single-block kernel instead of three launches:
// few chunks and bytes (one block then hashes them about as fast as a grid
// does, and a grid of one drops the kernel boundaries and every grid-wide
// round trip: a 64 KiB call takes 24 us instead of 32), payloads the staged
// hash can read, 64-bit or KEY16 keys, and no possible eviction (an evicting
// call scans the whole index, which wants the full grid).
bool small_call(const gleam_cache* c, bool aligned, uint64_t Ntot, uint64_t nbytes,
                int skip_block) {
  return Ntot > 0 && Ntot <= c->small_max_chunks && nbytes <= kSmallMaxBytes && aligned &&
         (c->C % 32 == 0 || Ntot == 1) && !(c->flags & GLEAM_PAPER_IDS) && skip_block < 0 &&
         (!(c->flags & GLEAM_EVICT_LRU) || c->slots_bound + Ntot <= c->nslots);
}

// After a call is enqueued: it stores at most Ntot new slots.
void note_call(gleam_cache* c, uint64_t Ntot) {
  c->slots_bound = std::min<uint64_t>(c->nslots, c->slots_bound + Ntot);
}

// Chained calls.  A call that leaves most of the GPU idle (at most
// kChainMaxChunks chunks and kChainMaxBytes bytes) launches its kernels with
// programmatic stream serialization: each kernel lets the next one on the
// stream be launched as soon as all of its blocks have started, so that a
// kernel's blocks are waiting on the GPU when the one before finishes instead
// of being launched then.  After the hash kernel, a call of one payload runs
// resolve, ranks, pack and publish as one launch (k_resolve_pack, one block
// per 256 chunks or kChainBytesPerBlock of payload, at most kChainPackBlocks);
// a batch runs the resolve kernel as a regular launch (a cooperative one is
// never launched early) on at most kChainDedupBlocks blocks and the pack
// kernel on at most kChainPackBlocks: every waiting block holds its SM
// resources.  With GLEAM_OVERLAP_CALLS the hash kernel also fingerprints
// before it waits (HashArgs::wait_late).  Evicting caches and the test hook
// that makes a block skip a barrier keep the plain launches.
#ifndef GLEAM_CHAIN_MAX_CHUNKS
#define GLEAM_CHAIN_MAX_CHUNKS 16384
#endif
#ifndef GLEAM_CHAIN_DEDUP_BLOCKS
#define GLEAM_CHAIN_DEDUP_BLOCKS 32
#endif
#ifndef GLEAM_CHAIN_PACK_BLOCKS
#define GLEAM_CHAIN_PACK_BLOCKS 76
#endif
constexpr uint64_t kChainMaxChunks = GLEAM_CHAIN_MAX_CHUNKS;
// A large payload keeps the full grids of the unchained path: its in-call
// duplicates (a 1 GiB payload of 64 KiB chunks, a quarter of them copies) are
// compared by every warp the resolve kernel has (0.47 ms with 456 blocks,
// 1.15 ms with 32).
constexpr uint64_t kChainMaxBytes = 256ull << 20;
constexpr int kChainDedupBlocks = GLEAM_CHAIN_DEDUP_BLOCKS;
constexpr int kChainPackBlocks = GLEAM_CHAIN_PACK_BLOCKS;
// Overlapping calls: a block of the one-launch kernel per 2 MiB of payload
// (Llama-3-8B, one call per tensor: 1,558-1,571 GB/s, against 1,480-1,495
// with 1 MiB), or per 512 KiB for calls under 4 MiB, whose copies would
// otherwise fall to one block (the 10,000-call stream's calls of 256 KiB-
// 1 MiB: 38.8 -> 34.2 us each).
#ifndef GLEAM_CHAIN_BYTES_PER_BLOCK
#define GLEAM_CHAIN_BYTES_PER_BLOCK (2ull << 20)
#endif
constexpr uint64_t kChainSmallCall = 4ull << 20;
constexpr uint64_t kChainBytesPerBlock = GLEAM_CHAIN_BYTES_PER_BLOCK;
// Without GLEAM_OVERLAP_CALLS a call overlaps the next only by the launch, so
// its one-launch resolve kernel may take a block per 512 KiB, up to one per SM
// (a 64 MiB call of 16,384 chunks: 0.101 -> 0.092 ms); with it, blocks that
// wait for an earlier call hold resources that the calls in flight want.
#ifndef GLEAM_SOLO_KIB_PER_BLOCK
#define GLEAM_SOLO_KIB_PER_BLOCK 512
#endif
#ifndef GLEAM_SOLO_CAP_DIV
#define GLEAM_SOLO_CAP_DIV 3
#endif
constexpr uint64_t kSoloBytesPerBlock = (uint64_t)GLEAM_SOLO_KIB_PER_BLOCK << 10;
#ifndef GLEAM_OVERLAP_COPY_GRAB
#define GLEAM_OVERLAP_COPY_GRAB 8
#endif
constexpr uint32_t kOverlapCopyGrab = GLEAM_OVERLAP_COPY_GRAB;
// the one-launch resolve kernel holds at most one chunk per thread
static_assert(kChainMaxChunks <= (uint64_t)kChainPackBlocks * 256, "chain limit");

bool chain_call(const gleam_cache* c, uint64_t Ntot, uint64_t nbytes, int skip_block) {
  return Ntot <= kChainMaxChunks && nbytes <= kChainMaxBytes && skip_block < 0 &&
         !(c->flags & GLEAM_EVICT_LRU);
}

// Orders a call on stream s after the cache's previous work: an event wait,
// unless that work ended on s itself (stream order already holds, and a wait
// between two kernels would keep the second from being launched early).
int order_after_done(gleam_cache* c, cudaStream_t s, unsigned long long* sid) {
  if (cudaStreamGetId(s, sid) != cudaSuccess) {
    cudaGetLastError();
    *sid = ~0ull;
  }
  if (*sid != ~0ull && *sid == c->done_stream) return GLEAM_OK;
  return cuda_err(cudaStreamWaitEvent(s, c->done, 0));
}

// Records the end of the cache's latest work on stream s.
int record_done(gleam_cache* c, cudaStream_t s, unsigned long long sid) {
  const int rc = cuda_err(cudaEventRecord(c->done, s));
  c->done_stream = rc == GLEAM_OK ? sid : ~0ull;
  return rc;
}

unsigned long long stream_id(cudaStream_t s) {
  unsigned long long id = ~0ull;
  if (cudaStreamGetId(s, &id) != cudaSuccess) {
    cudaGetLastError();
    id = ~0ull;
  }
  return id;
}

// The write-through fields of a call's kernel arguments.  It needs the staged
// hash (16-byte-aligned payloads, C a multiple of 32), 16-byte-aligned packed
// buffers (device or page-locked host memory), and 64-bit or KEY16 keys.  In the automatic
// mode the host launches the write-through variant of the hash kernel when
// the page-locked copy of the device state says it is on (as of the last call
// that finished: a call or two late at most, which a heuristic can afford),
// and every eligible call feeds the state back.
void set_spec(gleam_cache* c, HashArgs* h, DedupArgs* d, bool eligible) {
  h->spec_mode = 0;
  d->spec_active = 0;
  d->spec_state = nullptr;
  d->spec_mirror = nullptr;
  if (!eligible || c->C % 32 != 0 || (c->flags & GLEAM_PAPER_IDS) || c->spec_hook == 2) return;
  const bool on = c->spec_hook == 1 || *reinterpret_cast<volatile uint32_t*>(c->spec_mirror);
  h->spec_mode = on ? 1u : 0u;
  h->arena_w = c->arena;
  h->nslots = c->nslots;
  d->spec_active = h->spec_mode;
  if (c->spec_hook == 0) {
    d->spec_state = c->spec_state;
    d->spec_mirror = c->spec_mirror;
  }
}

// GLEAM_DEBUG_CHECKS: the index consistency check after a call.
int enqueue_index_check(gleam_cache* c, const DedupArgs& d, cudaStream_t s) {
  if (!(c->flags & GLEAM_DEBUG_CHECKS)) return GLEAM_OK;
  IndexCheckArgs k{};
  k.index = c->index;
  k.hints = c->hints;
  k.index_mask = c->index_cap - 1;
  k.slot_len = c->slot_len;
  k.dstats = c->dstats;
  k.count = c->dbg_count;
  k.flag = c->dbg_flag;
  k.table = d.table;
  k.one = d.one;
  k.npayloads = d.count;
  k.total = d.total;
  return cuda_err(launch_index_check(k, s));
}

// Enqueues one dedup call over `count` payloads on stream s, ordered after
// the cache's previous call.  Caller holds c->mu and the device.
int enqueue(gleam_cache* c, const gleam_payload_t* payloads, uint64_t count,
            gleam_result_t* d_total, cudaStream_t s, bool host_payloads = false,
            gleam_result_t* own_total = nullptr) {
  if (count == 0) return GLEAM_OK;
  if (count > 0xFFFFFFFEull) return GLEAM_ERR_INVALID_ARG;
  PtrChecker chk(c->device);
  int rc;
  if (d_total && (rc = chk.check(d_total, sizeof(gleam_result_t))) != GLEAM_OK) return rc;

  PayloadDesc one{};
  if (count > 1) {
    if ((rc = ensure_tables(c, count)) != GLEAM_OK) return rc;
    // the staging buffer may still feed the previous call's table copy
    if ((rc = cuda_err(cudaEventSynchronize(c->table_copied))) != GLEAM_OK) return rc;
  }
  uint64_t Ntot = 0, ncalls = 0, nbytes = 0;
  bool aligned = true, packed_aligned = true;
  for (uint64_t k = 0; k < count; ++k) {
    PayloadDesc* d = count > 1 ? &c->h_table[k] : &one;
    if ((rc = describe(c, chk, payloads[k], d, host_payloads)) != GLEAM_OK) return rc;
    d->chunk_base = Ntot;
    Ntot += d->nchunks;
    if (Ntot > kMaxChunks) return GLEAM_ERR_INVALID_ARG;
    if (d->n) {
      ++ncalls;
      nbytes += d->n;
      aligned = aligned && (reinterpret_cast<uintptr_t>(d->buf) % 16 == 0);
      packed_aligned = packed_aligned && (reinterpret_cast<uintptr_t>(d->packed) % 16 == 0);
    }
  }
  if ((rc = ensure_ws(c, std::max<uint64_t>(Ntot, 1))) != GLEAM_OK) return rc;

  unsigned long long sid = ~0ull;
  if ((rc = order_after_done(c, s, &sid)) != GLEAM_OK) return rc;
  if (count > 1) {
    if ((rc = cuda_err(cudaMemcpyAsync(c->d_table, c->h_table, count * sizeof(PayloadDesc),
                                       cudaMemcpyHostToDevice, s))) != GLEAM_OK)
      return rc;
    if ((rc = cuda_err(cudaEventRecord(c->table_copied, s))) != GLEAM_OK) return rc;
  }
  const uint64_t tcap =
      std::min<uint64_t>(c->tbl_cap, next_pow2(std::max<uint64_t>(64, 2 * Ntot)));
  // The group table and the control block start zeroed (at allocation) and
  // every call's dedup kernel leaves them zeroed for the next one.

  HashArgs h{};
  h.table = c->d_table;
  h.one = one;
  h.count = (uint32_t)count;
  h.Ntot = Ntot;
  h.C = c->C;
  h.fp_out = nullptr;
  h.index = c->index;
  h.index_mask = c->index_cap - 1;
  h.hints = c->hints;
  h.arena = c->arena;
  h.slot_key = c->slot_key;
  h.dstats = c->dstats;
  h.key16 = (c->flags & GLEAM_KEY16) ? 1u : 0u;
  h.paper = (c->flags & GLEAM_PAPER_IDS) ? 1u : 0u;
  h.ch = c->ch;
  h.ctl = c->ctl;
  // slots_bound: an upper bound of the used slots
  h.no_hints = c->slots_bound == 0 ||
                       (c->C <= kHintedMaxChunk && c->slots_bound * kHintedMinRatio < Ntot)
                   ? 1u : 0u;

  DedupArgs d{};
  d.table = c->d_table;
  d.one = one;
  d.count = (uint32_t)count;
  d.Ntot = Ntot;
  d.C = c->C;
  d.arena = c->arena;
  d.index = c->index;
  d.index_mask = c->index_cap - 1;
  d.hints = c->hints;
  d.nslots = c->nslots;
  d.slot_len = c->slot_len;
  d.slot_key = c->slot_key;
  d.dstats = c->dstats;
  d.ch = c->ch;
  d.pstart = count > 1 ? c->d_pstart : c->bcount + 2 * c->coop_max_blocks;
  d.paper = (c->flags & GLEAM_PAPER_IDS) ? 1u : 0u;
  d.key16 = (c->flags & GLEAM_KEY16) ? 1u : 0u;
  d.classes = d.key16 && !d.paper ? 1u : 0u;
  d.cls_tbl = c->cls_tbl;
  d.plain_copy = (host_payloads || chk.saw_managed()) ? 1u : 0u;
  d.tbl = c->tbl;
  d.tbl_mask = tcap - 1;
  d.bcount = c->bcount;
  d.ctl = c->ctl;
  // the call's result: the caller's device struct, else the library's own
  // (for gleam_dedup_copy, its page-locked one: read with no copy back)
  d.total = d_total ? d_total : own_total ? own_total : c->d_result;
  d.ncalls = ncalls;
  d.wait_ns = c->wait_ns;
  set_lru(c, &d, Ntot);
  d.skip_block = c->skip_block;
  c->skip_block = -1;  // the hook applies to one call
  int grid = dedup_grid(c, Ntot, nbytes);
  if (d.skip_block >= 0) {
    grid = std::max(grid, std::min(2, c->coop_max_blocks));  // someone must be left waiting
    if (d.skip_block >= grid) d.skip_block = grid - 1;
  }
  const bool fused = small_call(c, aligned, Ntot, nbytes, d.skip_block);
  const bool chain = chain_call(c, Ntot, nbytes, d.skip_block);
  // overlapping calls: the staged hash kernels fingerprint before they wait
  // (others ignore the field and wait first); the write-through stays off, as
  // it writes arena slots counted from a slot count that may still change
  h.wait_late = chain && (c->flags & GLEAM_OVERLAP_CALLS) && !(c->flags & GLEAM_PAPER_IDS) ? 1u : 0u;
  // host payloads too: a chunk written ahead then spares the pack a second
  // read over the CPU-GPU link (managed memory stays out)
  set_spec(c, &h, &d, aligned && packed_aligned && !chk.saw_managed() && !h.wait_late);
  // a payload resolved by the one-launch kernel: its staged hash kernel
  // claims the misses' groups as it records them
  const bool one_launch = !fused && chain && count == 1 && !d.classes;
  int rp_grid = 1;
  if (one_launch) {
    // at most one chunk per thread, and one block per kChainBytesPerBlock of
    // payload so that the misses' copies spread
    const bool solo = !(c->flags & GLEAM_OVERLAP_CALLS);
    const uint64_t per_block =
        solo || nbytes < kChainSmallCall ? kSoloBytesPerBlock : kChainBytesPerBlock;
    const uint64_t cap =
        solo ? (uint64_t)std::min(c->rp_max_blocks,
                                  std::max(kChainPackBlocks, c->coop_max_blocks / GLEAM_SOLO_CAP_DIV))
             : (uint64_t)kChainPackBlocks;
    const uint64_t want = std::max<uint64_t>((Ntot + dedup_threads() - 1) / dedup_threads(),
                                             (nbytes + per_block - 1) / per_block);
    rp_grid = (int)std::min<uint64_t>(std::max<uint64_t>(1, want), cap);
  }
  // (a grid of one block needs no barrier before its ranks anyway)
  // overlapping calls give the one-launch kernel few blocks (a block per
  // kChainBytesPerBlock): its warps then share the copies out as they go
  // (Llama-3-8B, one call per tensor: +1%, four layers of it: +3%), where an
  // equal share per warp suits the one-block-per-SM grid of a call on its own
  if (one_launch && rp_grid > 1 && (c->flags & GLEAM_OVERLAP_CALLS)) d.copy_grab = kOverlapCopyGrab;
  if (one_launch && rp_grid > 1 && hash_is_staged(h, aligned)) {
    h.claim_tbl = d.tbl;
    h.claim_mask = d.tbl_mask;
    d.pre_claimed = 1u;
  }

  cudaEvent_t ev[3] = {nullptr, nullptr, nullptr};
  if (c->profile) {
    while (c->ev_pool.size() < c->ev_used + 3) {
      cudaEvent_t e;
      if ((rc = cuda_err(cudaEventCreate(&e))) != GLEAM_OK) return rc;
      c->ev_pool.push_back(e);
    }
    for (int k = 0; k < 3; ++k) ev[k] = c->ev_pool[c->ev_used + k];
    c->ev_used += 3;
    cudaEventRecord(ev[0], s);
  }
  if (fused) {  // one kernel: all of its time is phase 0
    if ((rc = cuda_err(launch_small_call(h, d, s, chain))) != GLEAM_OK) return rc;
    if (ev[1]) cudaEventRecord(ev[1], s);
  } else {
    if ((rc = cuda_err(launch_hash(h, aligned, s, chain))) != GLEAM_OK) return rc;
    if (ev[1]) cudaEventRecord(ev[1], s);
    int pgrid = pack_grid(c, Ntot, nbytes);
    if (chain) {
      // one chunk per thread of the resolve kernel: a call of at most 256
      // chunks resolves in one block, without any grid-wide barrier
      grid = (int)std::min<uint64_t>(kChainDedupBlocks, (Ntot + 255) / 256);
      pgrid = std::min(pgrid, kChainPackBlocks);
    }
    if (one_launch) {
      rc = cuda_err(launch_resolve_pack(d, rp_grid, s));
    } else {
      rc = cuda_err(launch_dedup(d, grid, pgrid, s, chain));
    }
    if (rc != GLEAM_OK) {
      cudaMemsetAsync(c->ctl, 0, sizeof(DevCtl), s);  // the hash kernel may have flagged it
      if (d.pre_claimed)  // and claimed group entries
        cudaMemsetAsync(d.tbl, 0, (d.tbl_mask + 1) * sizeof(CallEntry), s);
      return rc;
    }
  }
  if (ev[2]) cudaEventRecord(ev[2], s);
  note_call(c, Ntot);
  if ((rc = enqueue_index_check(c, d, s)) != GLEAM_OK) return rc;
  return record_done(c, s, sid);
}

gleam_payload_t make_payload(const void* d_buf, size_t n, uint32_t* d_hit_mask,
                             uint32_t* d_miss_idx, void* d_miss_bytes, gleam_result_t* d_result) {
  gleam_payload_t p;
  p.d_buf = d_buf;
  p.n = n;
  p.d_hit_mask = d_hit_mask;
  p.d_miss_idx = d_miss_idx;
  p.d_miss_bytes = d_miss_bytes;
  p.d_result = d_result;
  p.d_chunk_slot = nullptr;
  return p;
}

// Device address of the allocation-free call's scratch array on the current
// GPU (defined with the entry point at the end of this file).
int noalloc_scratch(uint8_t** out);

}  // namespace

extern "C" {

const char* gleam_status_string(int status) {
  switch (status) {
    case GLEAM_OK: return "ok";
    case GLEAM_ERR_INVALID_ARG: return "invalid argument";
    case GLEAM_ERR_NOT_DEVICE_PTR: return "not a device pointer of the cache's GPU";
    case GLEAM_ERR_CUDA: return "CUDA error";
    case GLEAM_ERR_CAPACITY: return "cache capacity exceeded";
    case GLEAM_ERR_TIMEOUT: return "bounded device wait timed out";
    case GLEAM_ERR_NOMEM: return "device allocation failed";
    case GLEAM_ERR_INTERNAL: return "device consistency check failed";
    default: return "unknown status";
  }
}

int gleam_cache_create_ex(size_t capacity_bytes, size_t chunk_bytes, uint32_t flags,
                          gleam_cache_t** out) {
  if (out == nullptr) return GLEAM_ERR_INVALID_ARG;
  *out = nullptr;
  if (chunk_bytes < kMinChunk || chunk_bytes > kMaxChunk || chunk_bytes % 32 != 0)
    return GLEAM_ERR_INVALID_ARG;
  if ((flags & ~(GLEAM_KEY16 | GLEAM_DEBUG_CHECKS | GLEAM_PAPER_IDS | GLEAM_EVICT_LRU |
                 GLEAM_OVERLAP_CALLS)) != 0)
    return GLEAM_ERR_INVALID_ARG;
  const uint64_t nslots = capacity_bytes / chunk_bytes;
  if (nslots == 0 || nslots > 0xFFFFFFFEull) return GLEAM_ERR_INVALID_ARG;

  gleam_cache* c = new (std::nothrow) gleam_cache();
  if (!c) return GLEAM_ERR_NOMEM;
  if (cudaGetDevice(&c->device) != cudaSuccess) {
    cudaGetLastError();
    delete c;
    return GLEAM_ERR_CUDA;
  }
  c->capacity_bytes = capacity_bytes;
  c->C = chunk_bytes;
  c->nslots = nslots;
  c->flags = flags;
  c->index_cap = next_pow2(std::max<uint64_t>(1024, 2 * nslots));

  int rc = GLEAM_OK;
  auto step = [&](cudaError_t e) {
    if (rc == GLEAM_OK) rc = cuda_err(e);
  };
  step(cudaMalloc(&c->arena, nslots * chunk_bytes));
  step(cudaMalloc(&c->index, c->index_cap * sizeof(IndexEntry)));
  step(cudaMalloc(&c->hints, c->index_cap * sizeof(IndexEntry)));
  step(cudaMalloc(&c->slot_len, nslots * sizeof(uint32_t)));
  step(cudaMalloc(&c->slot_key, nslots * sizeof(unsigned long long)));
  step(cudaMalloc(&c->dstats, ST_COUNT * sizeof(unsigned long long)));
  if (flags & GLEAM_DEBUG_CHECKS) {
    step(cudaMalloc(&c->dbg_count, nslots * sizeof(uint32_t)));
    step(cudaMalloc(&c->dbg_flag, sizeof(uint32_t)));
  }
  if (flags & GLEAM_EVICT_LRU) {
    step(cudaMalloc(&c->last_use, nslots * sizeof(uint32_t)));
    step(cudaMalloc(&c->vflag, nslots));
    step(cudaMalloc(&c->victims, nslots * sizeof(uint32_t)));
    step(cudaMalloc(&c->bins, kLruBins * sizeof(uint32_t)));
  }
  step(cudaMalloc(&c->ctl, sizeof(DevCtl)));
  step(cudaMalloc(&c->spec_state, 2 * sizeof(uint32_t)));
  step(cudaHostAlloc(&c->spec_mirror, sizeof(uint32_t), cudaHostAllocMapped));
  step(cudaMalloc(&c->d_result, sizeof(gleam_result_t)));
  step(cudaHostAlloc(&c->h_result, sizeof(gleam_result_t), cudaHostAllocMapped));
  step(cudaHostGetDevicePointer(&c->h_result_dev, c->h_result, 0));
  step(cudaEventCreateWithFlags(&c->done, cudaEventDisableTiming));
  step(cudaEventCreateWithFlags(&c->table_copied, cudaEventDisableTiming));
  if (rc == GLEAM_OK) {
    int sms = 0;
    step(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device));
    const int per_sm = dedup_blocks_per_sm();
    c->coop_max_blocks = sms * per_sm;
    c->pack_max_blocks = sms * pack_blocks_per_sm();
    c->rp_max_blocks = sms * resolve_pack_blocks_per_sm();
    c->small_max_chunks = small_call_groups();
    if (c->coop_max_blocks <= 0 || c->pack_max_blocks <= 0 || c->rp_max_blocks < kChainPackBlocks)
      rc = GLEAM_ERR_CUDA;
  }
  // per-block miss and stored-miss counts, then one word used as the single
  // payload's start rank
  if (rc == GLEAM_OK)
    step(cudaMalloc(&c->bcount, (2 * c->coop_max_blocks + 1) * sizeof(uint32_t)));
  if (rc == GLEAM_OK) {
    step(cudaMemset(c->index, 0xFF, c->index_cap * sizeof(IndexEntry)));
    step(cudaMemset(c->hints, 0xFF, c->index_cap * sizeof(IndexEntry)));
    step(cudaMemset(c->dstats, 0, ST_COUNT * sizeof(unsigned long long)));
    step(cudaMemset(c->ctl, 0, sizeof(DevCtl)));
    const uint32_t spec0[2] = {1u, 0u};  // automatic write-through starts on
    step(cudaMemcpy(c->spec_state, spec0, sizeof(spec0), cudaMemcpyHostToDevice));
    if (rc == GLEAM_OK) *c->spec_mirror = 1u;
    if (flags & GLEAM_DEBUG_CHECKS) {
      step(cudaMemset(c->dbg_count, 0, nslots * sizeof(uint32_t)));
      step(cudaMemset(c->dbg_flag, 0, sizeof(uint32_t)));
    }
    if (flags & GLEAM_EVICT_LRU) {
      step(cudaMemset(c->last_use, 0, nslots * sizeof(uint32_t)));
      step(cudaMemset(c->vflag, 0, nslots));
      step(cudaMemset(c->bins, 0, kLruBins * sizeof(uint32_t)));
    }
    step(cudaEventRecord(c->done, nullptr));
    step(cudaEventRecord(c->table_copied, nullptr));
    step(cudaDeviceSynchronize());
  }
  // The allocation-free call's scratch array is looked up here, where the
  // device is current and allocating is allowed: the lookup may load this
  // file's device code on the GPU, which allocates the array.
  if (rc == GLEAM_OK) rc = noalloc_scratch(&c->na_scratch);
  if (rc == GLEAM_OK) step(load_hash_kernels());
  if (rc != GLEAM_OK) {
    destroy_cache(c);
    return rc;
  }
  *out = c;
  return GLEAM_OK;
}

int gleam_cache_create(size_t capacity_bytes, size_t chunk_bytes, gleam_cache_t** out) {
  return gleam_cache_create_ex(capacity_bytes, chunk_bytes, 0, out);
}

void gleam_cache_destroy(gleam_cache_t* cache) { destroy_cache(cache); }

int gleam_cache_reserve(gleam_cache_t* c, uint64_t max_chunks) {
  if (!c || max_chunks > kMaxChunks) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  return ensure_ws(c, max_chunks);
}

int gleam_fingerprint(const void* d_buf, size_t n, size_t chunk_bytes, uint64_t* d_out,
                      gleam_stream_t stream) {
  if (d_out == nullptr || (n > 0 && d_buf == nullptr)) return GLEAM_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return cuda_err(cudaErrorUnknown);
  uint64_t N, C;
  if (chunk_bytes == 0) {
    N = 1;
    C = n ? n : 1;
  } else {
    N = (n + chunk_bytes - 1) / chunk_bytes;
    C = chunk_bytes;
  }
  if (N == 0) return GLEAM_OK;
  if (N > kMaxChunks || C > 0xFFFFFFFFull) return GLEAM_ERR_INVALID_ARG;
  PtrChecker chk(dev);
  int rc;
  if ((rc = chk.check(d_out, N * 8)) != GLEAM_OK) return rc;
  if (n > 0 && (rc = chk.check(d_buf, n)) != GLEAM_OK) return rc;
  HashArgs h{};
  h.one.buf = static_cast<const uint8_t*>(d_buf);
  h.one.n = n;
  h.one.chunk_base = 0;
  h.one.nchunks = N;
  h.count = 1;
  h.Ntot = N;
  h.C = C;
  h.fp_out = reinterpret_cast<unsigned long long*>(d_out);
  const bool aligned = (reinterpret_cast<uintptr_t>(d_buf) % 16 == 0) && (N == 1 || C % 16 == 0);
  return cuda_err(launch_hash(h, aligned, reinterpret_cast<cudaStream_t>(stream)));
}

int gleam_dedup_copy_batch(gleam_cache_t* c, const gleam_payload_t* payloads, size_t count,
                           gleam_result_t* d_total, gleam_stream_t stream) {
  if (!c || (count > 0 && !payloads)) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  return enqueue(c, payloads, count, d_total, reinterpret_cast<cudaStream_t>(stream));
}

int gleam_dedup_copy_async(gleam_cache_t* c, const void* d_buf, size_t n, uint32_t* d_hit_mask,
                           uint32_t* d_miss_idx, void* d_miss_bytes, gleam_result_t* d_result,
                           gleam_stream_t stream) {
  if (!c) return GLEAM_ERR_INVALID_ARG;
  if (n == 0) return GLEAM_OK;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  const gleam_payload_t p = make_payload(d_buf, n, d_hit_mask, d_miss_idx, d_miss_bytes, d_result);
  return enqueue(c, &p, 1, nullptr, reinterpret_cast<cudaStream_t>(stream));
}

int64_t gleam_dedup_copy(gleam_cache_t* c, const void* d_buf, size_t n, uint32_t* d_hit_mask,
                         uint32_t* d_miss_idx, void* d_miss_bytes) {
  if (!c) return GLEAM_ERR_INVALID_ARG;
  if (n == 0) return 0;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  const gleam_payload_t p = make_payload(d_buf, n, d_hit_mask, d_miss_idx, d_miss_bytes, nullptr);
  // the last kernel writes the result straight into page-locked host memory
  int rc = enqueue(c, &p, 1, nullptr, nullptr, false, c->h_result_dev);
  if (rc != GLEAM_OK) return rc;
  rc = cuda_err(cudaStreamSynchronize(nullptr));
  if (rc != GLEAM_OK) return rc;
  const volatile gleam_result_t* r = c->h_result;
  if (r->status != 0) return r->status;
  return (int64_t)r->n_miss;
}

int gleam_dedup_copy_host_batch(gleam_cache_t* c, const gleam_payload_t* payloads, size_t count,
                                gleam_result_t* d_total, gleam_stream_t stream) {
  if (!c || (count > 0 && !payloads)) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  return enqueue(c, payloads, count, d_total, reinterpret_cast<cudaStream_t>(stream), true);
}

int gleam_dedup_copy_host_async(gleam_cache_t* c, const void* h_buf, size_t n,
                                uint32_t* d_hit_mask, uint32_t* d_miss_idx, void* d_miss_bytes,
                                gleam_result_t* d_result, gleam_stream_t stream) {
  if (!c) return GLEAM_ERR_INVALID_ARG;
  if (n == 0) return GLEAM_OK;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  const gleam_payload_t p = make_payload(h_buf, n, d_hit_mask, d_miss_idx, d_miss_bytes, d_result);
  return enqueue(c, &p, 1, nullptr, reinterpret_cast<cudaStream_t>(stream), true);
}

int gleam_block_check(const gleam_cache_t* c, const void* d_block, size_t block_bytes,
                      const uint64_t* d_offsets, const uint32_t* d_slots, size_t nrec,
                      uint8_t* d_mismatch, uint64_t* d_count, gleam_stream_t stream) {
  if (!c || !d_count) return GLEAM_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  PtrChecker chk(c->device);
  int rc;
  if ((rc = chk.check(d_count, sizeof(uint64_t))) != GLEAM_OK) return rc;
  if (nrec > 0) {
    if (block_bytes > 0 && (rc = chk.check(d_block, block_bytes)) != GLEAM_OK) return rc;
    if ((rc = chk.check(d_offsets, nrec * 8)) != GLEAM_OK) return rc;
    if ((rc = chk.check(d_slots, nrec * 4)) != GLEAM_OK) return rc;
    if (d_mismatch && (rc = chk.check(d_mismatch, nrec)) != GLEAM_OK) return rc;
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if ((rc = cuda_err(cudaStreamWaitEvent(s, c->done, 0))) != GLEAM_OK) return rc;
  if ((rc = cuda_err(cudaMemsetAsync(d_count, 0, sizeof(uint64_t), s))) != GLEAM_OK) return rc;
  BlockCheckArgs a{};
  a.block = static_cast<const uint8_t*>(d_block);
  a.block_bytes = block_bytes;
  a.offsets = reinterpret_cast<const unsigned long long*>(d_offsets);
  a.slots = d_slots;
  a.nrec = nrec;
  a.mismatch = d_mismatch;
  a.count = reinterpret_cast<unsigned long long*>(d_count);
  a.arena = c->arena;
  a.slot_len = c->slot_len;
  a.dstats = c->dstats;
  a.C = c->C;
  return cuda_err(launch_block_check(a, s));
}

int gleam_cache_stats(const gleam_cache_t* c, gleam_stats_t* out) {
  if (!c || !out) return GLEAM_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  int rc = wait_done(c);
  if (rc != GLEAM_OK) return rc;
  unsigned long long s[ST_COUNT];
  rc = cuda_err(cudaMemcpy(s, c->dstats, sizeof(s), cudaMemcpyDeviceToHost));
  if (rc != GLEAM_OK) return rc;
  out->calls = s[ST_CALLS];
  out->chunks = s[ST_CHUNKS];
  out->hits_cache = s[ST_HITS_CACHE];
  out->hits_intra = s[ST_HITS_INTRA];
  out->misses = s[ST_MISSES];
  out->inserts = s[ST_INSERTS];
  out->verify_rejects = s[ST_REJECTS];
  out->slots_used = s[ST_SLOTS_USED];
  out->bytes_used = s[ST_BYTES_USED];
  out->evictions = s[ST_EVICTIONS];
  out->spec_chunks = s[ST_SPEC_CHUNKS];
  out->capacity_bytes = c->capacity_bytes;
  out->nslots = c->nslots;
  out->chunk_bytes = c->C;
  return GLEAM_OK;
}

int gleam_cache_export(const gleam_cache_t* c, uint64_t* h_keys, uint32_t* h_lens, uint64_t max,
                       uint64_t* count) {
  if (!c || !count || (max > 0 && (!h_keys || !h_lens))) return GLEAM_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  int rc = wait_done(c);
  if (rc != GLEAM_OK) return rc;
  std::vector<IndexEntry> host(c->index_cap);
  rc = cuda_err(cudaMemcpy(host.data(), c->index, c->index_cap * sizeof(IndexEntry),
                           cudaMemcpyDeviceToHost));
  if (rc != GLEAM_OK) return rc;
  uint64_t cnt = 0;
  for (const IndexEntry& e : host) {
    if (e.slot == kEmptySlot) continue;
    ++cnt;
    if (e.slot < max) {
      h_keys[e.slot] = e.key;
      h_lens[e.slot] = e.len;
    }
  }
  *count = cnt;
  return GLEAM_OK;
}

int gleam_cache_read_slot(const gleam_cache_t* c, uint64_t slot, void* h_out, uint64_t max,
                          uint64_t* len) {
  if (!c || !len || (max > 0 && !h_out)) return GLEAM_ERR_INVALID_ARG;
  DeviceGuard g(c->device);
  int rc = wait_done(c);
  if (rc != GLEAM_OK) return rc;
  unsigned long long used = 0;
  rc = cuda_err(cudaMemcpy(&used, c->dstats + ST_SLOTS_USED, sizeof(used), cudaMemcpyDeviceToHost));
  if (rc != GLEAM_OK) return rc;
  if (slot >= used) return GLEAM_ERR_INVALID_ARG;
  uint32_t l = 0;
  rc = cuda_err(cudaMemcpy(&l, c->slot_len + slot, sizeof(l), cudaMemcpyDeviceToHost));
  if (rc != GLEAM_OK) return rc;
  *len = l;
  const uint64_t m = std::min<uint64_t>(l, max);
  if (m) rc = cuda_err(cudaMemcpy(h_out, c->arena + slot * c->C, m, cudaMemcpyDeviceToHost));
  return rc;
}

int gleam_cache_debug_insert(gleam_cache_t* c, uint64_t key, const void* d_bytes, size_t len) {
  if (!c || len == 0 || len > c->C) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  PtrChecker chk(c->device);
  int rc = chk.check(d_bytes, len);
  if (rc != GLEAM_OK) return rc;
  if ((rc = wait_done(c)) != GLEAM_OK) return rc;
  unsigned long long used = 0;
  rc = cuda_err(cudaMemcpy(&used, c->dstats + ST_SLOTS_USED, sizeof(used), cudaMemcpyDeviceToHost));
  if (rc != GLEAM_OK) return rc;
  if (used >= c->nslots) return GLEAM_ERR_CAPACITY;
  const unsigned long long k = (c->flags & GLEAM_KEY16) ? (key & 0xFFFFull) : key;
  rc = cuda_err(cudaMemcpy(c->arena + used * c->C, d_bytes, len, cudaMemcpyDeviceToDevice));
  if (rc == GLEAM_OK)
    rc = cuda_err(launch_debug_insert(c->index, c->index_cap - 1, c->slot_len, c->slot_key,
                                      c->dstats, k,
                                      (uint32_t)used, (uint32_t)len, c->ctl, c->last_use,
                                      c->last_use ? ++c->epoch : 0u, nullptr));
  if (rc == GLEAM_OK) rc = cuda_err(cudaDeviceSynchronize());
  if (rc == GLEAM_OK) rc = record_done(c, nullptr, stream_id(nullptr));
  if (rc == GLEAM_OK) note_call(c, 1);
  return rc;
}

int gleam_cache_debug_set(gleam_cache_t* c, int what, int64_t value) {
  if (!c) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  if (what == GLEAM_DEBUG_WAIT_LIMIT_NS) {
    if (value <= 0) return GLEAM_ERR_INVALID_ARG;
    c->wait_ns = (unsigned long long)value;
    return GLEAM_OK;
  }
  if (what == GLEAM_DEBUG_SKIP_ARRIVE) {
    c->skip_block = (int)value;
    return GLEAM_OK;
  }
  if (what == GLEAM_DEBUG_DROP_ENTRY) {  // damage the index on purpose (host side)
    DeviceGuard g(c->device);
    int rc = wait_done(c);
    if (rc != GLEAM_OK) return rc;
    std::vector<IndexEntry> host(c->index_cap);
    rc = cuda_err(cudaMemcpy(host.data(), c->index, c->index_cap * sizeof(IndexEntry),
                             cudaMemcpyDeviceToHost));
    if (rc != GLEAM_OK) return rc;
    for (uint64_t q = 0; q < c->index_cap; ++q)
      if (host[q].slot == (uint64_t)value) {
        const uint32_t empty = kEmptySlot;
        return cuda_err(cudaMemcpy(&c->index[q].slot, &empty, sizeof(empty),
                                   cudaMemcpyHostToDevice));
      }
    return GLEAM_ERR_INVALID_ARG;
  }
  if (what == GLEAM_DEBUG_SPECULATE) {
    if (value < 0 || value > 2) return GLEAM_ERR_INVALID_ARG;
    c->spec_hook = (int)value;
    return GLEAM_OK;
  }
  if (what == GLEAM_DEBUG_SMALL_CALLS) {
    if (value < 0 || value > (int64_t)kMaxChunks) return GLEAM_ERR_INVALID_ARG;
    c->small_max_chunks = (uint64_t)value;
    return GLEAM_OK;
  }
  if (what == GLEAM_DEBUG_CLOCK) {
    if (value < 0 || value > 0xFFFFFFFEll) return GLEAM_ERR_INVALID_ARG;
    c->epoch = (uint32_t)value;
    return GLEAM_OK;
  }
  return GLEAM_ERR_INVALID_ARG;
}

int gleam_cache_profile(gleam_cache_t* c, int enable) {
  if (!c) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  c->profile = enable != 0;
  return GLEAM_OK;
}

int gleam_cache_profile_read(gleam_cache_t* c, double* h_ms, uint64_t* h_launches, int nkernels) {
  if (!c || nkernels < 0 || (nkernels > 0 && (!h_ms || !h_launches))) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  int rc = wait_done(c);
  if (rc != GLEAM_OK) return rc;
  double ms[2] = {0.0, 0.0};
  for (size_t k = 0; k + 3 <= c->ev_used; k += 3) {
    float a = 0.f, b = 0.f;
    if ((rc = cuda_err(cudaEventElapsedTime(&a, c->ev_pool[k], c->ev_pool[k + 1]))) != GLEAM_OK)
      return rc;
    if ((rc = cuda_err(cudaEventElapsedTime(&b, c->ev_pool[k + 1], c->ev_pool[k + 2]))) != GLEAM_OK)
      return rc;
    ms[0] += a;
    ms[1] += b;
  }
  const uint64_t calls = c->ev_used / 3;
  for (int k = 0; k < nkernels; ++k) {
    h_ms[k] = k < 2 ? ms[k] : 0.0;
    h_launches[k] = k < 2 ? calls : 0;
  }
  c->ev_used = 0;
  return GLEAM_OK;
}

int gleam_cache_snapshot(gleam_cache_t* c, gleam_snapshot_t** out) {
  if (!c || !out) return GLEAM_ERR_INVALID_ARG;
  *out = nullptr;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  int rc = wait_done(c);
  if (rc != GLEAM_OK) return rc;
  gleam_snapshot* s = new (std::nothrow) gleam_snapshot();
  if (!s) return GLEAM_ERR_NOMEM;
  s->device = c->device;
  s->owner = c;
  s->index_cap = c->index_cap;
  s->slots_bound = c->slots_bound;
  rc = cuda_err(cudaMalloc(&s->index, c->index_cap * sizeof(IndexEntry)));
  if (rc == GLEAM_OK) rc = cuda_err(cudaMalloc(&s->hints, c->index_cap * sizeof(IndexEntry)));
  if (rc == GLEAM_OK) rc = cuda_err(cudaMalloc(&s->dstats, ST_COUNT * sizeof(unsigned long long)));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpy(s->index, c->index, c->index_cap * sizeof(IndexEntry),
                             cudaMemcpyDeviceToDevice));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpy(s->hints, c->hints, c->index_cap * sizeof(IndexEntry),
                             cudaMemcpyDeviceToDevice));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpy(s->dstats, c->dstats, ST_COUNT * sizeof(unsigned long long),
                             cudaMemcpyDeviceToDevice));
  if (rc == GLEAM_OK && c->last_use) {
    s->nslots = c->nslots;
    rc = cuda_err(cudaMalloc(&s->slot_len, c->nslots * sizeof(uint32_t)));
    if (rc == GLEAM_OK)
      rc = cuda_err(cudaMalloc(&s->slot_key, c->nslots * sizeof(unsigned long long)));
    if (rc == GLEAM_OK) rc = cuda_err(cudaMalloc(&s->last_use, c->nslots * sizeof(uint32_t)));
    if (rc == GLEAM_OK)
      rc = cuda_err(cudaMemcpy(s->slot_key, c->slot_key, c->nslots * sizeof(unsigned long long),
                               cudaMemcpyDeviceToDevice));
    if (rc == GLEAM_OK)
      rc = cuda_err(cudaMemcpy(s->slot_len, c->slot_len, c->nslots * sizeof(uint32_t),
                               cudaMemcpyDeviceToDevice));
    if (rc == GLEAM_OK)
      rc = cuda_err(cudaMemcpy(s->last_use, c->last_use, c->nslots * sizeof(uint32_t),
                               cudaMemcpyDeviceToDevice));
  }
  if (rc != GLEAM_OK) {
    gleam_snapshot_destroy(s);
    return rc;
  }
  *out = s;
  return GLEAM_OK;
}

// Stream-ordered on the legacy default stream: it orders after the cache's
// previous call, and later calls on blocking streams see the restored state.
int gleam_cache_restore(gleam_cache_t* c, const gleam_snapshot_t* s) {
  if (!c || !s || s->owner != c || s->index_cap != c->index_cap) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  int rc = cuda_err(cudaStreamWaitEvent(nullptr, c->done, 0));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpyAsync(c->index, s->index, c->index_cap * sizeof(IndexEntry),
                                  cudaMemcpyDeviceToDevice, nullptr));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpyAsync(c->hints, s->hints, c->index_cap * sizeof(IndexEntry),
                                  cudaMemcpyDeviceToDevice, nullptr));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpyAsync(c->dstats, s->dstats, ST_COUNT * sizeof(unsigned long long),
                                  cudaMemcpyDeviceToDevice, nullptr));
  if (rc == GLEAM_OK && s->last_use) {
    rc = cuda_err(cudaMemcpyAsync(c->slot_len, s->slot_len, s->nslots * sizeof(uint32_t),
                                  cudaMemcpyDeviceToDevice, nullptr));
    if (rc == GLEAM_OK)
      rc = cuda_err(cudaMemcpyAsync(c->slot_key, s->slot_key,
                                    s->nslots * sizeof(unsigned long long),
                                    cudaMemcpyDeviceToDevice, nullptr));
    if (rc == GLEAM_OK)
      rc = cuda_err(cudaMemcpyAsync(c->last_use, s->last_use, s->nslots * sizeof(uint32_t),
                                    cudaMemcpyDeviceToDevice, nullptr));
  }
  if (rc == GLEAM_OK) {
    c->slots_bound = s->slots_bound;
    rc = record_done(c, nullptr, stream_id(nullptr));
  }
  return rc;
}

void gleam_snapshot_destroy(gleam_snapshot_t* s) {
  if (!s) return;
  DeviceGuard g(s->device);
  cudaDeviceSynchronize();
  if (s->index) cudaFree(s->index);
  if (s->hints) cudaFree(s->hints);
  if (s->dstats) cudaFree(s->dstats);
  if (s->slot_len) cudaFree(s->slot_len);
  if (s->slot_key) cudaFree(s->slot_key);
  if (s->last_use) cudaFree(s->last_use);
  cudaGetLastError();
  delete s;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Dedup without allocation (gleam_dedup_copy_noalloc)
//
// For callers that must not allocate device memory while they run -- typically
// code that executes inside an intercepted CUDA call, such as the server side
// of an API-remoting layer handling a host-to-device copy, where calling
// cudaMalloc again would re-enter the interception or disturb the memory map
// it keeps for the application.  The per-call workspace of the normal path
// (grown with cudaMalloc on demand) is replaced here by one fixed array in the
// library's device image, so a call only launches kernels and memsets.
// ---------------------------------------------------------------------------
namespace {

constexpr uint64_t kNaChunks = GLEAM_NOALLOC_MAX_CHUNKS;  // chunks per call, at most
constexpr uint64_t kNaTable = 2 * kNaChunks;               // group-table entries (power of 2)
constexpr uint64_t kNaBlocks = 4096;                       // block-count words

constexpr uint64_t na_align(uint64_t x) { return (x + 255) & ~255ull; }
constexpr uint64_t kNaOffStatus = 0;
constexpr uint64_t kNaOffKey = kNaOffStatus + na_align(kNaChunks);
constexpr uint64_t kNaOffLen = kNaOffKey + na_align(kNaChunks * 8);
constexpr uint64_t kNaOffSrc = kNaOffLen + na_align(kNaChunks * 4);
constexpr uint64_t kNaOffPidx = kNaOffSrc + na_align(kNaChunks * 8);
constexpr uint64_t kNaOffRes = kNaOffPidx + na_align(kNaChunks * 4);
constexpr uint64_t kNaOffEnt = kNaOffRes + na_align(kNaChunks * 4);
constexpr uint64_t kNaOffRank = kNaOffEnt + na_align(kNaChunks * 4);
constexpr uint64_t kNaOffHint = kNaOffRank + na_align(kNaChunks * 4);
constexpr uint64_t kNaOffOrder = kNaOffHint + na_align(kNaChunks * 8);
constexpr uint64_t kNaOffSrank = kNaOffOrder + na_align(kNaChunks * 4);
constexpr uint64_t kNaOffOld = kNaOffSrank + na_align(kNaChunks * 4);
constexpr uint64_t kNaOffSpec = kNaOffOld + na_align(kNaChunks * 4);
constexpr uint64_t kNaOffTbl = kNaOffSpec + na_align(kNaChunks);
constexpr uint64_t kNaOffCls = kNaOffTbl + na_align(kNaTable * sizeof(CallEntry));
constexpr uint64_t kNaOffClsTbl = kNaOffCls + na_align(kNaChunks * 8);
constexpr uint64_t kNaOffCtl = kNaOffClsTbl + na_align(kNaTable * sizeof(ClassEntry));
constexpr uint64_t kNaOffBcount = kNaOffCtl + na_align(sizeof(DevCtl));
constexpr uint64_t kNaOffResult = kNaOffBcount + na_align((2 * kNaBlocks + 1) * 4);
constexpr uint64_t kNaBytes = kNaOffResult + na_align(sizeof(gleam_result_t));  // ~7.2 MiB

}  // namespace

// The scratch of every gleam_dedup_copy_noalloc call on this GPU.  Host code
// must not use this name as an address: it stands for the host-side shadow.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNaBytes];

namespace {

// Looks the array up on the current device.  Every cache keeps its own copy
// of the address, so nothing outlives the context the cache was made in.
int noalloc_scratch(uint8_t** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess || p == nullptr) return cuda_err(e == cudaSuccess ? cudaErrorUnknown : e);
  *out = static_cast<uint8_t*>(p);
  return GLEAM_OK;
}

}  // namespace

extern "C" int gleam_dedup_copy_noalloc(gleam_cache_t* c, const void* d_buf, size_t n,
                                        uint32_t* d_hit_mask, uint32_t* d_miss_idx,
                                        void* d_miss_bytes, gleam_result_t* d_result,
                                        gleam_stream_t stream) {
  if (!c) return GLEAM_ERR_INVALID_ARG;
  if (n == 0) return GLEAM_OK;
  const uint64_t N = (n + c->C - 1) / c->C;
  if (N > kNaChunks) return GLEAM_ERR_INVALID_ARG;  // beyond the fixed scratch
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  if ((uint64_t)c->coop_max_blocks + 1 > kNaBlocks) return GLEAM_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint8_t* const base = c->na_scratch;
  if (base == nullptr) return GLEAM_ERR_INTERNAL;

  const gleam_payload_t p = make_payload(d_buf, n, d_hit_mask, d_miss_idx, d_miss_bytes, d_result);
  PtrChecker chk(c->device);
  PayloadDesc one{};
  int rc;
  if ((rc = describe(c, chk, p, &one)) != GLEAM_OK) return rc;
  const bool aligned = reinterpret_cast<uintptr_t>(one.buf) % 16 == 0;

  ChunkArrays ch{};
  ch.status = base + kNaOffStatus;
  ch.key = reinterpret_cast<unsigned long long*>(base + kNaOffKey);
  ch.len = reinterpret_cast<uint32_t*>(base + kNaOffLen);
  ch.src = reinterpret_cast<unsigned long long*>(base + kNaOffSrc);
  ch.pidx = reinterpret_cast<uint32_t*>(base + kNaOffPidx);
  ch.res = reinterpret_cast<uint32_t*>(base + kNaOffRes);
  ch.ent = reinterpret_cast<uint32_t*>(base + kNaOffEnt);
  ch.rank = reinterpret_cast<uint32_t*>(base + kNaOffRank);
  ch.hint = reinterpret_cast<unsigned long long*>(base + kNaOffHint);
  ch.order = reinterpret_cast<uint32_t*>(base + kNaOffOrder);
  ch.srank = reinterpret_cast<uint32_t*>(base + kNaOffSrank);
  ch.old = reinterpret_cast<uint32_t*>(base + kNaOffOld);
  ch.spec = base + kNaOffSpec;
  ch.cls = reinterpret_cast<unsigned long long*>(base + kNaOffCls);
  CallEntry* tbl = reinterpret_cast<CallEntry*>(base + kNaOffTbl);
  ClassEntry* cls_tbl = reinterpret_cast<ClassEntry*>(base + kNaOffClsTbl);
  DevCtl* ctl = reinterpret_cast<DevCtl*>(base + kNaOffCtl);
  uint32_t* bcount = reinterpret_cast<uint32_t*>(base + kNaOffBcount);
  gleam_result_t* total = reinterpret_cast<gleam_result_t*>(base + kNaOffResult);
  const uint64_t tcap = std::min<uint64_t>(kNaTable, next_pow2(std::max<uint64_t>(64, 2 * N)));

  // the array keeps the previous call's contents: clear what must start at zero
  unsigned long long sid = ~0ull;
  if ((rc = order_after_done(c, s, &sid)) != GLEAM_OK) return rc;
  if ((rc = cuda_err(cudaMemsetAsync(ctl, 0, sizeof(DevCtl), s))) != GLEAM_OK) return rc;
  if ((rc = cuda_err(cudaMemsetAsync(tbl, 0, tcap * sizeof(CallEntry), s))) != GLEAM_OK) return rc;
  const bool classes = (c->flags & GLEAM_KEY16) && !(c->flags & GLEAM_PAPER_IDS);
  if (classes &&
      (rc = cuda_err(cudaMemsetAsync(cls_tbl, 0, tcap * sizeof(ClassEntry), s))) != GLEAM_OK)
    return rc;

  HashArgs h{};
  h.one = one;
  h.count = 1;
  h.Ntot = N;
  h.C = c->C;
  h.index = c->index;
  h.index_mask = c->index_cap - 1;
  h.hints = c->hints;
  h.arena = c->arena;
  h.slot_key = c->slot_key;
  h.dstats = c->dstats;
  h.key16 = (c->flags & GLEAM_KEY16) ? 1u : 0u;
  h.paper = (c->flags & GLEAM_PAPER_IDS) ? 1u : 0u;
  h.ch = ch;
  h.ctl = ctl;
  h.no_hints = c->slots_bound == 0 ||
                       (c->C <= kHintedMaxChunk && c->slots_bound * kHintedMinRatio < N)
                   ? 1u : 0u;

  DedupArgs d{};
  d.one = one;
  d.count = 1;
  d.Ntot = N;
  d.C = c->C;
  d.arena = c->arena;
  d.index = c->index;
  d.index_mask = c->index_cap - 1;
  d.hints = c->hints;
  d.nslots = c->nslots;
  d.slot_len = c->slot_len;
  d.slot_key = c->slot_key;
  d.dstats = c->dstats;
  d.ch = ch;
  d.pstart = bcount + 2 * kNaBlocks;
  d.paper = (c->flags & GLEAM_PAPER_IDS) ? 1u : 0u;
  d.key16 = (c->flags & GLEAM_KEY16) ? 1u : 0u;
  d.classes = classes ? 1u : 0u;
  d.cls_tbl = cls_tbl;
  d.tbl = tbl;
  d.tbl_mask = tcap - 1;
  d.bcount = bcount;
  d.ctl = ctl;
  d.total = total;
  d.ncalls = 1;
  d.wait_ns = c->wait_ns;
  d.plain_copy = chk.saw_managed() ? 1u : 0u;
  set_lru(c, &d, N);
  d.skip_block = c->skip_block;  // the test hook applies to this one call, as in enqueue()
  c->skip_block = -1;
  int grid = dedup_grid(c, N, n);
  if (d.skip_block >= 0) {
    grid = std::max(grid, std::min(2, c->coop_max_blocks));  // someone must be left waiting
    if (d.skip_block >= grid) d.skip_block = grid - 1;
  }
  set_spec(c, &h, &d,
           aligned && reinterpret_cast<uintptr_t>(one.packed) % 16 == 0 && !d.plain_copy);
  if (small_call(c, aligned, N, n, d.skip_block)) {
    if ((rc = cuda_err(launch_small_call(h, d, s))) != GLEAM_OK) return rc;
  } else {
    if ((rc = cuda_err(launch_hash(h, aligned, s))) != GLEAM_OK) return rc;
    if ((rc = cuda_err(launch_dedup(d, grid, pack_grid(c, N, n), s))) != GLEAM_OK) return rc;
  }
  note_call(c, N);
  if ((rc = enqueue_index_check(c, d, s)) != GLEAM_OK) return rc;
  return record_done(c, s, sid);
}
