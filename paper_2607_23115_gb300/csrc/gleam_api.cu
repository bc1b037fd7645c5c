// Host side of the C ABI declared in include/gleam.h: argument checks, the
// cache object (arena, index, counters, per-call workspace) and the launch
// sequence of one dedup call.  Every step of the path runs in the kernels of
// hash_probe.cu and dedup_compact.cu; nothing here touches payload bytes.
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
  uint64_t index_cap = 0;  // power of two >= 2 * nslots
  uint32_t* slot_len = nullptr;
  unsigned long long* dstats = nullptr;

  // per-call workspace
  uint64_t ws_chunks = 0;
  void* ws = nullptr;
  uint8_t* status = nullptr;
  unsigned long long* key = nullptr;
  uint32_t* res = nullptr;
  uint32_t* ent = nullptr;
  CallEntry* tbl = nullptr;
  uint64_t tbl_cap = 0;

  DevCtl* ctl = nullptr;
  uint32_t* bcount = nullptr;
  gleam_result_t* d_result = nullptr;
  gleam_result_t* h_result = nullptr;  // pinned
  int coop_max_blocks = 0;
  cudaEvent_t done = nullptr;

  unsigned long long wait_ns = 4000000000ULL;
  int skip_block = -1;

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
  uint64_t index_cap = 0;
  unsigned long long* dstats = nullptr;
};

namespace {

constexpr uint64_t kMinChunk = 32;
constexpr uint64_t kMaxChunk = 16ull << 20;

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

// GLEAM_OK iff p is device memory of `device` (or managed memory).
int check_device_ptr(const void* p, int device) {
  if (p == nullptr) return GLEAM_ERR_INVALID_ARG;
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return GLEAM_ERR_NOT_DEVICE_PTR;
  }
  if (at.type == cudaMemoryTypeManaged) return GLEAM_OK;
  if (at.type == cudaMemoryTypeDevice && at.device == device) return GLEAM_OK;
  return GLEAM_ERR_NOT_DEVICE_PTR;
}

void free_ws(gleam_cache* c) {
  if (c->ws) cudaFree(c->ws);
  c->ws = nullptr;
  c->ws_chunks = 0;
  c->tbl_cap = 0;
}

// Grows the per-call workspace to hold `nchunks` chunks (synchronises `s`).
int ensure_ws(gleam_cache* c, uint64_t nchunks, cudaStream_t s) {
  if (nchunks <= c->ws_chunks) return GLEAM_OK;
  uint64_t cap = std::max<uint64_t>({nchunks, 2 * c->ws_chunks, 4096});
  cap = std::min<uint64_t>(cap, 0xFFFFFFFFull);
  if (cap < nchunks) cap = nchunks;
  const uint64_t tcap = next_pow2(2 * cap);
  const uint64_t sz_status = align256(cap);
  const uint64_t sz_key = align256(cap * 8);
  const uint64_t sz_res = align256(cap * 4);
  const uint64_t sz_ent = align256(cap * 4);
  const uint64_t sz_tbl = align256(tcap * sizeof(CallEntry));
  if (s != nullptr) cudaStreamSynchronize(s);
  cudaStreamSynchronize(nullptr);
  free_ws(c);
  void* p = nullptr;
  int rc = cuda_err(cudaMalloc(&p, sz_status + sz_key + sz_res + sz_ent + sz_tbl));
  if (rc != GLEAM_OK) return rc;
  uint8_t* b = static_cast<uint8_t*>(p);
  c->ws = p;
  c->status = b;
  c->key = reinterpret_cast<unsigned long long*>(b + sz_status);
  c->res = reinterpret_cast<uint32_t*>(b + sz_status + sz_key);
  c->ent = reinterpret_cast<uint32_t*>(b + sz_status + sz_key + sz_res);
  c->tbl = reinterpret_cast<CallEntry*>(b + sz_status + sz_key + sz_res + sz_ent);
  c->tbl_cap = tcap;
  c->ws_chunks = cap;
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
    if (c->slot_len) cudaFree(c->slot_len);
    if (c->dstats) cudaFree(c->dstats);
    if (c->ctl) cudaFree(c->ctl);
    if (c->bcount) cudaFree(c->bcount);
    if (c->d_result) cudaFree(c->d_result);
    if (c->h_result) cudaFreeHost(c->h_result);
    if (c->done) cudaEventDestroy(c->done);
    for (cudaEvent_t e : c->ev_pool) cudaEventDestroy(e);
    cudaGetLastError();
  }
  delete c;
}

int wait_done(const gleam_cache* c) {
  return cuda_err(cudaEventSynchronize(c->done));
}

// Enqueues one dedup call on stream s.  Caller holds c->mu and the device.
int enqueue_dedup(gleam_cache* c, const void* d_buf, size_t n, uint32_t* d_hit_mask,
                  uint32_t* d_miss_idx, void* d_miss_bytes, gleam_result_t* d_result,
                  cudaStream_t s) {
  const uint64_t N = (n + c->C - 1) / c->C;
  if (N >= 0xFFFFFFFFull) return GLEAM_ERR_INVALID_ARG;
  int rc;
  if ((rc = check_device_ptr(d_buf, c->device)) != GLEAM_OK) return rc;
  if ((rc = check_device_ptr(d_hit_mask, c->device)) != GLEAM_OK) return rc;
  if ((rc = check_device_ptr(d_miss_idx, c->device)) != GLEAM_OK) return rc;
  if ((rc = check_device_ptr(d_miss_bytes, c->device)) != GLEAM_OK) return rc;
  if (d_result && (rc = check_device_ptr(d_result, c->device)) != GLEAM_OK) return rc;
  if ((rc = ensure_ws(c, N, s)) != GLEAM_OK) return rc;

  const uint64_t tcap = std::min<uint64_t>(c->tbl_cap, next_pow2(std::max<uint64_t>(64, 2 * N)));
  if ((rc = cuda_err(cudaMemsetAsync(c->ctl, 0, sizeof(DevCtl), s))) != GLEAM_OK) return rc;
  if ((rc = cuda_err(cudaMemsetAsync(c->tbl, 0, tcap * sizeof(CallEntry), s))) != GLEAM_OK)
    return rc;

  HashArgs h{};
  h.buf = static_cast<const uint8_t*>(d_buf);
  h.n = n;
  h.C = c->C;
  h.N = (uint32_t)N;
  h.fp_out = nullptr;
  h.index = c->index;
  h.index_mask = c->index_cap - 1;
  h.arena = c->arena;
  h.dstats = c->dstats;
  h.key16 = (c->flags & GLEAM_KEY16) ? 1u : 0u;
  h.status = c->status;
  h.key_out = c->key;
  h.ctl = c->ctl;
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
  if ((rc = cuda_err(launch_hash(h, s))) != GLEAM_OK) return rc;
  if (ev[1]) cudaEventRecord(ev[1], s);

  DedupArgs d{};
  d.buf = h.buf;
  d.n = n;
  d.C = c->C;
  d.N = (uint32_t)N;
  d.mask = d_hit_mask;
  d.miss_idx = d_miss_idx;
  d.packed = static_cast<uint8_t*>(d_miss_bytes);
  d.arena = c->arena;
  d.index = c->index;
  d.index_mask = c->index_cap - 1;
  d.nslots = c->nslots;
  d.slot_len = c->slot_len;
  d.dstats = c->dstats;
  d.status = c->status;
  d.key = c->key;
  d.res = c->res;
  d.ent = c->ent;
  d.tbl = c->tbl;
  d.tbl_mask = tcap - 1;
  d.bcount = c->bcount;
  d.ctl = c->ctl;
  d.result = d_result ? d_result : c->d_result;
  d.wait_ns = c->wait_ns;
  d.skip_block = c->skip_block;
  c->skip_block = -1;  // the hook applies to one call
  const int per_block = 4 * dedup_threads();
  int grid = (int)std::max<uint64_t>(
      1, std::min<uint64_t>(c->coop_max_blocks, (N + per_block - 1) / per_block));
  if (d.skip_block >= 0) {
    grid = std::max(grid, std::min(2, c->coop_max_blocks));  // someone must be left waiting
    if (d.skip_block >= grid) d.skip_block = grid - 1;
  }
  if ((rc = cuda_err(launch_dedup(d, grid, s))) != GLEAM_OK) return rc;
  if (ev[2]) cudaEventRecord(ev[2], s);
  return cuda_err(cudaEventRecord(c->done, s));
}

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
  if ((flags & ~(GLEAM_KEY16 | GLEAM_DEBUG_CHECKS)) != 0) return GLEAM_ERR_INVALID_ARG;
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
  step(cudaMalloc(&c->slot_len, nslots * sizeof(uint32_t)));
  step(cudaMalloc(&c->dstats, ST_COUNT * sizeof(unsigned long long)));
  step(cudaMalloc(&c->ctl, sizeof(DevCtl)));
  step(cudaMalloc(&c->d_result, sizeof(gleam_result_t)));
  step(cudaMallocHost(&c->h_result, sizeof(gleam_result_t)));
  step(cudaEventCreateWithFlags(&c->done, cudaEventDisableTiming));
  if (rc == GLEAM_OK) {
    int sms = 0;
    step(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device));
    const int per_sm = std::min(2, dedup_blocks_per_sm());
    c->coop_max_blocks = sms * per_sm;
    if (c->coop_max_blocks <= 0) rc = GLEAM_ERR_CUDA;
  }
  if (rc == GLEAM_OK) step(cudaMalloc(&c->bcount, c->coop_max_blocks * sizeof(uint32_t)));
  if (rc == GLEAM_OK) {
    step(cudaMemset(c->index, 0xFF, c->index_cap * sizeof(IndexEntry)));
    step(cudaMemset(c->dstats, 0, ST_COUNT * sizeof(unsigned long long)));
    step(cudaMemset(c->ctl, 0, sizeof(DevCtl)));
    step(cudaEventRecord(c->done, nullptr));
    step(cudaDeviceSynchronize());
  }
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
  if (!c || max_chunks >= 0xFFFFFFFFull) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  int rc = wait_done(c);
  if (rc != GLEAM_OK) return rc;
  return ensure_ws(c, max_chunks, nullptr);
}

int gleam_fingerprint(const void* d_buf, size_t n, size_t chunk_bytes, uint64_t* d_out,
                      gleam_stream_t stream) {
  if (d_out == nullptr || (n > 0 && d_buf == nullptr)) return GLEAM_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return cuda_err(cudaErrorUnknown);
  int rc;
  if ((rc = check_device_ptr(d_out, dev)) != GLEAM_OK) return rc;
  if (n > 0 && (rc = check_device_ptr(d_buf, dev)) != GLEAM_OK) return rc;
  uint64_t N, C;
  if (chunk_bytes == 0) {
    N = 1;
    C = n ? n : 1;
  } else {
    N = (n + chunk_bytes - 1) / chunk_bytes;
    C = chunk_bytes;
  }
  if (N == 0) return GLEAM_OK;
  if (N >= 0xFFFFFFFFull || C > 0xFFFFFFFFull) return GLEAM_ERR_INVALID_ARG;
  HashArgs h{};
  h.buf = static_cast<const uint8_t*>(d_buf);
  h.n = n;
  h.C = C;
  h.N = (uint32_t)N;
  h.fp_out = reinterpret_cast<unsigned long long*>(d_out);
  return cuda_err(launch_hash(h, reinterpret_cast<cudaStream_t>(stream)));
}

int gleam_dedup_copy_async(gleam_cache_t* c, const void* d_buf, size_t n, uint32_t* d_hit_mask,
                           uint32_t* d_miss_idx, void* d_miss_bytes, gleam_result_t* d_result,
                           gleam_stream_t stream) {
  if (!c) return GLEAM_ERR_INVALID_ARG;
  if (n == 0) return GLEAM_OK;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  return enqueue_dedup(c, d_buf, n, d_hit_mask, d_miss_idx, d_miss_bytes, d_result,
                       reinterpret_cast<cudaStream_t>(stream));
}

int64_t gleam_dedup_copy(gleam_cache_t* c, const void* d_buf, size_t n, uint32_t* d_hit_mask,
                         uint32_t* d_miss_idx, void* d_miss_bytes) {
  if (!c) return GLEAM_ERR_INVALID_ARG;
  if (n == 0) return 0;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  int rc = enqueue_dedup(c, d_buf, n, d_hit_mask, d_miss_idx, d_miss_bytes, c->d_result, nullptr);
  if (rc != GLEAM_OK) return rc;
  rc = cuda_err(cudaMemcpyAsync(c->h_result, c->d_result, sizeof(gleam_result_t),
                                cudaMemcpyDeviceToHost, nullptr));
  if (rc == GLEAM_OK) rc = cuda_err(cudaStreamSynchronize(nullptr));
  if (rc != GLEAM_OK) return rc;
  if (c->h_result->status != 0) return c->h_result->status;
  return (int64_t)c->h_result->n_miss;
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
  int rc = check_device_ptr(d_bytes, c->device);
  if (rc != GLEAM_OK) return rc;
  if ((rc = wait_done(c)) != GLEAM_OK) return rc;
  unsigned long long used = 0;
  rc = cuda_err(cudaMemcpy(&used, c->dstats + ST_SLOTS_USED, sizeof(used), cudaMemcpyDeviceToHost));
  if (rc != GLEAM_OK) return rc;
  if (used >= c->nslots) return GLEAM_ERR_CAPACITY;
  const unsigned long long k = (c->flags & GLEAM_KEY16) ? (key & 0xFFFFull) : key;
  rc = cuda_err(cudaMemcpy(c->arena + used * c->C, d_bytes, len, cudaMemcpyDeviceToDevice));
  if (rc == GLEAM_OK)
    rc = cuda_err(launch_debug_insert(c->index, c->index_cap - 1, c->slot_len, c->dstats, k,
                                      (uint32_t)used, (uint32_t)len, c->ctl, nullptr));
  if (rc == GLEAM_OK) rc = cuda_err(cudaDeviceSynchronize());
  if (rc == GLEAM_OK) rc = cuda_err(cudaEventRecord(c->done, nullptr));
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
  rc = cuda_err(cudaMalloc(&s->index, c->index_cap * sizeof(IndexEntry)));
  if (rc == GLEAM_OK) rc = cuda_err(cudaMalloc(&s->dstats, ST_COUNT * sizeof(unsigned long long)));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpy(s->index, c->index, c->index_cap * sizeof(IndexEntry),
                             cudaMemcpyDeviceToDevice));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpy(s->dstats, c->dstats, ST_COUNT * sizeof(unsigned long long),
                             cudaMemcpyDeviceToDevice));
  if (rc != GLEAM_OK) {
    gleam_snapshot_destroy(s);
    return rc;
  }
  *out = s;
  return GLEAM_OK;
}

// Stream-ordered on the legacy default stream: it orders after earlier work
// on every blocking stream, and later calls there see the restored state.
int gleam_cache_restore(gleam_cache_t* c, const gleam_snapshot_t* s) {
  if (!c || !s || s->owner != c || s->index_cap != c->index_cap) return GLEAM_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(c->mu);
  DeviceGuard g(c->device);
  int rc = cuda_err(cudaStreamWaitEvent(nullptr, c->done, 0));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpyAsync(c->index, s->index, c->index_cap * sizeof(IndexEntry),
                                  cudaMemcpyDeviceToDevice, nullptr));
  if (rc == GLEAM_OK)
    rc = cuda_err(cudaMemcpyAsync(c->dstats, s->dstats, ST_COUNT * sizeof(unsigned long long),
                                  cudaMemcpyDeviceToDevice, nullptr));
  if (rc == GLEAM_OK) rc = cuda_err(cudaEventRecord(c->done, nullptr));
  return rc;
}

void gleam_snapshot_destroy(gleam_snapshot_t* s) {
  if (!s) return;
  DeviceGuard g(s->device);
  cudaDeviceSynchronize();
  if (s->index) cudaFree(s->index);
  if (s->dstats) cudaFree(s->dstats);
  cudaGetLastError();
  delete s;
}

}  // extern "C"
