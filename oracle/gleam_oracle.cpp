// Gleam chunk-dedup ORACLE -- test infrastructure only.
//
// A plain, slow, single-threaded CPU statement of what the dedup hot path
// computes.  Only the test suite, the package's smoke check and the CPU
// baseline leg of the benchmark load this file's library; the product path
// never does.  It shares no code, header or table with the CUDA library.
//
// What it follows:
//  * Paper Sec. 4.1.2 ("Hash-based Weight Chunk Retrieval"): before a
//    host-to-device payload is forwarded, a hash of the source bytes is looked
//    up in the server's set of resident chunk identifiers; on a hit only
//    (hash, size) metadata crosses the network, otherwise the full chunk does
//    and it becomes reusable later.
//  * Paper App. B.1 ("Hash Cost and Collision"): the paper hashes a prefix with
//    MD5 and relies on never having seen a collision.  Here the identifier is
//    XXH64 (seed 0) of each fixed C-byte chunk, and every key match is
//    confirmed byte for byte so a collision can never alias two chunks.
//  * XXH64 itself is written from the public xxHash specification (the
//    "xxhash_spec" document): four accumulators over 32-byte stripes,
//    convergence, merge rounds, length, 8/4/1-byte tails, avalanche.
//
// Readings taken where the paper is silent:
//  R1 identifier = XXH64(seed 0) of the whole chunk, as a native u64.
//  R2 chunks are fixed C bytes; chunk_bytes == 0 in oracle_fingerprint means
//     one hash over the whole payload (the paper's per-payload identifier).
//  R3 the last chunk keeps its true length; length is part of equality.
//  R5 duplicates inside one call: chunks are decided strictly in ascending
//     order, so a later copy of an earlier miss is a hit on that fresh insert.
//  R6 verify_rejects counts chunks that had a key+length candidate and no
//     byte-equal candidate.
//  R7 running out of slots returns CAPACITY and leaves the cache unchanged.
//  R8 miss indices ascending, packed bytes in the same order at rank*C,
//     hit-mask bit i is bit (i % 32) of 32-bit word i / 32, trailing bits 0.
//  R10 KEY16 mode keys the index by the low 16 bits of the fingerprint.
//  R13 paper-identifier mode (App. B.1): the key is MD5 of the chunk's first
//      min(len, 128) bytes (first 8 digest bytes, little-endian); chunks under
//      1024 bytes are recorded but never cached: always misses, no slot, no
//      entry, no in-call dedup.  Verify is kept.
//  R12 a batch of payloads is its calls made in order (a chunk equal to an
//      earlier payload's miss is a cache hit for its own payload), except that
//      running out of slots fails the whole batch.
//  R16 LRU eviction (Sec. 4.1.3; caches created with the LRU flag): every call
//      (a batch counts as one call) takes the next value of a clock; the slots
//      it hits or fills get that value as their last use.  Hits and misses are
//      decided as without eviction.  If the call's stored misses exceed the
//      never-used slots, it evicts the missing number of slots among those it
//      did not hit, least recent last use first, ties by lower slot number;
//      if too few exist it fails with CAPACITY and changes nothing.  Evicted
//      slots lose their index entries; the call's new entries take the
//      evicted slots and then never-used ones, in ascending slot order, in the
//      order of the misses.
#include <algorithm>
#include <cmath>
#include <cstddef>
#include <cstdint>
#include <cstring>
#include <iterator>
#include <unordered_map>
#include <vector>

namespace {

// ---- XXH64, public xxHash specification ---------------------------------
const uint64_t kP1 = 0x9E3779B185EBCA87ULL;
const uint64_t kP2 = 0xC2B2AE3D27D4EB4FULL;
const uint64_t kP3 = 0x165667B19E3779F9ULL;
const uint64_t kP4 = 0x85EBCA77C2B2AE63ULL;
const uint64_t kP5 = 0x27D4EB2F165667C5ULL;

uint64_t rotl64(uint64_t x, int r) { return (x << r) | (x >> (64 - r)); }

// Inputs are read as little-endian words regardless of the host's byte order.
uint64_t read_le64(const uint8_t* p) {
  uint64_t v = 0;
  for (int k = 0; k < 8; ++k) v |= static_cast<uint64_t>(p[k]) << (8 * k);
  return v;
}

uint32_t read_le32(const uint8_t* p) {
  uint32_t v = 0;
  for (int k = 0; k < 4; ++k) v |= static_cast<uint32_t>(p[k]) << (8 * k);
  return v;
}

// One accumulator step: acc + input*P2, rotate left 31, times P1.
uint64_t xxh_round(uint64_t acc, uint64_t input) {
  acc += input * kP2;
  acc = rotl64(acc, 31);
  acc *= kP1;
  return acc;
}

// Folding one accumulator into the converged hash.
uint64_t xxh_merge(uint64_t h, uint64_t acc) {
  h ^= xxh_round(0, acc);
  h = h * kP1 + kP4;
  return h;
}

uint64_t xxh64(const uint8_t* p, size_t len, uint64_t seed) {
  size_t off = 0;
  uint64_t h;
  if (len >= 32) {
    // Step 1: accumulator initialisation.
    uint64_t v[4] = {seed + kP1 + kP2, seed + kP2, seed, seed - kP1};
    // Step 2: every full 32-byte stripe; lane l takes the word at 8*l.
    while (len - off >= 32) {
      for (int l = 0; l < 4; ++l) v[l] = xxh_round(v[l], read_le64(p + off + 8 * l));
      off += 32;
    }
    // Step 3: convergence.
    h = rotl64(v[0], 1) + rotl64(v[1], 7) + rotl64(v[2], 12) + rotl64(v[3], 18);
    // Step 4: merge every accumulator, in lane order.
    for (int l = 0; l < 4; ++l) h = xxh_merge(h, v[l]);
  } else {
    h = seed + kP5;  // short-input start value
  }
  // Step 5: total length.
  h += static_cast<uint64_t>(len);
  // Step 6: remaining input, 8 bytes, then 4, then single bytes.
  while (len - off >= 8) {
    h ^= xxh_round(0, read_le64(p + off));
    h = rotl64(h, 27) * kP1 + kP4;
    off += 8;
  }
  if (len - off >= 4) {
    h ^= static_cast<uint64_t>(read_le32(p + off)) * kP1;
    h = rotl64(h, 23) * kP2 + kP3;
    off += 4;
  }
  while (off < len) {
    h ^= static_cast<uint64_t>(p[off]) * kP5;
    h = rotl64(h, 11) * kP1;
    ++off;
  }
  // Step 7: avalanche.
  h ^= h >> 33;
  h *= kP2;
  h ^= h >> 29;
  h *= kP3;
  h ^= h >> 32;
  return h;
}

// ---- MD5, RFC 1321 ------------------------------------------------------------
// Used only for the paper's own identifier (App. B.1: MD5 of a chunk's first
// 1024 bits).  Per-step constants are floor(2^32 * |sin(i)|), i = 1..64.
struct Md5 {
  uint32_t k[64];
  Md5() {
    for (int i = 0; i < 64; ++i)
      k[i] = static_cast<uint32_t>(std::floor(std::fabs(std::sin(static_cast<double>(i + 1))) *
                                              4294967296.0));
  }
};

uint32_t rotl32(uint32_t x, int r) { return (x << r) | (x >> (32 - r)); }

void md5(const uint8_t* p, size_t len, uint8_t out[16]) {
  static const Md5 tab;
  static const int shift[4][4] = {{7, 12, 17, 22}, {5, 9, 14, 20}, {4, 11, 16, 23}, {6, 10, 15, 21}};
  // message + 0x80 + zero padding to 56 mod 64 + 64-bit little-endian bit length
  std::vector<uint8_t> m(p, p + len);
  m.push_back(0x80);
  while (m.size() % 64 != 56) m.push_back(0);
  const uint64_t bits = static_cast<uint64_t>(len) * 8;
  for (int k = 0; k < 8; ++k) m.push_back(static_cast<uint8_t>(bits >> (8 * k)));
  uint32_t a0 = 0x67452301u, b0 = 0xefcdab89u, c0 = 0x98badcfeu, d0 = 0x10325476u;
  for (size_t blk = 0; blk < m.size(); blk += 64) {
    uint32_t x[16];
    for (int j = 0; j < 16; ++j) x[j] = read_le32(&m[blk + 4 * j]);
    uint32_t a = a0, b = b0, c = c0, d = d0;
    for (int i = 0; i < 64; ++i) {
      const int round = i / 16;
      uint32_t f;
      int g;
      if (round == 0) {
        f = (b & c) | (~b & d);
        g = i;
      } else if (round == 1) {
        f = (d & b) | (~d & c);
        g = (5 * i + 1) % 16;
      } else if (round == 2) {
        f = b ^ c ^ d;
        g = (3 * i + 5) % 16;
      } else {
        f = c ^ (b | ~d);
        g = (7 * i) % 16;
      }
      const uint32_t t = d;
      d = c;
      c = b;
      b = b + rotl32(a + f + tab.k[i] + x[g], shift[round][i % 4]);
      a = t;
    }
    a0 += a;
    b0 += b;
    c0 += c;
    d0 += d;
  }
  const uint32_t w[4] = {a0, b0, c0, d0};
  for (int j = 0; j < 4; ++j)
    for (int k = 0; k < 4; ++k) out[4 * j + k] = static_cast<uint8_t>(w[j] >> (8 * k));
}

// The paper's identifier of a chunk: MD5 over its first min(len, 128) bytes,
// first 8 digest bytes as a little-endian u64.
uint64_t paper_key(const uint8_t* p, size_t len) {
  uint8_t d[16];
  md5(p, len < 128 ? len : 128, d);
  uint64_t k = 0;
  for (int i = 0; i < 8; ++i) k |= static_cast<uint64_t>(d[i]) << (8 * i);
  return k;
}

// ---- the weight cache -----------------------------------------------------
const int kOk = 0;
const int kErrInvalidArg = -1;
const int kErrCapacity = -4;
const uint32_t kFlagKey16 = 1u;
const uint32_t kFlagPaperIds = 4u;  // App. B.1 identifiers and small-chunk rule
const uint32_t kFlagEvictLru = 8u;  // Sec. 4.1.3 LRU eviction instead of CAPACITY
const size_t kPaperMinCached = 1024;
const uint32_t kNoSlot = 0xFFFFFFFFu;

struct Entry {
  uint64_t key;
  uint32_t len;
  uint32_t slot;
};

struct Cache {
  size_t capacity_bytes = 0;
  size_t chunk = 0;
  uint64_t nslots = 0;
  uint32_t flags = 0;
  std::unordered_multimap<uint64_t, Entry> index;  // key -> entries
  std::vector<std::vector<uint8_t>> slot_bytes;    // slot -> stored bytes
  std::vector<uint64_t> last_use;                  // slot -> clock of its last use
  uint64_t clock = 0;                              // one tick per call
  // statistics, same meaning as the CUDA library's
  uint64_t calls = 0, chunks = 0, hits_cache = 0, hits_intra = 0, misses = 0,
           inserts = 0, verify_rejects = 0, bytes_used = 0, evictions = 0;
};

// One payload of a call: its bytes, its outputs and its results.
struct Payload {
  const uint8_t* p;
  size_t n;
  uint32_t* hit_mask;
  uint32_t* miss_idx;
  uint8_t* packed;
  uint32_t* chunk_slot;  // may be null
  uint64_t n_miss = 0, hits_cache = 0, hits_intra = 0, rejects = 0, miss_bytes = 0;
};

uint64_t key_of(const Cache& c, uint64_t fp) {
  return (c.flags & kFlagKey16) ? (fp & 0xFFFFull) : fp;
}

// Index key of a chunk: XXH64 of the whole chunk, or in paper mode MD5 of its
// prefix; then the 16-bit truncation of the KEY16 test mode.
uint64_t chunk_key(const Cache& c, const uint8_t* p, size_t len) {
  return key_of(c, (c.flags & kFlagPaperIds) ? paper_key(p, len) : xxh64(p, len, 0));
}

bool bytes_equal(const std::vector<uint8_t>& stored, const uint8_t* p, size_t len) {
  return stored.size() == len && (len == 0 || std::memcmp(stored.data(), p, len) == 0);
}

}  // namespace

extern "C" {

uint64_t oracle_xxh64(const void* p, size_t n, uint64_t seed) {
  return xxh64(static_cast<const uint8_t*>(p), n, seed);
}

void oracle_md5(const void* p, size_t n, uint8_t* out16) {
  md5(static_cast<const uint8_t*>(p), n, out16);
}

// out[i] = XXH64 of chunk i; chunk_bytes == 0 -> out[0] = XXH64 of all n bytes.
int oracle_fingerprint(const void* buf, size_t n, size_t chunk_bytes, uint64_t* out) {
  const uint8_t* p = static_cast<const uint8_t*>(buf);
  if (chunk_bytes == 0) {
    out[0] = xxh64(p, n, 0);
    return kOk;
  }
  size_t nchunks = (n + chunk_bytes - 1) / chunk_bytes;
  for (size_t i = 0; i < nchunks; ++i) {
    size_t begin = i * chunk_bytes;
    size_t len = (n - begin < chunk_bytes) ? (n - begin) : chunk_bytes;
    out[i] = xxh64(p + begin, len, 0);
  }
  return kOk;
}

void* oracle_cache_create(size_t capacity_bytes, size_t chunk_bytes, uint32_t flags, int* err) {
  if (chunk_bytes < 32 || chunk_bytes % 32 != 0 || chunk_bytes > (16u << 20) ||
      (flags & ~(kFlagKey16 | kFlagPaperIds | kFlagEvictLru)) != 0 || capacity_bytes / (chunk_bytes ? chunk_bytes : 1) == 0 ||
      capacity_bytes / chunk_bytes > 0xFFFFFFFEull) {
    if (err) *err = kErrInvalidArg;
    return nullptr;
  }
  Cache* c = new Cache();
  c->capacity_bytes = capacity_bytes;
  c->chunk = chunk_bytes;
  c->nslots = capacity_bytes / chunk_bytes;
  c->flags = flags;
  if (err) *err = kOk;
  return c;
}

void oracle_cache_destroy(void* cache) { delete static_cast<Cache*>(cache); }

}  // extern "C"

namespace {

// The dedup of one call over `count` payloads (paper Sec. 4.1.2 with
// readings R1-R8, R12, R13, R16): chunks are decided one at a time, payload
// after payload, in ascending order.  Returns the number of misses, or a
// negative error code.  The cache is only changed when the whole call
// succeeds; on an error the outputs are unspecified.
int64_t dedup_calls(Cache* c, Payload* pays, size_t count) {
  const size_t C = c->chunk;
  uint64_t total_chunks = 0;
  for (size_t k = 0; k < count; ++k) {
    if (pays[k].n > 0 && pays[k].p == nullptr) return kErrInvalidArg;
    total_chunks += (pays[k].n + C - 1) / C;
  }
  if (total_chunks > 0xFFFFFFFEull) return kErrInvalidArg;
  if (total_chunks == 0) return 0;
  const uint64_t now = ++c->clock;

  // Entries inserted by this call, kept aside until the call commits.  Their
  // Entry.slot holds the insertion number r; the slot is decided at the end.
  std::unordered_multimap<uint64_t, Entry> fresh_index;
  std::vector<std::vector<uint8_t>> fresh_bytes;
  std::vector<size_t> fresh_payload;                      // payload that inserted r
  std::vector<std::pair<uint32_t*, uint64_t>> fresh_refs;  // chunk_slot cells naming r
  const uint64_t slots0 = c->slot_bytes.size();
  std::vector<char> used(slots0, 0);  // cached slots hit by this call
  const bool paper = (c->flags & kFlagPaperIds) != 0;
  uint64_t stored = 0;  // misses given a slot (all of them, except paper-mode small chunks)

  for (size_t k = 0; k < count; ++k) {
    Payload& P = pays[k];
    if (P.n == 0) continue;
    const uint64_t nchunks = (P.n + C - 1) / C;
    for (uint64_t w = 0; w < (nchunks + 31) / 32; ++w) P.hit_mask[w] = 0;
    uint64_t rank = 0;
    for (uint64_t i = 0; i < nchunks; ++i) {
      const uint8_t* chunk = P.p + i * C;
      const size_t len = (P.n - i * C < C) ? (P.n - i * C) : C;
      if (paper && len < kPaperMinCached) {
        // App. B.1: recorded but never cached -- always sent, never inserted
        P.miss_idx[rank] = static_cast<uint32_t>(i);
        if (P.chunk_slot) P.chunk_slot[i] = kNoSlot;
        std::memcpy(P.packed + rank * C, chunk, len);
        P.miss_bytes += len;
        ++rank;
        continue;
      }
      const uint64_t key = chunk_key(*c, chunk, len);

      bool candidate = false, hit = false, hit_is_fresh = false;
      uint64_t hit_slot = 0;
      auto look = [&](const std::unordered_multimap<uint64_t, Entry>& idx,
                      const std::vector<std::vector<uint8_t>>& store, bool fresh) {
        auto range = idx.equal_range(key);
        for (auto it = range.first; it != range.second; ++it) {
          if (it->second.len != len) continue;
          candidate = true;
          if (bytes_equal(store[it->second.slot], chunk, len)) {
            hit = true;
            hit_is_fresh = fresh;
            hit_slot = it->second.slot;
          }
        }
      };
      look(c->index, c->slot_bytes, false);
      look(fresh_index, fresh_bytes, true);

      if (hit) {
        P.hit_mask[i / 32] |= 1u << (i % 32);
        if (hit_is_fresh) {
          // an earlier miss of this payload, or of an earlier payload of the
          // batch, whose own call would have inserted it (R12)
          if (fresh_payload[hit_slot] == k) ++P.hits_intra; else ++P.hits_cache;
          if (P.chunk_slot) fresh_refs.emplace_back(P.chunk_slot + i, hit_slot);
        } else {
          ++P.hits_cache;
          used[hit_slot] = 1;
          if (P.chunk_slot) P.chunk_slot[i] = static_cast<uint32_t>(hit_slot);
        }
        continue;
      }
      if (candidate) ++P.rejects;
      P.miss_idx[rank] = static_cast<uint32_t>(i);
      if (P.chunk_slot) fresh_refs.emplace_back(P.chunk_slot + i, stored);
      std::memcpy(P.packed + rank * C, chunk, len);
      Entry e{key, static_cast<uint32_t>(len), static_cast<uint32_t>(stored)};
      fresh_index.emplace(key, e);
      fresh_bytes.emplace_back(chunk, chunk + len);
      fresh_payload.push_back(k);
      P.miss_bytes += len;
      ++rank;
      ++stored;
    }
    P.n_miss = rank;
  }

  // Slots for the new entries: never-used slots, and with LRU eviction the
  // least recently used slots this call did not hit (R7, R16).
  std::vector<uint64_t> victims;
  if (stored > c->nslots - slots0) {
    if (!(c->flags & kFlagEvictLru)) return kErrCapacity;  // nothing committed
    const uint64_t need = stored - (c->nslots - slots0);
    std::vector<uint64_t> cand;
    for (uint64_t s = 0; s < slots0; ++s)
      if (!used[s]) cand.push_back(s);
    if (cand.size() < need) return kErrCapacity;
    std::sort(cand.begin(), cand.end(), [&](uint64_t x, uint64_t y) {
      return c->last_use[x] != c->last_use[y] ? c->last_use[x] < c->last_use[y] : x < y;
    });
    victims.assign(cand.begin(), cand.begin() + need);
    std::sort(victims.begin(), victims.end());
  }
  std::vector<uint64_t> slot_of(stored);
  for (uint64_t r = 0; r < stored; ++r)
    slot_of[r] = r < victims.size() ? victims[r] : slots0 + (r - victims.size());

  // Commit: drop the victims' entries, then store the new ones.
  if (!victims.empty()) {
    std::vector<char> gone(slots0, 0);
    for (uint64_t v : victims) {
      gone[v] = 1;
      c->bytes_used -= c->slot_bytes[v].size();
    }
    for (auto it = c->index.begin(); it != c->index.end();)
      it = gone[it->second.slot] ? c->index.erase(it) : std::next(it);
  }
  for (auto& kv : fresh_index) {
    Entry e = kv.second;
    const uint64_t r = e.slot;
    e.slot = static_cast<uint32_t>(slot_of[r]);
    c->index.emplace(kv.first, e);
  }
  for (uint64_t r = 0; r < stored; ++r) {
    const uint64_t s = slot_of[r];
    c->bytes_used += fresh_bytes[r].size();
    if (s < c->slot_bytes.size()) {
      c->slot_bytes[s] = std::move(fresh_bytes[r]);
      c->last_use[s] = now;
    } else {
      c->slot_bytes.emplace_back(std::move(fresh_bytes[r]));
      c->last_use.push_back(now);
    }
  }
  for (uint64_t s = 0; s < slots0; ++s)
    if (used[s]) c->last_use[s] = now;
  for (auto& ref : fresh_refs) *ref.first = static_cast<uint32_t>(slot_of[ref.second]);

  uint64_t misses = 0;
  for (size_t k = 0; k < count; ++k) {
    const Payload& P = pays[k];
    if (P.n == 0) continue;
    c->calls += 1;
    c->chunks += (P.n + C - 1) / C;
    c->hits_cache += P.hits_cache;
    c->hits_intra += P.hits_intra;
    c->misses += P.n_miss;
    c->verify_rejects += P.rejects;
    misses += P.n_miss;
  }
  c->inserts += stored;
  c->evictions += victims.size();
  return static_cast<int64_t>(misses);
}

}  // namespace

extern "C" {

// The sequential dedup of one payload: a call of one payload.
int64_t oracle_dedup(void* cache, const void* buf, size_t n, uint32_t* hit_mask,
                     uint32_t* miss_idx, uint8_t* packed, uint32_t* chunk_slot) {
  Cache* c = static_cast<Cache*>(cache);
  if (c == nullptr) return kErrInvalidArg;
  Payload P{static_cast<const uint8_t*>(buf), n, hit_mask, miss_idx, packed, chunk_slot};
  return dedup_calls(c, &P, 1);
}

// A batch of payloads in one call.  results: count x 5 u64 (misses,
// cache hits, in-call hits, verify rejects, miss bytes) per payload.
int64_t oracle_dedup_batch(void* cache, size_t count, const void* const* bufs, const size_t* ns,
                           uint32_t* const* hit_masks, uint32_t* const* miss_idxs,
                           uint8_t* const* packeds, uint32_t* const* chunk_slots,
                           uint64_t* results) {
  Cache* c = static_cast<Cache*>(cache);
  if (c == nullptr || (count > 0 && (bufs == nullptr || ns == nullptr))) return kErrInvalidArg;
  std::vector<Payload> pays;
  for (size_t k = 0; k < count; ++k)
    pays.push_back(Payload{static_cast<const uint8_t*>(bufs[k]), ns[k], hit_masks[k],
                           miss_idxs[k], packeds[k], chunk_slots ? chunk_slots[k] : nullptr});
  const int64_t rc = dedup_calls(c, pays.data(), count);
  if (rc >= 0 && results)
    for (size_t k = 0; k < count; ++k) {
      results[5 * k + 0] = pays[k].n_miss;
      results[5 * k + 1] = pays[k].hits_cache;
      results[5 * k + 2] = pays[k].hits_intra;
      results[5 * k + 3] = pays[k].rejects;
      results[5 * k + 4] = pays[k].miss_bytes;
    }
  return rc;
}

// Weight-block identification at cudaFree time (paper Sec. 4.1.1): record r says
// that the block's bytes at offsets[r] were written by a host-to-device copy of
// the chunk stored in slots[r].  The block still holds weights iff every record
// matches the block's current bytes.  Writes mismatch[r] (1 = differs, or the
// record does not fit the block / names no stored slot) and returns how many
// records mismatch.
int64_t oracle_block_check(const void* cache, const void* block, uint64_t block_bytes,
                           const uint64_t* offsets, const uint32_t* slots, uint64_t nrec,
                           uint8_t* mismatch) {
  const Cache* c = static_cast<const Cache*>(cache);
  const uint8_t* b = static_cast<const uint8_t*>(block);
  int64_t bad = 0;
  for (uint64_t r = 0; r < nrec; ++r) {
    bool differs = true;
    if (slots[r] < c->slot_bytes.size()) {
      const std::vector<uint8_t>& stored = c->slot_bytes[slots[r]];
      if (offsets[r] <= block_bytes && stored.size() <= block_bytes - offsets[r])
        differs = !stored.empty() && std::memcmp(b + offsets[r], stored.data(), stored.size()) != 0;
    }
    mismatch[r] = differs ? 1 : 0;
    bad += differs ? 1 : 0;
  }
  return bad;
}

// Test hook: store `bytes` under an arbitrary key (crafted collisions).
int oracle_debug_insert(void* cache, uint64_t key, const void* bytes, size_t len) {
  Cache* c = static_cast<Cache*>(cache);
  if (c == nullptr || len == 0 || len > c->chunk || bytes == nullptr) return kErrInvalidArg;
  if (c->slot_bytes.size() >= c->nslots) return kErrCapacity;
  const uint8_t* b = static_cast<const uint8_t*>(bytes);
  Entry e{key_of(*c, key), static_cast<uint32_t>(len), static_cast<uint32_t>(c->slot_bytes.size())};
  c->index.emplace(e.key, e);
  c->slot_bytes.emplace_back(b, b + len);
  c->last_use.push_back(++c->clock);
  c->bytes_used += len;
  c->inserts += 1;
  return kOk;
}

// Stats in the CUDA library's field order:
// calls, chunks, hits_cache, hits_intra, misses, inserts, verify_rejects,
// slots_used, bytes_used, capacity_bytes, nslots, chunk_bytes, evictions.
void oracle_cache_stats(const void* cache, uint64_t* out) {
  const Cache* c = static_cast<const Cache*>(cache);
  out[0] = c->calls;
  out[1] = c->chunks;
  out[2] = c->hits_cache;
  out[3] = c->hits_intra;
  out[4] = c->misses;
  out[5] = c->inserts;
  out[6] = c->verify_rejects;
  out[7] = c->slot_bytes.size();
  out[8] = c->bytes_used;
  out[9] = c->capacity_bytes;
  out[10] = c->nslots;
  out[11] = c->chunk;
  out[12] = c->evictions;
}

// Index contents, ordered by slot: keys[s], lens[s] for s < slots_used.
uint64_t oracle_cache_entries(const void* cache, uint64_t* keys, uint32_t* lens, uint64_t max) {
  const Cache* c = static_cast<const Cache*>(cache);
  uint64_t count = 0;
  for (const auto& kv : c->index) {
    const Entry& e = kv.second;
    if (e.slot < max) {
      keys[e.slot] = e.key;
      lens[e.slot] = e.len;
    }
    ++count;
  }
  return count;
}

// Stored bytes of one slot; returns its length, or -1 for a bad slot.
int64_t oracle_slot_bytes(const void* cache, uint64_t slot, uint8_t* out, uint64_t max) {
  const Cache* c = static_cast<const Cache*>(cache);
  if (slot >= c->slot_bytes.size()) return -1;
  const auto& b = c->slot_bytes[slot];
  uint64_t m = b.size() < max ? b.size() : max;
  if (m) std::memcpy(out, b.data(), m);
  return static_cast<int64_t>(b.size());
}

}  // extern "C"
