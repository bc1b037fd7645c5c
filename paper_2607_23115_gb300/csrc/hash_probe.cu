// Fingerprint + index probe + byte verify of every chunk of a payload
// (paper Sec. 4.1.2: hash the source bytes, look the hash up in the set of
// resident chunks; App. B.1: confirm the match so collisions cannot alias).
//
// Mapping: a group of 4 consecutive threads owns one chunk; thread `lane`
// runs XXH64 accumulator lane `lane` on the 8-byte word at 8*lane of each
// 32-byte stripe, so a warp works on 8 chunks and every 32-byte sector it
// touches is used whole.  After the first 512 bytes the group looks its
// prefix hint up and, if a cached chunk began the same way, streams that copy
// alongside the payload and compares as it hashes (speculative verify).  The
// group then probes the index with the full fingerprint; the hinted slot is a
// hit if it is a key+length candidate and compared equal, and any other
// candidate is compared by re-reading both copies.
//
// Kernels: k_hash_probe_staged (16-byte-aligned payloads: chunks stream
// through shared memory by cp.async), k_hash_probe (any alignment: direct
// loads), and for the paper's identifiers k_probe_paper_staged /
// k_probe_paper (MD5 of the first 128 bytes as the key).
#include <algorithm>
#include <cmath>

#include "gleam_internal.cuh"
#include "xxh64_device.cuh"
#include "staged_hash.cuh"

namespace gleam {
namespace {

#ifndef GLEAM_HASH_THREADS
#define GLEAM_HASH_THREADS 256
#endif
#ifndef GLEAM_STAGED_HASH
#define GLEAM_STAGED_HASH 1
#endif
constexpr int kHashThreads = GLEAM_HASH_THREADS;


// Lane accumulator over `ns` stripes starting at p (p already offset by 8*lane).
template <bool kAligned>
__device__ __forceinline__ unsigned long long lane_stripes(unsigned long long acc,
                                                           const uint8_t* p, uint32_t ns) {
  uint32_t s = 0;
  if (ns >= kBatch) {
    unsigned long long x[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) x[u] = load_word<kAligned>(p + (uint64_t)u * 32);
    for (; s + 2 * kBatch <= ns; s += kBatch) {
      unsigned long long y[kBatch];
#pragma unroll
      for (int u = 0; u < kBatch; ++u)
        y[u] = load_word<kAligned>(p + (uint64_t)(s + kBatch + u) * 32);
#pragma unroll
      for (int u = 0; u < kBatch; ++u) acc = xstep(acc, x[u]);
#pragma unroll
      for (int u = 0; u < kBatch; ++u) x[u] = y[u];
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) acc = xstep(acc, x[u]);
    s += kBatch;
  }
  for (; s < ns; ++s) acc = xstep(acc, load_word<kAligned>(p + (uint64_t)s * 32));
  return acc;
}

// Lane accumulator over stripes [s0, s1) while comparing every payload word
// with the cached copy's word at q (p, q already offset by 8*lane).  `cmp`
// turns off, for the whole group, as soon as any word differs; diff then
// stays non-zero.  Loads of the next batch are issued before the current one
// is folded in.
template <bool kAligned>
__device__ __forceinline__ unsigned long long lane_stripes_cmp(
    unsigned long long acc, const uint8_t* p, const uint8_t* q, uint32_t s0, uint32_t s1,
    unsigned long long& diff, bool& cmp, unsigned gmask) {
  constexpr int B = kBatch;
  unsigned long long x[B], y[B];
  uint32_t s = s0;
  uint32_t m = min((uint32_t)B, s1 - s);
#pragma unroll
  for (int u = 0; u < B; ++u) {
    x[u] = (uint32_t)u < m ? load_word<kAligned>(p + (uint64_t)(s + u) * 32) : 0ULL;
    y[u] = (cmp && (uint32_t)u < m) ? load_arena_word(q + (uint64_t)(s + u) * 32) : x[u];
  }
  while (s < s1) {
    const uint32_t sn = s + m;
    const uint32_t mn = sn < s1 ? min((uint32_t)B, s1 - sn) : 0u;
    unsigned long long xn[B], yn[B];
#pragma unroll
    for (int u = 0; u < B; ++u) {
      xn[u] = (uint32_t)u < mn ? load_word<kAligned>(p + (uint64_t)(sn + u) * 32) : 0ULL;
      yn[u] = (cmp && (uint32_t)u < mn) ? load_arena_word(q + (uint64_t)(sn + u) * 32) : xn[u];
    }
    unsigned long long d = 0;
#pragma unroll
    for (int u = 0; u < B; ++u) {
      if ((uint32_t)u < m) {
        acc = xstep(acc, x[u]);
        d |= x[u] ^ y[u];
      }
    }
    if (cmp) {
      diff |= d;
      unsigned long long g = diff;
      g |= __shfl_xor_sync(gmask, g, 1);
      g |= __shfl_xor_sync(gmask, g, 2);
      if (g) {
        cmp = false;
        diff = 1;
      }
    }
#pragma unroll
    for (int u = 0; u < B; ++u) {
      x[u] = xn[u];
      y[u] = yn[u];
    }
    s = sn;
    m = mn;
  }
  return acc;
}



template <bool kAligned, bool kProbe>
__global__ void __launch_bounds__(kHashThreads) k_hash_probe(HashArgs a) {
  pdl_trigger();
  pdl_wait();  // this variant reads nothing before the previous call is complete
  const unsigned long long g = ((unsigned long long)blockIdx.x * blockDim.x + threadIdx.x) >> 2;
  __shared__ unsigned long long s_scratch[33];
  const uint32_t pid_b =
      a.count > 1 ? block_find_payload(a.table, a.count,
                                       ((unsigned long long)blockIdx.x * blockDim.x) >> 2, g,
                                       s_scratch)
                  : 0u;
  if (g >= a.Ntot) return;  // whole groups leave together
  const uint32_t lane = threadIdx.x & 3;
  const int gbase = threadIdx.x & 28;
  const unsigned gmask = 0xFu << gbase;

  uint32_t pid = 0;
  const uint8_t* buf;
  unsigned long long n, base;
  if (a.count > 1) {
    pid = pid_b;
    buf = a.table[pid].buf;
    n = a.table[pid].n;
    base = a.table[pid].chunk_base;
  } else {
    buf = a.one.buf;
    n = a.one.n;
    base = a.one.chunk_base;
  }
  const unsigned long long start = (g - base) * a.C;
  const uint32_t len = (uint32_t)min(a.C, n - start);
  const uint8_t* p = buf + start;
  const uint32_t ns = len >> 5;

  const bool speculate = kProbe && len >= kPrefixBytes;
  const unsigned long long slots_used = kProbe ? a.dstats[ST_SLOTS_USED] : 0ULL;
  unsigned long long hint = 0, diff = 0;
  uint32_t hint_slot = kEmptySlot;
  bool cmp = false;

  unsigned long long h;
  if (ns) {
    unsigned long long acc = xlane_start(lane);
    if (speculate) {
      constexpr uint32_t kPre = kPrefixBytes / 32;
      acc = lane_stripes<kAligned>(acc, p + 8 * lane, kPre);
      const unsigned long long b0 = group_shfl(acc, gmask, gbase + 0);
      const unsigned long long b1 = group_shfl(acc, gmask, gbase + 1);
      const unsigned long long b2 = group_shfl(acc, gmask, gbase + 2);
      const unsigned long long b3 = group_shfl(acc, gmask, gbase + 3);
      hint = b0 ^ xrotl(b1, 16) ^ xrotl(b2, 32) ^ xrotl(b3, 48);
      // an empty cache has no hints to look up
      hint_slot = slots_used ? hint_lookup(a.hints, a.index_mask, hint, len, slots_used)
                             : kEmptySlot;
      const uint8_t* q = a.arena + (unsigned long long)hint_slot * a.C;
      cmp = hint_slot != kEmptySlot;
      if (cmp) {  // the prefix, already hashed, is compared once (payload words from L2)
        unsigned long long d = 0;
#pragma unroll 4
        for (uint32_t s = 0; s < kPre; ++s) {
          const uint64_t off = (uint64_t)s * 32 + 8 * lane;
          d |= load_word<kAligned>(p + off) ^ load_arena_word(q + off);
        }
        d |= __shfl_xor_sync(gmask, d, 1);
        d |= __shfl_xor_sync(gmask, d, 2);
        if (d) {
          cmp = false;
          diff = 1;
        }
      }
      acc = lane_stripes_cmp<kAligned>(acc, p + 8 * lane, q + 8 * lane, kPre, ns, diff, cmp,
                                       gmask);
    } else {
      acc = lane_stripes<kAligned>(acc, p + 8 * lane, ns);
    }
    const unsigned long long a0 = group_shfl(acc, gmask, gbase + 0);
    const unsigned long long a1 = group_shfl(acc, gmask, gbase + 1);
    const unsigned long long a2 = group_shfl(acc, gmask, gbase + 2);
    const unsigned long long a3 = group_shfl(acc, gmask, gbase + 3);
    h = xconverge(a0, a1, a2, a3);
  } else {
    h = kXP5;
  }
  h += len;
  h = xfinish(h, p + (uint64_t)ns * 32, len & 31);

  if (a.fp_out != nullptr && lane == 0) a.fp_out[g] = h;
  if (!kProbe) return;

  // the bytes after the last full stripe, for the speculative compare
  bool spec_equal = false;
  if (speculate && hint_slot != kEmptySlot) {
    unsigned long long d = diff;
    if (cmp && lane == 0) {
      const uint8_t* q = a.arena + (unsigned long long)hint_slot * a.C;
      for (uint32_t k = ns * 32; k < len; ++k) d |= (unsigned long long)(p[k] ^ q[k]);
    }
    d |= __shfl_xor_sync(gmask, d, 1);
    d |= __shfl_xor_sync(gmask, d, 2);
    spec_equal = d == 0;
  }

  const unsigned long long key = a.key16 ? (h & 0xFFFFULL) : h;
  unsigned long long pos = mix64(key) & a.index_mask;
  bool hit = false, cand = false;
  uint32_t hit_slot = kEmptySlot;
  for (unsigned long long probe = 0; slots_used && probe <= a.index_mask; ++probe) {
    const IndexEntry e = a.index[pos];
    if (e.slot == kEmptySlot) break;
    if (e.key == key && e.len == len) {
      cand = true;
      if (e.slot >= slots_used) {
        // an entry pointing past the used slots: report, never read it
        if (lane == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
      } else if (e.slot == hint_slot) {
        if (spec_equal) {  // compared in the streaming pass
          hit = true;
          hit_slot = e.slot;
          break;
        }
      } else if (group_equal<kAligned>(p, a.arena + (uint64_t)e.slot * a.C, len, lane, gmask)) {
        hit = true;
        hit_slot = e.slot;
        break;
      }
    }
    pos = (pos + 1) & a.index_mask;
  }
  if (lane == 0) {
    a.ch.status[g] = hit ? kHit0 : (cand ? kMissCand : kMissNoCand);
    a.ch.key[g] = h;  // the group key: the whole fingerprint
    a.ch.len[g] = len;
    a.ch.src[g] = (unsigned long long)p;
    a.ch.pidx[g] = pid;
    a.ch.hint[g] = hint;
    if (hit) a.ch.ent[g] = hit_slot;
  }
}


template <bool kProbe, bool kAhead, bool kVerify, bool kPrefixAsync = false, int kS = kStage>
__global__ void __launch_bounds__(kStagedThreads) k_hash_probe_staged(HashArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  pdl_trigger();
  if (!a.wait_late) pdl_wait();  // else in staged_range, before the probe
  const unsigned long long nvb = (a.Ntot * 4 + kStagedThreads - 1) / kStagedThreads;
  for (unsigned long long vb = blockIdx.x; vb < nvb; vb += gridDim.x) {
    __syncthreads();  // the previous range's groups are done with the shared memory
    staged_range<kProbe, kAhead, kVerify, kPrefixAsync, kS>(a, vb, smem);
  }
}

// Blocks of the kS-stage variant resident at once on the whole GPU (0 if
// unknown); cached per instantiation (the machine's GPUs are all alike).
template <bool kProbe, bool kAhead, bool kVerify, int kS>
int staged_wave_blocks() {
  static int wave = -1;
  if (wave < 0) {
    constexpr int smem = (kStagedThreads / 4) * group_bytes(kVerify, kS);
    int dev = 0, nsm = 0, occ = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaFuncSetAttribute((const void*)k_hash_probe_staged<kProbe, kAhead, kVerify, false, kS>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(
            &occ, k_hash_probe_staged<kProbe, kAhead, kVerify, false, kS>, kStagedThreads, smem) !=
            cudaSuccess) {
      cudaGetLastError();
      return 0;
    }
    wave = nsm * occ;
  }
  return wave;
}

template <bool kProbe, bool kAhead, bool kVerify, bool kPrefixAsync = false, int kS = kStage>
cudaError_t launch_staged(const HashArgs& a, cudaStream_t s, bool pdl) {
  const unsigned long long threads = a.Ntot * 4;
  const unsigned sg = (unsigned)((threads + kStagedThreads - 1) / kStagedThreads);
  if constexpr (kS == kStage && kProbe && !kPrefixAsync) {
    // a call whose large chunks all fit one wave of the large-stage variant,
    // unless calls overlap (then the calls in flight share the SMs, and the
    // variant's larger blocks would crowd them out)
    if (a.C >= kBigStageMinChunk && !a.wait_late &&
        (unsigned long long)sg <= (unsigned long long)staged_wave_blocks<kProbe, kAhead, kVerify, kBigStage>())
      return launch_staged<kProbe, kAhead, kVerify, false, kBigStage>(a, s, pdl);
  }
  if constexpr (kVerify && !kPrefixAsync && kS == kStage) {
    if (a.C <= kPrefixAsyncMaxChunk)
      return launch_staged<kProbe, kAhead, kVerify, true>(a, s, pdl);
  }
  constexpr int smem = (kStagedThreads / 4) * group_bytes(kVerify, kS);
  // per device and cheap: set on every launch
  cudaFuncSetAttribute((const void*)k_hash_probe_staged<kProbe, kAhead, kVerify, kPrefixAsync, kS>,
                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  return launch_kernel(k_hash_probe_staged<kProbe, kAhead, kVerify, kPrefixAsync, kS>, dim3(sg),
                       dim3(kStagedThreads), smem, s, pdl, a);
}

// ---------------------------------------------------------------------------
// Paper-identifier mode (App. B.1): the key is MD5 (RFC 1321) of the chunk's
// first min(len, 128) bytes, computed by one lane; candidates are then
// compared with the payload directly, so no pass over the whole chunk is
// needed for the key and a chunk without candidates costs only its prefix.
// ---------------------------------------------------------------------------
struct Md5Table {
  uint32_t k[64];  // floor(2^32 * |sin(i + 1)|)
};

__device__ __forceinline__ uint32_t rotl32(uint32_t x, int r) { return (x << r) | (x >> (32 - r)); }

// First 8 digest bytes (little-endian) of MD5 over p[0, m), m <= 128.
__device__ unsigned long long md5_prefix_key(const uint8_t* p, uint32_t m, const uint32_t* K) {
  const uint32_t total = ((m + 8) / 64 + 1) * 64;  // message + 0x80 + padding + length
  const unsigned long long bits = (unsigned long long)m * 8;
  uint32_t a0 = 0x67452301u, b0 = 0xefcdab89u, c0 = 0x98badcfeu, d0 = 0x10325476u;
  for (uint32_t blk = 0; blk < total; blk += 64) {
    uint32_t x[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      uint32_t w = 0;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t q = blk + 4 * j + k;
        uint32_t byte;
        if (q < m) byte = p[q];
        else if (q == m) byte = 0x80u;
        else if (q >= total - 8) byte = (uint32_t)(bits >> (8 * (q - (total - 8)))) & 0xFFu;
        else byte = 0u;
        w |= byte << (8 * k);
      }
      x[j] = w;
    }
    uint32_t a = a0, b = b0, c = c0, d = d0;
#pragma unroll
    for (int i = 0; i < 64; ++i) {
      uint32_t f;
      int g, r;
      if (i < 16) {
        f = (b & c) | (~b & d);
        g = i;
        r = (i & 3) == 0 ? 7 : (i & 3) == 1 ? 12 : (i & 3) == 2 ? 17 : 22;
      } else if (i < 32) {
        f = (d & b) | (~d & c);
        g = (5 * i + 1) & 15;
        r = (i & 3) == 0 ? 5 : (i & 3) == 1 ? 9 : (i & 3) == 2 ? 14 : 20;
      } else if (i < 48) {
        f = b ^ c ^ d;
        g = (3 * i + 5) & 15;
        r = (i & 3) == 0 ? 4 : (i & 3) == 1 ? 11 : (i & 3) == 2 ? 16 : 23;
      } else {
        f = c ^ (b | ~d);
        g = (7 * i) & 15;
        r = (i & 3) == 0 ? 6 : (i & 3) == 1 ? 10 : (i & 3) == 2 ? 15 : 21;
      }
      const uint32_t t = d;
      d = c;
      c = b;
      b = b + rotl32(a + f + K[i] + x[g], r);
      a = t;
    }
    a0 += a;
    b0 += b;
    c0 += c;
    d0 += d;
  }
  return (unsigned long long)a0 | ((unsigned long long)b0 << 32);
}

template <bool kAligned>
__global__ void __launch_bounds__(kHashThreads) k_probe_paper(HashArgs a, Md5Table tab) {
  pdl_trigger();
  pdl_wait();
  const unsigned long long g = ((unsigned long long)blockIdx.x * blockDim.x + threadIdx.x) >> 2;
  __shared__ unsigned long long s_scratch[33];
  const uint32_t pid_b =
      a.count > 1 ? block_find_payload(a.table, a.count,
                                       ((unsigned long long)blockIdx.x * blockDim.x) >> 2, g,
                                       s_scratch)
                  : 0u;
  if (g >= a.Ntot) return;  // whole groups leave together
  const uint32_t lane = threadIdx.x & 3;
  const int gbase = threadIdx.x & 28;
  const unsigned gmask = 0xFu << gbase;

  uint32_t pid = 0;
  const uint8_t* buf;
  unsigned long long n, base;
  if (a.count > 1) {
    pid = pid_b;
    buf = a.table[pid].buf;
    n = a.table[pid].n;
    base = a.table[pid].chunk_base;
  } else {
    buf = a.one.buf;
    n = a.one.n;
    base = a.one.chunk_base;
  }
  const unsigned long long start = (g - base) * a.C;
  const uint32_t len = (uint32_t)min(a.C, n - start);
  const uint8_t* p = buf + start;

  unsigned long long key = 0;
  if (lane == 0) key = md5_prefix_key(p, min(len, 128u), tab.k);
  key = group_shfl(key, gmask, gbase);
  if (a.key16) key &= 0xFFFFULL;

  bool hit = false, cand = false;
  uint32_t hit_slot = kEmptySlot;
  if (len >= kPaperMinCached) {
    const unsigned long long slots_used = a.dstats[ST_SLOTS_USED];
    unsigned long long pos = mix64(key) & a.index_mask;
    for (unsigned long long probe = 0; probe <= a.index_mask; ++probe) {
      const IndexEntry e = a.index[pos];
      if (e.slot == kEmptySlot) break;
      if (e.key == key && e.len == len) {
        cand = true;
        if (e.slot >= slots_used) {
          if (lane == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
        } else if (group_equal<kAligned>(p, a.arena + (uint64_t)e.slot * a.C, len, lane, gmask)) {
          hit = true;
          hit_slot = e.slot;
          break;
        }
      }
      pos = (pos + 1) & a.index_mask;
    }
  }
  if (lane == 0) {
    a.ch.status[g] = len < kPaperMinCached ? kUncached : hit ? kHit0 : cand ? kMissCand : kMissNoCand;
    a.ch.key[g] = key;
    a.ch.len[g] = len;
    a.ch.src[g] = (unsigned long long)p;
    a.ch.pidx[g] = pid;
    a.ch.hint[g] = 0;
    if (hit) a.ch.ent[g] = hit_slot;
  }
}

// Staged variant of the paper-identifier probe for 16-byte-aligned payloads.
// Stage 0 of the chunk arrives by cp.async; one lane computes the MD5 key
// from shared memory, the group probes the index, and only if a key+length
// candidate exists do the rest of the chunk and the candidate's copy stream
// through two stages in flight and get compared (each lane compares the
// 16-byte pieces it copied itself, so no cross-lane sync is needed); the
// first difference ends the streaming.  A chunk without a candidate costs one
// stage; further candidates after a mismatch are compared by re-reading.
__global__ void __launch_bounds__(kStagedThreads) k_probe_paper_staged(HashArgs a, Md5Table tab) {
  extern __shared__ __align__(16) uint8_t smem[];
  pdl_trigger();
  pdl_wait();  // the key is known after the first stage: nothing to overlap
  const unsigned long long g = ((unsigned long long)blockIdx.x * blockDim.x + threadIdx.x) >> 2;
  const uint32_t pid_b =
      a.count > 1 ? block_find_payload(a.table, a.count,
                                       ((unsigned long long)blockIdx.x * blockDim.x) >> 2, g,
                                       reinterpret_cast<unsigned long long*>(smem))
                  : 0u;
  if (g >= a.Ntot) return;  // whole groups leave together
  const uint32_t lane = threadIdx.x & 3;
  const int gbase = threadIdx.x & 28;
  const unsigned gmask = 0xFu << gbase;
  uint8_t* region = smem + (threadIdx.x >> 2) * kGroupBytes;
  const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(region);

  uint32_t pid = 0;
  const uint8_t* buf;
  unsigned long long n, base;
  if (a.count > 1) {
    pid = pid_b;
    buf = a.table[pid].buf;
    n = a.table[pid].n;
    base = a.table[pid].chunk_base;
  } else {
    buf = a.one.buf;
    n = a.one.n;
    base = a.one.chunk_base;
  }
  const unsigned long long start = (g - base) * a.C;
  const uint32_t len = (uint32_t)min(a.C, n - start);
  const uint8_t* p = buf + start;
  const uint32_t full = (len >> 5) * 32;  // bytes in whole stripes
  const uint32_t nst = (full + kStage - 1) / kStage;
  auto sbytes = [&](uint32_t t) { return min((uint32_t)kStage, full - t * kStage); };

  unsigned long long key = 0;
  bool hit = false, cand = false;
  uint32_t hit_slot = kEmptySlot;
  if (len < kPaperMinCached) {  // recorded, never cached: only the key
    if (lane == 0) key = md5_prefix_key(p, min(len, 128u), tab.k);
    key = group_shfl(key, gmask, gbase);
    if (a.key16) key &= 0xFFFFULL;
  } else {
    // stage 0 (the first 512 bytes) -> MD5 of its first 128 bytes
    stage_copy(sbase, p, kStage, lane);
    cp_commit();
    cp_wait<0>();
    __syncwarp(gmask);
    if (lane == 0) key = md5_prefix_key(region, 128u, tab.k);
    key = group_shfl(key, gmask, gbase);
    if (a.key16) key &= 0xFFFFULL;

    // the first key+length candidate
    const unsigned long long slots_used = a.dstats[ST_SLOTS_USED];
    unsigned long long pos = mix64(key) & a.index_mask;
    uint32_t first = kEmptySlot;
    for (unsigned long long probe = 0; probe <= a.index_mask; ++probe) {
      const IndexEntry e = a.index[pos];
      if (e.slot == kEmptySlot) break;
      if (e.key == key && e.len == len) {
        if (e.slot >= slots_used) {
          if (lane == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
        } else {
          first = e.slot;
          break;
        }
      }
      pos = (pos + 1) & a.index_mask;
    }
    if (first != kEmptySlot) {
      cand = true;
      const uint8_t* q = a.arena + (unsigned long long)first * a.C;
      // stream the candidate (and the rest of the payload), two stages in flight
      stage_copy(sbase + kStage, q, kStage, lane);
      cp_commit();
      if (nst > 1) {
        stage_copy(sbase + 2 * kStage, p + kStage, sbytes(1), lane);
        stage_copy(sbase + 3 * kStage, q + kStage, sbytes(1), lane);
      }
      cp_commit();
      bool equal = true;
      for (uint32_t t = 0; t < nst; ++t) {
        cp_wait<1>();  // stage t's group; the one after it may still be in flight
        const uint32_t b = (t & 1) * 2 * kStage;
        unsigned long long d = 0;
#pragma unroll
        for (int j = 0; j < kStage / 64; ++j) {
          const uint32_t off = (uint32_t)j * 64 + lane * 16;
          if (off < sbytes(t)) {
            const uint4 x = *reinterpret_cast<const uint4*>(region + b + off);
            const uint4 y = *reinterpret_cast<const uint4*>(region + b + kStage + off);
            d |= (unsigned long long)((x.x ^ y.x) | (x.y ^ y.y) | (x.z ^ y.z) | (x.w ^ y.w));
          }
        }
        d |= __shfl_xor_sync(gmask, d, 1);
        d |= __shfl_xor_sync(gmask, d, 2);
        if (d) {
          equal = false;
          break;
        }
        if (t + 2 < nst) {  // into the buffers this lane has just read
          stage_copy(sbase + b, p + (unsigned long long)(t + 2) * kStage, sbytes(t + 2), lane);
          stage_copy(sbase + b + kStage, q + (unsigned long long)(t + 2) * kStage, sbytes(t + 2),
                     lane);
        }
        cp_commit();
      }
      cp_wait<0>();
      if (equal) {  // the bytes after the last whole stripe
        unsigned long long d = 0;
        if (lane == 0)
          for (uint32_t k = full; k < len; ++k) d |= (unsigned long long)(p[k] ^ q[k]);
        d |= __shfl_xor_sync(gmask, d, 1);
        d |= __shfl_xor_sync(gmask, d, 2);
        equal = d == 0;
      }
      if (equal) {
        hit = true;
        hit_slot = first;
      } else {  // any further candidates, by re-reading both copies
        pos = (pos + 1) & a.index_mask;
        for (unsigned long long probe = 0; probe <= a.index_mask && !hit; ++probe) {
          const IndexEntry e = a.index[pos];
          if (e.slot == kEmptySlot) break;
          if (e.key == key && e.len == len) {
            if (e.slot >= slots_used) {
              if (lane == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
            } else if (group_equal<true>(p, a.arena + (uint64_t)e.slot * a.C, len, lane, gmask)) {
              hit = true;
              hit_slot = e.slot;
            }
          }
          pos = (pos + 1) & a.index_mask;
        }
      }
    }
  }
  if (lane == 0) {
    a.ch.status[g] = len < kPaperMinCached ? kUncached : hit ? kHit0 : cand ? kMissCand : kMissNoCand;
    a.ch.key[g] = key;
    a.ch.len[g] = len;
    a.ch.src[g] = (unsigned long long)p;
    a.ch.pidx[g] = pid;
    a.ch.hint[g] = 0;
    if (hit) a.ch.ent[g] = hit_slot;
  }
}

Md5Table md5_table() {
  Md5Table t;
  for (int i = 0; i < 64; ++i)
    t.k[i] = (uint32_t)std::floor(std::fabs(std::sin((double)(i + 1))) * 4294967296.0);
  return t;
}

}  // namespace

// Loads this file's kernels on the current device (a query of one of them
// loads the module that holds them all, when the runtime loads modules lazily).
cudaError_t load_hash_kernels() {
  cudaFuncAttributes fa;
  return cudaFuncGetAttributes(&fa, k_hash_probe_staged<true, false, true>);
}

bool hash_is_staged(const HashArgs& a, bool aligned) {
#if GLEAM_STAGED_HASH
  return a.Ntot > 0 && !(a.index != nullptr && a.paper) && aligned && (a.C % 32 == 0 || a.Ntot == 1);
#else
  return false;
#endif
}

cudaError_t launch_hash(const HashArgs& a, bool aligned, cudaStream_t s, bool pdl) {
  if (a.Ntot == 0) return cudaSuccess;
  const unsigned long long threads = a.Ntot * 4;
  const unsigned grid = (unsigned)((threads + kHashThreads - 1) / kHashThreads);
  const bool probe = a.index != nullptr;
  if (probe && a.paper) {
    static const Md5Table tab = md5_table();
#if GLEAM_STAGED_HASH
    if (aligned && a.C % 32 == 0) {
      const unsigned sg = (unsigned)((threads + kStagedThreads - 1) / kStagedThreads);
      return launch_kernel(k_probe_paper_staged, dim3(sg), dim3(kStagedThreads), kStagedSmem, s,
                           pdl, a, tab);
    }
#endif
    return aligned ? launch_kernel(k_probe_paper<true>, dim3(grid), dim3(kHashThreads), 0, s,
                                   pdl, a, tab)
                   : launch_kernel(k_probe_paper<false>, dim3(grid), dim3(kHashThreads), 0, s,
                                   pdl, a, tab);
  }
#if GLEAM_STAGED_HASH
  if (aligned && (a.C % 32 == 0 || a.Ntot == 1)) {
    // no cached copy is streamed when only fingerprints are wanted or the
    // cache holds no chunk (or too few to be worth the hint lookups): the
    // variant without those buffers
    if (!probe) return launch_staged<false, false, false>(a, s, pdl);
    if (a.no_hints)
      return a.spec_mode ? launch_staged<true, true, false>(a, s, pdl)
                         : launch_staged<true, false, false>(a, s, pdl);
    return a.spec_mode ? launch_staged<true, true, true>(a, s, pdl)
                       : launch_staged<true, false, true>(a, s, pdl);
  }
#endif
  const dim3 g3(grid), b3(kHashThreads);
  if (aligned && probe) return launch_kernel(k_hash_probe<true, true>, g3, b3, 0, s, pdl, a);
  if (aligned) return launch_kernel(k_hash_probe<true, false>, g3, b3, 0, s, pdl, a);
  if (probe) return launch_kernel(k_hash_probe<false, true>, g3, b3, 0, s, pdl, a);
  return launch_kernel(k_hash_probe<false, false>, g3, b3, 0, s, pdl, a);
}

}  // namespace gleam
