// Fingerprint + index probe + byte verify of every chunk of a payload
// (paper Sec. 4.1.2: hash the source bytes, look the hash up in the set of
// resident chunks; App. B.1: confirm the match so collisions cannot alias).
//
// Mapping: a group of 4 consecutive threads owns one chunk; thread `lane`
// runs XXH64 accumulator lane `lane`, reading the 8-byte word at 8*lane of
// each 32-byte stripe straight from HBM (8 loads in flight per thread, the
// next batch issued before the current one is folded in).  A warp therefore
// streams 8 chunks at once and every 32-byte sector it touches is used whole.
// The group then probes the index and compares each key+length candidate
// with the cached copy, 8 bytes per thread per stripe.
#include "gleam_internal.cuh"
#include "xxh64_device.cuh"

namespace gleam {
namespace {

constexpr int kHashThreads = 256;
constexpr int kBatch = 8;  // stripes per thread in flight

// 8-byte load of read-only payload bytes, no L1 allocation, L2 fetches 256 B.
template <bool kAligned>
__device__ __forceinline__ unsigned long long load_word(const uint8_t* p) {
  if (kAligned) {
    unsigned long long v;
    asm("ld.global.nc.L1::no_allocate.L2::256B.u64 %0, [%1];" : "=l"(v) : "l"(p));
    return v;
  } else {
    return load_le64_bytes(p);
  }
}

__device__ __forceinline__ unsigned long long load_arena_word(const uint8_t* p) {
  unsigned long long v;
  asm("ld.global.nc.L1::no_allocate.L2::256B.u64 %0, [%1];" : "=l"(v) : "l"(p));
  return v;
}

__device__ __forceinline__ unsigned long long group_shfl(unsigned long long v, unsigned gmask,
                                                         int src) {
  return __shfl_sync(gmask, v, src);
}

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

// Byte equality of payload chunk p and cached chunk q over len bytes, by the
// 4-thread group; leaves early once any word differs.
template <bool kAligned>
__device__ __forceinline__ bool group_equal(const uint8_t* p, const uint8_t* q, uint32_t len,
                                            uint32_t lane, unsigned gmask) {
  const uint32_t ns = len >> 5;
  unsigned long long diff = 0;
  for (uint32_t s = 0; s < ns; s += kBatch) {
    const uint32_t m = min((uint32_t)kBatch, ns - s);
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      if ((uint32_t)u < m) {
        const uint64_t off = (uint64_t)(s + u) * 32 + 8 * lane;
        diff |= load_word<kAligned>(p + off) ^ load_arena_word(q + off);
      }
    }
    diff |= __shfl_xor_sync(gmask, diff, 1);
    diff |= __shfl_xor_sync(gmask, diff, 2);
    if (diff) return false;
  }
  if (lane == 0) {
    for (uint32_t k = ns * 32; k < len; ++k) diff |= (unsigned long long)(p[k] ^ q[k]);
  }
  diff |= __shfl_xor_sync(gmask, diff, 1);
  diff |= __shfl_xor_sync(gmask, diff, 2);
  return diff == 0;
}

template <bool kAligned, bool kProbe>
__global__ void __launch_bounds__(kHashThreads) k_hash_probe(HashArgs a) {
  const unsigned long long g = ((unsigned long long)blockIdx.x * blockDim.x + threadIdx.x) >> 2;
  if (g >= a.Ntot) return;  // whole groups leave together
  const uint32_t lane = threadIdx.x & 3;
  const int gbase = threadIdx.x & 28;
  const unsigned gmask = 0xFu << gbase;

  uint32_t pid = 0;
  const uint8_t* buf;
  unsigned long long n, base;
  if (a.count > 1) {
    pid = find_payload(a.table, a.count, g);
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

  unsigned long long h;
  if (ns) {
    const unsigned long long acc = lane_stripes<kAligned>(xlane_start(lane), p + 8 * lane, ns);
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

  const unsigned long long key = a.key16 ? (h & 0xFFFFULL) : h;
  const unsigned long long slots_used = a.dstats[ST_SLOTS_USED];
  unsigned long long pos = mix64(key) & a.index_mask;
  bool hit = false, cand = false;
  for (unsigned long long probe = 0; probe <= a.index_mask; ++probe) {
    const IndexEntry e = a.index[pos];
    if (e.slot == kEmptySlot) break;
    if (e.key == key && e.len == len) {
      cand = true;
      if (e.slot >= slots_used) {
        // an entry pointing past the used slots: report, never read it
        if (lane == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
      } else if (group_equal<kAligned>(p, a.arena + (uint64_t)e.slot * a.C, len, lane, gmask)) {
        hit = true;
        break;
      }
    }
    pos = (pos + 1) & a.index_mask;
  }
  if (lane == 0) {
    a.ch.status[g] = hit ? kHit0 : (cand ? kMissCand : kMissNoCand);
    a.ch.key[g] = key;
    a.ch.len[g] = len;
    a.ch.src[g] = (unsigned long long)p;
    a.ch.pidx[g] = pid;
  }
}

}  // namespace

cudaError_t launch_hash(const HashArgs& a, bool aligned, cudaStream_t s) {
  if (a.Ntot == 0) return cudaSuccess;
  const unsigned long long threads = a.Ntot * 4;
  const unsigned grid = (unsigned)((threads + kHashThreads - 1) / kHashThreads);
  const bool probe = a.index != nullptr;
  if (aligned && probe) k_hash_probe<true, true><<<grid, kHashThreads, 0, s>>>(a);
  else if (aligned) k_hash_probe<true, false><<<grid, kHashThreads, 0, s>>>(a);
  else if (probe) k_hash_probe<false, true><<<grid, kHashThreads, 0, s>>>(a);
  else k_hash_probe<false, false><<<grid, kHashThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace gleam
