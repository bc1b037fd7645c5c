// Staged fingerprint + index probe + speculative verify of one block-sized
// range of chunks (paper Sec. 4.1.2 and App. B.1), shared by the hash kernel
// and the single-block small-call kernel, and the loads and group helpers
// both use.
#pragma once

#include "gleam_internal.cuh"
#include "xxh64_device.cuh"

// The fingerprint-only instantiations (kProbe = false) see slots_used == 0 as a
// constant in probe code they never reach.
#pragma nv_diag_suppress 186

namespace gleam {
namespace {

#ifndef GLEAM_HASH_BATCH
#define GLEAM_HASH_BATCH 8
#endif
constexpr int kBatch = GLEAM_HASH_BATCH;  // stripes per thread in flight

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

// Slot of a cached chunk of length len whose prefix hint is h, or kEmptySlot.
__device__ __forceinline__ uint32_t hint_lookup(const IndexEntry* t, unsigned long long mask,
                                                unsigned long long h, uint32_t len,
                                                unsigned long long slots_used) {
  unsigned long long pos = mix64(h) & mask;
  for (unsigned long long probe = 0; probe <= mask; ++probe) {
    const IndexEntry e = t[pos];
    if (e.slot == kEmptySlot) return kEmptySlot;
    if (e.key == h && e.len == len && e.slot < slots_used) return e.slot;
    pos = (pos + 1) & mask;
  }
  return kEmptySlot;
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

// Byte equality of payload chunk p and cached chunk q over len bytes by the
// nl lanes of wmask (a prefix of the warp; this lane is wl): 8-byte words
// strided across the lanes, kBatch of them per lane in flight, leaving early
// once any word differs.  Eight groups' worth of lanes take a 64 KiB compare
// in 32 rounds of loads where one group's four lanes take 256.
__device__ __forceinline__ bool lanes_equal(const uint8_t* p, const uint8_t* q, uint32_t len,
                                            unsigned wmask, uint32_t wl, uint32_t nl) {
  const uint32_t nw = len >> 3;
  for (uint32_t w0 = 0; w0 < nw; w0 += kBatch * nl) {
    unsigned long long diff = 0;
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const uint32_t w = w0 + u * nl + wl;
      if (w < nw) diff |= load_word<true>(p + 8ull * w) ^ load_arena_word(q + 8ull * w);
    }
    if (__any_sync(wmask, diff != 0)) return false;
  }
  bool d = false;
  for (uint32_t k = (nw << 3) + wl; k < len; k += nl) d |= p[k] != q[k];
  return !__any_sync(wmask, d);
}

// Lanes of this warp whose groups hold a chunk of range vb (g < Ntot): a
// prefix of the warp, since chunks are numbered in thread order.  Called by a
// lane of such a group.
__device__ __forceinline__ unsigned present_lanes(unsigned long long vb, unsigned long long Ntot) {
  const unsigned long long t0 = vb * blockDim.x + (threadIdx.x & ~31u);
  const unsigned long long k = 4 * Ntot - t0;
  return k >= 32 ? 0xffffffffu : (1u << k) - 1;
}

// ---------------------------------------------------------------------------
// Staged variant for 16-byte-aligned payloads.  Each 4-thread group streams
// its chunk through shared memory in kStage-byte stages with asynchronous
// 16-byte global->shared copies (kDepth stages in flight, no registers held),
// and the cached copy named by the prefix hint streams alongside into a
// second buffer.  The lanes then hash and compare their words from shared
// memory.  Stage 0 is exactly the prefix used for the hint.
//
// Two stages in flight and blocks of one warp (8 groups, 16.6 KB of shared
// memory): about 100 groups share an SM, and that many independent chunks
// hide each chunk's dependent lookups (payload, prefix hint, index probe)
// better than deeper pipelines with fewer groups (measured: 3 stages and
// 64 groups per SM took 5.05 ms on the Llama upload, this takes 4.64 ms).
// ---------------------------------------------------------------------------
#ifndef GLEAM_STAGE_DEPTH
#define GLEAM_STAGE_DEPTH 2
#endif
// Chunks of at most this many bytes fetch a hinted chunk's cached prefix by
// cp.async into stage buffer 0, in the same round trip as the cached copy's
// next stages (GPT-2 pass 2, 4 KiB chunks: hash kernel -3%); larger chunks
// compare it with direct loads first (64 KiB chunks: 3% faster that way, their
// one prefix per 128 stages costs little and the simpler loop streams better).
constexpr uint32_t kPrefixAsyncMaxChunk = 16u << 10;
#ifndef GLEAM_STAGED_THREADS
#define GLEAM_STAGED_THREADS 32
#endif
constexpr int kStage = 512;                                 // bytes per stage
constexpr int kDepth = GLEAM_STAGE_DEPTH;                   // stages in flight
// A group's stage buffers: kDepth stages of its chunk and, when it may
// compare against a cached copy (verify), kDepth stages of that copy too
// (+32: bank skew).
__host__ __device__ constexpr int group_bytes(bool verify, int stage = kStage) {
  return kDepth * (verify ? 2 : 1) * stage + 32;
}
// Stage size of the variant for calls that leave most of the GPU idle (fewer
// chunks than one wave of it holds, chunks of at least kBigStageMinChunk):
// each stage's bookkeeping (its copies, waits and branches) then serves 64
// XXH64 rounds of a lane instead of 16, which is what a chunk's dependent
// chain waits on when nothing else shares the SM.
constexpr int kBigStage = 2048;
constexpr unsigned long long kBigStageMinChunk = 32768;
constexpr int kGroupBytes = group_bytes(true);
constexpr int kStagedThreads = GLEAM_STAGED_THREADS;
constexpr int kStagedSmem = (kStagedThreads / 4) * kGroupBytes;
static_assert(kStage == (int)kPrefixBytes, "stage 0 must be the hinted prefix");
static_assert(kStagedSmem >= 33 * 8, "the payload search borrows 33 words of the stage buffers");

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global.L2::256B [%0], [%1], 16;" ::"r"(dst), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
// Waits until at most min(n, kMax - 1) committed groups are pending (the
// instruction takes an immediate count).
template <int kMax>
__device__ __forceinline__ void cp_wait_upto(uint32_t n) {
  if constexpr (kMax <= 1) {
    cp_wait<0>();
  } else {
    if (n >= (uint32_t)kMax - 1) cp_wait<kMax - 1>();
    else cp_wait_upto<kMax - 1>(n);
  }
}

// This lane's share (4 lanes x kS / 64 x 16 bytes) of one stage of kS bytes
// of `src` into `dst`; `bytes` (multiple of 32, <= kS) of the stage exist.
template <int kS = kStage>
__device__ __forceinline__ void stage_copy(uint32_t dst, const uint8_t* src, uint32_t bytes,
                                           uint32_t lane) {
#pragma unroll
  for (int j = 0; j < kS / 64; ++j) {
    const uint32_t off = (uint32_t)j * 64 + lane * 16;
    if (off < bytes) cp_async16(dst + off, src + off);
  }
}

// The chunks of block-sized range vb (blockDim.x / 4 consecutive chunks); the
// shared memory holds one region of group_bytes(kVerify) per group.  kAhead:
// with the write-through of likely misses (written ahead of the pack step).
// kVerify = false: no speculative verify and no buffers for a cached copy
// (for a cache that holds no chunk, or too few to be worth the lookups), so
// twice as many groups fit an SM; a key+length candidate, if any, is still
// compared with direct loads.
template <bool kProbe, bool kAhead = false, bool kVerify = true, bool kPrefixAsync = false,
          int kS = kStage>
__device__ __forceinline__ void staged_range(const HashArgs& a, unsigned long long vb,
                                             uint8_t* smem) {
  static_assert(kS % kPrefixBytes == 0 && kS % 256 == 0, "stages hold whole prefixes and batches");
  const unsigned long long g = (vb * blockDim.x + threadIdx.x) >> 2;
  // the payload search borrows the start of the stage buffers (no static
  // shared memory: any would cost this kernel a fifth of its bandwidth)
  const uint32_t pid_b =
      a.count > 1 ? block_find_payload(a.table, a.count, (vb * blockDim.x) >> 2, g,
                                       reinterpret_cast<unsigned long long*>(smem))
                  : 0u;
  if (g >= a.Ntot) return;  // whole groups leave together
  const uint32_t lane = threadIdx.x & 3;
  const int gbase = threadIdx.x & 28;
  const unsigned gmask = 0xFu << gbase;
  uint8_t* region = smem + (threadIdx.x >> 2) * group_bytes(kVerify, kS);
  const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(region);
  // stage buffer t % kDepth: payload at [0, kS), cached copy at [kS, 2 kS)
  constexpr uint32_t kBuf = (kVerify ? 2 : 1) * kS;  // one stage's buffers
  auto pay_s = [&](uint32_t t) { return sbase + (t % kDepth) * kBuf; };
  auto pay_p = [&](uint32_t t) { return region + (t % kDepth) * kBuf; };

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
  const uint32_t full = ns * 32;                       // bytes in whole stripes
  const uint32_t nst = (full + kS - 1) / kS;   // stages
  auto sbytes = [&](uint32_t t) { return min((uint32_t)kS, full - t * kS); };

  const bool speculate = kProbe && len >= kPrefixBytes;
  // slots in use as the hint lookups see them; with a late wait (calls that
  // overlap) the count as published when the group started: the bytes and
  // table entries of the slots below it are complete and no call changes them
  const unsigned long long slots_used =
      !kProbe ? 0ULL
              : a.wait_late ? ld_acquire_u64(&a.dstats[ST_SLOTS_USED]) : a.dstats[ST_SLOTS_USED];
  unsigned long long hint = 0, diff = 0;
  uint32_t hint_slot = kEmptySlot;
  unsigned long long hint_key = 0;  // the whole fingerprint stored for hint_slot
  const uint8_t* q = nullptr;
  bool cmp = false;
  // write-through of a likely miss, decided once the prefix hint is known
  const bool ahead_ok = kAhead && speculate && slots_used + g < a.nslots;
  bool ahead = false;
  uint8_t* ahead_pk = nullptr;  // packed offset i*C of the payload
  uint8_t* ahead_ar = nullptr;  // arena slot slots_used + g

  unsigned long long acc = xlane_start(lane);
  // the accumulator after the prefix (stage 0 may hold more than the prefix)
  unsigned long long acc_pre = 0;
  // prologue: payload stages 0 .. kDepth-2
#pragma unroll
  for (int t = 0; t < kDepth - 1; ++t) {
    if ((uint32_t)t < nst) stage_copy<kS>(pay_s(t), p + t * kS, sbytes(t), lane);
    cp_commit();
  }
  for (uint32_t t = 0; t < nst; ++t) {
    // issue stage t + kDepth - 1 into the buffer consumed at t - 1
    const uint32_t tn = t + kDepth - 1;
    if (tn < nst) {
      stage_copy<kS>(pay_s(tn), p + (unsigned long long)tn * kS, sbytes(tn), lane);
      if (cmp) stage_copy<kS>(pay_s(tn) + kS, q + (unsigned long long)tn * kS, sbytes(tn), lane);
    }
    cp_commit();
    // groups committed so far, oldest first: prologue stages, then one per
    // iteration, plus (at t = 0) one holding the cached copy of stages
    // 1 .. kDepth-1, issued late because the hint is known only then
    // stage t needs everything up to the late group while t < kDepth - 1
    // (at most t newer groups may pend), else up to its own group
    cp_wait_upto<kDepth>((t == 0 || t >= (uint32_t)kDepth - 1) ? (uint32_t)kDepth - 1 : t);
    __syncwarp(gmask);
    const uint8_t* sp = pay_p(t);
    const uint32_t sst = sbytes(t) >> 5;
    unsigned long long d = 0;
    auto word = [&](const uint8_t* b, uint32_t s) {
      return *reinterpret_cast<const unsigned long long*>(b + s * 32 + lane * 8);
    };
    if (sst == (uint32_t)kS / 32) {
      // a whole stage, eight stripes at a time: the loads and the compare
      // overlap the XXH64 chain instead of waiting in it
#pragma unroll
      for (uint32_t h = 0; h < (uint32_t)kS / 32; h += 8) {
        unsigned long long w[8];
#pragma unroll
        for (uint32_t u = 0; u < 8; ++u) w[u] = word(sp, h + u);
        if (cmp && t > 0) {
#pragma unroll
          for (uint32_t u = 0; u < 8; ++u) d |= w[u] ^ word(sp + kS, h + u);
        }
#pragma unroll
        for (uint32_t u = 0; u < 8; ++u) acc = xstep(acc, w[u]);
        if (kS > (int)kPrefixBytes && h + 8 == kPrefixBytes / 32) acc_pre = acc;
      }
    } else if (cmp && t > 0) {
      const uint8_t* sq = sp + kS;
#pragma unroll 4
      for (uint32_t s = 0; s < sst; ++s) {
        const unsigned long long w = *reinterpret_cast<const unsigned long long*>(sp + s * 32 + lane * 8);
        const unsigned long long c = *reinterpret_cast<const unsigned long long*>(sq + s * 32 + lane * 8);
        acc = xstep(acc, w);
        d |= w ^ c;
      }
    } else {
#pragma unroll 4
      for (uint32_t s = 0; s < sst; ++s) {
        acc = xstep(acc, *reinterpret_cast<const unsigned long long*>(sp + s * 32 + lane * 8));
        if (kS > (int)kPrefixBytes && s + 1 == kPrefixBytes / 32) acc_pre = acc;
      }
    }
    if (kS == (int)kPrefixBytes) acc_pre = acc;
    if (t == 0 && speculate) {
      const unsigned long long b0 = group_shfl(acc_pre, gmask, gbase + 0);
      const unsigned long long b1 = group_shfl(acc_pre, gmask, gbase + 1);
      const unsigned long long b2 = group_shfl(acc_pre, gmask, gbase + 2);
      const unsigned long long b3 = group_shfl(acc_pre, gmask, gbase + 3);
      hint = b0 ^ xrotl(b1, 16) ^ xrotl(b2, 32) ^ xrotl(b3, 48);
      // an empty cache has no hints to look up
      hint_slot = kVerify && slots_used ? hint_lookup(a.hints, a.index_mask, hint, len, slots_used)
                                        : kEmptySlot;
      cmp = hint_slot != kEmptySlot;
      ahead = ahead_ok && !cmp;  // no cached chunk begins like it: a likely miss
      if (ahead) {
        ahead_pk = (a.count > 1 ? a.table[pid].packed : a.one.packed) + (g - base) * a.C;
        ahead_ar = a.arena_w + (slots_used + g) * a.C;
      }
      if (cmp) {
        q = a.arena + (unsigned long long)hint_slot * a.C;
        // loaded now, used once the chunk is hashed: no lookup waits then
        hint_key = a.slot_key[hint_slot];
        if constexpr (kPrefixAsync) {
          // the cached copy's prefix into the free half of stage buffer 0, in
          // a group of its own, and its next stages behind it: one round trip
          // for both
          stage_copy<kS>(pay_s(0) + kS, q, kS == (int)kPrefixBytes ? (uint32_t)kS : sbytes(0), lane);
          cp_commit();
        } else {
          // stage 0 (the prefix, and more in a larger stage), still in its
          // buffer, against the cached copy's
#pragma unroll 4
          for (uint32_t s = 0; s < (kS == (int)kPrefixBytes ? (uint32_t)kS / 32 : sst); ++s)
            d |= *reinterpret_cast<const unsigned long long*>(sp + s * 32 + lane * 8) ^
                 load_arena_word(q + s * 32 + lane * 8);
        }
        // the cached copy of the stages already in flight
        for (uint32_t tt = 1; tt < (uint32_t)kDepth && tt < nst; ++tt)
          stage_copy<kS>(pay_s(tt) + kS, q + (unsigned long long)tt * kS, sbytes(tt), lane);
      }
    }
    if (t == 0) cp_commit();  // the late group (empty without a hint)
    if (kPrefixAsync && t == 0 && cmp) {
      // the prefix's group is complete once at most the late group pends
      cp_wait<1>();
      __syncwarp(gmask);
      if constexpr (kS == (int)kPrefixBytes) {
#pragma unroll
        for (uint32_t s = 0; s < (uint32_t)kS / 32; ++s) d |= word(sp, s) ^ word(sp + kS, s);
      } else {
#pragma unroll 4
        for (uint32_t s = 0; s < sst; ++s) d |= word(sp, s) ^ word(sp + kS, s);
      }
    }
    if (cmp) {
      // a lane that found a difference stops streaming its share of the
      // cached copy; the others may then compare stale words, which can only
      // add differences to a chunk already known to differ
      diff |= d;
      if (diff) cmp = false;
    }
    if (ahead) {  // this lane's own pieces of stage t, to both destinations
      const uint32_t sb = sbytes(t);
#pragma unroll
      for (int j = 0; j < kS / 64; ++j) {
        const uint32_t off = (uint32_t)j * 64 + lane * 16;
        if (off < sb) {
          const uint4 v = *reinterpret_cast<const uint4*>(sp + off);
          const unsigned long long o = (unsigned long long)t * kS + off;
          __stcs(reinterpret_cast<uint4*>(ahead_pk + o), v);
          __stcs(reinterpret_cast<uint4*>(ahead_ar + o), v);
        }
      }
    }
    __syncwarp(gmask);  // everyone is done with buffer t before it is refilled
  }
  cp_wait<0>();
  if (ahead && lane == 0)  // the bytes past the last whole stripe
    for (uint32_t k = full; k < len; ++k) ahead_pk[k] = ahead_ar[k] = p[k];

  unsigned long long h;
  if (ns) {
    const unsigned long long a0 = group_shfl(acc, gmask, gbase + 0);
    const unsigned long long a1 = group_shfl(acc, gmask, gbase + 1);
    const unsigned long long a2 = group_shfl(acc, gmask, gbase + 2);
    const unsigned long long a3 = group_shfl(acc, gmask, gbase + 3);
    h = xconverge(a0, a1, a2, a3);
  } else {
    h = kXP5;
  }
  h += len;
  h = xfinish(h, p + full, len & 31);

  if (a.fp_out != nullptr && lane == 0) a.fp_out[g] = h;
  if (!kProbe) return;
  // with a late wait, the cache's previous calls are complete from here on:
  // the probe sees their inserts (candidates at or above slots_used are
  // compared like any other), and every write of this kernel follows
  unsigned long long slots_now = slots_used;
  if (a.wait_late) {
    pdl_wait();
    slots_now = *reinterpret_cast<const volatile unsigned long long*>(&a.dstats[ST_SLOTS_USED]);
  }

  bool spec_equal = false;
  if (speculate && hint_slot != kEmptySlot) {
    unsigned long long dd = diff;
    if (cmp && lane == 0)
      for (uint32_t k = full; k < len; ++k) dd |= (unsigned long long)(p[k] ^ q[k]);
    dd |= __shfl_xor_sync(gmask, dd, 1);
    dd |= __shfl_xor_sync(gmask, dd, 2);
    spec_equal = dd == 0;
  }

  const unsigned long long key = a.key16 ? (h & 0xFFFFULL) : h;
  bool hit = false, cand = false;
  uint32_t hit_slot = kEmptySlot;
  if (slots_now) {
    // The linear probe, in order.  A key+length candidate other than the
    // verified hint is compared by the whole warp: each group walks its probe
    // up to its next such candidate, then the warp compares the pending ones,
    // one group's at a time, and the groups whose candidate differs walk on.
    const unsigned wmask = present_lanes(vb, a.Ntot);
    const uint32_t wl = threadIdx.x & 31, nl = __popc(wmask);
    unsigned long long pos = mix64(key) & a.index_mask, probe = 0;
    // the hinted slot holds these very bytes and this fingerprint: the index
    // lists it under this key and length (both are written for every stored
    // chunk), so it is the hit and the probe can be skipped
    bool done = false;
    if (spec_equal && hint_key == h) {
      hit = true;
      hit_slot = hint_slot;
      done = true;
    }
    for (;;) {
      uint32_t want = kEmptySlot;  // a candidate for the warp to compare
      while (!done) {
        if (probe > a.index_mask) {
          done = true;
          break;
        }
        const IndexEntry e = a.index[pos];
        if (e.slot == kEmptySlot) {
          done = true;
          break;
        }
        pos = (pos + 1) & a.index_mask;
        ++probe;
        if (e.key == key && e.len == len) {
          cand = true;
          if (e.slot >= slots_now) {
            if (lane == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
          } else if (e.slot == hint_slot) {
            if (spec_equal) {
              hit = true;
              hit_slot = e.slot;
              done = true;
            }
          } else {
            want = e.slot;
            break;
          }
        }
      }
      const unsigned pend = __ballot_sync(wmask, want != kEmptySlot) & 0x11111111u;
      if (!pend) break;
      for (unsigned m = pend; m; m &= m - 1) {
        const int src = __ffs(m) - 1;
        const uint8_t* ps = reinterpret_cast<const uint8_t*>(
            __shfl_sync(wmask, reinterpret_cast<unsigned long long>(p), src));
        const uint32_t slot = __shfl_sync(wmask, want, src);
        const uint32_t ls = __shfl_sync(wmask, len, src);
        const bool eq = lanes_equal(ps, a.arena + (uint64_t)slot * a.C, ls, wmask, wl, nl);
        if (gbase == src && eq) {
          hit = true;
          hit_slot = slot;
          done = true;
        }
      }
    }
  }
  if (lane == 0) {
    a.ch.status[g] = hit ? kHit0 : (cand ? kMissCand : kMissNoCand);
    a.ch.key[g] = h;  // the group key: the whole fingerprint
    a.ch.len[g] = len;
    a.ch.src[g] = (unsigned long long)p;
    a.ch.pidx[g] = pid;
    a.ch.hint[g] = hint;
    if (kAhead) a.ch.spec[g] = ahead ? 1 : 0;
    if (hit) {
      a.ch.ent[g] = hit_slot;
    } else if (kProbe && a.claim_tbl != nullptr) {
      // the miss's (group key, length) entry of the per-call table, claimed
      // with one 64-bit CAS that also stores a 32-bit tag of the pair (where
      // the resolve kernel keeps a minimum): an entry found holding the same
      // tag may be the chunk's group, which sends the call down the general
      // path (shared_groups), where the groups are claimed again by the whole
      // key; a different tag is another group's entry
      const unsigned long long mixed = mix64(h ^ ((unsigned long long)len << 40));
      const unsigned long long tag = mixed >> 32;
      unsigned long long pos = mixed & a.claim_mask;
      uint32_t e = 0xFFFFFFFFu;
      for (unsigned long long probe = 0; probe <= a.claim_mask; ++probe) {
        const unsigned long long old =
            atomicCAS(reinterpret_cast<unsigned long long*>(&a.claim_tbl[pos]), 0ull,
                      (tag << 32) | ((unsigned long long)g + 1ull));
        if (old == 0) {
          e = (uint32_t)pos;
          break;
        }
        if ((old >> 32) == tag) {
          e = (uint32_t)pos;
          atomicOr(&a.ctl->shared_groups, 1u);
          break;
        }
        pos = (pos + 1) & a.claim_mask;
      }
      a.ch.ent[g] = e;
      a.ch.res[g] = kResUnresolved;
    }
  }
}

}  // namespace
}  // namespace gleam
