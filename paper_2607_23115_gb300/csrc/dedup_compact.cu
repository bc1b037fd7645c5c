// First-occurrence resolution, stream compaction, packing and insertion for
// one dedup call (paper Sec. 4.1.2: a chunk that is not resident "is
// transmitted in full" and becomes reusable).
//
// The result must equal deciding the chunks one at a time in ascending
// order.  Given the probe/verify outcome against the cache as it was at the
// start of the call (kHit0 or not), that sequential rule reduces to:
//   * a non-resident chunk is a hit iff an earlier chunk of the call has the
//     same bytes, and its leader is the first such chunk;
//   * the misses are the leaders, inserted in ascending order at
//     slot = slots_used + rank;
//   * a leader counts as a verify reject iff the cache had a key+length
//     candidate for it, or an earlier leader of the call has its key+length.
//
// One cooperative launch does it all, separated by bounded grid barriers:
//   A  every non-resident full chunk claims its key's entry in a per-call
//      table and posts its index as the group minimum;
//   B  each unresolved chunk compares itself (whole warp, 16-byte loads) with
//      its group's minimum: equal -> duplicate, index == minimum -> leader
//      of this round, else it stays for the next round (only different bytes
//      under one key: a true 64-bit collision, or KEY16 test mode);
//   C  group minima of the remaining chunks are reset and re-posted (A);
//   D  leaders are counted per contiguous block range, ranks come from the
//      block totals plus warp ballots, and the hit mask, miss indices,
//      packed bytes, arena copies and index entries are written.
// The last block to finish publishes the counters and the call result.
#include "gleam_internal.cuh"

namespace gleam {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

__device__ __forceinline__ uint32_t ldcg_u32(const uint32_t* p) { return __ldcg(p); }

__device__ __forceinline__ uint32_t chunk_len(const DedupArgs& a, uint32_t i) {
  const uint64_t start = (uint64_t)i * a.C;
  return (uint32_t)min(a.C, a.n - start);
}

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

// Whole-warp copy of one chunk to the packed output and to its arena slot.
__device__ void warp_copy2(uint8_t* d1, uint8_t* d2, const uint8_t* s, uint32_t len, bool vec) {
  const uint32_t lane = threadIdx.x & 31;
  uint32_t done = 0;
  if (vec) {
    const uint32_t nv = len >> 4;
    const uint4* sv = reinterpret_cast<const uint4*>(s);
    uint4* d1v = reinterpret_cast<uint4*>(d1);
    uint4* d2v = reinterpret_cast<uint4*>(d2);
    for (uint32_t k0 = 0; k0 < nv; k0 += 128) {
      uint4 u[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const uint32_t k = k0 + r * 32 + lane;
        if (k < nv) u[r] = __ldcs(sv + k);
      }
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const uint32_t k = k0 + r * 32 + lane;
        if (k < nv) {
          __stcs(d1v + k, u[r]);
          __stcs(d2v + k, u[r]);
        }
      }
    }
    done = nv << 4;
  }
  for (uint32_t k = done + lane; k < len; k += 32) {
    const uint8_t b = s[k];
    d1[k] = b;
    d2[k] = b;
  }
}

// Claims a free index entry for (key, slot, len); false if the table is full.
__device__ bool index_insert(IndexEntry* index, uint64_t mask, unsigned long long key,
                             uint32_t slot, uint32_t len) {
  uint64_t pos = mix64(key) & mask;
  for (uint64_t probe = 0; probe <= mask; ++probe) {
    const uint32_t old = atomicCAS(&index[pos].slot, kEmptySlot, slot);
    if (old == kEmptySlot) {
      index[pos].key = key;
      index[pos].len = len;
      return true;
    }
    pos = (pos + 1) & mask;
  }
  return false;
}

// Finds or claims the per-call table entry of a full chunk's key.
__device__ uint32_t group_entry(const DedupArgs& a, uint32_t i, unsigned long long k) {
  uint64_t pos = mix64(k) & a.tbl_mask;
  for (uint64_t probe = 0; probe <= a.tbl_mask; ++probe) {
    uint32_t o = ldcg_u32(&a.tbl[pos].owner);
    if (o == 0) {
      o = atomicCAS(&a.tbl[pos].owner, 0u, i + 1);
      if (o == 0) return (uint32_t)pos;
    }
    if (a.key[o - 1] == k) return (uint32_t)pos;
    pos = (pos + 1) & a.tbl_mask;
  }
  return 0xFFFFFFFFu;  // cannot happen: the table has >= 2N entries
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

__global__ void __launch_bounds__(kThreads) k_dedup(DedupArgs a) {
  __shared__ unsigned long long red64[kWarps];
  __shared__ uint32_t warp_cnt[kWarps];
  __shared__ uint32_t warp_off[kWarps];
  __shared__ uint32_t list_i[kThreads];
  __shared__ uint32_t list_r[kThreads];
  __shared__ unsigned long long s_slots0;

  const uint32_t G = gridDim.x;
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t tid = blockIdx.x * kThreads + threadIdx.x;
  const uint32_t nth = G * kThreads;
  const uint32_t N = a.N;
  const bool skip = (int)blockIdx.x == a.skip_block;
  const bool vec_buf = ((uintptr_t)a.buf % 16) == 0;

  if (threadIdx.x == 0) s_slots0 = *(volatile const unsigned long long*)&a.dstats[ST_SLOTS_USED];
  __syncthreads();
  const unsigned long long slots0 = s_slots0;

  // ---- A: round-1 claims -------------------------------------------------
  if (!skip) {
    for (uint32_t i = tid; i < N; i += nth) {
      if (a.status[i] == kHit0) {
        a.res[i] = kResHit0;
        continue;
      }
      if (chunk_len(a, i) != a.C) {  // the short last chunk: unique length
        a.res[i] = kResLeader | 1u;
        a.ent[i] = 0xFFFFFFFFu;
        continue;
      }
      const uint32_t e = group_entry(a, i, a.key[i]);
      if (e == 0xFFFFFFFFu) {
        atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
        a.res[i] = kResLeader | 1u;
        continue;
      }
      a.ent[i] = e;
      a.res[i] = kResUnresolved;
      atomicMax(&a.tbl[e].minv, ~i);
    }
  }
  bool ok = grid_barrier(a.ctl, G, a.wait_ns, skip);

  // ---- B/C: rounds until every chunk is a hit, duplicate or leader ---------
  uint32_t round = 1;
  while (ok) {
    if (tid == 0) atomicExch(&a.ctl->unres[(round + 1) % 3], 0u);
    const uint32_t nwarps = nth / 32;
    for (uint32_t base = (tid / 32) * 32; base < N; base += nwarps * 32) {
      const uint32_t i = base + lane;
      bool need = false;
      uint32_t m = 0;
      if (i < N && ldcg_u32(&a.res[i]) == kResUnresolved) {
        m = ~ldcg_u32(&a.tbl[a.ent[i]].minv);
        if (m == i) {
          a.res[i] = kResLeader | round;
        } else if (m > i) {  // the group minimum can only be below i: table damaged
          atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
          a.res[i] = kResLeader | round;
        } else {
          need = true;
        }
      }
      uint32_t todo = __ballot_sync(0xffffffffu, need);
      while (todo) {
        const int j = __ffs(todo) - 1;
        todo &= todo - 1;
        const uint32_t ii = base + j;
        const uint32_t mm = __shfl_sync(0xffffffffu, m, j);
        const bool eq = warp_equal(a.buf + (uint64_t)ii * a.C, a.buf + (uint64_t)mm * a.C,
                                   (uint32_t)a.C, vec_buf);
        if (lane == (uint32_t)j) {
          if (eq) a.res[ii] = kResDup;
          else atomicAdd(&a.ctl->unres[round % 3], 1u);
        }
      }
    }
    ok = grid_barrier(a.ctl, G, a.wait_ns, false);
    if (!ok) break;
    if (ldcg_u32(&a.ctl->unres[round % 3]) == 0) break;
    for (uint32_t i = tid; i < N; i += nth)
      if (ldcg_u32(&a.res[i]) == kResUnresolved) a.tbl[a.ent[i]].minv = 0;
    ok = grid_barrier(a.ctl, G, a.wait_ns, false);
    if (!ok) break;
    for (uint32_t i = tid; i < N; i += nth)
      if (ldcg_u32(&a.res[i]) == kResUnresolved) atomicMax(&a.tbl[a.ent[i]].minv, ~i);
    ok = grid_barrier(a.ctl, G, a.wait_ns, false);
    ++round;
  }

  // ---- D: count, rank, write ------------------------------------------------
  const uint64_t per = (((uint64_t)N + G - 1) / G + 31) & ~31ull;
  const uint32_t lo = (uint32_t)min((uint64_t)N, blockIdx.x * per);
  const uint32_t hi = (uint32_t)min((uint64_t)N, lo + per);
  if (ok) {
    uint32_t cnt = 0;
    for (uint32_t i = lo + threadIdx.x; i < hi; i += kThreads)
      cnt += (ldcg_u32(&a.res[i]) & kResLeader) ? 1u : 0u;
    const unsigned long long c = block_sum<unsigned long long>(cnt, red64);
    if (threadIdx.x == 0) a.bcount[blockIdx.x] = (uint32_t)c;
    ok = grid_barrier(a.ctl, G, a.wait_ns, false);
  }
  if (ok) {
    unsigned long long before = 0, total = 0;
    for (uint32_t j = threadIdx.x; j < G; j += kThreads) {
      const uint32_t v = ldcg_u32(&a.bcount[j]);
      total += v;
      if (j < blockIdx.x) before += v;
    }
    before = block_sum<unsigned long long>(before, red64);
    total = block_sum<unsigned long long>(total, red64);
    if (slots0 + total > a.nslots) {
      if (threadIdx.x == 0) atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_CAPACITY);
      ok = false;
    } else {
      const bool vec = vec_buf && ((uintptr_t)a.packed % 16) == 0;
      unsigned long long n_hc = 0, n_hi = 0, n_rej = 0, n_bytes = 0;
      unsigned long long running = before;
      for (uint32_t t = lo; t < hi; t += kThreads) {
        const uint32_t i = t + threadIdx.x;
        const bool valid = i < hi;
        const uint32_t r = valid ? ldcg_u32(&a.res[i]) : 0u;
        const bool miss = valid && (r & kResLeader);
        const bool hit = valid && (r & (kResHit0 | kResDup));
        const uint32_t mb = __ballot_sync(0xffffffffu, miss);
        const uint32_t hb = __ballot_sync(0xffffffffu, hit);
        const uint32_t g = t + w * 32;
        if (lane == 0 && g < hi) a.mask[g >> 5] = hb;
        if (lane == 0) warp_cnt[w] = __popc(mb);
        __syncthreads();
        if (threadIdx.x == 0) {
          uint32_t acc = 0;
          for (int k = 0; k < kWarps; ++k) {
            warp_off[k] = acc;
            acc += warp_cnt[k];
          }
          warp_cnt[0] = acc;  // tile total (read after the next barrier)
        }
        __syncthreads();
        const uint32_t tile_total = warp_cnt[0];
        if (miss) {
          const uint32_t local = warp_off[w] + __popc(mb & ((1u << lane) - 1u));
          const unsigned long long rank = running + local;
          a.miss_idx[rank] = i;
          list_i[local] = i;
          list_r[local] = (uint32_t)(rank - before);
          const uint32_t len = chunk_len(a, i);
          n_bytes += len;
          if ((r & kResRoundMask) > 1 || a.status[i] == kMissCand) ++n_rej;
        }
        if (valid && (r & kResHit0)) ++n_hc;
        if (valid && (r & kResDup)) ++n_hi;
        __syncthreads();
        for (uint32_t k = w; k < tile_total; k += kWarps) {
          const uint32_t ci = list_i[k];
          const unsigned long long rank = before + list_r[k];
          const uint32_t len = chunk_len(a, ci);
          const unsigned long long slot = slots0 + rank;
          warp_copy2(a.packed + rank * a.C, a.arena + slot * a.C, a.buf + (uint64_t)ci * a.C,
                     len, vec);
          if (lane == 0) {
            a.slot_len[slot] = len;
            if (!index_insert(a.index, a.index_mask, a.key[ci], (uint32_t)slot, len))
              atomicCAS(&a.ctl->err, 0, (int)GLEAM_ERR_INTERNAL);
          }
        }
        running += tile_total;
        __syncthreads();
      }
      n_hc = block_sum<unsigned long long>(n_hc, red64);
      n_hi = block_sum<unsigned long long>(n_hi, red64);
      n_rej = block_sum<unsigned long long>(n_rej, red64);
      n_bytes = block_sum<unsigned long long>(n_bytes, red64);
      if (threadIdx.x == 0) {
        atomicAdd(&a.ctl->acc_hits_cache, n_hc);
        atomicAdd(&a.ctl->acc_hits_intra, n_hi);
        atomicAdd(&a.ctl->acc_rejects, n_rej);
        atomicAdd(&a.ctl->acc_miss_bytes, n_bytes);
        if (blockIdx.x == 0) atomicExch(&a.ctl->acc_misses, total);
      }
    }
  }

  // ---- epilogue: the last block publishes ----------------------------------
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned int ticket = atomicAdd(&a.ctl->done, 1u);
    if (ticket == G - 1) {
      __threadfence();
      const int err = ld_volatile_s32(&a.ctl->err);
      const unsigned long long misses = __ldcg(&a.ctl->acc_misses);
      const unsigned long long hc = __ldcg(&a.ctl->acc_hits_cache);
      const unsigned long long hi2 = __ldcg(&a.ctl->acc_hits_intra);
      const unsigned long long rej = __ldcg(&a.ctl->acc_rejects);
      const unsigned long long mbytes = __ldcg(&a.ctl->acc_miss_bytes);
      if (err == 0) {
        a.dstats[ST_CALLS] += 1;
        a.dstats[ST_CHUNKS] += N;
        a.dstats[ST_HITS_CACHE] += hc;
        a.dstats[ST_HITS_INTRA] += hi2;
        a.dstats[ST_MISSES] += misses;
        a.dstats[ST_INSERTS] += misses;
        a.dstats[ST_REJECTS] += rej;
        a.dstats[ST_SLOTS_USED] = slots0 + misses;
        a.dstats[ST_BYTES_USED] += mbytes;
      }
      if (a.result != nullptr) {
        a.result->status = err;
        a.result->n_miss = err ? 0 : misses;
        a.result->n_hit_cache = err ? 0 : hc;
        a.result->n_hit_intra = err ? 0 : hi2;
        a.result->verify_rejects = err ? 0 : rej;
        a.result->miss_bytes = err ? 0 : mbytes;
      }
      __threadfence();
    }
  }
}

__global__ void k_debug_insert(IndexEntry* index, uint64_t index_mask, uint32_t* slot_len,
                               unsigned long long* dstats, unsigned long long key, uint32_t slot,
                               uint32_t len, DevCtl* ctl) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  if (!index_insert(index, index_mask, key, slot, len)) {
    ctl->err = GLEAM_ERR_INTERNAL;
    return;
  }
  slot_len[slot] = len;
  dstats[ST_SLOTS_USED] = (unsigned long long)slot + 1;
  dstats[ST_INSERTS] += 1;
  dstats[ST_BYTES_USED] += len;
}

}  // namespace

int dedup_threads() { return kThreads; }

int dedup_blocks_per_sm() {
  int nb = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k_dedup, kThreads, 0) != cudaSuccess)
    return 0;
  return nb;
}

cudaError_t launch_dedup(const DedupArgs& a, int grid, cudaStream_t s) {
  DedupArgs copy = a;
  void* args[] = {&copy};
  return cudaLaunchCooperativeKernel((void*)k_dedup, dim3(grid), dim3(kThreads), args, 0, s);
}

cudaError_t launch_debug_insert(IndexEntry* index, uint64_t index_mask, uint32_t* slot_len,
                                unsigned long long* dstats, unsigned long long key,
                                uint32_t slot, uint32_t len, DevCtl* ctl, cudaStream_t s) {
  k_debug_insert<<<1, 32, 0, s>>>(index, index_mask, slot_len, dstats, key, slot, len, ctl);
  return cudaGetLastError();
}

}  // namespace gleam
