// Least-recently-used slot replacement of one layer, run by one warp (internal).
//
// Section "Native Serving Path": on a miss the runtime materialises the expert block into an
// available slot and updates the route-to-slot metadata.  Accesses are processed one at a
// time in order: a resident expert hits (its slot becomes the most recently used); otherwise
// the lowest free slot is taken, or, with none free, the slot of the least recently used
// expert, which is evicted.  Accesses are grouped in waves of S consecutive accesses; within a
// wave no access evicts an expert accessed earlier in the same wave (those are the most recent
// and fewer than S), so each wave's experts occupy distinct slots when the wave is computed.
#pragma once

#include "mf_internal.cuh"

namespace mf {

constexpr int kMissBit = 1 << 30;  // in s_uslot until the record is written

// The record of every access (uniq, uslot, umiss, trace) and the counters, from s_uslot (slot,
// with kMissBit for a miss); clears the bit.  All 32 lanes of one warp call it; lane 0's clock
// and eviction count are the ones stored.
__device__ __forceinline__ void lru_records(const Dev& d, int layer, int U, const int* s_uniq, int* s_uslot,
                                            uint64_t clock, uint64_t evictions) {
  const int lane = threadIdx.x & 31, E = d.E, S = d.S_active;
  unsigned misses = 0;
  for (int u0 = 0; u0 < U; u0 += 32) {  // warp-uniform: every lane takes part in the ballot
    const int u = u0 + lane;
    const bool valid = u < U;
    int s = valid ? s_uslot[u] : 0;
    const bool miss = valid && (s & kMissBit);
    s &= ~kMissBit;
    misses += __popc(__ballot_sync(0xffffffffu, miss));
    if (valid) {
      const int e = s_uniq[u];
      s_uslot[u] = s;
      d.uniq[u] = e;
      d.uslot[u] = s;
      d.umiss[u] = miss ? 1 : 0;
      d.tr_expert[(size_t)layer * E + u] = e;
      d.tr_slot[(size_t)layer * E + u] = s;
      d.tr_hit[(size_t)layer * E + u] = miss ? 0 : 1;
    }
  }
  __syncwarp();
  if (lane == 0) {
    const uint64_t hits = (uint64_t)U - misses;
    d.clock[layer] = clock;
    unsigned long long* st = reinterpret_cast<unsigned long long*>(d.stats + (size_t)layer * 5);
    atomicAdd(st + 0, (unsigned long long)U);  // no return value used: fire-and-forget reductions
    atomicAdd(st + 1, (unsigned long long)hits);
    atomicAdd(st + 2, (unsigned long long)misses);
    atomicAdd(st + 3, (unsigned long long)evictions);
    atomicAdd(st + 4, (unsigned long long)((uint64_t)misses * d.lay.canonical));
    d.info[0] = U;
    d.info[1] = (U + S - 1) / S;
    d.tr_n[layer] = U;
  }
}

// State of the layer in shared memory: s_slot_of[E], s_expert_of[S_active], s_last[S_active].
// Writes the call's access record (uniq, uslot, umiss, trace), per-wave miss lists and counts,
// the counters and the clock.  All 32 lanes must call it.  The accesses are decided one after
// the other (lane 0 updates the state; the warp searches free and least-recently-used slots);
// the record of every access is then written by the whole warp at once.
__device__ __forceinline__ void lru_warp(const Dev& d, int layer, int U, const int* s_uniq, int* s_slot_of,
                                         int* s_expert_of, uint64_t* s_last, int* s_uslot, uint64_t clock) {
  const int lane = threadIdx.x & 31, S = d.S_active;  // the clock is kept by lane 0
  uint64_t evictions = 0;
  int wave = 0, wpos = 0, wave_miss = 0;  // wave of access u, u's position in it, misses so far in it
  // Every access a hit (the common case): nothing is placed or evicted, so the decisions are
  // independent -- access u just takes clock value clock + u + 1 -- and the warp applies them
  // together.  Any miss: the accesses are walked in order (a miss may evict the slot of a later
  // access of the same call).
  bool all_hit = true;
  for (int u0 = 0; u0 < U && all_hit; u0 += 32)
    all_hit = __all_sync(0xffffffffu, u0 + lane >= U || s_slot_of[s_uniq[u0 + lane]] >= 0);
  if (all_hit) {
    for (int u0 = 0; u0 < U; u0 += 32) {
      const int u = u0 + lane;
      if (u < U) {
        const int sl = s_slot_of[s_uniq[u]];
        s_last[sl] = clock + (uint64_t)u + 1;
        s_uslot[u] = sl;
      }
    }
    clock += (uint64_t)U;
    if (lane == 0)
      for (int w = 0; w * S < U; ++w) d.info[2 + w] = 0;
    __syncwarp();
  }
  for (int u = 0; u < U && !all_hit; ++u) {
    const int e = s_uniq[u];
    int s = s_slot_of[e];
    const bool hit = s >= 0;
    if (!hit) {
      int found = -1;
      for (int base = 0; base < S && found < 0; base += 32) {
        const int q = base + lane;
        const unsigned b = __ballot_sync(0xffffffffu, q < S && s_expert_of[q] < 0);
        if (b) found = base + __ffs(b) - 1;
      }
      if (found < 0) {  // no free slot: evict the least recently used
        uint64_t best = ~0ull;
        int bq = 0x7fffffff;
        for (int q = lane; q < S; q += 32)
          if (s_last[q] < best) {
            best = s_last[q];
            bq = q;
          }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const uint64_t ob = __shfl_xor_sync(0xffffffffu, best, off);
          const int oq = __shfl_xor_sync(0xffffffffu, bq, off);
          if (ob < best || (ob == best && oq < bq)) {
            best = ob;
            bq = oq;
          }
        }
        found = bq;
        if (lane == 0) s_slot_of[s_expert_of[found]] = -1;
        ++evictions;
      }
      s = found;
      if (lane == 0) {
        s_expert_of[s] = e;
        s_slot_of[e] = s;
        d.miss_list[wave * S + wave_miss] = u;
      }
      ++wave_miss;
    }
    if (lane == 0) {
      s_last[s] = ++clock;
      s_uslot[u] = hit ? s : (s | kMissBit);
    }
    if (++wpos == S || u == U - 1) {  // end of a wave: its miss count
      if (lane == 0) d.info[2 + wave] = wave_miss;
      ++wave;
      wpos = 0;
      wave_miss = 0;
    }
    __syncwarp();  // lane 0's shared-memory updates are seen by the whole warp at the next access
  }
  lru_records(d, layer, U, s_uniq, s_uslot, clock, evictions);
}


// The same replacement for many accesses (calls with T > 1), by a whole block: every thread
// calls it (it has block barriers).  The occupied slots are ordered by last use once, in
// parallel (rank counting on (last use, slot)), into a doubly linked list from least to most
// recently used, and the free slots in increasing order; thread 0 then walks the accesses with
// O(1) list operations (a hit moves its slot to the most-recent end; a miss takes the next free
// slot, else the list's head, whose expert is evicted).  Scratch: s_order, s_prev, s_next
// (S_active ints each), s_n (2 ints).  Same decisions as lru_warp.
__device__ __forceinline__ void lru_block(const Dev& d, int layer, int U, const int* s_uniq, int* s_slot_of,
                                          int* s_expert_of, uint64_t* s_last, int* s_uslot, uint64_t clock,
                                          int* s_order, int* s_prev, int* s_next, int* s_n) {
  const int S = d.S_active, tid = threadIdx.x, nt = blockDim.x;
  if (tid < 2) s_n[tid] = 0;
  __syncthreads();
  for (int q = tid; q < S; q += nt) {  // occupied: rank by (last use, slot); free: rank by slot
    const bool occ = s_expert_of[q] >= 0;
    const uint64_t lq = s_last[q];
    int r = 0;
    for (int q2 = 0; q2 < S; ++q2) {
      const bool occ2 = s_expert_of[q2] >= 0;
      if (occ2 != occ) continue;
      r += occ ? (s_last[q2] < lq || (s_last[q2] == lq && q2 < q)) : q2 < q;
    }
    if (occ) {
      s_order[r] = q;
      atomicAdd(&s_n[0], 1);
    } else {
      s_prev[r] = q;  // free slots in increasing order (s_prev is reused for the list below)
      atomicAdd(&s_n[1], 1);
    }
  }
  __syncthreads();
  const int n_occ = s_n[0], n_free = s_n[1];
  // the free slots move to the tail of s_order (after the occupied ones), freeing s_prev
  for (int r = tid; r < n_free; r += nt) s_order[n_occ + r] = s_prev[r];
  __syncthreads();
  for (int r = tid; r < n_occ; r += nt) {
    const int q = s_order[r];
    s_prev[q] = r > 0 ? s_order[r - 1] : -1;
    s_next[q] = r + 1 < n_occ ? s_order[r + 1] : -1;
  }
  __syncthreads();
  uint64_t evictions = 0;
  if (tid == 0) {
    int head = n_occ > 0 ? s_order[0] : -1, tail = n_occ > 0 ? s_order[n_occ - 1] : -1, fp = 0;
    int wave = 0, wpos = 0, wave_miss = 0;
    for (int u = 0; u < U; ++u) {
      const int e = s_uniq[u];
      int s = s_slot_of[e];
      const bool hit = s >= 0;
      if (hit) {  // unlink
        const int pv = s_prev[s], nx = s_next[s];
        if (pv >= 0) s_next[pv] = nx; else head = nx;
        if (nx >= 0) s_prev[nx] = pv; else tail = pv;
      } else {
        if (fp < n_free) {
          s = s_order[n_occ + fp++];
        } else {  // evict the least recently used (a wave never holds S accesses before this one)
          s = head;
          head = s_next[s];
          if (head >= 0) s_prev[head] = -1; else tail = -1;
          s_slot_of[s_expert_of[s]] = -1;
          ++evictions;
        }
        s_expert_of[s] = e;
        s_slot_of[e] = s;
        d.miss_list[wave * S + wave_miss++] = u;
      }
      s_prev[s] = tail;  // append as the most recently used
      s_next[s] = -1;
      if (tail >= 0) s_next[tail] = s; else head = s;
      tail = s;
      s_last[s] = ++clock;
      s_uslot[u] = hit ? s : (s | kMissBit);
      if (++wpos == S || u == U - 1) {  // end of a wave: its miss count
        d.info[2 + wave] = wave_miss;
        ++wave;
        wpos = 0;
        wave_miss = 0;
      }
    }
  }
  __syncthreads();
  if (tid < 32) lru_records(d, layer, U, s_uniq, s_uslot, __shfl_sync(0xffffffffu, clock, 0),
                            __shfl_sync(0xffffffffu, evictions, 0));
}

}  // namespace mf
