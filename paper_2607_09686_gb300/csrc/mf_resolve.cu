// Slot resolve: the per-layer bounded expert cache (section "Native Serving Path": a miss
// materialises the expert block into an available slot and updates the route-to-slot
// metadata).
//
// One block per call.  Steps:
//  1. the distinct experts of the call's T*k routes, in (token, rank) first-occurrence
//     order, and for each the list of assignments t*k+j it serves;
//  2. least-recently-used replacement over those accesses, one at a time (one warp):
//     resident -> hit; otherwise the lowest free slot, or the slot of the least recently
//     used expert, which is evicted;
//  3. accesses grouped in waves of S consecutive accesses (S = slots in use).  Within a
//     wave no access evicts an expert accessed earlier in the same wave (those are the
//     most recent ones and fewer than S), so each wave's experts end up in distinct
//     slots and the wave can be materialised and computed as one batch;
//  4. counters (accesses, hits, misses, evictions, bytes = misses * payload) and the
//     access record of the call.
#include "mf_internal.cuh"

namespace mf {
namespace {

__global__ void __launch_bounds__(256) k_resolve(Dev d, int layer, int T) {
  extern __shared__ unsigned char smem[];
  const int E = d.E, k = d.k, S = d.S_active, n = T * k;
  uint64_t* s_last = reinterpret_cast<uint64_t*>(smem);           // [S_alloc]
  int* firstpos = reinterpret_cast<int*>(s_last + d.S_alloc);       // [E]
  int* cnt = firstpos + E;                                          // [E]
  int* uidx = cnt + E;                                              // [E]
  int* fill = uidx + E;                                             // [E]
  int* s_slot_of = fill + E;                                        // [E]
  int* s_uniq = s_slot_of + E;                                      // [E]
  int* s_uslot = s_uniq + E;                                        // [E]
  int* s_expert_of = s_uslot + E;                                   // [S_alloc]
  __shared__ int s_U;

  const int tid = threadIdx.x, nt = blockDim.x;
  const int warp = tid >> 5, lane = tid & 31;
  int32_t* g_slot_of = d.slot_of + (size_t)layer * E;
  int32_t* g_expert_of = d.expert_of + (size_t)layer * d.S_alloc;
  uint64_t* g_last = d.last_use + (size_t)layer * d.S_alloc;

  for (int e = tid; e < E; e += nt) {
    firstpos[e] = 0x7fffffff;
    cnt[e] = 0;
    fill[e] = 0;
    s_slot_of[e] = g_slot_of[e];
  }
  for (int q = tid; q < S; q += nt) {
    s_expert_of[q] = g_expert_of[q];
    s_last[q] = g_last[q];
  }
  {  // every wave the host may launch for this call starts with no misses
    const int acc_max = n < E ? n : E;
    for (int w = tid; w < (acc_max + S - 1) / S; w += nt) d.info[2 + w] = 0;
  }
  __syncthreads();
  for (int p = tid; p < n; p += nt) {
    int e = d.idx[p];
    atomicMin(&firstpos[e], p);
    atomicAdd(&cnt[e], 1);
  }
  __syncthreads();
  // access order = order of first occurrence
  for (int e = tid; e < E; e += nt) {
    int fp = firstpos[e];
    if (fp == 0x7fffffff) continue;
    int r = 0;
    for (int e2 = 0; e2 < E; ++e2) r += firstpos[e2] < fp;
    uidx[e] = r;
    s_uniq[r] = e;
  }
  if (tid == 0) {
    int U = 0;
    for (int e = 0; e < E; ++e) U += firstpos[e] != 0x7fffffff;
    s_U = U;
  }
  __syncthreads();
  const int U = s_U;
  if (tid == 0) {  // assignment offsets, in access order
    int acc = 0;
    for (int u = 0; u < U; ++u) {
      d.asg_off[u] = acc;
      acc += cnt[s_uniq[u]];
    }
    d.asg_off[U] = acc;
  }
  __syncthreads();
  for (int p = tid; p < n; p += nt) {
    int u = uidx[d.idx[p]];
    int a = atomicAdd(&fill[u], 1);
    d.asg[d.asg_off[u] + a] = p;
  }

  // LRU, one access at a time
  if (warp == 0) {
    uint64_t clock = d.clock[layer];  // kept by lane 0
    uint64_t hits = 0, misses = 0, evictions = 0;
    int wave_miss = 0;
    for (int u = 0; u < U; ++u) {
      if (u % S == 0) wave_miss = 0;
      const int e = s_uniq[u];
      int s = s_slot_of[e];
      const bool hit = s >= 0;
      if (!hit) {
        int found = -1;
        for (int base = 0; base < S && found < 0; base += 32) {
          int q = base + lane;
          unsigned b = __ballot_sync(0xffffffffu, q < S && s_expert_of[q] < 0);
          if (b) found = base + __ffs(b) - 1;
        }
        if (found < 0) {
          uint64_t best = ~0ull;
          int bq = 0x7fffffff;
          for (int q = lane; q < S; q += 32)
            if (s_last[q] < best) {
              best = s_last[q];
              bq = q;
            }
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) {
            uint64_t ob = __shfl_xor_sync(0xffffffffu, best, off);
            int oq = __shfl_xor_sync(0xffffffffu, bq, off);
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
          d.miss_list[(u / S) * S + wave_miss] = u;
        }
        ++wave_miss;
        ++misses;
      } else {
        ++hits;
      }
      if (lane == 0 && (u % S == S - 1 || u == U - 1)) d.info[2 + u / S] = wave_miss;
      if (lane == 0) {
        s_last[s] = ++clock;
        s_uslot[u] = s;
        d.uniq[u] = e;
        d.uslot[u] = s;
        d.umiss[u] = hit ? 0 : 1;
        d.tr_expert[(size_t)layer * E + u] = e;
        d.tr_slot[(size_t)layer * E + u] = s;
        d.tr_hit[(size_t)layer * E + u] = hit ? 1 : 0;
      }
      __syncwarp();  // lane 0's shared-memory updates are seen by the whole warp next access
    }
    if (lane == 0) {
      d.clock[layer] = clock;
      uint64_t* st = d.stats + (size_t)layer * 5;
      st[0] += (uint64_t)U;
      st[1] += hits;
      st[2] += misses;
      st[3] += evictions;
      st[4] += misses * d.lay.canonical;
      d.info[0] = U;
      d.info[1] = (U + S - 1) / S;
      d.tr_n[layer] = U;
    }
  }
  __syncthreads();
  for (int p = tid; p < n; p += nt) d.pos_slot[p] = s_uslot[uidx[d.idx[p]]];
  for (int e = tid; e < E; e += nt) g_slot_of[e] = s_slot_of[e];
  for (int q = tid; q < S; q += nt) {
    g_expert_of[q] = s_expert_of[q];
    g_last[q] = s_last[q];
  }
}

__global__ void k_reset(Dev d) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t nE = (size_t)d.L * d.E, nS = (size_t)d.L * d.S_alloc;
  if (i < nE) d.slot_of[i] = -1;
  if (i < nS) {
    d.expert_of[i] = -1;
    d.last_use[i] = 0;
  }
  if (i < (size_t)d.L) {
    d.clock[i] = 0;
    d.tr_n[i] = 0;
  }
  if (i < (size_t)d.L * 5) d.stats[i] = 0;
}

}  // namespace

size_t resolve_smem_bytes(const Dev& d) {
  return (size_t)d.S_alloc * sizeof(uint64_t) + (size_t)7 * d.E * sizeof(int) + (size_t)d.S_alloc * sizeof(int);
}

cudaError_t launch_resolve(const Dev& d, int layer, int T, cudaStream_t s) {
  size_t smem = resolve_smem_bytes(d);
  k_resolve<<<1, 256, smem, s>>>(d, layer, T);
  return cudaGetLastError();
}

cudaError_t launch_reset(const Dev& d, cudaStream_t s) {
  size_t n = (size_t)d.L * (d.E > d.S_alloc ? d.E : d.S_alloc);
  if (n < (size_t)d.L * 5) n = (size_t)d.L * 5;
  k_reset<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(d);
  return cudaGetLastError();
}

}  // namespace mf
