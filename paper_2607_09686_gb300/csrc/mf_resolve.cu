// Slot resolve: the per-layer bounded expert cache (section "Native Serving Path": a miss
// materialises the expert block into an available slot and updates the route-to-slot
// metadata).
//
// One block per call.  Steps:
//  1. the distinct experts of the call's T*k routes, in (token, rank) first-occurrence
//     order, and for each the list of assignments t*k+j it serves;
//  2. least-recently-used replacement over those accesses in waves of S (lru_warp);
//  3. counters (accesses, hits, misses, evictions, bytes = misses * payload) and the
//     access record of the call.
// With one token per call the router's last block does this itself (mf_router.cu).
#include "mf_lru.cuh"

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
  const int warp = tid >> 5;
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
    int tiles = 0;  // 128-assignment blocks before each expert's (the grouped GEMMs' tile index)
    for (int u = 0; u < U; ++u) {
      d.tb_off[u] = tiles;
      tiles += (cnt[s_uniq[u]] + 127) / 128;
    }
    d.tb_off[U] = tiles;
  }
  __syncthreads();
  for (int p = tid; p < n; p += nt) {
    int u = uidx[d.idx[p]];
    int a = atomicAdd(&fill[u], 1);
    d.asg[d.asg_off[u] + a] = p;
  }

  // LRU, one access at a time
  if (warp == 0) lru_warp(d, layer, U, s_uniq, s_slot_of, s_expert_of, s_last, s_uslot, d.clock[layer]);
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
