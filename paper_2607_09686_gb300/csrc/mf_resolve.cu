// Slot resolve: the per-layer bounded expert cache (section "Native Serving Path": a miss
// materialises the expert block into an available slot and updates the route-to-slot
// metadata).
//
// One block of 1024 threads per call.  Steps:
//  1. the distinct experts of the call's T*k routes, in (token, rank) first-occurrence
//     order (or, with MF_ORDER_RESIDENT_FIRST, the resident ones first), and for each the list
//     of assignments t*k+j it serves;
//  2. least-recently-used replacement over those accesses in waves of S (lru_block);
//  3. counters (accesses, hits, misses, evictions, bytes = misses * payload) and the
//     access record of the call.
// Each warp counts its routes into its own copy of the per-expert counters, so that a hot
// expert's counter (skewed routing) is not contended across warps.
// With one token per call the router's last block does this itself (mf_router.cu).
#include "mf_lru.cuh"

namespace mf {
namespace {

constexpr int kThreadsRes = 1024;
constexpr int kRouteChunk = 8;  // routes a thread loads before using them (their loads overlap)

// histogram copies: one per warp where E allows (no two warps update the same counter), fewer
// for large E (shared memory)
__host__ __device__ inline int n_segments(int E) {
  const int n = 8192 / E;
  return n < 1 ? 1 : (n > kThreadsRes / 32 ? kThreadsRes / 32 : n);
}

__global__ void __launch_bounds__(kThreadsRes, 1) k_resolve(Dev d, int layer, int T) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int E = d.E, k = d.k, S = d.S_active, n = T * k, NSEG = n_segments(E);
  uint64_t* s_last = reinterpret_cast<uint64_t*>(smem);           // [S_alloc]
  int* seg_first = reinterpret_cast<int*>(s_last + d.S_alloc);     // [NSEG][E] first route per copy
  int* seg_cnt = seg_first + NSEG * E;                              // [NSEG][E] routes per copy
  int* seg_fill = seg_cnt + NSEG * E;                               // [NSEG][E] next assignment position
  int* cnt = seg_fill + NSEG * E;                                   // [E]
  int* uidx = cnt + E;                                              // [E]
  int* s_slot_of = uidx + E;                                        // [E]
  int* s_uniq = s_slot_of + E;                                      // [E]
  int* s_uslot = s_uniq + E;                                        // [E]
  int* firstpos = s_uslot + E;                                      // [E]
  int* s_expert_of = firstpos + E;                                  // [S_alloc]
  int* s_order = s_expert_of + d.S_alloc;                           // [S_alloc] LRU scratch
  int* s_prev = s_order + d.S_alloc;                                // [S_alloc]
  int* s_next = s_prev + d.S_alloc;                                 // [S_alloc]
  __shared__ int s_U, s_n[2];

  const int tid = threadIdx.x, nt = blockDim.x;
  const int seg = (tid >> 5) % NSEG;
  int32_t* g_slot_of = d.slot_of + (size_t)layer * E;
  int32_t* g_expert_of = d.expert_of + (size_t)layer * d.S_alloc;
  uint64_t* g_last = d.last_use + (size_t)layer * d.S_alloc;

  for (int i = tid; i < NSEG * E; i += nt) {
    seg_first[i] = 0x7fffffff;
    seg_cnt[i] = 0;
  }
  for (int e = tid; e < E; e += nt) s_slot_of[e] = g_slot_of[e];
  for (int q = tid; q < S; q += nt) {
    s_expert_of[q] = g_expert_of[q];
    s_last[q] = g_last[q];
  }
  {  // every wave the host may launch for this call starts with no misses
    const int acc_max = n < E ? n : E;
    for (int w = tid; w < (acc_max + S - 1) / S; w += nt) d.info[2 + w] = 0;
  }
  __syncthreads();
  // routes c0 + j * nt of this thread (j < kRouteChunk) are loaded first, then counted into
  // this warp's histogram copy (a warp's 32 consecutive routes hold an expert at most once per
  // token, so few lanes share a counter)
  for (int c0 = tid; c0 < n; c0 += nt * kRouteChunk) {
    int ev[kRouteChunk];
#pragma unroll
    for (int j = 0; j < kRouteChunk; ++j) {
      const int p = c0 + j * nt;
      ev[j] = p < n ? d.idx[p] : 0;
    }
#pragma unroll
    for (int j = 0; j < kRouteChunk; ++j) {
      const int p = c0 + j * nt;
      if (p < n) {
        atomicMin(&seg_first[seg * E + ev[j]], p);
        atomicAdd(&seg_cnt[seg * E + ev[j]], 1);
      }
    }
  }
  __syncthreads();
  for (int e = tid; e < E; e += nt) {
    int f = 0x7fffffff, c = 0;
    for (int g = 0; g < NSEG; ++g) {
      f = min(f, seg_first[g * E + e]);
      c += seg_cnt[g * E + e];
    }
    firstpos[e] = f;
    cnt[e] = c;
  }
  __syncthreads();
  // access order = order of first occurrence
  for (int e = tid; e < E; e += nt) {
    const int fp = firstpos[e];
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
  if (d.order == MF_ORDER_RESIDENT_FIRST) {  // stable: resident experts first, then the others
    int* tmp = s_uslot;                      // reused (written by the LRU below)
    for (int u = tid; u < U; u += nt) tmp[u] = s_uniq[u];
    __syncthreads();
    int n_res = 0;
    for (int v = 0; v < U; ++v) n_res += s_slot_of[tmp[v]] >= 0;
    for (int u = tid; u < U; u += nt) {
      const int e = tmp[u];
      const bool res = s_slot_of[e] >= 0;
      int r = res ? 0 : n_res;
      for (int v = 0; v < u; ++v) r += (s_slot_of[tmp[v]] >= 0) == res;
      s_uniq[r] = e;
      uidx[e] = r;
    }
    __syncthreads();
  }
  int* ucnt = firstpos;  // reused: routes of the u-th distinct expert
  for (int u = tid; u < U; u += nt) ucnt[u] = cnt[s_uniq[u]];
  __syncthreads();
  for (int u = tid; u <= U; u += nt) {  // assignment offsets and 128-assignment blocks, in access order
    int acc = 0, tiles = 0;
    for (int v = 0; v < u; ++v) {
      const int c = ucnt[v];
      acc += c;
      tiles += (c + 127) / 128;
    }
    d.asg_off[u] = acc;
    d.tb_off[u] = tiles;
    if (u < U) {  // where each histogram copy's routes of this expert start
      const int e = s_uniq[u];
      for (int g = 0; g < NSEG; ++g) {
        seg_fill[g * E + e] = acc;
        acc += seg_cnt[g * E + e];
      }
    }
  }
  __syncthreads();
  for (int c0 = tid; c0 < n; c0 += nt * kRouteChunk) {  // the same walk as the count
    int ev[kRouteChunk];
#pragma unroll
    for (int j = 0; j < kRouteChunk; ++j) {
      const int p = c0 + j * nt;
      ev[j] = p < n ? d.idx[p] : 0;
    }
#pragma unroll
    for (int j = 0; j < kRouteChunk; ++j) {
      const int p = c0 + j * nt;
      if (p < n) d.asg[atomicAdd(&seg_fill[seg * E + ev[j]], 1)] = p;
    }
  }

  lru_block(d, layer, U, s_uniq, s_slot_of, s_expert_of, s_last, s_uslot, d.clock[layer], s_order, s_prev, s_next,
            s_n);
  for (int c0 = tid; c0 < n; c0 += nt * kRouteChunk) {
    int ev[kRouteChunk];
#pragma unroll
    for (int j = 0; j < kRouteChunk; ++j) {
      const int p = c0 + j * nt;
      ev[j] = p < n ? d.idx[p] : 0;
    }
#pragma unroll
    for (int j = 0; j < kRouteChunk; ++j) {
      const int p = c0 + j * nt;
      if (p < n) d.pos_slot[p] = s_uslot[uidx[ev[j]]];
    }
  }
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
  return (size_t)d.S_alloc * sizeof(uint64_t) + ((size_t)3 * n_segments(d.E) + 6) * d.E * sizeof(int) +
         (size_t)4 * d.S_alloc * sizeof(int);
}

cudaError_t launch_resolve(const Dev& d, int layer, int T, cudaStream_t s) {
  const size_t smem = resolve_smem_bytes(d);
  cudaError_t e = cudaFuncSetAttribute(k_resolve, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_resolve<<<1, kThreadsRes, smem, s>>>(d, layer, T);
  return cudaGetLastError();
}

cudaError_t launch_reset(const Dev& d, cudaStream_t s) {
  size_t n = (size_t)d.L * (d.E > d.S_alloc ? d.E : d.S_alloc);
  if (n < (size_t)d.L * 5) n = (size_t)d.L * 5;
  k_reset<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(d);
  return cudaGetLastError();
}

}  // namespace mf
