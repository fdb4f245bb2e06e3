// Batch-1 decode expert FFN as two persistent, pipelined dequantising GEMV kernels.
//
//   gate/up:  h_j[r] = silu(Wg_j[r,:] . x) * (Wu_j[r,:] . x)        for the k routed experts j
//   down:     y[c]   = sum_j g_j (Wd_j[c,:] . h_j)                     (router-weighted combine)
// (SwiGLU experts with separate gate, up and down tensors, section "Native Serving Path";
// W = d*q for Q8_0, d*(n-8) for Q4_0; fp32 accumulation.)
//
// One CTA per SM.  A producer warp takes work items from a queue (an atomic counter zeroed by
// the router of the same call) and streams each item's quantised rows and scales from the HBM
// slots into a ring of shared-memory stages with bulk asynchronous copies completing on an
// mbarrier; eight consumer warps dequantise from shared memory and release each stage through
// a second mbarrier.  Memory traffic is decoupled from registers, so each SM keeps several
// items in flight.  Consumers hold the vector they multiply by (x, or their expert's h) in
// registers for the whole kernel: a lane always handles the same 16-byte column vectors.
//   gate/up item = 8 rows of one expert's gate and up tensors; consumer warp w owns row w.
//   down item    = R output rows of all k experts; consumer warp w owns expert w/(8/k); the
//                  last warp to finish an item (shared-memory counter) adds the k partial
//                  rows in rank order, so the combine is deterministic and atomic-free.
// Every wait is bounded; a wait that gives up sets the device error word and the CTA stops.
#include "mf_dequant.cuh"

namespace mf {
namespace {

using namespace dq;

constexpr int kConsumers = 8;
constexpr int kThreads = (kConsumers + 1) * 32;
constexpr int kMaxStages = 8;
constexpr int kGuRows = 8;  // gate/up rows per item, one per consumer warp
constexpr size_t kSmemBudget = 200 * 1024;

struct PipeCfg {
  int R;                 // rows per item
  int NS;                // stages
  uint32_t stage_bytes;  // bytes per item (= per stage)
  int n_items;
  uint32_t per_j;        // down: bytes of one expert's share of an item
};

struct Smem {
  unsigned char* stage0;
  uint64_t* full;
  uint64_t* empty;
  int* item;
  int* cnt;
  float* part;  // [kMaxStages][kMaxTopK][8]
};

__device__ __forceinline__ Smem carve(unsigned char* base, const PipeCfg& c) {
  Smem s;
  s.stage0 = base;
  unsigned char* p = base + (size_t)c.NS * c.stage_bytes;
  s.full = reinterpret_cast<uint64_t*>(p);
  s.empty = s.full + kMaxStages;
  s.item = reinterpret_cast<int*>(s.empty + kMaxStages);
  s.cnt = s.item + kMaxStages;
  s.part = reinterpret_cast<float*>(s.cnt + kMaxStages);
  return s;
}

size_t smem_bytes(const PipeCfg& c) {
  return (size_t)c.NS * c.stage_bytes + 2 * kMaxStages * sizeof(uint64_t) + 2 * kMaxStages * sizeof(int) +
         (size_t)kMaxStages * kMaxTopK * 8 * sizeof(float);
}

__device__ __forceinline__ const uint8_t* slot_ptr(const Dev& d, int layer, int slot) {
  return d.pool + ((size_t)layer * d.S_alloc + slot) * d.lay.stride;
}

// Producer: one thread.  Arms stage it % NS for item `it` (after the consumers released its
// previous use), or publishes -1 when the queue is empty.  Returns after waiting for every
// armed stage's copies, so no copy is in flight when the block exits.
template <class Issue>
__device__ void produce(const PipeCfg& c, const Smem& sm, unsigned* queue, unsigned* err, Issue issue) {
  int armed[kMaxStages];
#pragma unroll
  for (int s = 0; s < kMaxStages; ++s) armed[s] = 0;
  bool ok = true;
  for (int it = 0;; ++it) {
    const int s = it % c.NS;
    if (it >= c.NS && !mbar_wait(&sm.empty[s], ((it / c.NS) - 1) & 1)) {
      atomicExch(err, 1u);
      ok = false;
    }
    int item = ok ? (int)atomicAdd(queue, 1u) : -1;
    if (item >= c.n_items) item = -1;
    sm.item[s] = item;
    armed[s]++;
    if (item < 0) {
      mbar_arrive(&sm.full[s]);
      break;
    }
    mbar_arrive_tx(&sm.full[s], c.stage_bytes);
    issue(item, sm.stage0 + (size_t)s * c.stage_bytes, &sm.full[s]);
  }
  for (int s = 0; s < c.NS; ++s)
    if (armed[s] > 0 && !mbar_wait(&sm.full[s], (armed[s] - 1) & 1)) atomicExch(err, 2u);
}

__device__ __forceinline__ void init_barriers(const PipeCfg& c, const Smem& sm) {
  if (threadIdx.x == 0) {
    for (int s = 0; s < c.NS; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kConsumers);
      sm.cnt[s] = 0;
    }
    mbar_fence_init();
  }
  __syncthreads();
}

// ---------------------------------------------------------------- gate/up + SwiGLU, one token
template <int QT, int VPL>
__global__ void __launch_bounds__(kThreads, 1) k_gateup_pipe(Dev d, int layer, const float* __restrict__ x, PipeCfg c) {
  extern __shared__ __align__(128) unsigned char smem[];
  const Smem sm = carve(smem, c);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qrow = d.lay.qrow_gu, nb = d.lay.nb_gu, nvec = qrow / 16;
  const int nrb = d.I / kGuRows;
  init_barriers(c, sm);

  if (warp == kConsumers) {
    if (lane == 0)
      produce(c, sm, &d.work[0], d.err, [&](int item, unsigned char* st, uint64_t* bar) {
        const int u = item / nrb, rb = item % nrb;
        const uint8_t* base = slot_ptr(d, layer, d.uslot[u]);
        const uint32_t cb = kGuRows * qrow, sb = kGuRows * nb * 2;
        const size_t r0 = (size_t)rb * kGuRows;
        bulk_g2s(st, base + d.lay.gq + r0 * qrow, cb, bar);
        bulk_g2s(st + cb, base + d.lay.uq + r0 * qrow, cb, bar);
        bulk_g2s(st + 2 * cb, base + d.lay.gd + r0 * nb * 2, sb, bar);
        bulk_g2s(st + 2 * cb + sb, base + d.lay.ud + r0 * nb * 2, sb, bar);
      });
  } else {
    XV<QT> xr[VPL];
#pragma unroll
    for (int i = 0; i < VPL; ++i) {
      const int v = lane + 32 * i;
      if (v < nvec) xr[i] = load_x<QT>(x + v * Vec<QT>::kW);
    }
    const uint32_t cb = kGuRows * qrow, sb = kGuRows * nb * 2;
    for (int it = 0;; ++it) {
      const int s = it % c.NS;
      if (!mbar_wait(&sm.full[s], (it / c.NS) & 1)) {
        if (lane == 0) atomicExch(d.err, 3u);
        break;
      }
      const int item = sm.item[s];
      if (item < 0) break;
      const unsigned char* st = sm.stage0 + (size_t)s * c.stage_bytes;
      const unsigned char* gq = st + warp * qrow;
      const unsigned char* uq = st + cb + warp * qrow;
      const __half* gs = reinterpret_cast<const __half*>(st + 2 * cb) + warp * nb;
      const __half* us = reinterpret_cast<const __half*>(st + 2 * cb + sb) + warp * nb;
      float ag = 0.f, au = 0.f;
#pragma unroll
      for (int i = 0; i < VPL; ++i) {
        const int v = lane + 32 * i;
        if (v < nvec) {
          const uint4 wg = *reinterpret_cast<const uint4*>(gq + 16 * v);
          const uint4 wu = *reinterpret_cast<const uint4*>(uq + 16 * v);
          ag = fmaf(dot_vec<QT>(wg, xr[i]), __half2float(gs[scale_index<QT>(v)]), ag);
          au = fmaf(dot_vec<QT>(wu, xr[i]), __half2float(us[scale_index<QT>(v)]), au);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.empty[s]);
      ag = warp_sum(ag);
      au = warp_sum(au);
      if (lane == 0) {
        const int u = item / nrb, r = (item % nrb) * kGuRows + warp;
        d.h[(size_t)u * d.I + r] = ag / (1.0f + expf(-ag)) * au;
      }
    }
  }
  __syncthreads();
}

// ---------------------------------------------------------------- down + combine, one token
template <int QT, int VPLD>
__global__ void __launch_bounds__(kThreads, 1) k_down_pipe(Dev d, int layer, float* __restrict__ y, PipeCfg c) {
  extern __shared__ __align__(128) unsigned char smem[];
  const Smem sm = carve(smem, c);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = d.k, R = c.R;
  const int qrow = d.lay.qrow_d, nb = d.lay.nb_d, nvec = qrow / 16;
  init_barriers(c, sm);

  if (warp == kConsumers) {
    if (lane == 0)
      produce(c, sm, &d.work[1], d.err, [&](int item, unsigned char* st, uint64_t* bar) {
        const size_t c0 = (size_t)item * R;
        const uint32_t cbytes = (uint32_t)R * qrow, sbytes = (uint32_t)R * nb * 2;
        for (int j = 0; j < k; ++j) {
          const uint8_t* base = slot_ptr(d, layer, d.uslot[j]);
          bulk_g2s(st + j * c.per_j, base + d.lay.dq + c0 * qrow, cbytes, bar);
          bulk_g2s(st + j * c.per_j + cbytes, base + d.lay.dd + c0 * nb * 2, sbytes, bar);
        }
      });
  } else {
    const int nwe = kConsumers / k;  // warps per expert
    const int j = warp / nwe, sub = warp % nwe;
    const bool active = j < k;
    XV<QT> hr[VPLD];
    if (active) {
#pragma unroll
      for (int i = 0; i < VPLD; ++i) {
        const int v = lane + 32 * i;
        if (v < nvec) hr[i] = load_x<QT>(d.h + (size_t)j * d.I + v * Vec<QT>::kW);
      }
    }
    for (int it = 0;; ++it) {
      const int s = it % c.NS;
      if (!mbar_wait(&sm.full[s], (it / c.NS) & 1)) {
        if (lane == 0) atomicExch(d.err, 4u);
        break;
      }
      const int item = sm.item[s];
      if (item < 0) break;
      const unsigned char* st = sm.stage0 + (size_t)s * c.stage_bytes;
      float* part = sm.part + (size_t)s * kMaxTopK * 8;
      if (active) {
        const unsigned char* q = st + j * c.per_j;
        const __half* sc = reinterpret_cast<const __half*>(q + (size_t)R * qrow);
        for (int rho = sub; rho < R; rho += nwe) {
          float acc = 0.f;
#pragma unroll
          for (int i = 0; i < VPLD; ++i) {
            const int v = lane + 32 * i;
            if (v < nvec) {
              const uint4 w = *reinterpret_cast<const uint4*>(q + (size_t)rho * qrow + 16 * v);
              acc = fmaf(dot_vec<QT>(w, hr[i]), __half2float(sc[rho * nb + scale_index<QT>(v)]), acc);
            }
          }
          acc = warp_sum(acc);
          if (lane == 0) part[j * 8 + rho] = acc;
        }
      }
      __syncwarp();
      // the last warp to finish this item combines the k partial rows in rank order
      int last = 0;
      if (lane == 0) {
        __threadfence_block();
        last = atomicAdd(&sm.cnt[s], 1) == kConsumers - 1;
      }
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence_block();
        if (lane < R) {
          float acc = 0.f;
          for (int jj = 0; jj < k; ++jj) acc = fmaf(d.g[jj], part[jj * 8 + lane], acc);
          y[(size_t)item * R + lane] = acc;
        }
        if (lane == 0) sm.cnt[s] = 0;
        __syncwarp();
      }
      if (lane == 0) mbar_arrive(&sm.empty[s]);
    }
  }
  __syncthreads();
}

int pick_vpl(int nvec) {
  const int need = (nvec + 31) / 32;
  if (need <= 1) return 1;
  if (need <= 2) return 2;
  if (need <= 3) return 3;
  if (need <= 4) return 4;
  if (need <= 6) return 6;
  return 8;
}

int sm_count() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

PipeCfg gateup_cfg(const Dev& d) {
  PipeCfg c;
  c.R = kGuRows;
  c.stage_bytes = 2u * kGuRows * d.lay.qrow_gu + 2u * kGuRows * d.lay.nb_gu * 2;
  c.n_items = d.k * (d.I / kGuRows);
  c.per_j = 0;
  c.NS = (int)((kSmemBudget - 4096) / c.stage_bytes);
  if (c.NS > kMaxStages) c.NS = kMaxStages;
  return c;
}

PipeCfg down_cfg(const Dev& d) {
  PipeCfg c;
  c.R = 2;  // smallest row count whose scale block is a multiple of 16 bytes
  while ((c.R * d.I) % 256 != 0) c.R *= 2;
  c.per_j = (uint32_t)c.R * d.lay.qrow_d + (uint32_t)c.R * d.lay.nb_d * 2;
  c.stage_bytes = c.per_j * d.k;
  c.n_items = d.H / c.R;
  c.NS = (int)((kSmemBudget - 4096) / c.stage_bytes);
  if (c.NS > kMaxStages) c.NS = kMaxStages;
  return c;
}

template <int QT>
cudaError_t gateup_pipe_q(const Dev& d, int layer, const float* x, cudaStream_t s) {
  const PipeCfg c = gateup_cfg(d);
  const size_t smem = smem_bytes(c);
  const int grid = sm_count();
#define MF_GU(V)                                                                                     \
  {                                                                                                  \
    cudaError_t e = cudaFuncSetAttribute(k_gateup_pipe<QT, V>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                         (int)smem);                                                 \
    if (e != cudaSuccess) return e;                                                                  \
    k_gateup_pipe<QT, V><<<grid, kThreads, smem, s>>>(d, layer, x, c);                               \
    break;                                                                                           \
  }
  switch (pick_vpl(d.lay.qrow_gu / 16)) {
    case 1: MF_GU(1)
    case 2: MF_GU(2)
    case 3: MF_GU(3)
    case 4: MF_GU(4)
    default: MF_GU(6)
  }
#undef MF_GU
  return cudaGetLastError();
}

template <int QT>
cudaError_t down_pipe_q(const Dev& d, int layer, float* y, cudaStream_t s) {
  const PipeCfg c = down_cfg(d);
  const size_t smem = smem_bytes(c);
  const int grid = sm_count();
#define MF_DN(V)                                                                                   \
  {                                                                                                \
    cudaError_t e = cudaFuncSetAttribute(k_down_pipe<QT, V>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                         (int)smem);                                               \
    if (e != cudaSuccess) return e;                                                                \
    k_down_pipe<QT, V><<<grid, kThreads, smem, s>>>(d, layer, y, c);                               \
    break;                                                                                         \
  }
  switch (pick_vpl(d.lay.qrow_d / 16)) {
    case 1: MF_DN(1)
    default: MF_DN(2)
  }
#undef MF_DN
  return cudaGetLastError();
}

}  // namespace

// The pipelined kernels apply when the register-held vector fits (<= 96 floats for x,
// <= 64 for h) and at least two stages fit in shared memory.
bool decode_pipe_ok(const Dev& d) {
  const int kw = d.qtype == MF_Q8_0 ? 16 : 32;
  const int vx = pick_vpl(d.lay.qrow_gu / 16), vh = pick_vpl(d.lay.qrow_d / 16);
  if (vx * kw > 96 || vh > 2 || vh * kw > 64) return false;
  if (d.I % kGuRows != 0) return false;
  if (gateup_cfg(d).NS < 2 || down_cfg(d).NS < 2) return false;
  if (d.H % down_cfg(d).R != 0) return false;
  return true;
}

cudaError_t launch_gateup_single(const Dev& d, int layer, const float* x, cudaStream_t s) {
  return d.qtype == MF_Q8_0 ? gateup_pipe_q<kQ8>(d, layer, x, s) : gateup_pipe_q<kQ4>(d, layer, x, s);
}

cudaError_t launch_down_single_pipe(const Dev& d, int layer, float* y, cudaStream_t s) {
  return d.qtype == MF_Q8_0 ? down_pipe_q<kQ8>(d, layer, y, s) : down_pipe_q<kQ4>(d, layer, y, s);
}

size_t decode_smem_bytes(const Dev& d, int which) { return smem_bytes(which == 0 ? gateup_cfg(d) : down_cfg(d)); }

}  // namespace mf
