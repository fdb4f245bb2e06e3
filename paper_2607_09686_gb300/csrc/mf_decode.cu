// Batch-1 decode expert FFN as two persistent, pipelined dequantising GEMV kernels.
//
//   gate/up:  h_j[r] = silu(Wg_j[r,:] . x) * (Wu_j[r,:] . x)        for the k routed experts j
//   down:     y[c]   = sum_j g_j (Wd_j[c,:] . h_j)                     (router-weighted combine)
// (SwiGLU experts with separate gate, up and down tensors, section "Native Serving Path";
// W = d*q for Q8_0, d*(n-8) for Q4_0; fp32 accumulation.)
//
// One CTA per SM: one producer warp and sixteen consumer warps.  The producer takes the
// block's work items (round-robin over blocks: every item costs the same) and streams each
// item's quantised rows and scales from the HBM slots into a ring of shared-memory stages with
// bulk asynchronous copies completing on an mbarrier; the consumers dequantise from shared
// memory and release each stage through a second mbarrier.  Memory traffic is decoupled from
// registers: the ring holds most of an SM's share of a call, so nearly all of it is in flight
// at once.  Each consumer warp keeps the vector it multiplies by (its part of x, or its
// expert's h) in registers for the whole kernel: a lane always handles the same columns.
//   gate/up item = R rows of one expert's gate and up tensors; the 16 warps split the 2R rows
//                  into 16 / (2R) column ranges, and the last warp to finish the item forms
//                  h = silu(gate) * up for its R rows.
//   down item    = R output rows of all k experts; 16 / k warps per expert share its rows, and
//                  the last warp to finish the item adds the k partial rows in rank order.
// Partial results are combined in a fixed order, so results are deterministic and atomic-free
// in global memory.  Every wait is bounded; a wait that gives up sets the device error word
// and the block stops.
#include "mf_dequant.cuh"

namespace mf {
namespace {

using namespace dq;

constexpr int kConsumers = 16;
constexpr int kThreads = (kConsumers + 1) * 32;
constexpr int kMaxStages = 12;
constexpr int kPartSlots = 64;  // partial results kept per stage
constexpr size_t kSmemBudget = 200 * 1024;

struct PipeCfg {
  int R;                 // rows per item
  int NS;                // stages
  uint32_t stage_bytes;  // bytes per item (= per stage)
  int n_items;
  uint32_t per_j;        // down: bytes of one expert's share of an item
  int cs;                // gate/up: column ranges per row (16 / (2R))
};

struct Smem {
  unsigned char* stage0;
  uint64_t* full;
  uint64_t* empty;
  int* item;
  int* cnt;
  float* part;  // [kMaxStages][kPartSlots]
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
         (size_t)kMaxStages * kPartSlots * sizeof(float);
}

__device__ __forceinline__ const uint8_t* slot_ptr(const Dev& d, int layer, int slot) {
  return d.pool + ((size_t)layer * d.S_alloc + slot) * d.lay.stride;
}

// Producer: one thread.  Arms stage it % NS for item block + it * grid after the consumers
// released the stage's previous use, or publishes -1 when the block has no items left.
// Returns after waiting for every armed stage's copies, so no copy is in flight at exit.
template <class Issue>
__device__ void produce(const PipeCfg& c, const Smem& sm, unsigned* err, Issue issue) {
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
    int item = (int)blockIdx.x + it * (int)gridDim.x;
    if (!ok || item >= c.n_items) item = -1;
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

// After writing its partial results for the item a consumer warp counts itself in; the last
// one (true) may read every partial of the stage.
__device__ __forceinline__ bool last_of_item(const Smem& sm, int s, int lane) {
  int last = 0;
  if (lane == 0) {
    __threadfence_block();
    last = atomicAdd(&sm.cnt[s], 1) == kConsumers - 1;
  }
  last = __shfl_sync(0xffffffffu, last, 0);
  if (last) __threadfence_block();
  return last != 0;
}

// ---------------------------------------------------------------- gate/up + SwiGLU, one token
// Warp w: tensor w / (R*cs) (0 gate, 1 up), row (w / cs) % R, column range w % cs.
template <int QT, int VPL>
__global__ void __launch_bounds__(kThreads, 1) k_gateup_pipe(Dev d, int layer, const float* __restrict__ x, PipeCfg c) {
  extern __shared__ __align__(128) unsigned char smem[];
  const Smem sm = carve(smem, c);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qrow = d.lay.qrow_gu, nb = d.lay.nb_gu;
  const int R = c.R, cs = c.cs, nrb = d.I / R;
  const uint32_t cb = (uint32_t)R * qrow, sb = (uint32_t)R * nb * 2;
  init_barriers(c, sm);

  if (warp == kConsumers) {
    if (lane == 0)
      produce(c, sm, d.err, [&](int item, unsigned char* st, uint64_t* bar) {
        const int u = item / nrb, rb = item % nrb;
        const uint8_t* base = slot_ptr(d, layer, d.uslot[u]);
        const size_t r0 = (size_t)rb * R;
        bulk_g2s(st, base + d.lay.gq + r0 * qrow, cb, bar);
        bulk_g2s(st + cb, base + d.lay.uq + r0 * qrow, cb, bar);
        bulk_g2s(st + 2 * cb, base + d.lay.gd + r0 * nb * 2, sb, bar);
        bulk_g2s(st + 2 * cb + sb, base + d.lay.ud + r0 * nb * 2, sb, bar);
      });
  } else {
    const int ten = warp / (R * cs), row = (warp / cs) % R, col = warp % cs;
    const int nv = (qrow / 16) / cs;  // vectors in this warp's column range
    const int v0 = col * nv;
    XV<QT> xr[VPL];
#pragma unroll
    for (int i = 0; i < VPL; ++i) {
      const int v = lane + 32 * i;
      if (v < nv) xr[i] = load_x<QT>(x + (v0 + v) * Vec<QT>::kW);
    }
    for (int it = 0;; ++it) {
      const int s = it % c.NS;
      if (!mbar_wait(&sm.full[s], (it / c.NS) & 1)) {
        if (lane == 0) atomicExch(d.err, 3u);
        break;
      }
      const int item = sm.item[s];
      if (item < 0) break;
      const unsigned char* st = sm.stage0 + (size_t)s * c.stage_bytes;
      float* part = sm.part + (size_t)s * kPartSlots;
      const unsigned char* q = st + ten * cb + row * qrow + 16 * v0;
      const __half* sc = reinterpret_cast<const __half*>(st + 2 * cb + ten * sb) + row * nb;
      float acc = 0.f;
#pragma unroll
      for (int i = 0; i < VPL; ++i) {
        const int v = lane + 32 * i;
        if (v < nv)
          acc = fmaf(dot_vec<QT>(*reinterpret_cast<const uint4*>(q + 16 * v), xr[i]),
                     __half2float(sc[scale_index<QT>(v0 + v)]), acc);
      }
      acc = warp_sum(acc);
      if (lane == 0) part[warp] = acc;
      __syncwarp();
      if (last_of_item(sm, s, lane)) {
        if (lane < R) {
          float ag = 0.f, au = 0.f;
          for (int cc = 0; cc < cs; ++cc) {  // column ranges in order
            ag += part[(0 * R + lane) * cs + cc];
            au += part[(1 * R + lane) * cs + cc];
          }
          const int u = item / nrb, r = (item % nrb) * R + lane;
          d.h[(size_t)u * d.I + r] = ag / (1.0f + expf(-ag)) * au;
        }
        if (lane == 0) sm.cnt[s] = 0;
        __syncwarp();
      }
      if (lane == 0) mbar_arrive(&sm.empty[s]);
    }
  }
  __syncthreads();
}

// ---------------------------------------------------------------- down + combine, one token
template <int QT, int VPLD>
__global__ void __launch_bounds__(kThreads, 1) k_down_pipe(Dev d, int layer, float* __restrict__ y, PipeCfg c) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ float s_g[kMaxTopK];
  const Smem sm = carve(smem, c);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = d.k, R = c.R;
  const int qrow = d.lay.qrow_d, nb = d.lay.nb_d, nvec = qrow / 16;
  if (threadIdx.x < k) s_g[threadIdx.x] = d.g[threadIdx.x];
  init_barriers(c, sm);  // (its barrier also publishes s_g)

  if (warp == kConsumers) {
    if (lane == 0)
      produce(c, sm, d.err, [&](int item, unsigned char* st, uint64_t* bar) {
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
      float* part = sm.part + (size_t)s * kPartSlots;
      if (active) {
        const unsigned char* q = st + j * c.per_j;
        const __half* sc = reinterpret_cast<const __half*>(q + (size_t)R * qrow);
        for (int rho = sub; rho < R; rho += nwe) {
          float acc = 0.f;
#pragma unroll
          for (int i = 0; i < VPLD; ++i) {
            const int v = lane + 32 * i;
            if (v < nvec)
              acc = fmaf(dot_vec<QT>(*reinterpret_cast<const uint4*>(q + (size_t)rho * qrow + 16 * v), hr[i]),
                         __half2float(sc[rho * nb + scale_index<QT>(v)]), acc);
          }
          acc = warp_sum(acc);
          if (lane == 0) part[j * R + rho] = acc;
        }
      }
      __syncwarp();
      if (last_of_item(sm, s, lane)) {
        if (lane < R) {
          float acc = 0.f;
          for (int jj = 0; jj < k; ++jj) acc = fmaf(s_g[jj], part[jj * R + lane], acc);
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

int vpl_for(int nvec) {
  const int need = (nvec + 31) / 32;
  return need <= 1 ? 1 : need <= 2 ? 2 : need <= 3 ? 3 : need <= 4 ? 4 : 8;
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

int stages_for(uint32_t stage_bytes) {
  int ns = (int)((kSmemBudget - 4096) / stage_bytes);
  return ns > kMaxStages ? kMaxStages : ns;
}

PipeCfg gateup_cfg(const Dev& d) {
  PipeCfg c;
  const int nvec = d.lay.qrow_gu / 16;
  // 4 rows x 2 column ranges when 4 rows of scales are a multiple of 16 bytes and the row's
  // vectors split evenly; otherwise 8 whole rows
  if ((4 * d.lay.nb_gu * 2) % 16 == 0 && nvec % 2 == 0 && d.I % 4 == 0) {
    c.R = 4;
    c.cs = 2;
  } else {
    c.R = 8;
    c.cs = 1;
  }
  c.stage_bytes = 2u * c.R * d.lay.qrow_gu + 2u * c.R * d.lay.nb_gu * 2;
  c.n_items = d.k * (d.I / c.R);
  c.per_j = 0;
  c.NS = stages_for(c.stage_bytes);
  return c;
}

PipeCfg down_cfg(const Dev& d) {
  PipeCfg c;
  c.R = 2;  // smallest row count whose scale block is a multiple of 16 bytes
  while ((c.R * d.I) % 256 != 0) c.R *= 2;
  c.cs = 1;
  c.per_j = (uint32_t)c.R * d.lay.qrow_d + (uint32_t)c.R * d.lay.nb_d * 2;
  c.stage_bytes = c.per_j * d.k;
  c.n_items = d.H / c.R;
  c.NS = stages_for(c.stage_bytes);
  return c;
}

template <int QT>
cudaError_t gateup_pipe_q(const Dev& d, int layer, const float* x, cudaStream_t s) {
  const PipeCfg c = gateup_cfg(d);
  const size_t smem = smem_bytes(c);
  const int grid = sm_count();
#define MF_GU(V)                                                                                            \
  {                                                                                                         \
    cudaError_t e =                                                                                         \
        cudaFuncSetAttribute(k_gateup_pipe<QT, V>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
    if (e != cudaSuccess) return e;                                                                         \
    k_gateup_pipe<QT, V><<<grid, kThreads, smem, s>>>(d, layer, x, c);                                      \
    break;                                                                                                  \
  }
  switch (vpl_for((d.lay.qrow_gu / 16) / c.cs)) {
    case 1: MF_GU(1)
    case 2: MF_GU(2)
    case 3: MF_GU(3)
    default: MF_GU(4)
  }
#undef MF_GU
  return cudaGetLastError();
}

template <int QT>
cudaError_t down_pipe_q(const Dev& d, int layer, float* y, cudaStream_t s) {
  const PipeCfg c = down_cfg(d);
  const size_t smem = smem_bytes(c);
  const int grid = sm_count();
#define MF_DN(V)                                                                                          \
  {                                                                                                       \
    cudaError_t e =                                                                                       \
        cudaFuncSetAttribute(k_down_pipe<QT, V>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
    if (e != cudaSuccess) return e;                                                                       \
    k_down_pipe<QT, V><<<grid, kThreads, smem, s>>>(d, layer, y, c);                                      \
    break;                                                                                                \
  }
  switch (vpl_for(d.lay.qrow_d / 16)) {
    case 1: MF_DN(1)
    case 2: MF_DN(2)
    default: MF_DN(3)
  }
#undef MF_DN
  return cudaGetLastError();
}

}  // namespace

// The pipelined kernels apply when the register-held vectors fit without spills (Q8_0: at most
// 4 vectors per lane of x, 3 of h; Q4_0: 2 and 2), the work splits evenly and at least two
// stages fit in shared memory.
bool decode_pipe_ok(const Dev& d) {
  const PipeCfg gu = gateup_cfg(d), dn = down_cfg(d);
  const int max_vx = d.qtype == MF_Q8_0 ? 4 : 2, max_vh = d.qtype == MF_Q8_0 ? 3 : 2;  // no register spills
  if (((d.lay.qrow_gu / 16) / gu.cs + 31) / 32 > max_vx) return false;
  if ((d.lay.qrow_d / 16 + 31) / 32 > max_vh) return false;
  if (d.I % gu.R != 0 || d.H % dn.R != 0 || dn.R * d.k > kPartSlots) return false;
  if (gu.NS < 2 || dn.NS < 2) return false;
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
