// Batch-1 decode expert FFN as two persistent, pipelined dequantising GEMV kernels.
//
//   gate/up:  h_j[r] = silu(Wg_j[r,:] . x) * (Wu_j[r,:] . x)        for the k routed experts j
//   down:     y[c]   = sum_j g_j (Wd_j[c,:] . h_j)                     (router-weighted combine)
// (SwiGLU experts with separate gate, up and down tensors, section "Native Serving Path";
// W = d*q for Q8_0, d*(n-8) for Q4_0; fp32 accumulation.)
//
// One CTA per SM: one producer warp and sixteen consumer warps.  A block's work items are
// blockIdx.x, blockIdx.x + gridDim.x, ... (every item costs the same, so a static split is as
// balanced as a queue).  The producer streams each item's quantised rows and scales from the
// HBM slots into a ring of shared-memory stages with bulk asynchronous copies completing on an
// mbarrier; the consumers dequantise from shared memory and release each stage through a
// second mbarrier.  The producer loop is kept to a few instructions per item: it shares its
// scheduler with busy consumer warps, and its issue rate bounds the kernel's bandwidth.  Memory traffic is decoupled from
// registers: the ring holds most of an SM's share of a call, so nearly all of it is in flight
// at once.  Each consumer warp keeps the vector it multiplies by (its part of x, or its
// expert's h) in registers for the whole kernel: a lane always handles the same columns.
//   gate/up item = R rows of one expert's gate and up tensors; the 16 warps split the 2R rows
//                  into 16 / (2R) column ranges.
//   down item    = R output rows of all k experts; warp w owns (expert w / R, row w % R).
// Warps never wait for each other per item: each keeps its partial results of all the block's
// items in shared memory, and after one barrier at the end the block forms h = silu(gate) * up
// (column ranges added in order) or y = sum_j g_j part_j (experts in rank order).  Results are
// deterministic and need no atomics.  Every wait is bounded; a wait that gives up sets the device error word
// and the block stops.
#include "mf_dequant.cuh"

namespace mf {
namespace {

using namespace dq;

constexpr int kConsumers = 16;
constexpr int kThreads = (kConsumers + 1) * 32;
constexpr int kMaxStages = 12;
constexpr size_t kSmemBudget = 200 * 1024;

struct PipeCfg {
  int R;                 // rows per item
  int NS;                // stages
  uint32_t stage_bytes;  // bytes per item (= per stage)
  int n_items;
  uint32_t per_j;        // down: bytes of one expert's share of an item
  int cs;                // gate/up: column ranges per row (16 / (2R))
  int max_mine;          // most items any block gets
  int slots;             // partial results per item
  int n_vec;             // vectors split into int8 pieces at kernel start (x, or the k h's)
  uint32_t vq_bytes;     // their shared-memory bytes
};

struct Smem {
  unsigned char* stage0;
  uint64_t* full;
  uint64_t* empty;
  float* red;         // [max_mine][16 warps]: every partial result of the block, combined at the end
  unsigned char* vq;  // [n_vec] split vectors (XQ), written once by the consumers at kernel start
};

__device__ __forceinline__ Smem carve(unsigned char* base, const PipeCfg& c) {
  Smem s;
  s.stage0 = base;
  unsigned char* p = base + (size_t)c.NS * c.stage_bytes;
  s.full = reinterpret_cast<uint64_t*>(p);
  s.empty = s.full + kMaxStages;
  s.red = reinterpret_cast<float*>(s.empty + kMaxStages);
  s.vq = reinterpret_cast<unsigned char*>(s.red + c.max_mine * kConsumers);
  return s;
}

size_t part_bytes(int max_mine) { return (size_t)max_mine * kConsumers * sizeof(float); }

size_t smem_bytes(const PipeCfg& c) {
  return (size_t)c.NS * c.stage_bytes + 2 * kMaxStages * sizeof(uint64_t) + part_bytes(c.max_mine) + c.vq_bytes;
}

// The consumers split `n` vectors of kW values into int8 pieces, one vector per thread, into
// shared memory, then wait for each other (the producer keeps streaming meanwhile).
template <int QT>
__device__ __forceinline__ void split_vectors(const float* __restrict__ src, int n, XQ<QT>* dst) {
  for (int i = threadIdx.x; i < n; i += kConsumers * 32) dst[i] = quant_vec<QT>(src + (size_t)i * Vec<QT>::kW);
  named_bar_sync(1, kConsumers * 32);
}

// Items of this block: blockIdx.x, blockIdx.x + gridDim.x, ...  Producer and consumers both
// walk this sequence, so no item index is handed over; stage = iteration mod NS.
__device__ __forceinline__ int items_of_block(int n_items) {
  return (int)blockIdx.x < n_items ? (n_items - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x : 0;
}

// Stage/phase walk without divisions.
struct Ring {
  int s = 0;
  uint32_t phase = 0;
  __device__ __forceinline__ void next(int ns) {
    if (++s == ns) {
      s = 0;
      phase ^= 1u;
    }
  }
};

__device__ __forceinline__ void init_barriers(const PipeCfg& c, const Smem& sm) {
  if (threadIdx.x == 0) {
    for (int s = 0; s < c.NS; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kConsumers);
    }
    mbar_fence_init();
  }
  __syncthreads();
}

// Producer epilogue: wait (bounded) for the last use of every stage, so that no copy is in
// flight when the block exits even if the consumers stopped early.
__device__ __forceinline__ void drain(const PipeCfg& c, const Smem& sm, int mine, unsigned* err) {
  for (int s = 0; s < c.NS && s < mine; ++s) {
    const int uses = (mine - 1 - s) / c.NS + 1;  // iterations it < mine with it % NS == s
    if (!mbar_wait(&sm.full[s], (uint32_t)(uses - 1) & 1u)) atomicExch(err, 2u);
  }
}

// ---------------------------------------------------------------- gate/up + SwiGLU, one token
// Item i = (expert u = i / (I/R), row block i % (I/R)).  Warp w: tensor w / (R*cs) (0 gate,
// 1 up), row (w / cs) % R, column range w % cs.
template <int QT, int VPL>
__global__ void __launch_bounds__(kThreads, 1) k_gateup_pipe(Dev d, int layer, const float* __restrict__ x, PipeCfg c) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ const uint8_t* s_base[kMaxTopK];  // slot of each routed expert
  const Smem sm = carve(smem, c);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qrow = d.lay.qrow_gu;
  const int R = c.R, cs = c.cs, nrb = d.I / R;
  const uint32_t rs = d.lay.rs_gu;
  const int mine = items_of_block(c.n_items);
  if (threadIdx.x < d.k)
    s_base[threadIdx.x] = d.pool + ((size_t)layer * d.S_alloc + d.uslot[threadIdx.x]) * d.lay.stride;
  init_barriers(c, sm);

  if (warp == kConsumers) {
    if (lane == 0) {
      const int grid = (int)gridDim.x;
      int u = (int)blockIdx.x / nrb, rb = (int)blockIdx.x % nrb;
      Ring ring;
      for (int it = 0; it < mine; ++it) {
        if (it >= c.NS && !mbar_wait(&sm.empty[ring.s], ring.phase ^ 1u)) {
          atomicExch(d.err, 1u);
          break;
        }
        uint64_t* bar = &sm.full[ring.s];
        mbar_arrive_tx(bar, c.stage_bytes);  // R contiguous row records of expert u
        bulk_g2s(sm.stage0 + (size_t)ring.s * c.stage_bytes, s_base[u] + (size_t)rb * R * rs, c.stage_bytes, bar);
        ring.next(c.NS);
        rb += grid;  // next item of this block
        while (rb >= nrb) {
          rb -= nrb;
          ++u;
        }
      }
      drain(c, sm, mine, d.err);
    }
  } else {
    const int ten = warp / (R * cs), row = (warp / cs) % R, col = warp % cs;
    const int nv = (qrow / 16) / cs;  // vectors in this warp's column range
    const int v0 = col * nv;
    const XQ<QT>* xq = reinterpret_cast<const XQ<QT>*>(sm.vq);
    split_vectors<QT>(x, c.n_vec, reinterpret_cast<XQ<QT>*>(sm.vq));
    XQ<QT> xr[VPL];
#pragma unroll
    for (int i = 0; i < VPL; ++i) {
      const int v = lane + 32 * i;
      if (v < nv) xr[i] = xq[v0 + v];
    }
    Ring ring;
    for (int it = 0; it < mine; ++it) {
      if (!mbar_wait(&sm.full[ring.s], ring.phase)) {
        if (lane == 0) atomicExch(d.err, 3u);
        break;
      }
      const unsigned char* st = sm.stage0 + (size_t)ring.s * c.stage_bytes;
      const unsigned char* rec = st + row * rs;
      const unsigned char* q = rec + ten * d.lay.o_up + 16 * v0;
      const __half* sc = reinterpret_cast<const __half*>(rec + (ten ? d.lay.o_us : d.lay.o_gs));
      float acc = 0.f;
#pragma unroll
      for (int i = 0; i < VPL; ++i) {
        const int v = lane + 32 * i;
        if (v < nv)
          acc = fmaf(dot_q<QT>(*reinterpret_cast<const uint4*>(q + 16 * v), xr[i]),
                     __half2float(sc[scale_index<QT>(v0 + v)]), acc);
      }
      acc = warp_sum(acc);
      if (lane == 0) sm.red[it * kConsumers + warp] = acc;
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.empty[ring.s]);
      ring.next(c.NS);
    }
    // all partial results of the block are in shared memory: SwiGLU over (item, row), column
    // ranges added in order
    named_bar_sync(1, kConsumers * 32);
    for (int t = threadIdx.x; t < mine * R; t += kConsumers * 32) {
      const int it = t / R, r = t % R;
      const float* p = sm.red + it * kConsumers;
      float ag = 0.f, au = 0.f;
      for (int cc = 0; cc < cs; ++cc) {
        ag += p[(0 * R + r) * cs + cc];
        au += p[(1 * R + r) * cs + cc];
      }
      const int item = (int)blockIdx.x + it * (int)gridDim.x;
      d.h[(size_t)(item / nrb) * d.I + (item % nrb) * R + r] = ag / (1.0f + expf(-ag)) * au;
    }
  }
  __syncthreads();
}

// ---------------------------------------------------------------- down + combine, one token
// Item i = output rows [i*R, (i+1)*R) of all k experts.
template <int QT, int VPLD>
__global__ void __launch_bounds__(kThreads, 1) k_down_pipe(Dev d, int layer, float* __restrict__ y, PipeCfg c) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ float s_g[kMaxTopK];
  __shared__ const uint8_t* s_base[kMaxTopK];
  const Smem sm = carve(smem, c);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = d.k, R = c.R;
  const int qrow = d.lay.qrow_d, nvec = qrow / 16;
  const uint32_t rs = d.lay.rs_d;
  const int mine = items_of_block(c.n_items);
  if (threadIdx.x < k) {
    s_g[threadIdx.x] = d.g[threadIdx.x];
    s_base[threadIdx.x] = d.pool + ((size_t)layer * d.S_alloc + d.uslot[threadIdx.x]) * d.lay.stride + d.lay.d_off;
  }
  init_barriers(c, sm);  // (its barrier also publishes s_g and s_base)

  if (warp == kConsumers) {
    if (lane == 0) {
      const uint32_t per_j = c.per_j;  // R contiguous down records of each expert
      Ring ring;
      size_t c0 = (size_t)blockIdx.x * R;
      const size_t c_step = (size_t)gridDim.x * R;
      for (int it = 0; it < mine; ++it) {
        if (it >= c.NS && !mbar_wait(&sm.empty[ring.s], ring.phase ^ 1u)) {
          atomicExch(d.err, 1u);
          break;
        }
        unsigned char* st = sm.stage0 + (size_t)ring.s * c.stage_bytes;
        uint64_t* bar = &sm.full[ring.s];
        mbar_arrive_tx(bar, c.stage_bytes);
        for (int j = 0; j < k; ++j) bulk_g2s(st + j * per_j, s_base[j] + c0 * rs, per_j, bar);
        ring.next(c.NS);
        c0 += c_step;
      }
      drain(c, sm, mine, d.err);
    }
  } else {
    const int j = warp / R, rho = warp % R;  // one (expert, row) task per warp: k * R <= 16
    const bool active = j < k;
    const XQ<QT>* hq = reinterpret_cast<const XQ<QT>*>(sm.vq);
    split_vectors<QT>(d.h, c.n_vec, reinterpret_cast<XQ<QT>*>(sm.vq));  // h of all k experts
    XQ<QT> hr[VPLD];
    if (active) {
#pragma unroll
      for (int i = 0; i < VPLD; ++i) {
        const int v = lane + 32 * i;
        if (v < nvec) hr[i] = hq[j * nvec + v];
      }
    }
    Ring ring;
    for (int it = 0; it < mine; ++it) {
      if (!mbar_wait(&sm.full[ring.s], ring.phase)) {
        if (lane == 0) atomicExch(d.err, 4u);
        break;
      }
      const unsigned char* st = sm.stage0 + (size_t)ring.s * c.stage_bytes;
      float acc = 0.f;
      if (active) {
        const unsigned char* q = st + j * c.per_j + (size_t)rho * rs;
        const __half* sc = reinterpret_cast<const __half*>(q + d.lay.o_ds);
#pragma unroll
        for (int i = 0; i < VPLD; ++i) {
          const int v = lane + 32 * i;
          if (v < nvec)
            acc = fmaf(dot_q<QT>(*reinterpret_cast<const uint4*>(q + 16 * v), hr[i]),
                       __half2float(sc[scale_index<QT>(v)]), acc);
        }
      }
      acc = warp_sum(acc);
      if (lane == 0) sm.red[it * kConsumers + warp] = acc;
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.empty[ring.s]);
      ring.next(c.NS);
    }
    // combine the k experts of each output row in rank order
    named_bar_sync(1, kConsumers * 32);
    for (int t = threadIdx.x; t < mine * R; t += kConsumers * 32) {
      const int it = t / R, r = t % R;
      const float* p = sm.red + it * kConsumers;
      float acc = 0.f;
      for (int jj = 0; jj < k; ++jj) acc = fmaf(s_g[jj], p[jj * R + r], acc);
      y[((size_t)blockIdx.x + (size_t)it * gridDim.x) * R + r] = acc;
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

int stages_for(uint32_t stage_bytes, size_t part_bytes) {
  if (part_bytes + 4096 >= kSmemBudget) return 0;
  int ns = (int)((kSmemBudget - 4096 - part_bytes) / stage_bytes);
  return ns > kMaxStages ? kMaxStages : ns;
}

PipeCfg gateup_cfg(const Dev& d) {
  PipeCfg c;
  const int nvec = d.lay.qrow_gu / 16;
  // 4 rows x 2 column ranges when the row's vectors split evenly, else 8 whole rows
  if (nvec % 2 == 0 && d.I % 4 == 0) {
    c.R = 4;
    c.cs = 2;
  } else {
    c.R = 8;
    c.cs = 1;
  }
  c.stage_bytes = (uint32_t)c.R * d.lay.rs_gu;
  c.n_items = d.k * (d.I / c.R);
  c.per_j = 0;
  c.slots = kConsumers;
  c.max_mine = (c.n_items + sm_count() - 1) / sm_count();
  c.n_vec = d.lay.qrow_gu / 16;
  c.vq_bytes = (uint32_t)(c.n_vec * (d.qtype == MF_Q8_0 ? sizeof(XQ<kQ8>) : sizeof(XQ<kQ4>)));
  c.NS = stages_for(c.stage_bytes, part_bytes(c.max_mine) + c.vq_bytes);
  return c;
}

PipeCfg down_cfg(const Dev& d) {
  PipeCfg c;
  c.R = 2;
  c.cs = 1;
  c.per_j = (uint32_t)c.R * d.lay.rs_d;
  c.stage_bytes = c.per_j * d.k;
  c.n_items = d.H / c.R;
  c.slots = kConsumers;
  c.max_mine = (c.n_items + sm_count() - 1) / sm_count();
  c.n_vec = d.k * (d.lay.qrow_d / 16);
  c.vq_bytes = (uint32_t)(c.n_vec * (d.qtype == MF_Q8_0 ? sizeof(XQ<kQ8>) : sizeof(XQ<kQ4>)));
  c.NS = stages_for(c.stage_bytes, part_bytes(c.max_mine) + c.vq_bytes);
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
  const int max_vx = d.qtype == MF_Q8_0 ? 4 : 2, max_vh = d.qtype == MF_Q8_0 ? 3 : 2;  // registers: no spills
  if (((d.lay.qrow_gu / 16) / gu.cs + 31) / 32 > max_vx) return false;
  if ((d.lay.qrow_d / 16 + 31) / 32 > max_vh) return false;
  if (d.I % gu.R != 0 || d.H % dn.R != 0 || d.k * dn.R > kConsumers) return false;
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
