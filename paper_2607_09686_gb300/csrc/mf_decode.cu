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
constexpr int kThreadsF = (kConsumers + 2) * 32;  // fused kernel: + a link warp
constexpr int kMaxStages = 12;
constexpr size_t kSmemBudget = 200 * 1024;
constexpr size_t kFusedSmem = 224 * 1024;  // the fused kernel's dynamic + static shared memory
constexpr int kMaxItemsF = 64;            // gate/up items one block of the fused kernel may take

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

// The consumers split `n` groups of kW values into int8 pieces in shared memory (XQ).  Groups
// [r * per, (r + 1) * per) form one vector r (x, or one expert's h), split as if scaled by one
// power of two: each group is split with its own exponent, the vector's exponent e_r (the largest,
// a shared-memory atomic max) goes to s_exp[r], and each group's s is then rescaled to it.
// s_max[r] must hold kNoExp on entry; n <= 4 * 512.  The producer keeps streaming meanwhile.
template <int QT, bool kCoherent = false>
__device__ __forceinline__ void split_vectors(const float* __restrict__ src, int n, int per, XQ<QT>* dst,
                                              int* s_max, int* s_exp) {
  constexpr int kW = Vec<QT>::kW;
  const int nt = kConsumers * 32, i0 = (int)threadIdx.x;
  int eg[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = i0 + q * nt;
    if (i < n) {
      float v[kW];
      load_group<QT, kCoherent>(src + (size_t)i * kW, v);
      eg[q] = group_exponent(group_absmax<QT>(v));
      dst[i] = quant_vals<QT>(v, eg[q] == kNoExp ? 0 : -eg[q]);
      atomicMax(&s_max[i / per], eg[q]);
    }
  }
  named_bar_sync(1, nt);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = i0 + q * nt;
    if (i < n) rescale_group<QT>(dst[i], eg[q], vector_exponent(s_max[i / per]));
  }
  for (int r = i0; r * per < n; r += nt) s_exp[r] = vector_exponent(s_max[r]);
  named_bar_sync(1, nt);
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
__device__ __forceinline__ void drain(const PipeCfg& c, const Smem& sm, int mine, unsigned* err, uint64_t limit_ns) {
  for (int s = 0; s < c.NS && s < mine; ++s) {
    const int uses = (mine - 1 - s) / c.NS + 1;  // iterations it < mine with it % NS == s
    if (!mbar_wait(&sm.full[s], (uint32_t)(uses - 1) & 1u, limit_ns)) atomicExch(err, 2u);
  }
}

// ---------------------------------------------------------------- gate/up + SwiGLU, one token
// Item i = (expert u = i / (I/R), row block i % (I/R)).  Warp w: tensor w / (R*cs) (0 gate,
// 1 up), row (w / cs) % R, column range w % cs.
template <int QT, int VPL>
__global__ void __launch_bounds__(kThreads, 1) k_gateup_pipe(Dev d, int layer, const float* __restrict__ x, PipeCfg c) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ const uint8_t* s_base[kMaxTopK];  // slot of each routed expert
  __shared__ int s_xmax;
  __shared__ int s_xexp;
  const Smem sm = carve(smem, c);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qrow = d.lay.qrow_gu;
  const int R = c.R, cs = c.cs, nrb = d.I / R;
  const uint32_t rs = d.lay.rs_gu;
  const int mine = items_of_block(c.n_items);
  if (threadIdx.x < d.k)
    s_base[threadIdx.x] = d.pool + ((size_t)layer * d.S_alloc + d.uslot[threadIdx.x]) * d.lay.stride;
  if (threadIdx.x == 0) s_xmax = kNoExp;
  init_barriers(c, sm);

  if (warp == kConsumers) {
    if (lane == 0) {
      const int grid = (int)gridDim.x;
      int u = (int)blockIdx.x / nrb, rb = (int)blockIdx.x % nrb;
      Ring ring;
      for (int it = 0; it < mine; ++it) {
        if (it >= c.NS && !mbar_wait(&sm.empty[ring.s], ring.phase ^ 1u, d.wait_ns)) {
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
      drain(c, sm, mine, d.err, d.wait_ns);
    }
  } else {
    const int ten = warp / (R * cs), row = (warp / cs) % R, col = warp % cs;
    const int nv = (qrow / 16) / cs;  // vectors in this warp's column range
    const int v0 = col * nv;
    const XQ<QT>* xq = reinterpret_cast<const XQ<QT>*>(sm.vq);
    split_vectors<QT>(x, c.n_vec, c.n_vec, reinterpret_cast<XQ<QT>*>(sm.vq), &s_xmax, &s_xexp);
    XQ<QT> xr[VPL];
#pragma unroll
    for (int i = 0; i < VPL; ++i) {
      const int v = lane + 32 * i;
      if (v < nv) xr[i] = xq[v0 + v];
    }
    const int ex = s_xexp;
    Ring ring;
    for (int it = 0; it < mine; ++it) {
      if (!mbar_wait(&sm.full[ring.s], ring.phase, d.wait_ns)) {
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
    // ranges added in order, times 2^ex (x was split scaled by 2^-ex)
    named_bar_sync(1, kConsumers * 32);
    for (int t = threadIdx.x; t < mine * R; t += kConsumers * 32) {
      const int it = t / R, r = t % R;
      const float* p = sm.red + it * kConsumers;
      float ag = 0.f, au = 0.f;
      for (int cc = 0; cc < cs; ++cc) {
        ag += p[(0 * R + r) * cs + cc];
        au += p[(1 * R + r) * cs + cc];
      }
      ag = scale2(ag, ex);
      au = scale2(au, ex);
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
  __shared__ int s_hmax[kMaxTopK];
  __shared__ int s_hexp[kMaxTopK];
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
  if (threadIdx.x < kMaxTopK) s_hmax[threadIdx.x] = kNoExp;
  init_barriers(c, sm);  // (its barrier also publishes s_g, s_base and s_hmax)

  if (warp == kConsumers) {
    if (lane == 0) {
      const uint32_t per_j = c.per_j;  // R contiguous down records of each expert
      Ring ring;
      size_t c0 = (size_t)blockIdx.x * R;
      const size_t c_step = (size_t)gridDim.x * R;
      for (int it = 0; it < mine; ++it) {
        if (it >= c.NS && !mbar_wait(&sm.empty[ring.s], ring.phase ^ 1u, d.wait_ns)) {
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
      drain(c, sm, mine, d.err, d.wait_ns);
    }
  } else {
    const int j = warp / R, rho = warp % R;  // one (expert, row) task per warp: k * R <= 16
    const bool active = j < k;
    const XQ<QT>* hq = reinterpret_cast<const XQ<QT>*>(sm.vq);
    split_vectors<QT>(d.h, c.n_vec, nvec, reinterpret_cast<XQ<QT>*>(sm.vq), s_hmax, s_hexp);  // h of all k experts
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
      if (!mbar_wait(&sm.full[ring.s], ring.phase, d.wait_ns)) {
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
    // combine the k experts of each output row in rank order (expert j's partial times 2^e_j:
    // its h was split scaled by 2^-e_j)
    named_bar_sync(1, kConsumers * 32);
    for (int t = threadIdx.x; t < mine * R; t += kConsumers * 32) {
      const int it = t / R, r = t % R;
      const float* p = sm.red + it * kConsumers;
      float acc = 0.f;
      for (int jj = 0; jj < k; ++jj) acc = fmaf(s_g[jj], scale2(p[jj * R + r], s_hexp[jj]), acc);
      y[((size_t)blockIdx.x + (size_t)it * gridDim.x) * R + r] = acc;
    }
  }
  __syncthreads();
}

// ---------------------------------------------------------------- fused gate/up + down, one token
// Both projections in one persistent launch, which also materialises the call's missed
// experts.  The gate/up items are dealt round-robin over the blocks from a list that holds the
// resident experts' items first, so every block gets an equal share (+-1) of the missed ones.
// The producer warp streams the resident items from HBM through ring A; a link warp, from the
// first cycle, reads the missed items straight from the pinned pack (16-byte loads over the host
// link) into the stages of a small ring B and writes each through to the expert's new HBM slot,
// then does the same for the missed experts' down records, so the link transfer overlaps the
// resident data and all compute.  The consumers take ring A's items, then ring B's.  A block's
// down work is a contiguous range of rpc output rows: its item j is expert j's rpc down records,
// one bulk copy into a buffer of its own.  The producer requests those k copies right after the
// first gate/up items (the down weights do not depend on h), then streams the rest of the gate/up
// items through the ring, so the whole call's weights are in flight from the start.  The
// consumers form h = silu(gate) * up for their gate/up items, publish it, meet every other block
// at a grid-wide arrival counter (bounded wait), and then take the down items with the k experts'
// h.  The counter never resets: each launch adds one arrival per block, and a block waits for the
// multiple of gridDim.x that completes its launch.
//
// Missed experts' bytes, by the whole warp: host_pull issues `bytes` (a multiple of 16) from the
// pinned pack into shared memory as 16-byte cp.async pieces (every piece in flight at once; the
// caller commits and waits); once they have landed, slot_write_through makes the warp's
// writes visible to the async proxy and lane 0 writes the buffer through to the expert's HBM
// slot with one bulk copy (completion awaited before the buffer is refilled and before the
// block exits).
__device__ __forceinline__ void host_pull(unsigned char* dst, const uint8_t* pack, uint32_t bytes, int lane) {
  const int n = (int)(bytes / 16);
  for (int i = lane; i < n; i += 32)
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst + (size_t)i * 16)),
                 "l"(pack + (size_t)i * 16)
                 : "memory");
}
__device__ __forceinline__ void slot_write_through(unsigned char* src, uint8_t* slot, uint32_t bytes, int lane) {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // before the bulk copy reads them
  __syncwarp();
  if (lane == 0) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(slot), "r"(smem_u32(src)),
                 "r"(bytes)
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
  }
}
// lane 0: the stage-to-slot copies issued so far have read their source (the stage may be refilled)
__device__ __forceinline__ void slot_writes_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// ... and have completed
__device__ __forceinline__ void slot_writes_done() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

struct FusedCfg {
  PipeCfg g;
  int rpc;               // down: output rows per block (a contiguous range)
  uint32_t dn_bytes;     // down item: one expert's rpc down records (one bulk copy, own buffer)
  int n_hvec;            // h vectors of the k experts, split into int8 pieces
  int NS;                // gate/up ring stages
  uint32_t stage_bytes;  // gate/up item
  int red_floats;        // partial results: gate/up items x 16 warps, then k x rpc down rows
  uint32_t vq_bytes;
  // shared memory: [NS gate/up stages | k down buffers | full | empty | full_d | red | vq]
  size_t off_dn, off_bar, off_red, off_vq, total;
};
constexpr int kFusedBars = 2 * kMaxStages + kMaxTopK;

// The arrival is a release (the block's h, written before it and published to this thread by the
// block barrier, becomes visible with it); the polling loads acquire.  Bounded in time.
__device__ __forceinline__ bool grid_arrive_wait(unsigned long long* arrive, unsigned* err, uint64_t limit_ns) {
  unsigned long long old;
  asm volatile("atom.add.release.gpu.global.u64 %0, [%1], 1;" : "=l"(old) : "l"(arrive) : "memory");
  const unsigned long long target = (old / gridDim.x + 1) * gridDim.x;
  if (counter_wait(arrive, target, limit_ns)) return true;
  atomicExch(err, 5u);
  return false;
}

template <int QT, int VPL, int VPLD>
__global__ void __launch_bounds__(kThreadsF, 1)
    k_ffn_pipe(Dev d, int layer, const float* __restrict__ x, float* __restrict__ y, FusedCfg f) {
  constexpr int kW = Vec<QT>::kW;
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ uint8_t* s_gu[kMaxTopK];  // each expert's HBM slot: gate/up region, down region
  __shared__ uint8_t* s_dn[kMaxTopK];
  __shared__ const uint8_t* s_hgu[kMaxTopK];  // its payload in host memory (missed experts)
  __shared__ float s_g[kMaxTopK];
  __shared__ int s_miss[kMaxTopK];
  __shared__ int s_gord[kMaxItemsF];  // the block's gate/up items: resident experts' first
  __shared__ const uint8_t* s_gsrc[kMaxItemsF];  // ... their HBM records (resident items)
  __shared__ int s_nres, s_nb;        // how many of them are resident; ring B's stages
  __shared__ int s_xmax, s_xexp;      // exponent of x's largest magnitude (split scale)
  __shared__ int s_hmax[kMaxTopK], s_hexp[kMaxTopK];  // the same for each expert's h
  const PipeCfg& cg = f.g;
  Smem sm;
  sm.stage0 = smem;
  sm.full = reinterpret_cast<uint64_t*>(smem + f.off_bar);
  sm.empty = sm.full + kMaxStages;
  uint64_t* full_d = sm.empty + kMaxStages;  // [kMaxTopK] down buffers, one use each
  unsigned char* dbuf = smem + f.off_dn;
  sm.red = reinterpret_cast<float*>(smem + f.off_red);
  sm.vq = smem + f.off_vq;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = d.k;
  const int mine_g = items_of_block(cg.n_items);
  const int r0 = (int)blockIdx.x * f.rpc, nrows = max(0, min(d.H - r0, f.rpc));  // this block's down rows
  const int mine_d = nrows > 0 ? k : 0;
  // prologue: this block's shared memory only (with a programmatic launch it overlaps the router)
  if (threadIdx.x == 0) {
    for (int s = 0; s < f.NS; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kConsumers);
    }
    for (int j = 0; j < k; ++j) mbar_init(&full_d[j], 1);
    mbar_fence_init();
    s_xmax = kNoExp;
  }
  if (threadIdx.x < kMaxTopK) s_hmax[threadIdx.x] = kNoExp;
  pdl_wait();  // the router's outputs (and the caller's x) are complete and visible
  // x split by kG = kW / 4 threads per group (consecutive lanes), each one word of four values,
  // where x has at most 512 words (H <= 2048); consumer thread t's word is requested while the
  // block sets up.  Larger x: one group per thread (split_vectors).
  constexpr int kG = kW / 4;
  const bool x_words = cg.n_vec * kG <= kConsumers * 32;
  const bool x_mine = x_words && warp < kConsumers && (int)threadIdx.x < cg.n_vec * kG;
  float4 xv = make_float4(0.f, 0.f, 0.f, 0.f);
  if (x_mine) xv = __ldg(reinterpret_cast<const float4*>(x) + threadIdx.x);
  if (threadIdx.x < k) {  // one token: access u = rank j
    uint8_t* slot = d.pool + ((size_t)layer * d.S_alloc + d.uslot[threadIdx.x]) * d.lay.stride;
    s_gu[threadIdx.x] = slot;
    s_dn[threadIdx.x] = slot + d.lay.d_off;
    s_hgu[threadIdx.x] = d.fstage ? d.fstage + (size_t)threadIdx.x * d.fstride  // staged from the file
                                  : d.pack + ((size_t)layer * d.E + d.uniq[threadIdx.x]) * d.lay.stride;
    s_g[threadIdx.x] = d.g[threadIdx.x];
    s_miss[threadIdx.x] = d.umiss[threadIdx.x];
  }
  __syncthreads();
  if (warp == 0) {
    // list position p = blockIdx.x + t * gridDim.x (lane t); the list holds the resident experts'
    // items, then the missed experts' (ranks in order within each); item id = rank * (I / R) + row
    // block.  Position q of the expert list: the q-th resident rank, or the (q - n_res)-th missed one.
    const int nrb = d.I / cg.R;
    const unsigned kmask = (1u << k) - 1u;
    const unsigned res = __ballot_sync(0xffffffffu, lane < k && !s_miss[lane]);
    const int n_res_e = __popc(res);
    for (int t = lane; t < mine_g; t += 32) {
      const int p = (int)blockIdx.x + t * (int)gridDim.x, q = p / nrb;
      unsigned m = q < n_res_e ? res : (~res & kmask);
      for (int c = q < n_res_e ? q : q - n_res_e; c > 0; --c) m &= m - 1u;  // drop the c lowest ranks
      const int u = __ffs(m) - 1, rb = p % nrb;
      s_gord[t] = u * nrb + rb;
      s_gsrc[t] = s_gu[u] + (size_t)rb * cg.R * d.lay.rs_gu;
    }
    if (lane == 0) {
      const int lim = n_res_e * nrb - (int)blockIdx.x;  // items t with p < n_res_e * nrb
      s_nres = lim <= 0 ? 0 : min(mine_g, (lim + (int)gridDim.x - 1) / (int)gridDim.x);
      s_nb = n_res_e < k ? 2 : 0;  // ring B only when the call has a missed expert (NS >= 4)
    }
  }
  __syncthreads();

  const int nres = s_nres, NB = s_nb, NA = f.NS - NB;  // ring A: stages [0, NA); ring B: [NA, NS)
  if (warp == kConsumers) {
    // ---- producer warp: lane 0 streams the resident experts' items and down records (none while
    // the context's test hold is set)
    Ring ring;
    int it = 0;
    bool ok = true;
    const int R = cg.R, nrb = d.I / R;
    const uint32_t bytes = cg.stage_bytes, rs = d.lay.rs_gu;
    const uint32_t dbytes = (uint32_t)nrows * d.lay.rs_d;
    const size_t doff = (size_t)r0 * d.lay.rs_d;
    const int n_issue = d.hold ? 0 : nres;
    // the resident experts' down records go after the first two gate/up items
    const int first = min(n_issue, min(2, NA));
    const uint64_t pol = l2_evict_first();  // read once per call: keep L2 for what is reused
    bool d_issued = false;
    auto issue_down_hits = [&]() {
      if (lane == 0)
        for (int j = 0; j < mine_d; ++j)
          if (!s_miss[j]) {
            mbar_arrive_tx(&full_d[j], dbytes);
            bulk_g2s_hint(dbuf + (size_t)j * f.dn_bytes, s_dn[j] + doff, dbytes, &full_d[j], pol);
          }
      d_issued = true;
    };
    if (lane == 0) {
      for (int t = 0; t < n_issue; ++t, ++it) {
        if (t == first) issue_down_hits();
        if (it >= NA && !(ok = mbar_wait(&sm.empty[ring.s], ring.phase ^ 1u, d.wait_ns))) break;
        uint64_t* bar = &sm.full[ring.s];
        mbar_arrive_tx(bar, bytes);
        bulk_g2s_hint(sm.stage0 + (size_t)ring.s * f.stage_bytes, s_gsrc[t], bytes, bar, pol);
        ring.next(NA);
      }
      if (ok && !d_issued && !d.hold) issue_down_hits();
      if (!ok) atomicExch(d.err, 1u);
      // no copy may be in flight when the block exits: wait for the last use of every stage
      for (int s = 0; s < NA && s < it; ++s) {
        const int uses = (it - 1 - s) / NA + 1;
        if (!mbar_wait(&sm.full[s], (uint32_t)(uses - 1) & 1u, d.wait_ns)) atomicExch(d.err, 2u);
      }
      if (d_issued)
        for (int j = 0; j < mine_d; ++j)
          if (!s_miss[j] && !mbar_wait(&full_d[j], 0, d.wait_ns)) atomicExch(d.err, 2u);
    }
  } else if (warp == kConsumers + 1) {
    // ---- link warp: the missed experts' items through ring B (both stages in flight at once),
    // then all their down records at once (after the items: the grid barrier and the h split
    // overlap that transfer)
    bool ok = true;
    const int R = cg.R, nrb = d.I / R, n_li = mine_g - nres;
    const uint32_t bytes = cg.stage_bytes, rs = d.lay.rs_gu;
    const uint32_t dbytes = (uint32_t)nrows * d.lay.rs_d;
    const size_t doff = (size_t)r0 * d.lay.rs_d;
    auto issue_item = [&](int t, int s) {  // the block's link item t into ring B stage s: one group
      const int item = s_gord[nres + t], u = item / nrb, rb = item % nrb;
      const size_t off = (size_t)rb * R * rs;
      host_pull(sm.stage0 + (size_t)(NA + s) * f.stage_bytes, s_hgu[u] + off, bytes, lane);
      asm volatile("cp.async.commit_group;" ::: "memory");
    };
    int issued = 0;
    for (; issued < n_li && issued < NB; ++issued) issue_item(issued, issued);
    for (int t = 0; t < n_li; ++t) {
      const int s = t % NB;
      if (issued > t + 1)  // item t's group is complete once at most the later one is pending
        asm volatile("cp.async.wait_group 1;" ::: "memory");
      else
        asm volatile("cp.async.wait_group 0;" ::: "memory");
      const int item = s_gord[nres + t], u = item / nrb, rb = item % nrb;
      slot_write_through(sm.stage0 + (size_t)(NA + s) * f.stage_bytes, s_gu[u] + (size_t)rb * R * rs, bytes, lane);
      if (lane == 0) mbar_arrive(&sm.full[NA + s]);  // release: every lane's stage writes
      if (issued < n_li) {  // refill the stage once the consumers are done with item t
        int w = 1;
        if (lane == 0) {
          w = mbar_wait(&sm.empty[NA + s], (uint32_t)(t / NB) & 1u, d.wait_ns);
          slot_writes_read();  // and its write-through has read it
        }
        if (!__shfl_sync(0xffffffffu, w, 0)) {
          ok = false;
          break;
        }
        issue_item(issued, s);
        ++issued;
      }
    }
    if (!ok) asm volatile("cp.async.wait_all;" ::: "memory");  // nothing of ours in flight at exit
    if (ok) {
      bool any = false;
      for (int j = 0; j < mine_d; ++j)
        if (s_miss[j]) {
          host_pull(dbuf + (size_t)j * f.dn_bytes, s_hgu[j] + d.lay.d_off + doff, dbytes, lane);
          any = true;
        }
      if (any) {
        asm volatile("cp.async.wait_all;" ::: "memory");
        for (int j = 0; j < mine_d; ++j)
          if (s_miss[j]) {
            slot_write_through(dbuf + (size_t)j * f.dn_bytes, s_dn[j] + doff, dbytes, lane);
            if (lane == 0) mbar_arrive(&full_d[j]);
          }
      }
    }
    if (lane == 0) {
      if (!ok) atomicExch(d.err, 1u);
      slot_writes_done();  // every write-through complete before the block exits
    }
  } else {
    Ring ring, ring_b;
    bool ok = true;
    // ---- gate/up: warp w: tensor w / (R*cs), row (w / cs) % R, column range w % cs
    {
      const int R = cg.R, cs = cg.cs, nrb = d.I / R;
      const uint32_t rs = d.lay.rs_gu;
      const int ten = warp / (R * cs), row = (warp / cs) % R, col = warp % cs;
      const int nv = (d.lay.qrow_gu / 16) / cs;
      const int v0 = col * nv;
      const XQ<QT>* xq = reinterpret_cast<const XQ<QT>*>(sm.vq);
      if (x_words) {  // x split into int8 pieces, scaled by the power of two of its largest magnitude:
                      // the same pieces as quant_vals of the whole group (the group's largest
                      // magnitude m by shuffles, each value scaled by 2^-e_g and split by
                      // 127 / (m 2^-e_g), the piece sums added over the kG threads), then the
                      // vector's exponent and rescale_group as in split_vectors
        XQ<QT>* dst = reinterpret_cast<XQ<QT>*>(sm.vq);
        const int gi = threadIdx.x / kG, part = threadIdx.x % kG;
        float m = fmaxf(fmaxf(fabsf(xv.x), fabsf(xv.y)), fmaxf(fabsf(xv.z), fabsf(xv.w)));
#pragma unroll
        for (int o = 1; o < kG; o <<= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        const int eg = group_exponent(m), ne = eg == kNoExp ? 0 : -eg;
        const float sa = pow2i(ne / 2), sb = pow2i(ne - ne / 2);
        const float ms = m * sa * sb;  // exact: the largest value scaled by a power of two
        const float inv = ms > 0x1p-100f ? 127.f / ms : 0.f;
        const float vv[4] = {xv.x * sa * sb, xv.y * sa * sb, xv.z * sa * sb, xv.w * sa * sb};
        uint32_t b1 = 0, b2 = 0, b3 = 0;
        int s1 = 0, s2 = 0, s3 = 0;
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
          const float t = vv[jj] * inv;
          const int a = __float2int_rn(t);
          const float e = (t - (float)a) * 127.f;
          const int b = __float2int_rn(e);
          const int c = __float2int_rn((e - (float)b) * 127.f);
          s1 += a;
          s2 += b;
          s3 += c;
          b1 |= (uint32_t)(a & 0xFF) << (8 * jj);
          b2 |= (uint32_t)(b & 0xFF) << (8 * jj);
          b3 |= (uint32_t)(c & 0xFF) << (8 * jj);
        }
#pragma unroll
        for (int o = 1; o < kG; o <<= 1) {
          s1 += __shfl_xor_sync(0xffffffffu, s1, o);
          s2 += __shfl_xor_sync(0xffffffffu, s2, o);
          s3 += __shfl_xor_sync(0xffffffffu, s3, o);
        }
        if (x_mine) {
          dst[gi].p1[part] = b1;
          dst[gi].p2[part] = b2;
          dst[gi].p3[part] = b3;
          if (part == 0) {
            constexpr int off = QT == kQ8 ? 128 : 8;
            dst[gi].k12 = off * (s1 * 127 + s2);
            dst[gi].k3 = off * s3;
            dst[gi].sf = inv > 0.f ? ms / 127.f / 16129.f : 0.f;
            atomicMax(&s_xmax, eg);
          }
        }
        named_bar_sync(1, kConsumers * 32);
        if (x_mine && part == 0) rescale_group<QT>(dst[gi], eg, vector_exponent(s_xmax));
        if (threadIdx.x == 0) s_xexp = vector_exponent(s_xmax);
        named_bar_sync(1, kConsumers * 32);
      } else {
        split_vectors<QT>(x, cg.n_vec, cg.n_vec, reinterpret_cast<XQ<QT>*>(sm.vq), &s_xmax, &s_xexp);
      }
      XQ<QT> xr[VPL];
#pragma unroll
      for (int i = 0; i < VPL; ++i) {
        const int v = lane + 32 * i;
        if (v < nv) xr[i] = xq[v0 + v];
      }
      for (int it = 0; it < mine_g; ++it) {
        const bool link = it >= nres;  // a missed expert's item: ring B
        const int bi = link ? NA + ring_b.s : ring.s;
        if (!(ok = mbar_wait(&sm.full[bi], link ? ring_b.phase : ring.phase, d.wait_ns))) break;
        const unsigned char* rec = sm.stage0 + (size_t)bi * f.stage_bytes + row * rs;
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
        if (lane == 0) mbar_arrive(&sm.empty[bi]);
        if (link)
          ring_b.next(NB);
        else
          ring.next(NA);
      }
      // SwiGLU of the block's items (column ranges added in order, times 2^ex: x was split
      // scaled by 2^-ex)
      named_bar_sync(1, kConsumers * 32);
      const int ex = s_xexp;
      for (int t = threadIdx.x; t < mine_g * R; t += kConsumers * 32) {
        const int it = t / R, r = t % R;
        const float* p = sm.red + it * kConsumers;
        float ag = 0.f, au = 0.f;
        for (int cc = 0; cc < cs; ++cc) {
          ag += p[(0 * R + r) * cs + cc];
          au += p[(1 * R + r) * cs + cc];
        }
        ag = scale2(ag, ex);
        au = scale2(au, ex);
        const int item = s_gord[it];
        d.h[(size_t)(item / nrb) * d.I + (item % nrb) * R + r] = ag / (1.0f + expf(-ag)) * au;
      }
      named_bar_sync(1, kConsumers * 32);  // the block's h written
    }
    if (!ok && lane == 0) atomicExch(d.err, 3u);
    // ---- every block's h published (one arrival per block, always, so launches stay aligned)
    if (threadIdx.x == 0 && !grid_arrive_wait(d.work, d.err, d.wait_ns)) ok = false;
    named_bar_sync(1, kConsumers * 32);
    // ---- down: warp w holds expert j = w / (16 / k)'s h in registers for the whole phase and
    // takes rows sub, sub + 16 / k, ... of that expert's item (sub = w % (16 / k))
    {
      const int nvec = d.lay.qrow_d / 16;
      const uint32_t rs = d.lay.rs_d;
      const XQ<QT>* hq = reinterpret_cast<const XQ<QT>*>(sm.vq);
      split_vectors<QT, true>(d.h, f.n_hvec, nvec, reinterpret_cast<XQ<QT>*>(sm.vq), s_hmax, s_hexp);  // other blocks wrote h
      float* red = sm.red + cg.max_mine * kConsumers;  // [k][rpc]
      const int wpe = kConsumers / k, j = warp / wpe, sub = warp % wpe;
      if (QT == kQ8 && j < mine_d && ok && nvec > 32 && nvec <= 48) {
        // rows of at most 48 vectors: half-warp h (lanes 16 h ..) takes row 2 p + h of the warp's
        // row pairs p = sub, sub + wpe, ..., each lane three vectors: no idle lanes, a 16-lane sum
        const int hl = lane & 15, half = lane >> 4;
        XQ<QT> hr3[3];
#pragma unroll
        for (int i = 0; i < 3; ++i) {
          const int v = hl + 16 * i;
          if (v < nvec) hr3[i] = hq[j * nvec + v];
        }
        const int e = s_hexp[j];
        if ((ok = mbar_wait(&full_d[j], 0, d.wait_ns))) {
          const unsigned char* st = dbuf + (size_t)j * f.dn_bytes;
          for (int p0 = sub; 2 * p0 < nrows; p0 += 2 * wpe) {  // two row pairs at a time
            float acc[2];
#pragma unroll
            for (int pp = 0; pp < 2; ++pp) {
              const int row = 2 * (p0 + pp * wpe) + half;
              acc[pp] = 0.f;
              if (row < nrows) {
                const unsigned char* q = st + (size_t)row * rs;
                const __half* sc = reinterpret_cast<const __half*>(q + d.lay.o_ds);
#pragma unroll
                for (int i = 0; i < 3; ++i) {
                  const int v = hl + 16 * i;
                  if (v < nvec)
                    acc[pp] = fmaf(dot_q<QT>(*reinterpret_cast<const uint4*>(q + 16 * v), hr3[i]),
                                   __half2float(sc[scale_index<QT>(v)]), acc[pp]);
                }
              }
            }
#pragma unroll
            for (int o = 8; o > 0; o >>= 1)
#pragma unroll
              for (int pp = 0; pp < 2; ++pp) acc[pp] += __shfl_xor_sync(0xffffffffu, acc[pp], o);
            if (hl == 0)
#pragma unroll
              for (int pp = 0; pp < 2; ++pp) {
                const int row = 2 * (p0 + pp * wpe) + half;
                if (row < nrows) red[j * f.rpc + row] = scale2(acc[pp], e);
              }
          }
        }
      } else if (j < mine_d && ok) {
        XQ<QT> hr[VPLD];
#pragma unroll
        for (int i = 0; i < VPLD; ++i) {
          const int v = lane + 32 * i;
          if (v < nvec) hr[i] = hq[j * nvec + v];
        }
        const int e = s_hexp[j];
        if ((ok = mbar_wait(&full_d[j], 0, d.wait_ns))) {
          const unsigned char* st = dbuf + (size_t)j * f.dn_bytes;
          // four rows at a time: independent dot products and interleaved reductions
          for (int row0 = sub; row0 < nrows; row0 += 4 * wpe) {
            float acc[4];
#pragma unroll
            for (int rr = 0; rr < 4; ++rr) {
              const int row = row0 + rr * wpe;
              acc[rr] = 0.f;
              if (row < nrows) {
                const unsigned char* q = st + (size_t)row * rs;
                const __half* sc = reinterpret_cast<const __half*>(q + d.lay.o_ds);
#pragma unroll
                for (int i = 0; i < VPLD; ++i) {
                  const int v = lane + 32 * i;
                  if (v < nvec)
                    acc[rr] = fmaf(dot_q<QT>(*reinterpret_cast<const uint4*>(q + 16 * v), hr[i]),
                                   __half2float(sc[scale_index<QT>(v)]), acc[rr]);
                }
              }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1)
#pragma unroll
              for (int rr = 0; rr < 4; ++rr) acc[rr] += __shfl_xor_sync(0xffffffffu, acc[rr], o);
            if (lane == 0)
#pragma unroll
              for (int rr = 0; rr < 4; ++rr)
                if (row0 + rr * wpe < nrows) red[j * f.rpc + row0 + rr * wpe] = scale2(acc[rr], e);
          }
        }
      }
      if (!ok && lane == 0) atomicExch(d.err, 3u);
      named_bar_sync(1, kConsumers * 32);
      // combine the k experts of each row in rank order
      for (int row = threadIdx.x; row < nrows; row += kConsumers * 32) {
        float acc = 0.f;
        for (int jj = 0; jj < k; ++jj) acc = fmaf(s_g[jj], red[jj * f.rpc + row], acc);
        y[r0 + row] = acc;
      }
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

FusedCfg fused_cfg(const Dev& d) {
  FusedCfg f;
  f.g = gateup_cfg(d);
  f.rpc = (d.H + sm_count() - 1) / sm_count();
  f.dn_bytes = (uint32_t)f.rpc * d.lay.rs_d;
  f.n_hvec = d.k * (d.lay.qrow_d / 16);
  const uint32_t hv_bytes = (uint32_t)(f.n_hvec * (d.qtype == MF_Q8_0 ? sizeof(XQ<kQ8>) : sizeof(XQ<kQ4>)));
  f.stage_bytes = f.g.stage_bytes;
  f.red_floats = f.g.max_mine * kConsumers + d.k * f.rpc;
  f.vq_bytes = f.g.vq_bytes > hv_bytes ? f.g.vq_bytes : hv_bytes;
  const size_t fixed = (size_t)d.k * f.dn_bytes + kFusedBars * sizeof(uint64_t) +
                       (size_t)f.red_floats * sizeof(float) + f.vq_bytes;
  const size_t budget = kFusedSmem - 1024;  // - the kernel's static shared memory
  const size_t ns = fixed < budget ? (budget - fixed) / f.stage_bytes : 0;
  f.NS = (int)(ns > (size_t)kMaxStages ? kMaxStages : ns);
  f.off_dn = (size_t)f.NS * f.stage_bytes;
  f.off_bar = f.off_dn + (size_t)d.k * f.dn_bytes;
  f.off_red = f.off_bar + kFusedBars * sizeof(uint64_t);
  f.off_vq = f.off_red + (((size_t)f.red_floats * sizeof(float) + 15) & ~(size_t)15);
  f.total = f.off_vq + f.vq_bytes;
  return f;
}

size_t fused_smem(const FusedCfg& f) { return f.total; }

// One block per SM.  The launch is programmatic (it may begin while the router finishes: the
// kernel's prologue touches only shared memory and it waits for the router before reading
// anything else); where the driver refuses that, a cooperative launch.  Blocks wait for each
// other only through bounded waits.
template <class Kern>
cudaError_t launch_ffn(Kern kern, size_t smem, cudaStream_t s, const Dev& d, int layer, const float* x, float* y,
                       const FusedCfg& f) {
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(sm_count());
  cfg.blockDim = dim3(kThreadsF);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  static bool pdl_ok = true;
  if (pdl_ok) {
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    e = cudaLaunchKernelEx(&cfg, kern, d, layer, x, y, f);
    if (e == cudaSuccess) return e;
    cudaGetLastError();
    pdl_ok = false;
  }
  attr[0].id = cudaLaunchAttributeCooperative;  // every block resident: they wait for each other
  attr[0].val.cooperative = 1;
  return cudaLaunchKernelEx(&cfg, kern, d, layer, x, y, f);
}

template <int QT>
cudaError_t ffn_pipe_q(const Dev& d, int layer, const float* x, float* y, cudaStream_t s) {
  const FusedCfg f = fused_cfg(d);
  const size_t smem = fused_smem(f);
  const int vx = vpl_for((d.lay.qrow_gu / 16) / f.g.cs), vh = vpl_for(d.lay.qrow_d / 16);
#define MF_FF(A, B) \
  if (vx == A && vh == B) return launch_ffn(k_ffn_pipe<QT, A, B>, smem, s, d, layer, x, y, f);
  MF_FF(1, 1) MF_FF(1, 2) MF_FF(2, 1) MF_FF(2, 2)
  if constexpr (QT == kQ8) {  // Q4_0 takes at most two vectors per lane (decode_pipe_ok)
    MF_FF(1, 3) MF_FF(2, 3) MF_FF(3, 1) MF_FF(3, 2) MF_FF(3, 3) MF_FF(4, 1) MF_FF(4, 2) MF_FF(4, 3)
  }
#undef MF_FF
  return cudaErrorInvalidConfiguration;
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

bool ffn_fused_ok(const Dev& d) {
  const FusedCfg f = fused_cfg(d);
  return decode_pipe_ok(d) && f.NS >= 4 && f.g.max_mine <= kMaxItemsF;
}

cudaError_t launch_ffn_single(const Dev& d, int layer, const float* x, float* y, cudaStream_t s) {
  return d.qtype == MF_Q8_0 ? ffn_pipe_q<kQ8>(d, layer, x, y, s) : ffn_pipe_q<kQ4>(d, layer, x, y, s);
}

}  // namespace mf
