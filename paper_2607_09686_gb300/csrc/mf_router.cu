// Router: logits z = W_r x (+ bias), top-k by (z desc, id asc), softmax over the chosen.
//
// MoE routing selects a subset of experts per token (Background section of the paper).
// Logits are computed with a compensated dot product (Ogita, Rump & Oishi, "Accurate sum and
// dot product", SIAM J. Sci. Comput. 2005, algorithm Dot2): every product is split exactly
// into value + error with an FMA, the running sum is kept as an unevaluated pair, and the pair
// is rounded to fp32 once.  The result is the fp32 rounding of the exact dot product except
// where the exact value lies within ~n*2^-48 relative of a rounding boundary, so selection does
// not depend on the summation order.
//
// One thread-block cluster of 16 blocks per token (8 where the GPU does not schedule clusters of
// 16): block r computes the logits of experts [r*ceil(E/nc), (r+1)*ceil(E/nc)), with
// 16 / ceil(E/nc) warps per expert
// when the block has fewer experts than warps (each warp a lane-interleaved share of the row,
// its loads issued together; the warps' compensated pairs are then added with the same
// error-free steps), and stores them straight into block 0's shared memory.  After
// a cluster barrier, block 0 gathers all logits through distributed shared memory, ranks each
// expert by counting the experts ahead of it, and keeps the k first.  With one token per call,
// block 0 then runs the layer's slot resolve (lru_warp) on cache state it prefetched into
// registers while the logits were being computed.  No global atomics or fences on the path.
//
// Calls with many tokens (T >= kTiledMinT) compute the logits as a tiled product instead, so
// that W_r is read once per 32 tokens rather than once per token: see k_logits_tiled.
#include <cooperative_groups.h>

#include "mf_lru.cuh"

namespace cg = cooperative_groups;

namespace mf {
namespace {

constexpr int kThreadsR = 512;
constexpr int kWarpsR = kThreadsR / 32;
constexpr int kChunk = 8;  // float4 loads of W (and of x) a lane issues before using them
constexpr int kPre = kMaxExperts / kThreadsR;  // prefetched cache-state entries per thread

struct F2 {
  float hi, lo;
};

__device__ __forceinline__ F2 two_sum(float a, float b) {
  float s = __fadd_rn(a, b);
  float bb = __fsub_rn(s, a);
  float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return {s, e};
}

// (s, c) += a * b, error-free product split plus compensated running sum
__device__ __forceinline__ void dot2(float& s, float& c, float a, float b) {
  float p = __fmul_rn(a, b);
  float pe = __fmaf_rn(a, b, -p);
  F2 t = two_sum(s, p);
  s = t.hi;
  c = __fadd_rn(c, __fadd_rn(t.lo, pe));
}

// (s, c) += (s2, c2) for compensated pairs
__device__ __forceinline__ void pair_add(float& s, float& c, float s2, float c2) {
  const F2 t = two_sum(s, s2);
  s = t.hi;
  c = __fadd_rn(__fadd_rn(c, c2), t.lo);
}

// The first chunk of logit_part's W loads, issued before x is in shared memory.
__device__ __forceinline__ void w_preload(const float* __restrict__ w, int n4, int first, int step, float4* a) {
  const float4* w4 = reinterpret_cast<const float4*>(w);
  const uint64_t pol = l2_evict_last();  // W_r is read again by the layer's next call
#pragma unroll
  for (int u = 0; u < kChunk; ++u) {
    const int q = first + u * step;
    if (q < n4) a[u] = ld_hint(w4 + q, pol);
  }
}

// Compensated partial dot product of one expert row with x (in shared memory) over the float4
// indices q = first, first + step, ... (< H / 4), summed over the warp; returns the pair in (s, c).
// `pre` holds the first chunk's W values (w_preload).
__device__ __forceinline__ void logit_part(const float* __restrict__ w, const float* xs, int n4, int first, int step,
                                           const float4* pre, float& s, float& c) {
  s = 0.f;
  c = 0.f;
  const float4* w4 = reinterpret_cast<const float4*>(w);
  const float4* x4 = reinterpret_cast<const float4*>(xs);
  for (int q0 = first; q0 < n4; q0 += kChunk * step) {
    float4 a[kChunk], b[kChunk];
#pragma unroll
    for (int u = 0; u < kChunk; ++u) {  // all loads of the chunk first
      const int q = q0 + u * step;
      if (q < n4) {
        a[u] = q0 == first ? pre[u] : ld_hint(w4 + q, l2_evict_last());
        b[u] = x4[q];
      }
    }
#pragma unroll
    for (int u = 0; u < kChunk; ++u) {
      if (q0 + u * step < n4) {
        dot2(s, c, a[u].x, b[u].x);
        dot2(s, c, a[u].y, b[u].y);
        dot2(s, c, a[u].z, b[u].z);
        dot2(s, c, a[u].w, b[u].w);
      }
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float so = __shfl_xor_sync(0xffffffffu, s, off);
    const float co = __shfl_xor_sync(0xffffffffu, c, off);
    pair_add(s, c, so, co);
  }
}

__device__ __forceinline__ bool cluster_rank_zero() {
  uint32_t r;
  asm("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r == 0;
}

__global__ void __launch_bounds__(kThreadsR)
    k_router(Dev d, const float* __restrict__ x, const float* __restrict__ wr, const float* __restrict__ bias, int T,
             int layer, int fuse_resolve, float* __restrict__ x_copy, int nc) {
  extern __shared__ __align__(16) float s_x[];  // the token's x, read once per block
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int t = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int H = d.H, E = d.E, k = d.k, S = d.S_active;
  const int epc = (E + nc - 1) / nc;
  // this warp's first expert and its first W chunk, requested before x is staged
  const int e0 = rank * epc, e1 = min(E, e0 + epc);
  const int wpe = epc >= kWarpsR ? 1 : kWarpsR / epc;  // warps per expert
  const int ew = kWarpsR / wpe;                         // experts per pass
  const int part = warp % wpe, n4 = H / 4;
  // a programmatic launch may begin during the previous kernel: nothing above touched global memory
  pdl_wait();
  float4 pre[kChunk];
  if (e0 + warp / wpe < e1 && warp / wpe < ew) w_preload(wr + (size_t)(e0 + warp / wpe) * H, n4, part * 32 + lane, wpe * 32, pre);
  {  // x may be pinned host memory read over the CPU-GPU link: once per block
    const float4* x4 = reinterpret_cast<const float4*>(x + (size_t)t * H);
    float4* sx4 = reinterpret_cast<float4*>(s_x);
    for (int i = threadIdx.x; i < H / 4; i += kThreadsR) {
      const float4 v = x4[i];
      sx4[i] = v;
      if (x_copy && cluster_rank_zero()) reinterpret_cast<float4*>(x_copy + (size_t)t * H)[i] = v;  // for the FFN
    }
  }
  __syncthreads();

  __shared__ __align__(16) float s_z[kMaxExperts];  // block 0: every logit (the blocks store theirs)
  __shared__ float s_ps[kWarpsR], s_pc[kWarpsR];  // each warp's compensated partial
  __shared__ int s_sel[kMaxTopK];
  __shared__ float s_zsel[kMaxTopK];
  __shared__ int s_slot_of[kMaxExperts];
  __shared__ int s_expert_of[kMaxExperts];
  __shared__ uint64_t s_lastuse[kMaxExperts];
  __shared__ int s_uslot[kMaxTopK];

  // block 0 of a one-token call: start loading the layer's cache state now (used after the logits)
  const bool resolve = fuse_resolve && rank == 0;
  int pre_slot[kPre], pre_exp[kPre];
  uint64_t pre_last[kPre], clock0 = 0;
  if (resolve) {
    const int32_t* g_slot_of = d.slot_of + (size_t)layer * E;
    const int32_t* g_expert_of = d.expert_of + (size_t)layer * d.S_alloc;
    const uint64_t* g_last = d.last_use + (size_t)layer * d.S_alloc;
#pragma unroll
    for (int i = 0; i < kPre; ++i) {
      const int e = tid + i * kThreadsR;
      pre_slot[i] = e < E ? g_slot_of[e] : -1;
      pre_exp[i] = e < S ? g_expert_of[e] : -1;
      pre_last[i] = e < S ? g_last[e] : 0;
    }
    if (tid == 0) clock0 = d.clock[layer];
  }

  float* z0 = rank == 0 ? s_z : cluster.map_shared_rank(s_z, 0);  // block 0's logits
  for (int eb = e0; eb < e1; eb += ew) {  // block-uniform passes
    const int e = eb + warp / wpe;
    float ps = 0.f, pc = 0.f;
    if (e < e1 && warp / wpe < ew) {
      if (eb != e0) w_preload(wr + (size_t)e * H, n4, part * 32 + lane, wpe * 32, pre);
      logit_part(wr + (size_t)e * H, s_x, n4, part * 32 + lane, wpe * 32, pre, ps, pc);
    }
    if (lane == 0) {
      s_ps[warp] = ps;
      s_pc[warp] = pc;
    }
    __syncthreads();
    if (lane == 0 && part == 0 && e < e1 && warp / wpe < ew) {
      float zs = s_ps[warp], zc = s_pc[warp];
      for (int p = 1; p < wpe; ++p) pair_add(zs, zc, s_ps[warp + p], s_pc[warp + p]);
      float z = __fadd_rn(zs, zc);
      if (bias) z = __fadd_rn(z, bias[(size_t)t * E + e]);
      z0[e] = z;  // distributed shared memory store into block 0
    }
    __syncthreads();
  }
  if (resolve) {  // the prefetched cache state into shared memory (the loads have long landed)
#pragma unroll
    for (int i = 0; i < kPre; ++i) {
      const int e = tid + i * kThreadsR;
      if (e < E) s_slot_of[e] = pre_slot[i];
      if (e < S) {
        s_expert_of[e] = pre_exp[i];
        s_lastuse[e] = pre_last[i];
      }
    }
  }
  // the logits are stored: the expert FFN (a programmatic launch) may start its prologue
  pdl_trigger();
  // every block's logits stores, before block 0 reads them; the other blocks leave
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  if (rank != 0) return;
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");

  // rank by counting: position of expert e = experts with a larger logit, or equal and lower id
  // (s_sel starts as 0..k-1: a valid choice even where the logits are not ordered, e.g. NaN).
  // tpe consecutive lanes share an expert, each counting over every tpe-th other expert.
  if (tid < k) s_sel[tid] = tid;
  __syncthreads();
  {
    int tpe = 1;
    while (tpe < 32 && tpe * 2 * E <= kThreadsR) tpe *= 2;
    const int per_pass = kThreadsR / tpe, part = tid % tpe;
    for (int e0 = 0; e0 < E; e0 += per_pass) {  // block-uniform
      const int e = e0 + tid / tpe;
      const bool valid = e < E;
      const float z = valid ? s_z[e] : 0.f;
      int r = 0;
      if (valid)
        for (int e2 = part; e2 < E; e2 += tpe) {
          const float z2 = s_z[e2];
          r += (z2 > z) || (z2 == z && e2 < e);
        }
      for (int off = tpe >> 1; off > 0; off >>= 1) r += __shfl_xor_sync(0xffffffffu, r, off);
      if (valid && part == 0 && r < k) {
        s_sel[r] = e;
        s_zsel[r] = z;
      }
    }
  }
  __syncthreads();
  if (warp == 0) {  // softmax over the chosen: lane j < k holds exp(z_j - z_0); fixed shuffle-tree sum
    const float ex = lane < k ? expf(s_zsel[lane] - s_zsel[0]) : 0.f;
    float den = ex;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) den += __shfl_xor_sync(0xffffffffu, den, off);
    if (lane < k) {
      d.idx[(size_t)t * k + lane] = s_sel[lane];
      d.g[(size_t)t * k + lane] = ex / den;
    }
  }
  if (!resolve) return;

  // One token per call: the k chosen experts are distinct, so the accesses are the chosen
  // experts in rank order, all in one wave.
  if (tid == 0) d.info[2] = 0;
  __syncthreads();
  if (warp == 0) lru_warp(d, layer, k, s_sel, s_slot_of, s_expert_of, s_lastuse, s_uslot, __shfl_sync(0xffffffffu, clock0, 0));
  __syncthreads();
  if (tid < k) {  // one assignment per distinct expert: t = 0, j = u
    d.pos_slot[tid] = s_uslot[tid];
    d.asg[tid] = tid;
    d.asg_off[tid] = tid;
  }
  if (tid == 0) d.asg_off[k] = k;
  int32_t* g_slot_of = d.slot_of + (size_t)layer * E;
  int32_t* g_expert_of = d.expert_of + (size_t)layer * d.S_alloc;
  uint64_t* g_last = d.last_use + (size_t)layer * d.S_alloc;
  for (int e = tid; e < E; e += kThreadsR) g_slot_of[e] = s_slot_of[e];
  for (int q = tid; q < S; q += kThreadsR) {
    g_expert_of[q] = s_expert_of[q];
    g_last[q] = s_lastuse[q];
  }
}


// ---------------------------------------------------------------- many tokens per call
// k_logits_tiled: block (expert tile, token tile, K split) computes the compensated pairs of a
// 32-token x 64-expert tile over its range of H, from shared-memory tiles of x and W_r that
// cp.async fills 32 columns at a time (double-buffered).  Thread (ty, tx) owns tokens 2ty, 2ty+1
// and experts tx + 16j (j < 4).  Columns are taken two at a time with f32x2 arithmetic (the same
// IEEE operations as dot2, on two lanes): each output keeps one compensated pair for its even
// and one for its odd columns, added error-free at the end.  The pairs of every K split go to
// scratch; k_topk_tiled (one warp per token) adds them in split order, rounds once, adds the
// bias, ranks and takes the softmax exactly as the one-token path does.
constexpr int kTT = 32, kTE = 64, kHC = 32, kThreadsT = 256;
constexpr int kPadT = kHC + 4;  // shared row stride in floats: 16 rows read together hit 2 bank phases

__device__ __forceinline__ uint64_t f2_op_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t f2_op_sub(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t f2_op_mul(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t f2_op_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2_of(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ float2 f2_split(uint64_t a) {
  float lo, hi;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(a));
  return make_float2(lo, hi);
}

// dot2 on two lanes: (s, c) += a * b, product split exactly by an FMA, two-sum into s
__device__ __forceinline__ void dot2x2(uint64_t& s, uint64_t& c, uint64_t a, uint64_t b) {
  const uint64_t p = f2_op_mul(a, b);
  const uint64_t pe = f2_op_fma(a, b, p ^ 0x8000000080000000ull);  // a * b - p, exact
  const uint64_t s1 = f2_op_add(s, p);
  const uint64_t bb = f2_op_sub(s1, s);
  const uint64_t e = f2_op_add(f2_op_sub(s, f2_op_sub(s1, bb)), f2_op_sub(p, bb));
  s = s1;
  c = f2_op_add(c, f2_op_add(e, pe));
}

__device__ __forceinline__ void cp_async16_zfill(void* dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(valid ? 16 : 0)
               : "memory");
}

__global__ void __launch_bounds__(kThreadsT)
    k_logits_tiled(const float* __restrict__ x, const float* __restrict__ wr, int T, int E, int H, int cps,
                   float2* __restrict__ part) {
  __shared__ __align__(16) float s_x[2][kTT][kPadT];
  __shared__ __align__(16) float s_w[2][kTE][kPadT];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int e0 = (int)blockIdx.x * kTE, t0 = (int)blockIdx.y * kTT;
  const int c0 = (int)blockIdx.z * cps, c1 = min(H / kHC, c0 + cps);
  // one 16-byte piece of the x tile and two of the W tile per thread; rows past T or E read zeros
  auto load = [&](int ch, int buf) {
    {
      const int r = tid >> 3, q = tid & 7, t = t0 + r;
      cp_async16_zfill(&s_x[buf][r][4 * q], x + (size_t)min(t, T - 1) * H + ch * kHC + 4 * q, t < T);
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int id = tid + i * kThreadsT, r = id >> 3, q = id & 7, e = e0 + r;
      cp_async16_zfill(&s_w[buf][r][4 * q], wr + (size_t)min(e, E - 1) * H + ch * kHC + 4 * q, e < E);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  uint64_t S[2][4], C[2][4];  // [token][expert]: (even-column, odd-column) pairs
#pragma unroll
  for (int a = 0; a < 2; ++a)
#pragma unroll
    for (int j = 0; j < 4; ++j) S[a][j] = C[a][j] = 0;
  if (c0 < c1) load(c0, 0);
  for (int ch = c0; ch < c1; ++ch) {
    const int buf = (ch - c0) & 1;
    if (ch + 1 < c1) {
      load(ch + 1, buf ^ 1);  // that buffer was released by the barrier ending the previous chunk
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
#pragma unroll
    for (int k4 = 0; k4 < kHC; k4 += 4) {
      const float4 xa = *reinterpret_cast<const float4*>(&s_x[buf][2 * ty][k4]);
      const float4 xb = *reinterpret_cast<const float4*>(&s_x[buf][2 * ty + 1][k4]);
      const uint64_t xa01 = f2_of(xa.x, xa.y), xa23 = f2_of(xa.z, xa.w);
      const uint64_t xb01 = f2_of(xb.x, xb.y), xb23 = f2_of(xb.z, xb.w);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float4 w = *reinterpret_cast<const float4*>(&s_w[buf][tx + 16 * j][k4]);
        const uint64_t w01 = f2_of(w.x, w.y), w23 = f2_of(w.z, w.w);
        dot2x2(S[0][j], C[0][j], w01, xa01);
        dot2x2(S[0][j], C[0][j], w23, xa23);
        dot2x2(S[1][j], C[1][j], w01, xb01);
        dot2x2(S[1][j], C[1][j], w23, xb23);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int a = 0; a < 2; ++a) {
    const int t = t0 + 2 * ty + a;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int e = e0 + tx + 16 * j;
      const float2 sv = f2_split(S[a][j]), cv = f2_split(C[a][j]);
      float ss = sv.x, cc = cv.x;
      pair_add(ss, cc, sv.y, cv.y);
      if (t < T && e < E) part[((size_t)blockIdx.z * T + t) * E + e] = make_float2(ss, cc);
    }
  }
}

constexpr int kTokW = 8;  // tokens (warps) per block of k_topk_tiled

__global__ void __launch_bounds__(kTokW * 32)
    k_topk_tiled(Dev d, const float2* __restrict__ part, const float* __restrict__ bias, int T, int ks) {
  extern __shared__ __align__(16) float s_zt[];  // [kTokW][E]
  __shared__ int s_sel[kTokW][kMaxTopK];
  __shared__ float s_zs[kTokW][kMaxTopK];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = (int)blockIdx.x * kTokW + warp;
  if (t >= T) return;  // warp-uniform; no block-wide barrier below
  const int E = d.E, k = d.k;
  float* z = s_zt + (size_t)warp * E;
  for (int e = lane; e < E; e += 32) {
    float2 p = part[(size_t)t * E + e];
    for (int sp = 1; sp < ks; ++sp) {
      const float2 q = part[((size_t)sp * T + t) * E + e];
      pair_add(p.x, p.y, q.x, q.y);
    }
    float v = __fadd_rn(p.x, p.y);
    if (bias) v = __fadd_rn(v, bias[(size_t)t * E + e]);
    z[e] = v;
  }
  __syncwarp();
  if (lane < k) s_sel[warp][lane] = lane;  // valid even where the logits are not ordered (NaN)
  __syncwarp();
  for (int e = lane; e < E; e += 32) {  // rank by counting, ties to the lower id
    const float v = z[e];
    int r = 0;
    for (int e2 = 0; e2 < E; ++e2) {
      const float v2 = z[e2];
      r += (v2 > v) || (v2 == v && e2 < e);
    }
    if (r < k) {
      s_sel[warp][r] = e;
      s_zs[warp][r] = v;
    }
  }
  __syncwarp();
  const float ex = lane < k ? expf(s_zs[warp][lane] - s_zs[warp][0]) : 0.f;
  float den = ex;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) den += __shfl_xor_sync(0xffffffffu, den, off);
  if (lane < k) {
    d.idx[(size_t)t * k + lane] = s_sel[warp][lane];
    d.g[(size_t)t * k + lane] = ex / den;
  }
}

// K splits for T tokens: about kTiledBlocks blocks when the tiles alone are fewer.  A constant
// (two blocks per SM of a 152-SM part), not the device's count, so that the planner, which runs
// without a GPU, sizes the scratch exactly as the context does.
constexpr int kTiledBlocks = 304;
int tiled_splits(int T, int E, int H) {
  const int tiles = ((T + kTT - 1) / kTT) * ((E + kTE - 1) / kTE);
  const int nch = H / kHC;
  int want = (kTiledBlocks + tiles - 1) / tiles;
  if (want < 1) want = 1;
  const int cps = (nch + want - 1) / want;
  return (nch + cps - 1) / cps;
}

cudaError_t launch_router_tiled(const Dev& d, const float* x, const float* wr, const float* bias, int T,
                                cudaStream_t s) {
  const int ks = tiled_splits(T, d.E, d.H);
  const int nch = d.H / kHC, cps = (nch + ks - 1) / ks;
  k_logits_tiled<<<dim3((d.E + kTE - 1) / kTE, (T + kTT - 1) / kTT, ks), kThreadsT, 0, s>>>(x, wr, T, d.E, d.H, cps,
                                                                                            d.zpart);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t smem = (size_t)kTokW * d.E * sizeof(float);
  if (smem > 48 * 1024) {
    e = cudaFuncSetAttribute(k_topk_tiled, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  k_topk_tiled<<<(T + kTokW - 1) / kTokW, kTokW * 32, smem, s>>>(d, d.zpart, bias, T, ks);
  return cudaGetLastError();
}

}  // namespace

size_t router_part_pairs(int T_max, int E, int H) {
  size_t most = 0;
  for (int T = kTiledMinT; T <= T_max; ++T) {
    const size_t n = (size_t)tiled_splits(T, E, H) * T * E;
    if (n > most) most = n;
  }
  return most;
}

cudaError_t launch_router(const Dev& d, const float* x, const float* wr, const float* bias, int T, int layer,
                          cudaStream_t s, float* x_copy) {
  if (T >= kTiledMinT) return launch_router_tiled(d, x, wr, bias, T, s);
  const size_t smem = (size_t)d.H * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(k_router, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kThreadsR);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // cluster size: 16 where the GPU can hold such a cluster (asked once), else the portable 8
  static int nc = 0;
  if (nc == 0) {
    nc = 8;
    if (cudaFuncSetAttribute(k_router, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess) {
      cfg.gridDim = dim3(16, 1);
      attr[0].val.clusterDim.x = 16;
      int clusters = 0;
      if (cudaOccupancyMaxActiveClusters(&clusters, k_router, &cfg) == cudaSuccess && clusters >= 1) nc = 16;
    }
    cudaGetLastError();
  }
  cfg.gridDim = dim3(nc, T);
  attr[0].val.clusterDim.x = nc;
  // programmatic: the launch may begin while the previous kernel of the stream finishes (the
  // kernel waits for it before touching global memory); plain where the driver refuses that
  static bool pdl_ok = true;
  if (pdl_ok) {
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.numAttrs = 2;
    e = cudaLaunchKernelEx(&cfg, k_router, d, x, wr, bias, T, layer, T == 1 ? 1 : 0, x_copy, nc);
    if (e == cudaSuccess) return e;
    cudaGetLastError();
    pdl_ok = false;
    cfg.numAttrs = 1;
  }
  e = cudaLaunchKernelEx(&cfg, k_router, d, x, wr, bias, T, layer, T == 1 ? 1 : 0, x_copy, nc);
  return e;
}

}  // namespace mf
