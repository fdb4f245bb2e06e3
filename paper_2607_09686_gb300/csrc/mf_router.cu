// Router: logits z = W_r x (+ bias), top-k by (z desc, id asc), softmax over the chosen.
//
// MoE routing selects a subset of experts per token (Background section of the paper).
// Logits are computed with a compensated dot product (Ogita, Rump & Oishi, "Accurate
// sum and dot product", SIAM J. Sci. Comput. 2005, algorithm Dot2): every product is split
// exactly into value + error with an FMA, the running sum is kept as an unevaluated pair,
// and the pair is rounded to fp32 once.  The result is the fp32 rounding of the exact dot
// product except where the exact value lies within ~n*2^-48 relative of a rounding
// boundary, so selection does not depend on the summation order.
//
// Launch: grid (ceil(E / 8), T) (at most 4 blocks per token when T > 1), 256 threads; each
// warp owns whole experts.  The last block to finish a token (ticket counter) selects its
// top-k; with one token per call that block then runs the layer's slot resolve (lru_warp).
#include "mf_lru.cuh"

namespace mf {
namespace {

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

__global__ void __launch_bounds__(256) k_router(Dev d, const float* __restrict__ x, const float* __restrict__ wr,
                                                const float* __restrict__ bias, int T, int layer, int fuse_resolve) {
  const int t = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int H = d.H, E = d.E, k = d.k;
  const float* xt = x + (size_t)t * H;

  for (int e = blockIdx.x * 8 + warp; e < E; e += gridDim.x * 8) {
    const float* w = wr + (size_t)e * H;
    float s = 0.f, c = 0.f;
    for (int i = lane * 4; i < H; i += 128) {
      float4 a = __ldg(reinterpret_cast<const float4*>(w + i));
      float4 b = __ldg(reinterpret_cast<const float4*>(xt + i));
      dot2(s, c, a.x, b.x);
      dot2(s, c, a.y, b.y);
      dot2(s, c, a.z, b.z);
      dot2(s, c, a.w, b.w);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      float so = __shfl_xor_sync(0xffffffffu, s, off);
      float co = __shfl_xor_sync(0xffffffffu, c, off);
      F2 t2 = two_sum(s, so);
      s = t2.hi;
      c = __fadd_rn(__fadd_rn(c, co), t2.lo);
    }
    if (lane == 0) {
      float z = __fadd_rn(s, c);
      if (bias) z = __fadd_rn(z, bias[(size_t)t * E + e]);
      d.logits[(size_t)t * E + e] = z;
    }
  }

  // the last block of this token selects
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    int last = 1;
    if (gridDim.x > 1) {
      unsigned prev = atomicAdd(&d.ticket[t], 1u);
      last = prev == gridDim.x - 1;
      if (last) d.ticket[t] = 0u;
    }
    s_last = last;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  __shared__ float s_z[kMaxExperts];
  __shared__ unsigned char s_taken[kMaxExperts];
  __shared__ int s_sel[kMaxTopK];
  if (warp == 0) {
    for (int e = lane; e < E; e += 32) {
      s_z[e] = __ldcg(d.logits + (size_t)t * E + e);
      s_taken[e] = 0;
    }
    __syncwarp();
    float zsel[kMaxTopK];
    int isel[kMaxTopK];
    for (int j = 0; j < k; ++j) {
      float bz = -INFINITY;
      int bi = 0x7fffffff;
      for (int e = lane; e < E; e += 32) {
        if (s_taken[e]) continue;
        float z = s_z[e];
        if (z > bz || (z == bz && e < bi)) {
          bz = z;
          bi = e;
        }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        float oz = __shfl_xor_sync(0xffffffffu, bz, off);
        int oi = __shfl_xor_sync(0xffffffffu, bi, off);
        if (oz > bz || (oz == bz && oi < bi)) {
          bz = oz;
          bi = oi;
        }
      }
      zsel[j] = bz;
      isel[j] = bi;
      if (lane == 0) s_taken[bi] = 1;
      __syncwarp();
    }
    if (lane == 0) {
      float den = 0.f, ex[kMaxTopK];
      for (int j = 0; j < k; ++j) {
        ex[j] = expf(zsel[j] - zsel[0]);
        den += ex[j];
      }
      for (int j = 0; j < k; ++j) {
        d.idx[(size_t)t * k + j] = isel[j];
        d.g[(size_t)t * k + j] = ex[j] / den;
        s_sel[j] = isel[j];
      }
    }
  }
  if (!fuse_resolve) return;

  // One token per call: this block also runs the layer's slot resolve.  The k chosen experts
  // are distinct, so the accesses are the chosen experts in rank order, all in one wave.
  __shared__ int s_slot_of[kMaxExperts];
  __shared__ int s_expert_of[kMaxExperts];
  __shared__ uint64_t s_lastuse[kMaxExperts];
  __shared__ int s_uslot[kMaxTopK];
  const int S = d.S_active;
  int32_t* g_slot_of = d.slot_of + (size_t)layer * E;
  int32_t* g_expert_of = d.expert_of + (size_t)layer * d.S_alloc;
  uint64_t* g_last = d.last_use + (size_t)layer * d.S_alloc;
  for (int e = threadIdx.x; e < E; e += blockDim.x) s_slot_of[e] = g_slot_of[e];
  for (int q = threadIdx.x; q < S; q += blockDim.x) {
    s_expert_of[q] = g_expert_of[q];
    s_lastuse[q] = g_last[q];
  }
  if (threadIdx.x == 0) {
    d.info[2] = 0;
    d.work[0] = 0u;  // work queues of the pipelined gate/up and down kernels of this call
    d.work[1] = 0u;
  }
  __syncthreads();
  if (warp == 0) lru_warp(d, layer, k, s_sel, s_slot_of, s_expert_of, s_lastuse, s_uslot);
  __syncthreads();
  if (threadIdx.x < k) {  // one assignment per distinct expert: t = 0, j = u
    d.pos_slot[threadIdx.x] = s_uslot[threadIdx.x];
    d.asg[threadIdx.x] = threadIdx.x;
    d.asg_off[threadIdx.x] = threadIdx.x;
  }
  if (threadIdx.x == 0) d.asg_off[k] = k;
  for (int e = threadIdx.x; e < E; e += blockDim.x) g_slot_of[e] = s_slot_of[e];
  for (int q = threadIdx.x; q < S; q += blockDim.x) {
    g_expert_of[q] = s_expert_of[q];
    g_last[q] = s_lastuse[q];
  }
}

}  // namespace

cudaError_t launch_router(const Dev& d, const float* x, const float* wr, const float* bias, int T, int layer,
                          cudaStream_t s) {
  int blocks_e = (d.E + 7) / 8;
  if (T > 1 && blocks_e > 4) blocks_e = 4;  // with many tokens, fewer blocks per token
  dim3 grid(blocks_e, T);
  k_router<<<grid, 256, 0, s>>>(d, x, wr, bias, T, layer, T == 1 ? 1 : 0);
  return cudaGetLastError();
}

}  // namespace mf
