// Router arithmetic shared by the router kernels and the fused one-token kernel (internal).
//
// MoE routing selects a subset of experts per token (Background section of the paper): logits
// z = W_r x (+ bias), the k largest by (z desc, id asc), softmax over the chosen.  Logits use a
// compensated dot product (Ogita, Rump & Oishi, "Accurate sum and dot product", SIAM J. Sci.
// Comput. 2005, algorithm Dot2): every product is split exactly into value + error with an FMA,
// the running sum is kept as an unevaluated pair, and the pair is rounded to fp32 once.  The
// result is the fp32 rounding of the exact dot product except where the exact value lies within
// ~n*2^-48 relative of a rounding boundary, so the selection does not depend on the order in
// which a kernel sums.
#pragma once

#include "mf_internal.cuh"

namespace mf {

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

// The k largest of E logits in shared memory, ranked by counting: the position of expert e is the
// number of experts with a larger logit, or an equal one and a lower id.  s_sel[r] / s_zsel[r]
// receive the expert of rank r < k and its logit; s_sel starts as 0..k-1, a valid choice even
// where the logits are not ordered (NaN).  tpe consecutive lanes share an expert, each counting
// over every tpe-th other expert.  Every thread of the block calls it (block barriers inside);
// the logits must be stored before the call.
__device__ __forceinline__ void rank_topk(const float* s_z, int E, int k, int* s_sel, float* s_zsel) {
  const int tid = threadIdx.x, nt = blockDim.x;
  if (tid < k) s_sel[tid] = tid;
  __syncthreads();
  int tpe = 1;
  while (tpe < 32 && tpe * 2 * E <= nt) tpe *= 2;
  const int per_pass = nt / tpe, part = tid % tpe;
  for (int e0 = 0; e0 < E; e0 += per_pass) {  // block-uniform
    const int e = e0 + tid / tpe;
    const bool valid = e < E;
    const float z = valid ? s_z[e] : 0.f;
    int r = 0;
    if (valid) {
      int e2 = part;
      for (; e2 + 7 * tpe < E; e2 += 8 * tpe) {  // eight loads in flight
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int ee = e2 + u * tpe;
          const float z2 = s_z[ee];
          r += (z2 > z) || (z2 == z && ee < e);
        }
      }
      for (; e2 < E; e2 += tpe) {
        const float z2 = s_z[e2];
        r += (z2 > z) || (z2 == z && e2 < e);
      }
    }
    for (int off = tpe >> 1; off > 0; off >>= 1) r += __shfl_xor_sync(0xffffffffu, r, off);
    if (valid && part == 0 && r < k) {
      s_sel[r] = e;
      s_zsel[r] = z;
    }
  }
  __syncthreads();
}

// Softmax over the chosen, by one whole warp: lane j < k returns exp(z_j - z_0) / sum over the
// chosen (a fixed shuffle tree, so every kernel that calls it gets the same bits); others 0.
__device__ __forceinline__ float topk_softmax(const float* s_zsel, int k) {
  const int lane = threadIdx.x & 31;
  const float ex = lane < k ? expf(s_zsel[lane] - s_zsel[0]) : 0.f;
  float den = ex;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) den += __shfl_xor_sync(0xffffffffu, den, off);
  return lane < k ? ex / den : 0.f;
}

}  // namespace mf
