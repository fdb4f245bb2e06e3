// Decode expert FFN: grouped dequantising GEMV over the experts resident in HBM slots.
//
//   h[t,j][r] = silu(sum_c Wg_e[r,c] x_t[c]) * sum_c Wu_e[r,c] x_t[c]     (gate/up + SwiGLU)
//   y[t][c]   = sum_j g[t,j] * sum_r Wd_e[c,r] h[t,j][r]                  (down + combine)
// with e = the expert routed at (t, j), W = d * q (Q8_0) or d * (n - 8) (Q4_0), silu(v) =
// v / (1 + e^-v) (SwiGLU expert FFN with separate gate, up and down tensors, section
// "Native Serving Path").  fp32 accumulation throughout.
//
// One warp per weight row.  Each lane holds whole 16-byte vectors of the row's codes in
// registers (Q8_0: 16 weights, Q4_0: one 32-weight block) and reuses them for every token
// the expert serves.  The down projection of a call with several tokens runs 8 or 16 rows per
// block and stages the h vectors of up to kChunkT of the expert's assignments at a time in
// shared memory, arranged so that the lanes' loads of one vector part are contiguous, for all
// its rows to read.  Codes are turned into floats exactly by placing each byte (or
// nibble) in the low mantissa bits of 2^23 with a byte permute and subtracting 2^23 plus
// the code offset (the int8 -> float "magic number" conversion of Kim et al., "Who says
// elephants can't run", 2022), which costs one PRMT and one FADD per weight instead of an
// integer-to-float conversion.  The scale multiplies each vector's partial dot product.
// Cross-lane sums use a fixed xor-shuffle tree, so results are deterministic.
#include "mf_dequant.cuh"

namespace mf {
namespace {

using namespace dq;

__device__ __forceinline__ const uint8_t* slot_base(const Dev& d, int layer, int slot) {
  return d.pool + ((size_t)layer * d.S_alloc + slot) * d.lay.stride;
}

// rows (warps) per block of the many-token kernels: 16 where the row's registers fit in 128 per
// thread, else 8
template <int QT, int VPL>
__host__ __device__ constexpr int rows_per_block() {
  return (QT == kQ8 && (VPL <= 3 || VPL == 6)) ? 16 : 8;
}
constexpr int kChunkT = 8;           // tokens whose activations are staged at once
constexpr int kStageFloats = 24576;  // at most 96 KB of staged activations

// Shared-memory order of a staged vector of n floats (n = nvec * kW): float4 j of vector v at
// float4 index j * nvec + v, so that lane-consecutive vectors v read consecutive float4s.
template <int QT>
__device__ __forceinline__ void stage_vec(float4* dst, const float* __restrict__ src, int nvec) {
  constexpr int kP = Vec<QT>::kW / 4;  // float4 parts per vector
  for (int q = threadIdx.x; q < nvec * kP; q += blockDim.x) {
    const float4 f = __ldg(reinterpret_cast<const float4*>(src) + q);
    dst[(q % kP) * nvec + q / kP] = f;
  }
}
template <int QT>
__device__ __forceinline__ XV<QT> staged_x(const float4* xs, int nvec, int v) {
  XV<QT> r;
#pragma unroll
  for (int j = 0; j < Vec<QT>::kW / 4; ++j) {
    const float4 f = xs[j * nvec + v];
    r.p[2 * j] = f2_pack(__float_as_uint(f.x), __float_as_uint(f.y));
    r.p[2 * j + 1] = f2_pack(__float_as_uint(f.z), __float_as_uint(f.w));
  }
  return r;
}
// tokens staged per chunk for vectors of n floats
__host__ __device__ __forceinline__ int chunk_tokens(int n) {
  const int c = kStageFloats / n;
  return c < 1 ? 1 : (c > kChunkT ? kChunkT : c);
}

// ---------------------------------------------------------------- gate/up + SwiGLU
// grid (ceil(I / 8), wave width); block 256 = 8 warps = 8 rows of gate and up.
template <int QT, int VPL>
__global__ void __launch_bounds__(256) k_gateup(Dev d, int layer, int wave, const float* __restrict__ x) {
  const int u = wave * d.S_active + blockIdx.y;
  if (u >= d.info[0]) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * 8 + warp;
  if (r >= d.I) return;
  const uint8_t* slot = slot_base(d, layer, d.uslot[u]);
  const uint8_t* gq = slot + (size_t)r * d.lay.rs_gu;  // row record: gate, up codes; gate, up scales
  const uint8_t* uq = gq + d.lay.o_up;
  const __half* gd = reinterpret_cast<const __half*>(gq + d.lay.o_gs);
  const __half* ud = reinterpret_cast<const __half*>(gq + d.lay.o_us);
  const int nvec = d.lay.qrow_gu / 16;

  uint4 wg[VPL], wu[VPL];
  float sg[VPL], su[VPL];
#pragma unroll
  for (int i = 0; i < VPL; ++i) {
    const int v = lane + 32 * i;
    if (v < nvec) {
      wg[i] = ld_stream(gq + 16 * v);
      wu[i] = ld_stream(uq + 16 * v);
      sg[i] = __half2float(gd[scale_index<QT>(v)]);
      su[i] = __half2float(ud[scale_index<QT>(v)]);
    }
  }
  const int a0 = d.asg_off[u], a1 = d.asg_off[u + 1];
  for (int a = a0; a < a1; ++a) {
    const int pos = d.asg[a];
    const float* xt = x + (size_t)(pos / d.k) * d.H;
    float ag = 0.f, au = 0.f;
#pragma unroll
    for (int i = 0; i < VPL; ++i) {
      const int v = lane + 32 * i;
      if (v < nvec) {
        const XV<QT> xv = load_x<QT>(xt + v * Vec<QT>::kW);
        ag = fmaf(dot_vec<QT>(wg[i], xv), sg[i], ag);
        au = fmaf(dot_vec<QT>(wu[i], xv), su[i], au);
      }
    }
    ag = warp_sum(ag);
    au = warp_sum(au);
    if (lane == 0) d.h[(size_t)pos * d.I + r] = ag / (1.0f + expf(-ag)) * au;
  }
}

// ---------------------------------------------------------------- down + combine, one token
// grid ceil(H / 8); block 256 = 8 warps = 8 output rows; JB experts' rows held at once.
template <int QT, int VPL, int JB>
__global__ void __launch_bounds__(256) k_down_single(Dev d, int layer, float* __restrict__ y) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x * 8 + warp;
  if (c >= d.H) return;
  const int k = d.k, nvec = d.lay.qrow_d / 16;
  float acc = 0.f;
  for (int j0 = 0; j0 < k; j0 += JB) {
    uint4 w[JB][VPL];
    float sc[JB][VPL];
#pragma unroll
    for (int jj = 0; jj < JB; ++jj) {
      const int j = j0 + jj;
      if (j < k) {
        const uint8_t* slot = slot_base(d, layer, d.pos_slot[j]);
        const uint8_t* q = slot + d.lay.d_off + (size_t)c * d.lay.rs_d;
        const __half* s = reinterpret_cast<const __half*>(q + d.lay.o_ds);
#pragma unroll
        for (int i = 0; i < VPL; ++i) {
          const int v = lane + 32 * i;
          if (v < nvec) {
            w[jj][i] = ld_stream(q + 16 * v);
            sc[jj][i] = __half2float(s[scale_index<QT>(v)]);
          }
        }
      }
    }
#pragma unroll
    for (int jj = 0; jj < JB; ++jj) {
      const int j = j0 + jj;
      if (j < k) {
        const float* hj = d.h + (size_t)j * d.I;
        float part = 0.f;
#pragma unroll
        for (int i = 0; i < VPL; ++i) {
          const int v = lane + 32 * i;
          if (v < nvec) part = fmaf(dot_vec<QT>(w[jj][i], load_x<QT>(hj + v * Vec<QT>::kW)), sc[jj][i], part);
        }
        acc = fmaf(d.g[j], part, acc);
      }
    }
  }
  acc = warp_sum(acc);
  if (lane == 0) y[c] = acc;
}

// ---------------------------------------------------------------- down, per assignment (T > 1)
// grid (ceil(H / RB), wave width): part[t*k+j][c] = sum_r Wd[c,r] h[t*k+j][r]; h of the
// expert's assignments staged chunk by chunk.
template <int QT, int VPL>
__global__ void __launch_bounds__(rows_per_block<QT, VPL>() * 32, 1) k_down_partial(Dev d, int layer, int wave) {
  extern __shared__ float4 s_hs[];  // [chunk][I / 4] in staged order
  const int u = wave * d.S_active + blockIdx.y;
  if (u >= d.info[0]) return;  // block-uniform
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x * rows_per_block<QT, VPL>() + warp;
  const bool row_ok = c < d.H;
  const uint8_t* slot = slot_base(d, layer, d.uslot[u]);
  const uint8_t* q = slot + d.lay.d_off + (size_t)(row_ok ? c : 0) * d.lay.rs_d;
  const __half* s = reinterpret_cast<const __half*>(q + d.lay.o_ds);
  const int nvec = d.lay.qrow_d / 16, I = d.I, nq = I / 4;
  uint4 w[VPL];
  float sc[VPL];
#pragma unroll
  for (int i = 0; i < VPL; ++i) {
    const int v = lane + 32 * i;
    if (row_ok && v < nvec) {
      w[i] = ld_stream(q + 16 * v);
      sc[i] = __half2float(s[scale_index<QT>(v)]);
    }
  }
  const int a0 = d.asg_off[u], a1 = d.asg_off[u + 1], ct = chunk_tokens(I);
  for (int c0 = a0; c0 < a1; c0 += ct) {
    const int n = min(ct, a1 - c0);
    __syncthreads();
    for (int t = 0; t < n; ++t) stage_vec<QT>(s_hs + (size_t)t * nq, d.h + (size_t)d.asg[c0 + t] * I, nvec);
    __syncthreads();
    if (!row_ok) continue;
    for (int t = 0; t < n; ++t) {
      const float4* hs = s_hs + (size_t)t * nq;
      float part = 0.f;
#pragma unroll
      for (int i = 0; i < VPL; ++i) {
        const int v = lane + 32 * i;
        if (v < nvec) part = fmaf(dot_vec<QT>(w[i], staged_x<QT>(hs, nvec, v)), sc[i], part);
      }
      part = warp_sum(part);
      if (lane == 0) d.part[(size_t)d.asg[c0 + t] * d.H + c] = part;
    }
  }
}

// y[t][c] = sum_j g[t,j] part[t*k+j][c], j in rank order
__global__ void k_combine(Dev d, int T, float* __restrict__ y) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (size_t)T * d.H) return;
  const int t = (int)(i / d.H), c = (int)(i % d.H);
  float acc = 0.f;
  for (int j = 0; j < d.k; ++j) acc = fmaf(d.g[t * d.k + j], d.part[((size_t)t * d.k + j) * d.H + c], acc);
  y[i] = acc;
}

// Kernels of calls with several waves run beside the side stream's materialiser, which asks for
// the largest shared-memory carveout (an SM holds blocks of one carveout at a time): they ask
// for the same, once per kernel.
template <class K>
cudaError_t same_carveout(K kern) {
  static cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                                              cudaSharedmemCarveoutMaxShared);
  return e;
}

// smallest instantiated vectors-per-lane count covering `nvec` vectors
int pick_vpl(int nvec) {
  const int need = (nvec + 31) / 32;
  if (need <= 1) return 1;
  if (need <= 2) return 2;
  if (need <= 3) return 3;
  if (need <= 4) return 4;
  if (need <= 6) return 6;
  return 8;
}

template <int QT, int VPL>
cudaError_t launch_gateup_v(const Dev& d, int layer, int wave, int width, const float* x, cudaStream_t s) {
  const cudaError_t e = same_carveout(k_gateup<QT, VPL>);
  if (e != cudaSuccess) return e;
  k_gateup<QT, VPL><<<dim3((d.I + 7) / 8, width), 256, 0, s>>>(d, layer, wave, x);
  return cudaGetLastError();
}

template <int QT>
cudaError_t gateup_q(const Dev& d, int layer, int wave, int width, const float* x, cudaStream_t s) {
  switch (pick_vpl(d.lay.qrow_gu / 16)) {
    case 1: return launch_gateup_v<QT, 1>(d, layer, wave, width, x, s);
    case 2: return launch_gateup_v<QT, 2>(d, layer, wave, width, x, s);
    case 3: return launch_gateup_v<QT, 3>(d, layer, wave, width, x, s);
    case 4: return launch_gateup_v<QT, 4>(d, layer, wave, width, x, s);
    case 6: return launch_gateup_v<QT, 6>(d, layer, wave, width, x, s);
    default: return launch_gateup_v<QT, 8>(d, layer, wave, width, x, s);
  }
}

template <int QT>
cudaError_t down_single_q(const Dev& d, int layer, float* y, cudaStream_t s) {
  dim3 grid((d.H + 7) / 8);
  switch (pick_vpl(d.lay.qrow_d / 16)) {
    case 1: k_down_single<QT, 1, 8><<<grid, 256, 0, s>>>(d, layer, y); break;
    case 2: k_down_single<QT, 2, 8><<<grid, 256, 0, s>>>(d, layer, y); break;
    case 3: k_down_single<QT, 3, 8><<<grid, 256, 0, s>>>(d, layer, y); break;
    case 4: k_down_single<QT, 4, 4><<<grid, 256, 0, s>>>(d, layer, y); break;
    case 6: k_down_single<QT, 6, 2><<<grid, 256, 0, s>>>(d, layer, y); break;
    default: k_down_single<QT, 8, 2><<<grid, 256, 0, s>>>(d, layer, y); break;
  }
  return cudaGetLastError();
}

template <int QT, int VPL>
cudaError_t launch_down_partial_v(const Dev& d, int layer, int wave, int width, cudaStream_t s) {
  constexpr int RB = rows_per_block<QT, VPL>();
  const size_t smem = (size_t)chunk_tokens(d.I) * d.I * sizeof(float);
  cudaError_t e =
      cudaFuncSetAttribute(k_down_partial<QT, VPL>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) e = same_carveout(k_down_partial<QT, VPL>);
  if (e != cudaSuccess) return e;
  k_down_partial<QT, VPL><<<dim3((d.H + RB - 1) / RB, width), RB * 32, smem, s>>>(d, layer, wave);
  return cudaGetLastError();
}

template <int QT>
cudaError_t down_partial_q(const Dev& d, int layer, int wave, int width, cudaStream_t s) {
  switch (pick_vpl(d.lay.qrow_d / 16)) {
    case 1: return launch_down_partial_v<QT, 1>(d, layer, wave, width, s);
    case 2: return launch_down_partial_v<QT, 2>(d, layer, wave, width, s);
    case 3: return launch_down_partial_v<QT, 3>(d, layer, wave, width, s);
    case 4: return launch_down_partial_v<QT, 4>(d, layer, wave, width, s);
    case 6: return launch_down_partial_v<QT, 6>(d, layer, wave, width, s);
    default: return launch_down_partial_v<QT, 8>(d, layer, wave, width, s);
  }
}

}  // namespace

cudaError_t launch_gateup(const Dev& d, int layer, int wave, int width, const float* x, cudaStream_t s) {
  return d.qtype == kQ8 ? gateup_q<kQ8>(d, layer, wave, width, x, s) : gateup_q<kQ4>(d, layer, wave, width, x, s);
}

cudaError_t launch_down_single(const Dev& d, int layer, float* y, cudaStream_t s) {
  return d.qtype == kQ8 ? down_single_q<kQ8>(d, layer, y, s) : down_single_q<kQ4>(d, layer, y, s);
}

cudaError_t launch_down_partial(const Dev& d, int layer, int wave, int width, cudaStream_t s) {
  return d.qtype == kQ8 ? down_partial_q<kQ8>(d, layer, wave, width, s) : down_partial_q<kQ4>(d, layer, wave, width, s);
}

cudaError_t launch_combine(const Dev& d, int T, float* y, cudaStream_t s) {
  const size_t n = (size_t)T * d.H;
  same_carveout(k_combine);
  k_combine<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(d, T, y);
  return cudaGetLastError();
}

}  // namespace mf
