// Dequantising dot products shared by the decode kernels (internal).
//
// Codes become floats exactly by placing each byte (Q8_0: code + 128; Q4_0: the 4-bit code) in
// the low mantissa bits of 2^23 with a byte permute and subtracting 2^23 plus the offset (the
// integer -> float "magic number" conversion of Kim et al., "Who says elephants can't run",
// 2022): one PRMT and one FADD per weight instead of an integer-to-float conversion.
#pragma once

#include "mf_internal.cuh"

namespace mf {
namespace dq {

constexpr int kQ8 = MF_Q8_0;
constexpr int kQ4 = MF_Q4_0;

// four signed int8 codes of w dotted with x[0..3]
__device__ __forceinline__ float dot4_q8(uint32_t w, float4 x, float acc) {
  const uint32_t u = w ^ 0x80808080u;  // code + 128 in each byte
  const float f0 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7540)) - 8388736.0f;  // 2^23 + 128
  const float f1 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7541)) - 8388736.0f;
  const float f2 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7542)) - 8388736.0f;
  const float f3 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7543)) - 8388736.0f;
  acc = fmaf(f0, x.x, acc);
  acc = fmaf(f1, x.y, acc);
  acc = fmaf(f2, x.z, acc);
  acc = fmaf(f3, x.w, acc);
  return acc;
}

// four 4-bit codes (one per byte, already masked) dotted with x[0..3]; weight = n - 8
__device__ __forceinline__ float dot4_q4(uint32_t n, float4 x, float acc) {
  const float f0 = __uint_as_float(__byte_perm(n, 0x4B000000u, 0x7540)) - 8388616.0f;  // 2^23 + 8
  const float f1 = __uint_as_float(__byte_perm(n, 0x4B000000u, 0x7541)) - 8388616.0f;
  const float f2 = __uint_as_float(__byte_perm(n, 0x4B000000u, 0x7542)) - 8388616.0f;
  const float f3 = __uint_as_float(__byte_perm(n, 0x4B000000u, 0x7543)) - 8388616.0f;
  acc = fmaf(f0, x.x, acc);
  acc = fmaf(f1, x.y, acc);
  acc = fmaf(f2, x.z, acc);
  acc = fmaf(f3, x.w, acc);
  return acc;
}

// weights covered by one 16-byte vector
template <int QT>
struct Vec {
  static constexpr int kW = QT == kQ8 ? 16 : 32;
};

// x values of vector v: Q8_0 16 contiguous floats; Q4_0 the 32 floats of block v
template <int QT>
struct XV {
  float4 a[Vec<QT>::kW / 4];
};

template <int QT>
__device__ __forceinline__ XV<QT> load_x(const float* __restrict__ xv) {
  XV<QT> r;
#pragma unroll
  for (int i = 0; i < Vec<QT>::kW / 4; ++i) r.a[i] = __ldg(reinterpret_cast<const float4*>(xv) + i);
  return r;
}

// unscaled dot product of one code vector with its x values
template <int QT>
__device__ __forceinline__ float dot_vec(uint4 w, const XV<QT>& x) {
  float acc = 0.f;
  if constexpr (QT == kQ8) {
    acc = dot4_q8(w.x, x.a[0], acc);
    acc = dot4_q8(w.y, x.a[1], acc);
    acc = dot4_q8(w.z, x.a[2], acc);
    acc = dot4_q8(w.w, x.a[3], acc);
  } else {
    // byte j: element j (low nibble), element j + 16 (high nibble)
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      acc = dot4_q4(ws[i] & 0x0F0F0F0Fu, x.a[i], acc);
      acc = dot4_q4((ws[i] >> 4) & 0x0F0F0F0Fu, x.a[4 + i], acc);
    }
  }
  return acc;
}

template <int QT>
__device__ __forceinline__ int scale_index(int v) {
  return QT == kQ8 ? (v >> 1) : v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

}  // namespace dq
}  // namespace mf
