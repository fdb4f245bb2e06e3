// Dequantising dot products shared by the decode kernels (internal).
//
// Codes become floats exactly by placing each byte (Q8_0: code + 128, the form the pack stores;
// Q4_0: the 4-bit code) in the low mantissa bits of 2^23 with a byte permute and subtracting
// 2^23 plus the offset (the integer -> float "magic number" conversion of Kim et al., "Who says
// elephants can't run", 2022).  Subtractions and FMAs use packed f32x2 arithmetic: about two
// instructions per weight.  Every product and sum is an ordinary fp32 operation.
#pragma once

#include "mf_internal.cuh"

namespace mf {
namespace dq {

constexpr int kQ8 = MF_Q8_0;
constexpr int kQ4 = MF_Q4_0;

// Packed pair of fp32 values (Blackwell f32x2 arithmetic: two FMAs / adds per instruction).
__device__ __forceinline__ uint64_t f2_pack(uint32_t lo, uint32_t hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(lo), "r"(hi));
  return r;
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ float f2_sum(uint64_t a) {
  uint32_t lo, hi;
  asm("mov.b64 {%0, %1}, %2;" : "=r"(lo), "=r"(hi) : "l"(a));
  return __uint_as_float(lo) + __uint_as_float(hi);
}

// Four unsigned byte codes c_i of w (Q8_0 codes are stored as q + 128; Q4_0 nibbles already
// masked to bytes), dotted with x[0..3] into the packed accumulator: each byte is placed in the
// low mantissa bits of 2^23 (value 2^23 + c), the offset 2^23 + off is subtracted exactly, and
// the result multiplies x.  acc.lo collects elements 0 and 2, acc.hi elements 1 and 3.
template <uint32_t kOffBits>
__device__ __forceinline__ uint64_t dot4_u8(uint32_t w, uint64_t x01, uint64_t x23, uint64_t acc) {
  const uint64_t neg = f2_pack(kOffBits | 0x80000000u, kOffBits | 0x80000000u);  // -(2^23 + off)
  const uint64_t f01 = f2_add(f2_pack(__byte_perm(w, 0x4B000000u, 0x7540), __byte_perm(w, 0x4B000000u, 0x7541)), neg);
  const uint64_t f23 = f2_add(f2_pack(__byte_perm(w, 0x4B000000u, 0x7542), __byte_perm(w, 0x4B000000u, 0x7543)), neg);
  acc = f2_fma(f01, x01, acc);
  return f2_fma(f23, x23, acc);
}
constexpr uint32_t kOffQ8 = 0x4B000080u;  // bits of 2^23 + 128
constexpr uint32_t kOffQ4 = 0x4B000008u;  // bits of 2^23 + 8

// weights covered by one 16-byte vector
template <int QT>
struct Vec {
  static constexpr int kW = QT == kQ8 ? 16 : 32;
};

// x values of one vector as packed pairs: Q8_0 16 contiguous floats; Q4_0 the 32 of a block
template <int QT>
struct XV {
  uint64_t p[Vec<QT>::kW / 2];
};

template <int QT>
__device__ __forceinline__ XV<QT> load_x(const float* __restrict__ xv) {
  XV<QT> r;
#pragma unroll
  for (int i = 0; i < Vec<QT>::kW / 4; ++i) {
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(xv) + i);
    r.p[2 * i] = f2_pack(v.x, v.y);
    r.p[2 * i + 1] = f2_pack(v.z, v.w);
  }
  return r;
}

// unscaled dot product of one code vector with its x values (two independent accumulators)
template <int QT>
__device__ __forceinline__ float dot_vec(uint4 w, const XV<QT>& x) {
  uint64_t a = 0, b = 0;
  if constexpr (QT == kQ8) {
    a = dot4_u8<kOffQ8>(w.x, x.p[0], x.p[1], a);
    b = dot4_u8<kOffQ8>(w.y, x.p[2], x.p[3], b);
    a = dot4_u8<kOffQ8>(w.z, x.p[4], x.p[5], a);
    b = dot4_u8<kOffQ8>(w.w, x.p[6], x.p[7], b);
  } else {
    // byte j of the block: element j (low nibble), element j + 16 (high nibble)
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      a = dot4_u8<kOffQ4>(ws[i] & 0x0F0F0F0Fu, x.p[2 * i], x.p[2 * i + 1], a);
      b = dot4_u8<kOffQ4>((ws[i] >> 4) & 0x0F0F0F0Fu, x.p[8 + 2 * i], x.p[8 + 2 * i + 1], b);
    }
  }
  return f2_sum(f2_add(a, b));
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
