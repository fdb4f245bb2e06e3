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

// ---- exact integer dot products for vectors held in registers across many rows
//
// A vector of kW fp32 values v (x, or h) is split once into three int8 pieces
//   v ~= s * (p1 + p2 / 127 + p3 / 127^2),  s = max|v| / 127,
// so that |v - that| <= max|v| * 2^-22.  A row's codes c then give the exact integer sums
// P_i = sum_j c_j p_i[j] with dp4a (4 byte products per instruction), and
//   sum_j (c_j - off) v_j ~= s * ((P1 * 127 + P2 - off * (S1 * 127 + S2)) * 127 + P3 - off * S3) / 127^2
// where S_i = sum_j p_i[j] and off is the code offset (128 for Q8_0's stored q + 128, 8 for Q4_0).
// Every integer sum is exact (|P1 * 127| < 2^27); fp32 rounds only the final combination.
//
// Range: every group of one logical vector (all of x, or one expert's h) is split as if first
// multiplied by the same power of two 2^-e, e the binary exponent of the vector's largest
// magnitude, so the largest group maximum lies in [0.5, 1): 127 / max never overflows and s stays
// a normal number for any finite input, however small or large.  Scaling by a power of two is
// exact, so the pieces (and every product) are those of the unscaled vector; a result is
// multiplied back by 2^e once per output row (scale2).  A group whose maximum is below 2^-100 of
// the vector's is taken as zero (its contribution is below 2^-88 of the row's largest term).
template <int QT>
struct XQ {
  static constexpr int kWords = Vec<QT>::kW / 4;  // words of four values: 4 (Q8_0) or 8 (Q4_0)
  uint32_t p1[kWords], p2[kWords], p3[kWords];
  int k12, k3;  // offset corrections: off * (S1 * 127 + S2), off * S3
  float sf;     // s / 127^2
};

// 2^n as a binary32 value, for -126 <= n <= 127
__device__ __forceinline__ float pow2i(int n) { return __uint_as_float((uint32_t)(127 + n) << 23); }
// v * 2^n, exact unless the result leaves the binary32 range (|n| <= 252: two normal factors)
__device__ __forceinline__ float scale2(float v, int n) {
  const int a = n / 2;
  return v * pow2i(a) * pow2i(n - a);
}
// the exponent e of m = f * 2^e with 0.5 <= f < 1, from m's binary32 fields (0 for m = 0; m >= 0,
// finite; subnormal m from its leading bit)
__device__ __forceinline__ int vec_exponent(float m) {
  const uint32_t b = __float_as_uint(m) & 0x7fffffffu;
  if (b == 0) return 0;
  const int be = (int)(b >> 23);
  if (be > 0) return be - 126;
  return (31 - __clz((int)b)) - 148;
}

// Splitting group by group: each group is split scaled by its own exponent e_g (quant_vals(v,
// -e_g)), then, once the vector's exponent e is known (the largest e_g), its s is multiplied by
// 2^(e_g - e) (rescale_group): the same pieces and s as splitting the group scaled by 2^-e, without
// keeping the values.  kNoExp stands for the exponent of an all-zero group.
constexpr int kNoExp = -100000;
__device__ __forceinline__ int group_exponent(float m) { return m > 0.f ? vec_exponent(m) : kNoExp; }
__device__ __forceinline__ int vector_exponent(int e_max) { return e_max == kNoExp ? 0 : e_max; }
template <int QT>
__device__ __forceinline__ void rescale_group(XQ<QT>& q, int e_g, int e) {
  q.sf = e_g - e >= -100 ? scale2(q.sf, e_g - e) : 0.f;  // groups below 2^-100 of the vector: zero
}

// the kW values of one group (kCoherent: read through L2 only, for values other blocks wrote)
template <int QT, bool kCoherent = false>
__device__ __forceinline__ void load_group(const float* __restrict__ vp, float (&v)[Vec<QT>::kW]) {
#pragma unroll
  for (int i = 0; i < Vec<QT>::kW / 4; ++i) {
    const float4 f =
        kCoherent ? __ldcg(reinterpret_cast<const float4*>(vp) + i) : __ldg(reinterpret_cast<const float4*>(vp) + i);
    v[4 * i] = f.x;
    v[4 * i + 1] = f.y;
    v[4 * i + 2] = f.z;
    v[4 * i + 3] = f.w;
  }
}

template <int QT>
__device__ __forceinline__ float group_absmax(const float (&v)[Vec<QT>::kW]) {
  float m = 0.f;
#pragma unroll
  for (int j = 0; j < Vec<QT>::kW; ++j) m = fmaxf(m, fabsf(v[j]));
  return m;
}

// the pieces of one group, after multiplying its values by 2^ne (ne = -e of the whole vector)
template <int QT>
__device__ __forceinline__ XQ<QT> quant_vals(const float (&v0)[Vec<QT>::kW], int ne) {
  constexpr int kW = Vec<QT>::kW;
  float v[kW];
  const float sa = pow2i(ne / 2), sb = pow2i(ne - ne / 2);
#pragma unroll
  for (int j = 0; j < kW; ++j) v[j] = v0[j] * sa * sb;
  float m = 0.f;
#pragma unroll
  for (int j = 0; j < kW; ++j) m = fmaxf(m, fabsf(v[j]));
  const float inv = m > 0x1p-100f ? 127.f / m : 0.f;
  XQ<QT> r;
  int s1 = 0, s2 = 0, s3 = 0;
#pragma unroll
  for (int w = 0; w < XQ<QT>::kWords; ++w) {
    uint32_t b1 = 0, b2 = 0, b3 = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float t = v[4 * w + j] * inv;
      const int a = __float2int_rn(t);
      const float e = (t - (float)a) * 127.f;
      const int b = __float2int_rn(e);
      const int c = __float2int_rn((e - (float)b) * 127.f);
      s1 += a;
      s2 += b;
      s3 += c;
      b1 |= (uint32_t)(a & 0xFF) << (8 * j);
      b2 |= (uint32_t)(b & 0xFF) << (8 * j);
      b3 |= (uint32_t)(c & 0xFF) << (8 * j);
    }
    r.p1[w] = b1;
    r.p2[w] = b2;
    r.p3[w] = b3;
  }
  constexpr int off = QT == kQ8 ? 128 : 8;
  r.k12 = off * (s1 * 127 + s2);
  r.k3 = off * s3;
  r.sf = inv > 0.f ? m / 127.f / 16129.f : 0.f;
  return r;
}

// sum of four unsigned byte x signed byte products, added to c
__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c) {
  int d;
  asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// unscaled dot product of one code vector with a split vector
template <int QT>
__device__ __forceinline__ float dot_q(uint4 w, const XQ<QT>& x) {
  int a = 0, b = 0, c = 0;
  const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
  if constexpr (QT == kQ8) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      a = dp4a_us(ws[i], x.p1[i], a);
      b = dp4a_us(ws[i], x.p2[i], b);
      c = dp4a_us(ws[i], x.p3[i], c);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {  // byte j: element j (low nibble), element j + 16 (high nibble)
      const uint32_t lo = ws[i] & 0x0F0F0F0Fu, hi = (ws[i] >> 4) & 0x0F0F0F0Fu;
      a = dp4a_us(lo, x.p1[i], a);
      a = dp4a_us(hi, x.p1[4 + i], a);
      b = dp4a_us(lo, x.p2[i], b);
      b = dp4a_us(hi, x.p2[4 + i], b);
      c = dp4a_us(lo, x.p3[i], c);
      c = dp4a_us(hi, x.p3[4 + i], c);
    }
  }
  const int p12 = a * 127 + b - x.k12;
  const int p3 = c - x.k3;
  return fmaf((float)p12, 127.f, (float)p3) * x.sf;
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
