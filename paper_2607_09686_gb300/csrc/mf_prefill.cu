// Prefill expert FFN: grouped GEMMs on the fifth-generation tensor cores (tcgen05).
//
// When many tokens route to each expert (a prefill chunk), the expert FFN of a wave is a set
// of dense products, one per expert e of the wave with the n_e assignments it serves:
//   gate/up:  G = Wg_e X_e^T, U = Wu_e X_e^T,  h = silu(G) * U                 [I x n_e]
//   down:     P = Wd_e h                                                        [H x n_e]
// then y[t] = sum_j g[t,j] P_{e_j}[:, t] (the batched combine kernel).  (SwiGLU experts with
// separate gate, up and down tensors, section "Native Serving Path".)
//
// Precision.  Operands are split into two bfloat16 parts, v = hi + lo with hi = bf16(v) and
// lo = bf16(v - hi), so hi + lo carries 16 significant bits (relative error <= 2^-17).  Each
// product is formed as hi*hi + hi*lo + lo*hi with fp32 accumulation in tensor memory; the
// dropped lo*lo term is below 2^-16 of the product.  Per product the relative error is thus
// a few times 1e-5, far inside the output tolerance, while the tensor cores do the work.
//
// Work unit = (expert of the wave, block of 128 assignments, block of 128 weight rows).  One
// CTA per SM walks the units.  For each 64-wide K chunk all 256 threads dequantise the weight
// tiles and gather the assignment tiles into one of two shared-memory stages (no-swizzle
// K-major core-matrix layout); thread 0 then issues the MMAs (M = 128, N = 128, K = 16 each)
// and commits them to the stage's mbarrier, so filling stage s+1 overlaps the MMAs of stage s.
// The epilogue (warps 0-3, one TMEM lane = one weight row each) reads the accumulators with
// tcgen05.ld.  Every wait is bounded and taken by thread 0, which publishes the outcome
// before the block acts on it; after a wait gives up the block sets the device error word,
// waits (bounded) for its MMAs and frees its tensor memory before returning.
#include <cuda_bf16.h>

#include "mf_internal.cuh"

namespace mf {
namespace {

constexpr int kBM = 128, kBN = 128, kBK = 64;
constexpr int kThreadsP = 256;
constexpr uint32_t kTileBytes = kBM * kBK * 2;  // one bf16 tile: 128 rows x 64 k
constexpr uint32_t kWaitLimit = 1u << 26;

// Byte offset of element (row r, k) in a K-major no-swizzle tile of 128 x 64: 8x8 core
// matrices of 128 contiguous bytes, K-adjacent core matrices 128 B apart (the descriptor's
// leading byte offset), 8-row groups 1024 B apart (its stride byte offset).
__device__ __forceinline__ uint32_t core_off(int r, int k) {
  return (uint32_t)((r >> 3) * 1024 + (k >> 3) * 128 + (r & 7) * 16 + (k & 7) * 2);
}

// shared-memory matrix descriptor: start >> 4, LBO >> 4 at bit 16, SBO >> 4 at bit 32,
// descriptor version 1 at bit 46, no swizzle
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
  return (uint64_t)((addr >> 4) & 0x3FFF) | ((uint64_t)(128u >> 4) << 16) | ((uint64_t)(1024u >> 4) << 32) |
         ((uint64_t)1 << 46);
}

// kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B, both K-major, M x N
constexpr uint32_t kIdesc =
    (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kBN >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.u32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(kIdesc), "r"(accumulate));
}
// arrive on `bar` once every MMA this thread issued so far has completed
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// generic-proxy shared-memory writes become visible to the tensor cores' (async proxy) reads
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// 16 consecutive fp32 accumulator columns of this thread's TMEM lane
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void split_bf16(float v, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(v);
  lo = __float2bfloat16_rn(v - __bfloat162float(hi));
}

// 8 consecutive K values of one row -> a 16-byte chunk of the hi tile and of the lo tile
__device__ __forceinline__ void store8(unsigned char* hi_tile, unsigned char* lo_tile, uint32_t off, const float* w) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __nv_bfloat16 h0, l0, h1, l1;
    split_bf16(w[2 * i], h0, l0);
    split_bf16(w[2 * i + 1], h1, l1);
    h[i] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
    l[i] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
  }
  *reinterpret_cast<uint4*>(hi_tile + off) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4*>(lo_tile + off) = make_uint4(l[0], l[1], l[2], l[3]);
}

// Dequantise one 32-weight block of a slot row record (codes + binary16 scale) into row r of
// the hi / lo tiles at K = kb*32 .. kb*32 + 31 of the 64-wide chunk.
template <int QT>
__device__ __forceinline__ void dequant_block(const uint8_t* codes, const __half* scale, unsigned char* hi,
                                              unsigned char* lo, int r, int kb) {
  const float d = __half2float(*scale);
  float w[32];
  if constexpr (QT == MF_Q8_0) {  // stored as q + 128
    const uint4 c0 = *reinterpret_cast<const uint4*>(codes), c1 = *reinterpret_cast<const uint4*>(codes + 16);
    const uint32_t ws[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
#pragma unroll
    for (int i = 0; i < 32; ++i) w[i] = d * (float)((int)((ws[i >> 2] >> (8 * (i & 3))) & 0xFF) - 128);
  } else {  // byte j: element j in the low nibble, element j + 16 in the high nibble
    const uint4 c = *reinterpret_cast<const uint4*>(codes);
    const uint32_t ws[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const uint32_t b = (ws[j >> 2] >> (8 * (j & 3))) & 0xFF;
      w[j] = d * (float)((int)(b & 0xF) - 8);
      w[j + 16] = d * (float)((int)(b >> 4) - 8);
    }
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) store8(hi, lo, core_off(r, kb * 32 + q * 8), w + q * 8);
}

struct Unit {
  int u;   // unique-expert index (access order)
  int tb;  // block of 128 assignments
  int rb;  // block of 128 weight rows
};

// The wave's units, expert by expert: expert u0 + e has ceil(n / 128) assignment blocks times
// `nrb` row blocks, row blocks innermost (CTAs working on the same assignment block at once
// share its gathered activations in L2).
struct UnitMap {
  int u0, nu, nrb, total;
  const int* pre;  // [nu + 1] exclusive prefix of the experts' unit counts
  __device__ __forceinline__ Unit at(int i) const {
    int lo = 0, hi = nu - 1;
    while (lo < hi) {  // last expert with pre[e] <= i
      const int mid = (lo + hi + 1) >> 1;
      if (pre[mid] <= i) lo = mid;
      else hi = mid - 1;
    }
    const int rel = i - pre[lo];
    return {u0 + lo, rel / nrb, rel % nrb};
  }
};

__device__ __forceinline__ UnitMap build_units(const Dev& d, int wave, int nrb, int* s_pre) {
  const int U = d.info[0], S = d.S_active;
  UnitMap m;
  m.u0 = wave * S;
  m.nu = max(0, min(S, U - m.u0));
  m.nrb = nrb;
  m.pre = s_pre;
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int e = 0; e < m.nu; ++e) {
      s_pre[e] = acc;
      const int n = d.asg_off[m.u0 + e + 1] - d.asg_off[m.u0 + e];
      acc += (n + kBN - 1) / kBN * nrb;
    }
    s_pre[m.nu] = acc;
  }
  __syncthreads();
  m.total = s_pre[m.nu];
  return m;
}

// Shared memory: two stages of [NA weight tiles | 2 activation tiles], then the barriers,
// the assignment of each accumulator column, the unit prefix, the TMEM base and a flag.
struct PSmem {
  unsigned char* stage[2];
  uint64_t* mma_done;   // [2] the MMAs reading stage s have completed
  uint64_t* acc_ready;  // [1] every MMA issued so far has completed
  int* pos;             // [kBN] assignment t*k+j of each accumulator column, -1 past the end
  int* pre;             // [kMaxExperts + 1]
  uint32_t* tmem;       // [1]
  int* flag;            // [1] nonzero once a wait gave up
};

template <int NA>
__host__ __device__ constexpr uint32_t stage_bytes() {
  return (NA + 2) * kTileBytes;
}

template <int NA>
constexpr size_t prefill_smem() {
  return 2 * (size_t)stage_bytes<NA>() + 3 * sizeof(uint64_t) + kBN * sizeof(int) + (kMaxExperts + 1) * sizeof(int) +
         2 * sizeof(uint32_t);
}

template <int NA>
__device__ __forceinline__ PSmem carve_p(unsigned char* base) {
  PSmem s;
  s.stage[0] = base;
  s.stage[1] = base + stage_bytes<NA>();
  unsigned char* p = base + 2 * stage_bytes<NA>();
  s.mma_done = reinterpret_cast<uint64_t*>(p);
  s.acc_ready = s.mma_done + 2;
  s.pos = reinterpret_cast<int*>(s.acc_ready + 1);
  s.pre = s.pos + kBN;
  s.tmem = reinterpret_cast<uint32_t*>(s.pre + kMaxExperts + 1);
  s.flag = reinterpret_cast<int*>(s.tmem + 1);
  return s;
}

// Thread 0 waits (bounded) for the phase of `bar` with the given parity; the whole block then
// learns the outcome.  Returns false once any wait of the block has given up.
__device__ __forceinline__ bool block_wait(uint64_t* bar, uint32_t parity, const PSmem& sm, unsigned* err,
                                           unsigned code) {
  if (threadIdx.x == 0 && !*sm.flag && !mbar_wait(bar, parity, kWaitLimit)) {
    *sm.flag = 1;
    atomicExch(err, code);
  }
  __syncthreads();
  return *reinterpret_cast<volatile int*>(sm.flag) == 0;
}

template <uint32_t kCols>
__device__ __forceinline__ void tmem_alloc(const PSmem& sm) {
  if (threadIdx.x < 32) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(sm.tmem)),
                 "r"(kCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
}
template <uint32_t kCols>
__device__ __forceinline__ void tmem_free(uint32_t taddr) {
  if (threadIdx.x < 32) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(kCols));
}

// Barriers, flag and tensor memory at kernel start.
template <uint32_t kCols>
__device__ __forceinline__ uint32_t prologue(const PSmem& sm) {
  if (threadIdx.x == 0) {
    mbar_init(&sm.mma_done[0], 1);
    mbar_init(&sm.mma_done[1], 1);
    mbar_init(sm.acc_ready, 1);
    *sm.flag = 0;
    mbar_fence_init();
  }
  tmem_alloc<kCols>(sm);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  return *sm.tmem;
}

// At kernel end: wait (bounded) until no MMA is in flight, then free the tensor memory.
template <uint32_t kCols>
__device__ __forceinline__ void epilogue_free(const PSmem& sm, uint32_t taddr, uint32_t n_acc, unsigned* err) {
  if (threadIdx.x == 0) {
    mma_commit(sm.acc_ready);
    if (!mbar_wait(sm.acc_ready, n_acc & 1, kWaitLimit)) atomicExch(err, 7u);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  tmem_free<kCols>(taddr);
}

// Gather the unit's activation rows (bf16 hi/lo [rows][ld]; row = assignment / kdiv) for K
// chunk c into the B tiles; columns past the unit's n assignments are zero.  Lanes 0-7 of
// each group of eight take eight consecutive columns, so each 16-byte store of a warp quarter
// covers all 32 banks.  With `record`, also notes each column's assignment.
__device__ __forceinline__ void gather_bf16(const uint16_t* __restrict__ src_hi, const uint16_t* __restrict__ src_lo,
                                            int ld, int kdiv, const int32_t* __restrict__ asg, int a0, int n, int c,
                                            unsigned char* bhi, unsigned char* blo, int* pos, bool record) {
  for (int i = threadIdx.x; i < kBN * 8; i += kThreadsP) {
    const int col = (i & 7) | ((i >> 6) << 3), g = (i >> 3) & 7;
    uint4 vh = make_uint4(0, 0, 0, 0), vl = make_uint4(0, 0, 0, 0);
    int p = -1;
    if (col < n) {
      p = asg[a0 + col];
      const size_t off = (size_t)(p / kdiv) * ld + c * kBK + g * 8;
      vh = *reinterpret_cast<const uint4*>(src_hi + off);
      vl = *reinterpret_cast<const uint4*>(src_lo + off);
    }
    if (record && g == 0) pos[col] = p;
    *reinterpret_cast<uint4*>(bhi + core_off(col, g * 8)) = vh;
    *reinterpret_cast<uint4*>(blo + core_off(col, g * 8)) = vl;
  }
}

// Same from an fp32 [rows][ld] matrix indexed by assignment (the SwiGLU output h), split on
// the fly.
__device__ __forceinline__ void gather_f32(const float* __restrict__ src, int ld, const int32_t* __restrict__ asg,
                                           int a0, int n, int c, unsigned char* bhi, unsigned char* blo, int* pos,
                                           bool record) {
  for (int i = threadIdx.x; i < kBN * 8; i += kThreadsP) {
    const int col = (i & 7) | ((i >> 6) << 3), g = (i >> 3) & 7;
    float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    int p = -1;
    if (col < n) {
      p = asg[a0 + col];
      const float4* s = reinterpret_cast<const float4*>(src + (size_t)p * ld + c * kBK + g * 8);
      const float4 f0 = s[0], f1 = s[1];
      v[0] = f0.x, v[1] = f0.y, v[2] = f0.z, v[3] = f0.w;
      v[4] = f1.x, v[5] = f1.y, v[6] = f1.z, v[7] = f1.w;
    }
    if (record && g == 0) pos[col] = p;
    store8(bhi, blo, core_off(col, g * 8), v);
  }
}

// ---------------------------------------------------------------- gate/up GEMM + SwiGLU
// h[p][r] = silu(sum_c Wg[r,c] x[p/k][c]) * sum_c Wu[r,c] x[p/k][c] for the wave's assignments
template <int QT>
__global__ void __launch_bounds__(kThreadsP, 1) k_prefill_gateup(Dev d, int layer, int wave) {
  extern __shared__ __align__(1024) unsigned char smem[];
  const PSmem sm = carve_p<4>(smem);  // weights: gate hi, gate lo, up hi, up lo; then x hi, x lo
  const uint32_t taddr = prologue<256>(sm);  // columns 0..127 gate, 128..255 up
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const UnitMap um = build_units(d, wave, d.I / kBM, sm.pre);
  const int nchunk = d.H / kBK;
  constexpr int kCodeBytes = QT == MF_Q8_0 ? 32 : 16;  // per 32-weight block
  uint32_t gc = 0, n_acc = 0;                           // chunks filled, accumulator commits
  for (int ui = blockIdx.x; ui < um.total; ui += gridDim.x) {
    const Unit un = um.at(ui);
    const uint8_t* slot = d.pool + ((size_t)layer * d.S_alloc + d.uslot[un.u]) * d.lay.stride;
    const int a0 = d.asg_off[un.u] + un.tb * kBN;
    const int n = min(kBN, d.asg_off[un.u + 1] - a0);
    bool ok = true;
    for (int c = 0; c < nchunk; ++c, ++gc) {
      const int st_i = (int)(gc & 1);
      unsigned char* st = sm.stage[st_i];
      // the MMAs that last read this stage (two chunks ago) must be done before it is refilled
      if (gc >= 2 && !(ok = block_wait(&sm.mma_done[st_i], ((gc >> 1) - 1) & 1, sm, d.err, 5u))) break;
      for (int t = threadIdx.x; t < kBM * 4; t += kThreadsP) {  // (row, 32-block, tensor)
        const int r = t >> 2, kb = (t >> 1) & 1, ten = t & 1;
        const uint8_t* rec = slot + (size_t)(un.rb * kBM + r) * d.lay.rs_gu;
        const int blk = c * 2 + kb;
        const uint8_t* codes = rec + (ten ? d.lay.o_up : 0u) + (size_t)blk * kCodeBytes;
        const __half* sc = reinterpret_cast<const __half*>(rec + (ten ? d.lay.o_us : d.lay.o_gs)) + blk;
        dequant_block<QT>(codes, sc, st + (2 * ten) * kTileBytes, st + (2 * ten + 1) * kTileBytes, r, kb);
      }
      gather_bf16(d.xh, d.xl, d.H, d.k, d.asg, a0, n, c, st + 4 * kTileBytes, st + 5 * kTileBytes, sm.pos, c == 0);
      fence_async_smem();
      __syncthreads();
      if (threadIdx.x == 0) {
        tc_fence_after();
        const uint32_t base = smem_u32(st);
#pragma unroll
        for (int ks = 0; ks < kBK / 16; ++ks) {
          const uint32_t ko = ks * 256;  // K = 16 spans two core matrices
          const uint64_t bh = smem_desc(base + 4 * kTileBytes + ko), bl = smem_desc(base + 5 * kTileBytes + ko);
#pragma unroll
          for (int ten = 0; ten < 2; ++ten) {
            const uint64_t ah = smem_desc(base + (2 * ten) * kTileBytes + ko);
            const uint64_t al = smem_desc(base + (2 * ten + 1) * kTileBytes + ko);
            const uint32_t dt = taddr + ten * kBN;
            mma_bf16(dt, ah, bh, (c | ks) != 0);
            mma_bf16(dt, ah, bl, 1);
            mma_bf16(dt, al, bh, 1);
          }
        }
        mma_commit(&sm.mma_done[st_i]);
      }
    }
    if (!ok) break;
    // every MMA of the unit done -> h = silu(gate) * up
    if (threadIdx.x == 0) mma_commit(sm.acc_ready);
    if (!block_wait(sm.acc_ready, n_acc & 1, sm, d.err, 6u)) break;
    ++n_acc;
    tc_fence_after();
    if (warp < 4) {
      const int r = un.rb * kBM + warp * 32 + lane;
      const uint32_t lane_addr = taddr + ((uint32_t)(warp * 32) << 16);
      for (int c0 = 0; c0 < n; c0 += 16) {
        float g[16], u[16];
        tmem_ld16(lane_addr + c0, g);
        tmem_ld16(lane_addr + kBN + c0, u);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int p = sm.pos[c0 + j];
          if (p >= 0) d.h[(size_t)p * d.I + r] = g[j] / (1.0f + expf(-g[j])) * u[j];
        }
      }
    }
    tc_fence_before();
    __syncthreads();  // accumulators read before the next unit's first MMA overwrites them
  }
  epilogue_free<256>(sm, taddr, n_acc, d.err);
}

// ---------------------------------------------------------------- down GEMM
// part[p][c] = sum_r Wd[c,r] h[p][r] for the wave's assignments
template <int QT>
__global__ void __launch_bounds__(kThreadsP, 1) k_prefill_down(Dev d, int layer, int wave) {
  extern __shared__ __align__(1024) unsigned char smem[];
  const PSmem sm = carve_p<2>(smem);  // weights: down hi, down lo; then h hi, h lo
  const uint32_t taddr = prologue<128>(sm);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const UnitMap um = build_units(d, wave, d.H / kBM, sm.pre);
  const int nchunk = d.I / kBK;
  constexpr int kCodeBytes = QT == MF_Q8_0 ? 32 : 16;
  uint32_t gc = 0, n_acc = 0;
  for (int ui = blockIdx.x; ui < um.total; ui += gridDim.x) {
    const Unit un = um.at(ui);
    const uint8_t* slot = d.pool + ((size_t)layer * d.S_alloc + d.uslot[un.u]) * d.lay.stride + d.lay.d_off;
    const int a0 = d.asg_off[un.u] + un.tb * kBN;
    const int n = min(kBN, d.asg_off[un.u + 1] - a0);
    bool ok = true;
    for (int c = 0; c < nchunk; ++c, ++gc) {
      const int st_i = (int)(gc & 1);
      unsigned char* st = sm.stage[st_i];
      if (gc >= 2 && !(ok = block_wait(&sm.mma_done[st_i], ((gc >> 1) - 1) & 1, sm, d.err, 5u))) break;
      for (int t = threadIdx.x; t < kBM * 2; t += kThreadsP) {  // (row, 32-block)
        const int r = t >> 1, kb = t & 1;
        const uint8_t* rec = slot + (size_t)(un.rb * kBM + r) * d.lay.rs_d;
        const int blk = c * 2 + kb;
        dequant_block<QT>(rec + (size_t)blk * kCodeBytes, reinterpret_cast<const __half*>(rec + d.lay.o_ds) + blk, st,
                          st + kTileBytes, r, kb);
      }
      gather_f32(d.h, d.I, d.asg, a0, n, c, st + 2 * kTileBytes, st + 3 * kTileBytes, sm.pos, c == 0);
      fence_async_smem();
      __syncthreads();
      if (threadIdx.x == 0) {
        tc_fence_after();
        const uint32_t base = smem_u32(st);
#pragma unroll
        for (int ks = 0; ks < kBK / 16; ++ks) {
          const uint32_t ko = ks * 256;
          const uint64_t ah = smem_desc(base + ko), al = smem_desc(base + kTileBytes + ko);
          const uint64_t bh = smem_desc(base + 2 * kTileBytes + ko), bl = smem_desc(base + 3 * kTileBytes + ko);
          mma_bf16(taddr, ah, bh, (c | ks) != 0);
          mma_bf16(taddr, ah, bl, 1);
          mma_bf16(taddr, al, bh, 1);
        }
        mma_commit(&sm.mma_done[st_i]);
      }
    }
    if (!ok) break;
    if (threadIdx.x == 0) mma_commit(sm.acc_ready);
    if (!block_wait(sm.acc_ready, n_acc & 1, sm, d.err, 6u)) break;
    ++n_acc;
    tc_fence_after();
    if (warp < 4) {
      const int r = un.rb * kBM + warp * 32 + lane;  // output feature
      const uint32_t lane_addr = taddr + ((uint32_t)(warp * 32) << 16);
      for (int c0 = 0; c0 < n; c0 += 16) {
        float v[16];
        tmem_ld16(lane_addr + c0, v);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int p = sm.pos[c0 + j];
          if (p >= 0) d.part[(size_t)p * d.H + r] = v[j];
        }
      }
    }
    tc_fence_before();
    __syncthreads();
  }
  epilogue_free<128>(sm, taddr, n_acc, d.err);
}

// x (fp32 [T][H]) -> bf16 hi and lo parts, once per call
__global__ void k_split_x(const float4* __restrict__ x, size_t n4, uint2* __restrict__ hi, uint2* __restrict__ lo) {
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += (size_t)gridDim.x * blockDim.x) {
    const float4 v = x[i];
    const float f[4] = {v.x, v.y, v.z, v.w};
    uint32_t h[2], l[2];
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      __nv_bfloat16 h0, l0, h1, l1;
      split_bf16(f[2 * q], h0, l0);
      split_bf16(f[2 * q + 1], h1, l1);
      h[q] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
      l[q] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
    }
    hi[i] = make_uint2(h[0], h[1]);
    lo[i] = make_uint2(l[0], l[1]);
  }
}

int sm_count_p() {
  static int n = 0;
  if (!n) {
    int dev = 0, v = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
    n = v > 0 ? v : 1;
  }
  return n;
}

template <class K>
cudaError_t launch_persistent(K kernel, size_t smem, const Dev& d, int layer, int wave, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kernel<<<sm_count_p(), kThreadsP, smem, s>>>(d, layer, wave);
  return cudaGetLastError();
}

}  // namespace

bool prefill_shape_ok(int H, int I) { return H > 0 && I > 0 && H % kBM == 0 && I % kBM == 0; }

cudaError_t launch_split_x(const Dev& d, const float* x, int T, cudaStream_t s) {
  const size_t n4 = (size_t)T * d.H / 4;
  k_split_x<<<2 * sm_count_p(), 256, 0, s>>>(reinterpret_cast<const float4*>(x), n4, reinterpret_cast<uint2*>(d.xh),
                                             reinterpret_cast<uint2*>(d.xl));
  return cudaGetLastError();
}

cudaError_t launch_prefill_gateup(const Dev& d, int layer, int wave, cudaStream_t s) {
  return d.qtype == MF_Q8_0 ? launch_persistent(k_prefill_gateup<MF_Q8_0>, prefill_smem<4>(), d, layer, wave, s)
                            : launch_persistent(k_prefill_gateup<MF_Q4_0>, prefill_smem<4>(), d, layer, wave, s);
}

cudaError_t launch_prefill_down(const Dev& d, int layer, int wave, cudaStream_t s) {
  return d.qtype == MF_Q8_0 ? launch_persistent(k_prefill_down<MF_Q8_0>, prefill_smem<2>(), d, layer, wave, s)
                            : launch_persistent(k_prefill_down<MF_Q4_0>, prefill_smem<2>(), d, layer, wave, s);
}

}  // namespace mf
