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
// Operand B never needs a gather inside the GEMM: once per call k_tile_x writes x, split, in
// the MMA's shared-memory order per (128-assignment block, K step of 32) -- 16 KiB tiles that
// one bulk copy moves -- and the gate/up epilogue writes h the same way for the down GEMM.
//
// Work unit = (expert of the wave, block of 128 assignments, block of 128 weight rows); one
// CTA of 14 warps per SM walks its units as a flat sequence of K steps of 32 (one quantisation
// block), with warp-specialised roles linked by mbarriers:
//   producer (1 warp)    per step: one TMA load per weight tensor (the 128 rows' codes of the
//                        block, from a 3-D tensor map over the slot pool) into a 3-slot raw ring,
//                        every 8 steps one TMA load per tensor of the rows' next 8 scales into a
//                        2-group scale ring, and one bulk copy of the B tile into operand stage
//                        s % 4 (lane 0 issues the copies);
//   converters (8 warps) dequantise the raw codes exactly into the stage's A tiles (hi / lo,
//                        no-swizzle K-major core-matrix layout): byte -> float by the
//                        magic-number conversion, times the binary16 scale, split with packed
//                        bf16x2 conversions;
//   MMA (1 thread)       issues the step's tcgen05.mma (M = 128, K = 16, N = the block's assignments
//                        rounded up to a multiple of 16) into one of two
//                        TMEM accumulators and commits them to the stage's mbarrier;
//   epilogue (4 warps)   reads a finished accumulator with tcgen05.ld (warp w: TMEM lanes
//                        32 (w % 4) .. +31) while the MMAs of the next unit use the other one.
// Every wait is bounded; a wait that gives up sets the block's flag and the device error word,
// the roles leave their loops, and the block drains its copies and MMAs (bounded) and frees
// its tensor memory before returning.
#include <cuda_bf16.h>

#include "mf_dequant.cuh"

namespace mf {
namespace {

using dq::f2_add;
using dq::f2_fma;
using dq::f2_pack;

constexpr int kBM = 128, kBN = 128, kBK = 32;
constexpr int kStages = 4;  // operand stages (A + B tiles)
constexpr int kRaw = 3;     // raw-code ring slots
constexpr uint32_t kTile = kBM * kBK * 2;  // one bf16 tile: 128 rows x 32 k = 8 KiB
constexpr uint32_t kBTile = 2 * kTile;     // B hi + lo, one bulk copy

// warp roles of the 448-thread CTA
constexpr int kConvWarps = 8;  // warps 0-7: dequantise A tiles
constexpr int kProdWarp = 8;   // warp 8: copies
constexpr int kMmaWarp = 9;    // warp 9, lane 0: MMA issue
constexpr int kEpiWarp0 = 10;  // warps 10-13: epilogue; TMEM lane quarter = warp % 4
constexpr int kThreadsW = 14 * 32;
static_assert(kEpiWarp0 == kMmaWarp + 1 && kEpiWarp0 + 4 == kThreadsW / 32, "warp roles");

// Byte offset of element (row r, k) in a K-major no-swizzle tile of 128 x 32: 8x8 core
// matrices of 128 contiguous bytes, K-adjacent core matrices 128 B apart (the descriptor's
// leading byte offset), 8-row groups 512 B apart (its stride byte offset).
__host__ __device__ __forceinline__ uint32_t core_off(int r, int k) {
  return (uint32_t)((r >> 3) * 512 + (k >> 3) * 128 + (r & 7) * 16 + (k & 7) * 2);
}

// shared-memory matrix descriptor: start >> 4, LBO >> 4 at bit 16, SBO >> 4 at bit 32,
// descriptor version 1 at bit 46, no swizzle
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr) {
  return (uint64_t)((addr >> 4) & 0x3FFF) | ((uint64_t)(128u >> 4) << 16) | ((uint64_t)(512u >> 4) << 32) |
         ((uint64_t)1 << 46);
}

// kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B, both K-major, M = 128 x N
// (N a multiple of 16, at most 128 here)
__device__ __forceinline__ uint32_t idesc_n(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
}
// the MMA width of a block with n assignments: n rounded up to a multiple of 16
__device__ __forceinline__ int n_eff(int n) { return max(16, (n + 15) & ~15); }

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.u32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(accumulate));
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

// 3-D tiled TMA load of a box at (x, y, z) of `tmap` into shared memory, completing on `bar`
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* tmap, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

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

__device__ __forceinline__ uint32_t bf2_bits(__nv_bfloat162 v) { return *reinterpret_cast<uint32_t*>(&v); }

__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// Two values (packed fp32 pair) -> bf16x2 words hi = bf16(v), lo = bf16(v - hi).
__device__ __forceinline__ void split2(uint64_t w, uint32_t& hi, uint32_t& lo) {
  uint32_t a, b;
  asm("mov.b64 {%0, %1}, %2;" : "=r"(a), "=r"(b) : "l"(w));
  const __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(a), __uint_as_float(b));
  const float2 hf = __bfloat1622float2(h);
  const uint64_t r = f2_fma(f2_pack(__float_as_uint(hf.x), __float_as_uint(hf.y)), f2_pack(0xBF800000u, 0xBF800000u), w);
  uint32_t ra, rb;
  asm("mov.b64 {%0, %1}, %2;" : "=r"(ra), "=r"(rb) : "l"(r));
  hi = bf2_bits(h);
  lo = bf2_bits(__floats2bfloat162_rn(__uint_as_float(ra), __uint_as_float(rb)));
}

// Eight byte codes c (two words; Q8_0 c = q + 128, Q4_0 nibbles masked to bytes) times the
// scale dd = (d, d) -> one 16-byte chunk of the hi tile and of the lo tile at `off`.
template <uint32_t kOffBits>
__device__ __forceinline__ void dequant8(uint32_t w0, uint32_t w1, uint64_t dd, unsigned char* hi_t,
                                         unsigned char* lo_t, uint32_t off) {
  const uint64_t neg = f2_pack(kOffBits | 0x80000000u, kOffBits | 0x80000000u);  // -(2^23 + offset)
  const uint32_t ws[2] = {w0, w1};
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const uint64_t q01 =
        f2_add(f2_pack(__byte_perm(ws[i], 0x4B000000u, 0x7650), __byte_perm(ws[i], 0x4B000000u, 0x7651)), neg);
    const uint64_t q23 =
        f2_add(f2_pack(__byte_perm(ws[i], 0x4B000000u, 0x7652), __byte_perm(ws[i], 0x4B000000u, 0x7653)), neg);
    split2(f2_mul(q01, dd), h[2 * i], l[2 * i]);
    split2(f2_mul(q23, dd), h[2 * i + 1], l[2 * i + 1]);
  }
  *reinterpret_cast<uint4*>(hi_t + off) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4*>(lo_t + off) = make_uint4(l[0], l[1], l[2], l[3]);
}

struct Unit {
  int u;   // unique-expert index (access order)
  int tb;  // block of 128 assignments
  int rb;  // block of 128 weight rows
};

// The wave's units, expert by expert: expert u0 + e has ceil(n / 128) assignment blocks times
// `nrb` row blocks, row blocks innermost (CTAs working on the same assignment block at once
// share its B tiles in L2).  Unit i is row block i % nrb of the wave's assignment block i / nrb,
// found in the exclusive prefix of assignment blocks per unique expert (tb_off).
struct UnitMap {
  int u0, nu, nrb, total;
  const int* tb_off;
  __device__ __forceinline__ Unit at(int i) const {
    const int ti = __ldg(&tb_off[u0]) + i / nrb;
    int lo = u0, hi = u0 + nu - 1;
    while (lo < hi) {  // last expert whose first assignment block is at or before ti
      const int mid = (lo + hi + 1) >> 1;
      if (__ldg(&tb_off[mid]) <= ti) lo = mid;
      else hi = mid - 1;
    }
    return {lo, ti - __ldg(&tb_off[lo]), i % nrb};
  }
};

// Scales travel in groups of kGroup K steps: one 16-byte TMA box per (tensor, row) holds the
// group's 8 binary16 scales.  A group's buffer is loaded again two groups later, once the
// producer has seen the raw slot of a step of the group in between freed; every group but a
// unit's last has 8 steps and the last has 4 or 8 (K is a multiple of 128), so that step lies
// inside the group in between whenever the raw ring has at most 4 slots.
constexpr int kGroup = 8;
constexpr uint32_t kScaleBox = 16;
static_assert(kRaw <= 4 && kGroup * 2 == (int)kScaleBox, "scale groups");

// Shared memory of one CTA: operand stages, raw ring, scale ring, barriers.
template <int NT, int CB>  // tensors per step (2: gate and up, 1: down), code bytes per 32-weight block
struct PLayout {
  static constexpr int kNA = 2 * NT;                          // A tiles per stage: hi / lo per tensor
  static constexpr uint32_t kStage = kNA * kTile + kBTile;    // + B hi / lo
  static constexpr uint32_t kRawSlot = NT * kBM * CB;         // codes of one step (TMA boxes)
  static constexpr uint32_t kScaleBuf = NT * kBM * kScaleBox;  // scales of one group (TMA boxes)
  static constexpr int kBars = 2 * kRaw + 2 * kStages + 2 * 2 + 1;
  static constexpr uint32_t kOffRaw = kStages * kStage;
  static constexpr uint32_t kOffScale = kOffRaw + kRaw * kRawSlot;
  static constexpr uint32_t kOffBar = kOffScale + 2 * kScaleBuf;
  static constexpr uint32_t kOffMisc = kOffBar + kBars * 8;
  static constexpr uint32_t kBytes = kOffMisc + 16;
  static_assert(kRawSlot % 128 == 0 && kOffRaw % 128 == 0 && kOffScale % 128 == 0 && kScaleBuf % 128 == 0,
                "TMA destinations are 128-byte aligned");
};

// Gate/up (NT = 2) or down (NT = 1) projection of wave `wave` for every assignment of the wave.
//   gate/up: A = gate / up rows of the slot's gate/up region, B = x tiles; epilogue
//            h = silu(G) * U, split, into the h tiles
//   down:    A = down rows, B = h tiles; epilogue part[assignment][hidden]
// Pipeline (mbarriers): producer --full--> converters --a_ready--> MMA --mma_done--> producer
// (B slot) and converters (A slot); converters --raw_free--> producer; MMA --acc_full-->
// epilogue --acc_empty--> MMA, with two TMEM accumulators.
template <int QT, int NT>
__global__ void __launch_bounds__(kThreadsW, 1)
    k_prefill(const __grid_constant__ CUtensorMap tmap, const __grid_constant__ CUtensorMap smap, Dev d, int layer,
              int wave) {
  constexpr int CB = QT == MF_Q8_0 ? 32 : 16;
  using PL = PLayout<NT, CB>;
  constexpr uint32_t kAcc = NT * kBN;  // TMEM columns of one accumulator (gate | up, or down)
  constexpr uint32_t kCols = 2 * kAcc;
  constexpr uint32_t kOffBits = QT == MF_Q8_0 ? dq::kOffQ8 : dq::kOffQ4;
  extern __shared__ __align__(1024) unsigned char smem[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + PL::kOffBar);
  uint64_t* full = bars;                    // [kRaw]    1 expect-tx arrival (codes, scales, B tile)
  uint64_t* raw_free = full + kRaw;         // [kRaw]    one arrival per converter warp
  uint64_t* a_ready = raw_free + kRaw;      // [kStages] one arrival per converter warp
  uint64_t* mma_done = a_ready + kStages;   // [kStages] tcgen05.commit
  uint64_t* acc_full = mma_done + kStages;  // [2]       tcgen05.commit
  uint64_t* acc_empty = acc_full + 2;       // [2]       one arrival per epilogue warp
  uint64_t* drain = acc_empty + 2;          // [1]       tcgen05.commit
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(smem + PL::kOffMisc);
  volatile int* s_flag = reinterpret_cast<volatile int*>(smem + PL::kOffMisc + 4);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  const int K = NT == 2 ? d.H : d.I;            // reduction length
  const int nk = K / kBK;                       // steps per unit
  const int nrb = (NT == 2 ? d.I : d.H) / kBM;  // row blocks per expert

  // ---- prologue: barriers, tensor memory, the wave's unit prefix
  if (tid == 0) {
    for (int i = 0; i < kRaw; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&raw_free[i], kConvWarps);
    }
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&a_ready[i], kConvWarps);
      mbar_init(&mma_done[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 4);
    }
    mbar_init(drain, 1);
    *s_flag = 0;
    mbar_fence_init();
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(s_tmem)),
                 "r"(kCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  UnitMap um;
  um.u0 = wave * d.S_active;
  um.nu = max(0, min(d.S_active, d.info[0] - um.u0));
  um.nrb = nrb;
  um.tb_off = d.tb_off;
  um.total = um.nu > 0 ? (d.tb_off[um.u0 + um.nu] - d.tb_off[um.u0]) * nrb : 0;
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem0 = *s_tmem;
  const int bid = (int)blockIdx.x, nb = (int)gridDim.x;
  const int n_units = um.total > bid ? (um.total - 1 - bid) / nb + 1 : 0;
  const int n_steps = n_units * nk;

  // bounded wait; false (and the block's flag and the device error word set) once any wait gave up
  auto wait = [&](uint64_t* bar, uint32_t parity, unsigned code) -> bool {
    if (mbar_try_wait(bar, parity)) return true;  // the common case: no flag read on the fast path
    if (*s_flag) return false;
    if (mbar_wait(bar, parity, d.wait_ns)) return true;
    *s_flag = 1;
    atomicExch(d.err, code);
    return false;
  };
  // the same for a whole warp: lane 0 polls, the warp synchronises and shares the outcome
  auto warp_wait = [&](uint64_t* bar, uint32_t parity, unsigned code) -> bool { return wait(bar, parity, code); };

  if (warp < kConvWarps) {
    // ================= converters: raw codes of step s -> A tiles of stage s % kStages
    // gate/up: thread = (tensor, row), 32 weights; down: thread = (half, row), 16 weights
    const int r = tid & (kBM - 1), part = tid >> 7;
    const int ten = NT == 2 ? part : 0, tr = ten * kBM + r;
    constexpr int kGroups = NT == 2 ? 4 : 2;  // 8-weight groups of this thread
    const int g0 = NT == 2 ? 0 : part * 2;
    int kk = 0, slot = 0, stage = 0, gb = 1;
    uint32_t rph = 0, sph = 0;  // phase parities of the raw ring and of the stage ring
    uint4 sv = make_uint4(0, 0, 0, 0);  // this row's scales of the current group
    for (int s = 0; s < n_steps; ++s) {
      if (!warp_wait(&full[slot], rph, 1u)) break;
      if (s >= kStages && !warp_wait(&mma_done[stage], sph ^ 1, 2u)) break;
      const unsigned char* raw = smem + PL::kOffRaw + slot * PL::kRawSlot;
      unsigned char* a_hi = smem + stage * PL::kStage + (2 * ten) * kTile;
      unsigned char* a_lo = a_hi + kTile;
      if ((kk & (kGroup - 1)) == 0) {  // first step of a group: its scales arrived with this step's codes
        gb ^= 1;
        sv = *reinterpret_cast<const uint4*>(smem + PL::kOffScale + gb * PL::kScaleBuf + tr * kScaleBox);
      }
      const int q = (kk >> 1) & 3;
      const uint32_t sw = q == 0 ? sv.x : q == 1 ? sv.y : q == 2 ? sv.z : sv.w;
      const float dsc = __half2float(__ushort_as_half((unsigned short)((kk & 1) ? (sw >> 16) : (sw & 0xFFFFu))));
      const uint64_t dd = f2_pack(__float_as_uint(dsc), __float_as_uint(dsc));
      const unsigned char* codes = raw + (size_t)tr * CB;
      if constexpr (QT == MF_Q8_0) {
#pragma unroll
        for (int g = 0; g < kGroups; ++g) {
          const uint2 w = *reinterpret_cast<const uint2*>(codes + (g0 + g) * 8);
          dequant8<kOffBits>(w.x, w.y, dd, a_hi, a_lo, core_off(r, (g0 + g) * 8));
        }
      } else {
        // byte j: element j (low nibble), element j + 16 (high nibble): groups 0 and 1 are the
        // low nibbles of bytes 0-7 and 8-15, groups 2 and 3 their high nibbles
        const uint4 c = *reinterpret_cast<const uint4*>(codes);
        const uint32_t ws[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
        for (int g = 0; g < kGroups; ++g) {
          const int gg = g0 + g;
          const int sh = gg >= 2 ? 4 : 0, wb = (gg & 1) * 2;
          dequant8<kOffBits>((ws[wb] >> sh) & 0x0F0F0F0Fu, (ws[wb + 1] >> sh) & 0x0F0F0F0Fu, dd, a_hi, a_lo,
                             core_off(r, gg * 8));
        }
      }
      fence_async_smem();  // this thread's A writes, before the MMAs read them
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&a_ready[stage]);
        mbar_arrive(&raw_free[slot]);
      }
      if (++kk == nk) kk = 0;
      if (++slot == kRaw) slot = 0, rph ^= 1;
      if (++stage == kStages) stage = 0, sph ^= 1;
    }
  } else if (warp == kProdWarp) {
    // ================= producer (lane 0; the warp's other lanes have no role): TMA boxes of codes
    // and scales, bulk B tile
    if (lane == 0) {
    const uint8_t* tiles = NT == 2 ? d.xt : d.ht;
    int y0 = 0, z0 = 0;    // the unit's TMA coordinates: first row, slot plane
    size_t b0 = 0;         // its first B tile
    uint32_t b_bytes = 0;  // bytes of each B half the MMAs read: n_eff columns
    int kk = 0, slot = 0, stage = 0, j = 0, gb = 1;
    uint32_t rph = 0, sph = 0;
    for (int s = 0; s < n_steps; ++s) {
      if (kk == 0) {
        const Unit un = um.at(bid + j * nb);
        z0 = layer * d.S_alloc + d.uslot[un.u];
        y0 = un.rb * kBM;
        b0 = (size_t)(d.tb_off[un.u] + un.tb) * nk;
        const int a0 = d.asg_off[un.u] + un.tb * kBN;
        b_bytes = (uint32_t)n_eff(min(kBN, d.asg_off[un.u + 1] - a0)) * (kBK * 2);
      }
      if (s >= kRaw && !wait(&raw_free[slot], rph ^ 1, 3u)) break;
      if (s >= kStages && !wait(&mma_done[stage], sph ^ 1, 4u)) break;
      unsigned char* raw = smem + PL::kOffRaw + slot * PL::kRawSlot;
      const bool group = (kk & (kGroup - 1)) == 0;
      if (group) gb ^= 1;
      {
        mbar_arrive_tx(&full[slot], NT * kBM * CB + 2 * b_bytes + (group ? PL::kScaleBuf : 0u));
#pragma unroll
        for (int tn = 0; tn < NT; ++tn)
          tma_load_3d(raw + tn * kBM * CB, &tmap, (tn ? (int)d.lay.o_up : 0) + kk * CB, y0, z0, &full[slot]);
        if (group) {
          // x = the scale region's start (16-byte aligned in the slot layout) + 16 bytes per group
#pragma unroll
          for (int tn = 0; tn < NT; ++tn) {
            const uint32_t so = NT == 2 ? (tn ? d.lay.o_us : d.lay.o_gs) : d.lay.o_ds;
            tma_load_3d(smem + PL::kOffScale + gb * PL::kScaleBuf + tn * kBM * kScaleBox, &smap,
                        (int)(so + (uint32_t)(kk / kGroup) * kScaleBox), y0, z0, &full[slot]);
          }
        }
        unsigned char* bdst = smem + stage * PL::kStage + PL::kNA * kTile;
        const uint8_t* bsrc = tiles + (b0 + kk) * kBTile;
        bulk_g2s(bdst, bsrc, b_bytes, &full[slot]);                  // hi: the first n_eff columns
        bulk_g2s(bdst + kTile, bsrc + kTile, b_bytes, &full[slot]);  // lo
      }
      if (++kk == nk) kk = 0, ++j;
      if (++slot == kRaw) slot = 0, rph ^= 1;
      if (++stage == kStages) stage = 0, sph ^= 1;
    }
    }
  } else if (warp == kMmaWarp) {
    // ================= MMA issue (one thread)
    if (lane == 0) {
      int kk = 0, stage = 0, j = 0;
      uint32_t sph = 0, idesc = 0;
      for (int s = 0; s < n_steps; ++s) {
        const uint32_t acc = tmem0 + (uint32_t)(j & 1) * kAcc;
        if (kk == 0) {
          const Unit un = um.at(bid + j * nb);
          const int a0 = d.asg_off[un.u] + un.tb * kBN;
          idesc = idesc_n(n_eff(min(kBN, d.asg_off[un.u + 1] - a0)));
        }
        if (kk == 0 && j >= 2 && !wait(&acc_empty[j & 1], ((j >> 1) - 1) & 1, 8u)) break;
        if (!wait(&a_ready[stage], sph, 9u)) break;
        tc_fence_after();
        const uint32_t base = smem_u32(smem + stage * PL::kStage);
        const uint64_t bh = smem_desc(base + PL::kNA * kTile), bl = smem_desc(base + PL::kNA * kTile + kTile);
#pragma unroll
        for (int ks = 0; ks < kBK / 16; ++ks) {
          const uint64_t ko = (ks * 256) >> 4;  // K = 16 spans two core matrices
#pragma unroll
          for (int tn = 0; tn < NT; ++tn) {
            const uint64_t ah = smem_desc(base + (2 * tn) * kTile) + ko;
            const uint64_t al = smem_desc(base + (2 * tn + 1) * kTile) + ko;
            const uint32_t dt = acc + tn * kBN;
            mma_bf16(dt, ah, bh + ko, idesc, (kk | ks) != 0);
            mma_bf16(dt, ah, bl + ko, idesc, 1);
            mma_bf16(dt, al, bh + ko, idesc, 1);
          }
        }
        mma_commit(&mma_done[stage]);
        if (kk == nk - 1) mma_commit(&acc_full[j & 1]);
        if (++kk == nk) kk = 0, ++j;
        if (++stage == kStages) stage = 0, sph ^= 1;
      }
      // nothing may be in flight when the tensor memory is freed
      mma_commit(drain);
      if (!mbar_wait(drain, 0, d.wait_ns)) atomicExch(d.err, 10u);
    }
  } else {
    // ================= epilogue: accumulator j & 1 -> outputs
    const int q4 = warp & 3;  // TMEM lanes 32 q4 .. 32 q4 + 31 = weight rows of the block
    for (int j = 0; j < n_units; ++j) {
      if (!warp_wait(&acc_full[j & 1], (j >> 1) & 1, 11u)) break;
      tc_fence_after();
      const Unit un = um.at(bid + j * nb);
      const int a0 = d.asg_off[un.u] + un.tb * kBN;
      const int n = min(kBN, d.asg_off[un.u + 1] - a0);
      const int r = un.rb * kBM + q4 * 32 + lane;  // weight row = output feature
      const uint32_t lane_addr = tmem0 + (uint32_t)(j & 1) * kAcc + ((uint32_t)(q4 * 32) << 16);
      if constexpr (NT == 2) {
        // h tile of K step r / 32 of the down GEMM: this lane's row is its k = r % 32
        uint8_t* ht = d.ht + ((size_t)(d.tb_off[un.u] + un.tb) * (d.I / kBK) + (r >> 5)) * kBTile;
        for (int c0 = 0; c0 < n_eff(n); c0 += 16) {  // the columns the down MMAs read
          float g[16], u[16];
          tmem_ld16(lane_addr + c0, g);
          tmem_ld16(lane_addr + kBN + c0, u);
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const int col = c0 + q;
            const float hv = col < n ? g[q] / (1.0f + expf(-g[q])) * u[q] : 0.0f;
            const __nv_bfloat16 hi = __float2bfloat16_rn(hv);
            const uint32_t o = core_off(col, r & 31);
            *reinterpret_cast<uint16_t*>(ht + o) = __bfloat16_as_ushort(hi);
            *reinterpret_cast<uint16_t*>(ht + kTile + o) =
                __bfloat16_as_ushort(__float2bfloat16_rn(hv - __bfloat162float(hi)));
          }
        }
      } else {
        for (int c0 = 0; c0 < n; c0 += 32) {
          const int pl = c0 + lane < n ? __ldg(&d.asg[a0 + c0 + lane]) : -1;  // assignment of column c0 + lane
#pragma unroll
          for (int hlf = 0; hlf < 2; ++hlf) {
            if (c0 + hlf * 16 >= n) break;
            float v[16];
            tmem_ld16(lane_addr + c0 + hlf * 16, v);
#pragma unroll
            for (int q = 0; q < 16; ++q) {
              const int p = __shfl_sync(0xffffffffu, pl, hlf * 16 + q);
              if (p >= 0) d.part[(size_t)p * d.H + r] = v[q];
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[j & 1]);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem0), "r"(kCols));
}

// x (fp32 [T][H]) -> the x tiles of every 128-assignment block of the call: block t (of unique
// expert u, assignments asg_off[u] + 128 tb ..), K step kk: column c = assignment, row k,
// split into bf16 hi and lo; columns past the expert's assignments are zero.
__global__ void __launch_bounds__(256) k_tile_x(Dev d, const float* __restrict__ x) {
  __shared__ int s_row[kBN];
  __shared__ int s_u, s_tb;
  const int t = blockIdx.x;
  const int U = d.info[0];
  if (t >= d.tb_off[U]) return;
  if (threadIdx.x == 0) {
    int lo = 0, hi = U - 1;
    while (lo < hi) {  // last expert with tb_off[u] <= t
      const int mid = (lo + hi + 1) >> 1;
      if (d.tb_off[mid] <= t) lo = mid;
      else hi = mid - 1;
    }
    s_u = lo;
    s_tb = t - d.tb_off[lo];
  }
  __syncthreads();
  const int a0 = d.asg_off[s_u] + s_tb * kBN, n = min(kBN, d.asg_off[s_u + 1] - a0);
  for (int c = threadIdx.x; c < kBN; c += blockDim.x) s_row[c] = c < n ? d.asg[a0 + c] / d.k : -1;
  __syncthreads();
  const int nk = d.H / kBK;
  uint8_t* tile0 = d.xt + (size_t)t * nk * kBTile;
  // item i = (column i >> 2, 8-value group i & 3) of one K step: 512 per step
  for (int it = threadIdx.x; it < nk * 512; it += blockDim.x) {
    const int kk = it >> 9, i = it & 511, col = i >> 2, g = i & 3;
    uint32_t h[4] = {0, 0, 0, 0}, l[4] = {0, 0, 0, 0};
    const int row = s_row[col];
    if (row >= 0) {
      const float4* src = reinterpret_cast<const float4*>(x + (size_t)row * d.H + kk * kBK + g * 8);
      const float4 v0 = __ldg(src), v1 = __ldg(src + 1);
      split2(f2_pack(__float_as_uint(v0.x), __float_as_uint(v0.y)), h[0], l[0]);
      split2(f2_pack(__float_as_uint(v0.z), __float_as_uint(v0.w)), h[1], l[1]);
      split2(f2_pack(__float_as_uint(v1.x), __float_as_uint(v1.y)), h[2], l[2]);
      split2(f2_pack(__float_as_uint(v1.z), __float_as_uint(v1.w)), h[3], l[3]);
    }
    uint8_t* tile = tile0 + (size_t)kk * kBTile + core_off(col, g * 8);
    *reinterpret_cast<uint4*>(tile) = make_uint4(h[0], h[1], h[2], h[3]);
    *reinterpret_cast<uint4*>(tile + kTile) = make_uint4(l[0], l[1], l[2], l[3]);
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

template <int QT, int NT>
cudaError_t launch_k(const Dev& d, const CUtensorMap* tm, int layer, int wave, cudaStream_t s) {
  constexpr size_t smem = PLayout<NT, QT == MF_Q8_0 ? 32 : 16>::kBytes;
  static_assert(smem <= 232448, "shared memory per block");
  cudaError_t e = cudaFuncSetAttribute(k_prefill<QT, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_prefill<QT, NT><<<sm_count_p(), kThreadsW, smem, s>>>(tm[0], tm[1], d, layer, wave);
  return cudaGetLastError();
}

using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                 const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// One region of every slot as a 3-D byte tensor: (byte in row record, row, slot plane).
int encode_region(EncodeTiled enc, CUtensorMap* tm, void* base, uint64_t rec_bytes, uint64_t rows, uint64_t planes,
                  uint64_t plane_stride, uint32_t box_bytes) {
  const cuuint64_t dims[3] = {rec_bytes, rows, planes};
  const cuuint64_t strides[2] = {rec_bytes, plane_stride};
  const cuuint32_t box[3] = {box_bytes, (cuuint32_t)kBM, 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  return enc(tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
                 CUDA_SUCCESS
             ? 0
             : -1;
}

}  // namespace

// shapes the GEMM path serves: whole 128-row blocks in both projections (which also makes the
// scale words read in pairs lie inside each row's scales)
bool prefill_shape_ok(int H, int I) { return H > 0 && I > 0 && H % kBM == 0 && I % kBM == 0; }

// Each unique expert adds at most one partial block: sum_u ceil(n_u / 128) <= T k / 128 + min(E, T k).
uint64_t prefill_tiles_max(int T, int k, int E) {
  const uint64_t a = (uint64_t)T * k;
  return a / kBN + (a < (uint64_t)E ? a : (uint64_t)E);
}

uint64_t prefill_scratch_bytes(int T_max, int k, int E, int H, int I) {
  return prefill_tiles_max(T_max, k, E) * (uint64_t)kBN * (uint64_t)(H + I) * 4;  // hi + lo bf16
}

int prefill_tensor_maps(mf_ctx* c) {
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess || !fn)
    return -1;
  const EncodeTiled enc = reinterpret_cast<EncodeTiled>(fn);
  const Dev& d = c->d;
  const uint32_t cb = d.qtype == MF_Q8_0 ? 32 : 16;
  const uint64_t planes = (uint64_t)d.L * d.S_alloc;
  for (int m = 0; m < 2; ++m) {  // code boxes (one step), scale boxes (one group)
    const uint32_t box = m ? kScaleBox : cb;
    if (encode_region(enc, &c->tm_gu[m], d.pool, d.lay.rs_gu, (uint64_t)d.I, planes, d.lay.stride, box)) return -1;
    if (encode_region(enc, &c->tm_d[m], d.pool + d.lay.d_off, d.lay.rs_d, (uint64_t)d.H, planes, d.lay.stride, box))
      return -1;
  }
  return 0;
}

cudaError_t launch_tile_x(const Dev& d, const float* x, int T, cudaStream_t s) {
  const uint64_t blocks = prefill_tiles_max(T, d.k, d.E);
  k_tile_x<<<(unsigned)blocks, 256, 0, s>>>(d, x);
  return cudaGetLastError();
}

cudaError_t launch_prefill_gateup(const Dev& d, const CUtensorMap* tm, int layer, int wave, cudaStream_t s) {
  return d.qtype == MF_Q8_0 ? launch_k<MF_Q8_0, 2>(d, tm, layer, wave, s) : launch_k<MF_Q4_0, 2>(d, tm, layer, wave, s);
}

cudaError_t launch_prefill_down(const Dev& d, const CUtensorMap* tm, int layer, int wave, cudaStream_t s) {
  return d.qtype == MF_Q8_0 ? launch_k<MF_Q8_0, 1>(d, tm, layer, wave, s) : launch_k<MF_Q4_0, 1>(d, tm, layer, wave, s);
}

}  // namespace mf
