// Internal declarations of the GB300 routed-expert library (not part of the C ABI).
#pragma once

#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "mawforge.h"

namespace mf {

constexpr int kMaxTopK = 8;
constexpr int kMaxExperts = 1024;
constexpr int kTimerClasses = 7;
constexpr uint64_t kDefaultWaitNs = 1000000000ull;  // bounded device waits give up after 1 s by default
enum TimerClass { kTRouter = 0, kTResolve = 1, kTMaterialize = 2, kTGateUp = 3, kTDown = 4, kTPrefill = 5, kTFfn = 6 };

// Layout of one expert slot, identical in the pinned pack and in the HBM pool: row records.
// Gate/up region: I records, record r = [gate codes row r | up codes row r | gate scales row r,
// padded to 16 bytes | up scales row r], padded to 16 bytes.  Down region: H records, record
// c = [down codes row c | down scales row c], padded to 16 bytes.  Codes: Q8_0 one byte per weight stored as
// q + 128; Q4_0 the 16 code bytes of each block in GGUF order.  Scales: binary16, one per 32
// weights.  Rows that are computed together are contiguous, so a work item is one copy.
struct Layout {
  uint64_t d_off;       // byte offset of the down region (the gate/up region starts at 0)
  uint32_t rs_gu, rs_d;  // bytes per gate/up record and per down record
  uint32_t o_up, o_gs, o_us;  // inside a gate/up record: up codes, gate scales, up scales
  uint32_t o_ds;        // inside a down record: scales
  uint64_t stride;      // bytes per slot (a multiple of 256)
  uint64_t canonical;   // canonical GGUF payload bytes (what a miss accounts for)
  int qrow_gu, qrow_d;  // code bytes per row: gate/up rows (hidden weights), down rows (inter weights)
  int nb_gu, nb_d;      // 32-weight blocks per row
};

// Everything a kernel needs, passed by value.
struct Dev {
  // model
  int L, H, E, k, I, qtype;
  int S_alloc, S_active, T_max;
  int order;  // access order of calls with T > 1 (MF_ORDER_*)
  Layout lay;
  // memory
  const uint8_t* pack;  // pinned host pack [L][E] slots, device-addressable (null for a file-backed pack)
  const uint8_t* fstage;  // file-backed pack: pinned staging the host reads a call's misses into
  uint64_t fstride;       // ... bytes per staged payload (a multiple of 4096); miss r of a one-token
                          //     call (its rank r), or miss m of a wave, at fstage + index * fstride
  uint8_t* pool;        // HBM slot pool [L][S_alloc] slots
  // per-layer cache state
  int32_t* slot_of;    // [L][E]        expert -> slot or -1
  int32_t* expert_of;  // [L][S_alloc]  slot -> expert or -1
  uint64_t* last_use;  // [L][S_alloc]  LRU time of the slot's last access
  uint64_t* clock;     // [L]
  uint64_t* stats;     // [L][5]        accesses, hits, misses, evictions, bytes
  // trace of each layer's latest call
  int32_t* tr_n;       // [L]
  int32_t* tr_expert;  // [L][E]
  int32_t* tr_slot;    // [L][E]
  uint8_t* tr_hit;     // [L][E]
  // per-call scratch
  float2* zpart;       // router, T >= kTiledMinT: compensated logit pairs [K split][T][E]
  int32_t* idx;        // [T_max][k]
  float* g;            // [T_max][k]
  int32_t* uniq;       // [E]           distinct experts in access order
  int32_t* uslot;      // [E]           their slots
  int32_t* umiss;      // [E]           1 if the access missed
  int32_t* asg_off;    // [E + 1]       assignments of unique expert u: asg[asg_off[u] .. asg_off[u+1])
  int32_t* asg;        // [T_max * k]   assignment = t * k + j
  int32_t* pos_slot;   // [T_max * k]   slot serving assignment t * k + j
  int32_t* info;       // [2 + E]       U, number of waves, misses of wave w at 2 + w
  int32_t* miss_list;  // [E + S_alloc] unique index of miss m of wave w at w * S_active + m
  float* h;            // [T_max * k][I]  SwiGLU activations
  float* part;         // [T_max * k][H]  per-assignment down outputs (T > 1)
  int32_t* tb_off;     // [E + 1]       128-assignment blocks before unique expert u (T > 1)
  // tensor-core path (many tokens per expert): operand tiles in the MMA's shared-memory order,
  // per 128-assignment block t and K step kk of 32: [bf16 hi 8 KiB | bf16 lo 8 KiB]
  uint8_t* xt;         // x tiles:  t * (H / 32) + kk
  uint8_t* ht;         // h tiles:  t * (I / 32) + kk
  uint8_t* stage;      // [S_alloc] payloads: a wave's misses staged while the previous wave computes (T_max > 1)
  unsigned long long* work;  // [16]     arrival counter of the fused one-token FFN kernel (word 0)
  unsigned* err;       // [1]           nonzero after a bounded wait gave up (see MF_E_TIMEOUT)
  uint64_t wait_ns;    // time limit of every bounded device wait (mf_wait_limit)
  int hold;            // test hold (mf_test_hold): the fused FFN's producer issues no copies
};

// ---- shared-memory pipeline primitives (mbarrier + bulk asynchronous copy, PTX ISA 8.x)
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Nanoseconds of the GPU's global timer.
__device__ __forceinline__ uint64_t gtimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Poll-count backstop of every bounded wait, should the global timer not advance.
constexpr uint32_t kWaitPolls = 1u << 26;
// try_wait that may suspend the thread for up to `hint_ns` (it resumes as soon as the phase
// completes): a waiting warp then takes no issue slots from the warps doing the work.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3; selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}
// Bounded wait for the phase with the given parity; false once `limit_ns` nanoseconds have passed
// since the first failed poll (an error, never a hang: the caller records it and stops using the
// pipeline).  Between polls the thread sleeps in the barrier (at most 20 us per poll).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = gtimer_ns();
  for (uint32_t i = 0; i < kWaitPolls; ++i) {
    if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
    if (gtimer_ns() - t0 > limit_ns) return false;
  }
  return false;
}
// Bounded wait until the 64-bit counter reaches `target` (acquire: what the adders released
// before their additions is visible afterwards); false once `limit_ns` nanoseconds have passed.
__device__ __forceinline__ bool counter_wait(const unsigned long long* cnt, unsigned long long target,
                                             uint64_t limit_ns) {
  uint64_t t0 = 0;
  for (uint32_t i = 0; i < kWaitPolls; ++i) {
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(cnt) : "memory");
    if (v >= target) return true;
    if (i == 0) t0 = gtimer_ns();
    if (i >= 32) {
      if (gtimer_ns() - t0 > limit_ns) return false;
      __nanosleep(32);
    }
  }
  return false;
}
// Programmatic dependent launch (PTX griddepcontrol).  pdl_wait: block until the grid this launch
// depends on has completed and its memory operations are visible (returns at once when the
// launch was not programmatic); everything before it may overlap the predecessor's tail and must
// touch no global memory the predecessor or the caller's earlier work could write.
// pdl_trigger: allow the dependent launch to be scheduled (its blocks start as SMs free up).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
// bulk copy global -> this CTA's shared memory, completing `bytes` on the mbarrier
// (addresses 16-byte aligned, bytes a multiple of 16)
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}
// L2 eviction-priority policies for cache hints: expert weights are streamed once per call
// (evict first), router weights are read again by the next call of the layer (evict last)
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// bulk_g2s with an L2 cache-hint policy
__device__ __forceinline__ void bulk_g2s_hint(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                              uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
      : "memory");
}
// read-only 16-byte load with an L2 cache-hint policy
__device__ __forceinline__ float4 ld_hint(const float4* p, uint64_t pol) {
  float4 v;
  asm volatile("ld.global.nc.L2::cache_hint.v4.f32 {%0,%1,%2,%3}, [%4], %5;"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ void named_bar_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// 16-byte streaming load that does not allocate in L1 (weights are read once per call)
__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

}  // namespace mf

namespace mf {
struct PackFile;  // mf_packfile.cu
}

struct mf_ctx {
  mf_model_t model;
  mf_plan_t plan;
  int device;
  mf::Dev d;
  uint8_t* pack_host;      // cudaHostAlloc'ed pack (host pointer; null for a file-backed pack)
  mf::PackFile* file;      // the split-pack file of a file-backed context (else null)
  unsigned char* put_map;  // [L][E] which payloads have been put
  int64_t n_put;
  cudaStream_t side;       // materialisation stream
  int max_waves;
  cudaEvent_t* ev_fork;    // [max_waves + 1]
  cudaEvent_t* ev_join;    // [max_waves + 1]
  // staging for mf_moe_forward_host
  float* stage_x;
  float* stage_bias;
  float* stage_y;
  int32_t* stage_idx;
  float* stage_w;
  // event timing
  unsigned timing;  // bit i set: kernel class i is timed
  int timer_cap;
  int timer_n[mf::kTimerClasses];
  int64_t timer_dropped;
  cudaEvent_t* timer_ev[mf::kTimerClasses];  // pairs: [2 * i], [2 * i + 1]
  uint64_t overhead_bytes;
  bool decode_pipe;  // batch-1 calls use the pipelined decode kernels
  bool ffn_fused;    // ... fused into one cooperative launch
  int prefill_min_t;  // calls with T >= this use the tensor-core grouped GEMMs (0 = never)
  uint8_t* gemm_scratch;  // x and h tiles of the tensor-core path (allocated when first enabled)
  bool tmaps_ok;
  CUtensorMap tm_gu[2], tm_d[2];  // the slot pool's gate/up and down row records as 3-D byte tensors:
                                  // [0] boxes of one step's codes, [1] boxes of one scale group
};

namespace mf {

// layout of a slot for a model shape
Layout make_layout(const mf_model_t& m);
uint64_t canonical_payload_bytes(const mf_model_t& m);

// kernel launchers (each returns the launch status)
// x and bias may be pinned host memory; with x_copy, the router also writes x there (device)
// calls with at least this many tokens take the tiled router (W_r read once per 32 tokens)
constexpr int kTiledMinT = 16;
// pairs of zpart the tiled router needs for any T in [kTiledMinT, T_max] (0 below that)
size_t router_part_pairs(int T_max, int E, int H);
cudaError_t launch_router(const Dev& d, const float* x, const float* wr, const float* bias, int T, int layer,
                          cudaStream_t s, float* x_copy = nullptr);
cudaError_t launch_resolve(const Dev& d, int layer, int T, cudaStream_t s);
// dst_stage null: each miss into its slot; else miss m of the wave to dst_stage + m * stride.
// spread: one small block per SM (beside the persistent GEMM kernels), else a few large blocks
cudaError_t launch_materialize(const Dev& d, int layer, int wave, int max_miss, cudaStream_t s,
                               uint8_t* dst_stage = nullptr, bool spread = false);
// the wave's staged payloads into their slots
cudaError_t launch_stage_commit(const Dev& d, int layer, int wave, const uint8_t* stage, cudaStream_t s);
cudaError_t launch_gateup(const Dev& d, int layer, int wave, int wave_width, const float* x, cudaStream_t s);
cudaError_t launch_down_single(const Dev& d, int layer, float* y, cudaStream_t s);
cudaError_t launch_down_partial(const Dev& d, int layer, int wave, int wave_width, cudaStream_t s);
cudaError_t launch_combine(const Dev& d, int T, float* y, cudaStream_t s);
cudaError_t launch_reset(const Dev& d, cudaStream_t s);
// batch-1 decode: pipelined gate/up + SwiGLU and down + combine (shared-memory bulk-copy stages)
cudaError_t launch_gateup_single(const Dev& d, int layer, const float* x, cudaStream_t s);
cudaError_t launch_down_single_pipe(const Dev& d, int layer, float* y, cudaStream_t s);
size_t decode_smem_bytes(const Dev& d, int which);
bool decode_pipe_ok(const Dev& d);
// both projections of one token in one cooperative launch (d.work holds its arrival counter)
bool ffn_fused_ok(const Dev& d);
cudaError_t launch_ffn_single(const Dev& d, int layer, const float* x, float* y, cudaStream_t s);
// many tokens per expert: tcgen05 grouped GEMMs (gate/up + SwiGLU, down) per wave
constexpr int kPrefillMinTokens = 256;
bool prefill_shape_ok(int hidden, int inter);
uint64_t prefill_tiles_max(int T, int k, int E);  // bound on the 128-assignment blocks of a call
uint64_t prefill_scratch_bytes(int T_max, int k, int E, int hidden, int inter);
int prefill_tensor_maps(mf_ctx* c);  // encode tm_gu / tm_d for the context's pool; 0 on success
cudaError_t launch_tile_x(const Dev& d, const float* x, int T, cudaStream_t s);
cudaError_t launch_prefill_gateup(const Dev& d, const CUtensorMap* tm, int layer, int wave, cudaStream_t s);
cudaError_t launch_prefill_down(const Dev& d, const CUtensorMap* tm, int layer, int wave, cudaStream_t s);
// file-backed split-pack (mf_packfile.cu)
int open_pack_file(mf_ctx* c, const char* path);  // MF_OK or an MF_E_* code
void close_pack_file(mf_ctx* c);
int pack_file_error(mf_ctx* c);  // errno of a failed read since the last call (0: none), cleared
// a host function on `s` that reads the missed records of `layer` (one token: the call's misses
// by rank; else wave `wave`'s misses in order) from the file into the staging
cudaError_t enqueue_file_reads(mf_ctx* c, int layer, int wave, bool one_token, cudaStream_t s);

}  // namespace mf
