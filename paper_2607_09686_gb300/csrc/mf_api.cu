// C ABI entry points: static plan, context and pinned split-pack, the routed-expert step,
// counters, trace and per-kernel event timing.  Declarations and contracts: mawforge.h.
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>

#include "mf_internal.cuh"

namespace mf {

size_t resolve_smem_bytes(const Dev& d);

namespace {

thread_local char g_cuda_err[256] = "";

int cuda_fail(cudaError_t e, const char* what) {
  snprintf(g_cuda_err, sizeof(g_cuda_err), "%s: %s", what, cudaGetErrorString(e));
  return e == cudaErrorMemoryAllocation ? MF_E_OOM : MF_E_CUDA;
}

#define MF_CUDA(call)                                 \
  do {                                                \
    cudaError_t e_ = (call);                          \
    if (e_ != cudaSuccess) return cuda_fail(e_, #call); \
  } while (0)

struct DevGuard {
  int prev = -1;
  bool ok = true;
  explicit DevGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) {
      prev = -1;
      ok = cudaSetDevice(dev) == cudaSuccess;
      return;
    }
    if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DevGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

uint64_t block_bytes(int qtype) { return qtype == MF_Q8_0 ? 34 : (qtype == MF_Q4_0 ? 18 : 0); }

bool valid_model(const mf_model_t* m) {
  if (!m) return false;
  if (m->n_layers <= 0 || m->hidden <= 0 || m->inter <= 0) return false;
  if (m->hidden % 32 || m->inter % 32) return false;
  if (m->top_k < 1 || m->top_k > kMaxTopK || m->n_experts < m->top_k || m->n_experts > kMaxExperts) return false;
  if (!block_bytes(m->qtype)) return false;
  // the decode kernels hold at most 8 16-byte code vectors per lane and row
  const int vec_w = m->qtype == MF_Q8_0 ? 16 : 32;
  if (m->hidden / vec_w > 8 * 32 || m->inter / vec_w > 8 * 32) return false;
  return true;
}

uint64_t align256(uint64_t v) { return (v + 255) & ~uint64_t(255); }

int slots_for(const mf_model_t& m, double pct) {
  int S = (int)std::floor(pct * (double)m.n_experts / 100.0 + 1e-9);
  if (S < m.top_k) S = m.top_k;
  if (S > m.n_experts) S = m.n_experts;
  return S;
}

int waves_upper_bound(const mf_model_t& m, int Tm, int S) {
  long long acc = (long long)Tm * m.top_k;
  if (acc > m.n_experts) acc = m.n_experts;
  return (int)((acc + S - 1) / S);
}

// device scratch carved from one allocation
struct Carve {
  uint64_t off = 0;
  template <class T>
  uint64_t take(uint64_t count) {
    uint64_t o = off;
    off = align256(off + count * sizeof(T));
    return o;
  }
};

struct ScratchOffsets {
  uint64_t slot_of, expert_of, last_use, clock, stats, tr_n, tr_expert, tr_slot, tr_hit;
  uint64_t zpart, idx, g, uniq, uslot, umiss, asg_off, asg, pos_slot, info, miss_list, h, part;
  uint64_t work, err, tb_off, sx, sb, sy, sidx, sw, stage;
  uint64_t total;
};

ScratchOffsets scratch_layout(const mf_model_t& m, int S, int Tm) {
  ScratchOffsets o;
  Carve c;
  const uint64_t L = m.n_layers, E = m.n_experts, k = m.top_k, H = m.hidden, I = m.inter;
  o.slot_of = c.take<int32_t>(L * E);
  o.expert_of = c.take<int32_t>(L * S);
  o.last_use = c.take<uint64_t>(L * S);
  o.clock = c.take<uint64_t>(L);
  o.stats = c.take<uint64_t>(L * 5);
  o.tr_n = c.take<int32_t>(L);
  o.tr_expert = c.take<int32_t>(L * E);
  o.tr_slot = c.take<int32_t>(L * E);
  o.tr_hit = c.take<uint8_t>(L * E);
  o.zpart = c.take<float2>(router_part_pairs(Tm, (int)E, (int)H));
  o.idx = c.take<int32_t>((uint64_t)Tm * k);
  o.g = c.take<float>((uint64_t)Tm * k);
  o.uniq = c.take<int32_t>(E);
  o.uslot = c.take<int32_t>(E);
  o.umiss = c.take<int32_t>(E);
  o.asg_off = c.take<int32_t>(E + 1);
  o.asg = c.take<int32_t>((uint64_t)Tm * k);
  o.pos_slot = c.take<int32_t>((uint64_t)Tm * k);
  o.info = c.take<int32_t>(2 + E);
  o.miss_list = c.take<int32_t>(E + S);
  o.h = c.take<float>((uint64_t)Tm * k * I);
  o.part = c.take<float>(Tm > 1 ? (uint64_t)Tm * k * H : 1);
  o.work = c.take<uint64_t>(16);  // the fused FFN's grid arrival counter, alone on its 128-byte line
  o.err = c.take<unsigned>(1);
  o.tb_off = c.take<int32_t>(E + 1);
  o.sx = c.take<float>((uint64_t)Tm * H);
  o.sb = c.take<float>((uint64_t)Tm * E);
  o.sy = c.take<float>((uint64_t)Tm * H);
  o.sidx = c.take<int32_t>((uint64_t)Tm * k);
  o.sw = c.take<float>((uint64_t)Tm * k);
  // calls with several waves stage the next wave's misses: one payload per slot (T_max > 1)
  o.stage = c.take<uint8_t>(Tm > 1 ? (uint64_t)S * make_layout(m).stride : 0);
  o.total = c.off;
  return o;
}

// the tensor-core path's operand tiles are allocated with the context when max_tokens reaches
// the default threshold (else on first enabling it)
bool gemm_at_create(const mf_model_t& m, int Tm) { return Tm >= kPrefillMinTokens && prefill_shape_ok(m.hidden, m.inter); }

uint64_t overhead_bytes(const mf_model_t& m, int S, int Tm) {
  const Layout lay = make_layout(m);
  const uint64_t padding = (uint64_t)m.n_layers * S * (lay.stride - lay.canonical);
  const uint64_t gemm =
      gemm_at_create(m, Tm) ? prefill_scratch_bytes(Tm, m.top_k, m.n_experts, m.hidden, m.inter) : 0;
  return scratch_layout(m, S, Tm).total + padding + gemm;
}

int alloc_gemm_scratch(mf_ctx* c) {
  if (c->gemm_scratch) return MF_OK;
  Dev& d = c->d;
  const uint64_t tiles = prefill_tiles_max(d.T_max, d.k, d.E);
  uint8_t* p = nullptr;
  cudaError_t e = cudaMalloc((void**)&p, prefill_scratch_bytes(d.T_max, d.k, d.E, d.H, d.I));
  if (e != cudaSuccess) {
    cuda_fail(e, "cudaMalloc(GEMM tiles)");
    return MF_E_OOM;
  }
  c->gemm_scratch = p;
  d.xt = p;
  d.ht = p + tiles * (uint64_t)128 * d.H * 4;
  return MF_OK;
}

// ---- per-kernel event timing
void timer_mark(mf_ctx* c, int cls, int which, cudaStream_t s) {
  if (!(c->timing & (1u << cls))) return;
  int n = c->timer_n[cls];
  if (n >= c->timer_cap) {
    if (which == 1) c->timer_dropped++;
    return;
  }
  // inside stream capture the record must become a graph node that records on every replay
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  cudaStreamIsCapturing(s, &cap);
  if (cap == cudaStreamCaptureStatusActive)
    cudaEventRecordWithFlags(c->timer_ev[cls][2 * n + which], s, cudaEventRecordExternal);
  else
    cudaEventRecord(c->timer_ev[cls][2 * n + which], s);
  if (which == 1) c->timer_n[cls] = n + 1;
}

void free_ctx(mf_ctx* c) {
  if (!c) return;
  if (c->side) cudaStreamSynchronize(c->side);
  cudaDeviceSynchronize();
  for (int i = 0; i < kTimerClasses; ++i) {
    if (c->timer_ev[i]) {
      for (int j = 0; j < 2 * c->timer_cap; ++j)
        if (c->timer_ev[i][j]) cudaEventDestroy(c->timer_ev[i][j]);
      free(c->timer_ev[i]);
    }
  }
  if (c->ev_fork) {
    for (int w = 0; w <= c->max_waves; ++w)
      if (c->ev_fork[w]) cudaEventDestroy(c->ev_fork[w]);
    free(c->ev_fork);
  }
  if (c->ev_join) {
    for (int w = 0; w <= c->max_waves; ++w)
      if (c->ev_join[w]) cudaEventDestroy(c->ev_join[w]);
    free(c->ev_join);
  }
  if (c->side) cudaStreamDestroy(c->side);
  if (c->d.slot_of) cudaFree(c->d.slot_of);  // base of the scratch allocation
  if (c->d.pool) cudaFree(c->d.pool);
  if (c->gemm_scratch) cudaFree(c->gemm_scratch);
  if (c->pack_host) cudaFreeHost(c->pack_host);
  close_pack_file(c);
  free(c->put_map);
  delete c;
}

// Repack one canonical GGUF tensor [rows x cols] into row records: the codes of row r go to
// rec0 + r * rstride + codes_off, its binary16 scales to rec0 + r * rstride + scales_off.
// Q8_0 codes are stored offset to unsigned (q + 128), which the dequantising kernels expect.
void repack_tensor(const uint8_t* src, int rows, int cols, int qtype, uint8_t* rec0, uint32_t rstride,
                   uint32_t codes_off, uint32_t scales_off) {
  const int nb = cols / 32;
  const int bb = (int)block_bytes(qtype);
  const int cb = qtype == MF_Q8_0 ? 32 : 16;
  for (int r = 0; r < rows; ++r) {
    uint8_t* rec = rec0 + (size_t)r * rstride;
    for (int b = 0; b < nb; ++b) {
      const uint8_t* blk = src + ((size_t)r * nb + b) * bb;
      rec[scales_off + 2 * b] = blk[0];
      rec[scales_off + 2 * b + 1] = blk[1];
      uint8_t* dst = rec + codes_off + (size_t)b * cb;
      if (qtype == MF_Q8_0)
        for (int i = 0; i < cb; ++i) dst[i] = (uint8_t)(blk[2 + i] ^ 0x80u);  // q + 128, unsigned
      else
        memcpy(dst, blk + 2, (size_t)cb);
    }
  }
}

}  // namespace

uint64_t canonical_payload_bytes(const mf_model_t& m) {
  const uint64_t bb = block_bytes(m.qtype);
  return (2ull * m.inter * (m.hidden / 32) + (uint64_t)m.hidden * (m.inter / 32)) * bb;
}

Layout make_layout(const mf_model_t& m) {
  Layout l;
  const uint64_t H = m.hidden, I = m.inter;
  l.qrow_gu = m.qtype == MF_Q8_0 ? (int)H : (int)(H / 2);
  l.qrow_d = m.qtype == MF_Q8_0 ? (int)I : (int)(I / 2);
  l.nb_gu = (int)(H / 32);
  l.nb_d = (int)(I / 32);
  l.o_up = (uint32_t)l.qrow_gu;
  l.o_gs = 2u * l.qrow_gu;
  l.o_us = l.o_gs + ((2u * l.nb_gu + 15) & ~15u);  // 16-byte aligned: the GEMMs load scales by TMA box
  l.rs_gu = (uint32_t)((l.o_us + 2u * l.nb_gu + 15) & ~15u);
  l.o_ds = (uint32_t)l.qrow_d;
  l.rs_d = (uint32_t)((l.qrow_d + 2u * l.nb_d + 15) & ~15u);
  l.d_off = align256(I * l.rs_gu);
  l.stride = align256(l.d_off + H * l.rs_d);
  l.canonical = canonical_payload_bytes(m);
  return l;
}

}  // namespace mf

namespace mf {
namespace {
// A context with its pinned pack (with_pack) or, for a file-backed split-pack, without one.
int create_ctx(mf_ctx_t** out, const mf_model_t* m, const mf_plan_t* p, int device, bool with_pack) {
  if (!out || !valid_model(m) || !p) return MF_E_INVAL;
  *out = nullptr;
  if (!p->accepted) return MF_E_BUDGET;
  if (p->payload_bytes != canonical_payload_bytes(*m) || p->slots_per_layer < m->top_k ||
      p->slots_per_layer > m->n_experts || p->max_tokens < 1 || p->max_tokens > 65535)
    return MF_E_INVAL;
  DevGuard guard(device);
  if (!guard.ok) return cuda_fail(cudaSetDevice(device), "cudaSetDevice");

  mf_ctx* c = new (std::nothrow) mf_ctx();
  if (!c) return MF_E_OOM;
  c->model = *m;
  c->plan = *p;
  c->device = device;
  const int S = p->slots_per_layer, Tm = p->max_tokens;
  Dev& d = c->d;
  d.L = m->n_layers;
  d.H = m->hidden;
  d.E = m->n_experts;
  d.k = m->top_k;
  d.I = m->inter;
  d.qtype = m->qtype;
  d.S_alloc = S;
  d.S_active = S;
  d.T_max = Tm;
  d.order = MF_ORDER_FIRST_OCCURRENCE;
  d.lay = make_layout(*m);
  d.wait_ns = kDefaultWaitNs;
  d.hold = 0;

  int rc = MF_OK;
  cudaError_t e;
  if (with_pack) {
    const uint64_t pack_bytes = (uint64_t)d.L * d.E * d.lay.stride;
    e = cudaHostAlloc((void**)&c->pack_host, pack_bytes, cudaHostAllocMapped | cudaHostAllocPortable);
    if (e != cudaSuccess) {
      rc = cuda_fail(e, "cudaHostAlloc(pack)");
      if (rc == MF_E_CUDA) rc = MF_E_OOM;
      c->pack_host = nullptr;
      free_ctx(c);
      return rc;
    }
    void* dev_pack = nullptr;
    e = cudaHostGetDevicePointer(&dev_pack, c->pack_host, 0);
    if (e != cudaSuccess) {
      rc = cuda_fail(e, "cudaHostGetDevicePointer");
      free_ctx(c);
      return rc;
    }
    d.pack = static_cast<const uint8_t*>(dev_pack);
  }
  c->put_map = static_cast<unsigned char*>(calloc((size_t)d.L * d.E, 1));
  if (!c->put_map) {
    free_ctx(c);
    return MF_E_OOM;
  }
  e = cudaMalloc((void**)&d.pool, (uint64_t)d.L * S * d.lay.stride);
  if (e != cudaSuccess) {
    d.pool = nullptr;
    rc = cuda_fail(e, "cudaMalloc(pool)");
    free_ctx(c);
    return rc == MF_E_CUDA ? MF_E_OOM : rc;
  }
  const ScratchOffsets so = scratch_layout(*m, S, Tm);
  uint8_t* base = nullptr;
  e = cudaMalloc((void**)&base, so.total);
  if (e != cudaSuccess) {
    rc = cuda_fail(e, "cudaMalloc(scratch)");
    free_ctx(c);
    return rc == MF_E_CUDA ? MF_E_OOM : rc;
  }
  d.slot_of = reinterpret_cast<int32_t*>(base + so.slot_of);
  d.expert_of = reinterpret_cast<int32_t*>(base + so.expert_of);
  d.last_use = reinterpret_cast<uint64_t*>(base + so.last_use);
  d.clock = reinterpret_cast<uint64_t*>(base + so.clock);
  d.stats = reinterpret_cast<uint64_t*>(base + so.stats);
  d.tr_n = reinterpret_cast<int32_t*>(base + so.tr_n);
  d.tr_expert = reinterpret_cast<int32_t*>(base + so.tr_expert);
  d.tr_slot = reinterpret_cast<int32_t*>(base + so.tr_slot);
  d.tr_hit = reinterpret_cast<uint8_t*>(base + so.tr_hit);
  d.zpart = reinterpret_cast<float2*>(base + so.zpart);
  d.idx = reinterpret_cast<int32_t*>(base + so.idx);
  d.g = reinterpret_cast<float*>(base + so.g);
  d.uniq = reinterpret_cast<int32_t*>(base + so.uniq);
  d.uslot = reinterpret_cast<int32_t*>(base + so.uslot);
  d.umiss = reinterpret_cast<int32_t*>(base + so.umiss);
  d.asg_off = reinterpret_cast<int32_t*>(base + so.asg_off);
  d.asg = reinterpret_cast<int32_t*>(base + so.asg);
  d.pos_slot = reinterpret_cast<int32_t*>(base + so.pos_slot);
  d.info = reinterpret_cast<int32_t*>(base + so.info);
  d.miss_list = reinterpret_cast<int32_t*>(base + so.miss_list);
  d.h = reinterpret_cast<float*>(base + so.h);
  d.part = reinterpret_cast<float*>(base + so.part);
  d.work = reinterpret_cast<unsigned long long*>(base + so.work);
  d.stage = Tm > 1 ? base + so.stage : nullptr;
  d.err = reinterpret_cast<unsigned*>(base + so.err);
  d.tb_off = reinterpret_cast<int32_t*>(base + so.tb_off);
  c->stage_x = reinterpret_cast<float*>(base + so.sx);
  c->stage_bias = reinterpret_cast<float*>(base + so.sb);
  c->stage_y = reinterpret_cast<float*>(base + so.sy);
  c->stage_idx = reinterpret_cast<int32_t*>(base + so.sidx);
  c->stage_w = reinterpret_cast<float*>(base + so.sw);
  c->overhead_bytes = so.total;

  if ((e = cudaMemset(base, 0, so.total)) != cudaSuccess ||
      (e = cudaStreamCreateWithFlags(&c->side, cudaStreamNonBlocking)) != cudaSuccess) {
    rc = cuda_fail(e, "scratch init / side stream");
    free_ctx(c);
    return rc;
  }
  c->max_waves = waves_upper_bound(*m, Tm, m->top_k);
  c->ev_fork = static_cast<cudaEvent_t*>(calloc((size_t)c->max_waves + 1, sizeof(cudaEvent_t)));
  c->ev_join = static_cast<cudaEvent_t*>(calloc((size_t)c->max_waves + 1, sizeof(cudaEvent_t)));
  if (!c->ev_fork || !c->ev_join) {
    free_ctx(c);
    return MF_E_OOM;
  }
  for (int w = 0; w <= c->max_waves; ++w) {
    if ((e = cudaEventCreateWithFlags(&c->ev_fork[w], cudaEventDisableTiming)) != cudaSuccess ||
        (e = cudaEventCreateWithFlags(&c->ev_join[w], cudaEventDisableTiming)) != cudaSuccess) {
      rc = cuda_fail(e, "cudaEventCreate");
      free_ctx(c);
      return rc;
    }
  }
  if ((e = launch_reset(d, c->side)) != cudaSuccess || (e = cudaStreamSynchronize(c->side)) != cudaSuccess) {
    rc = cuda_fail(e, "reset");
    free_ctx(c);
    return rc;
  }
  size_t smem = resolve_smem_bytes(d);
  if (smem > 232448) {  // the resolve kernel's shared memory (at most 1024 experts and slots: 144 KB)
    free_ctx(c);
    return MF_E_INVAL;
  }
  c->decode_pipe = decode_pipe_ok(d) && getenv("MF_DECODE_SIMPLE") == nullptr;
  c->ffn_fused = c->decode_pipe && ffn_fused_ok(d) && getenv("MF_DECODE_UNFUSED") == nullptr;
  c->tmaps_ok = prefill_shape_ok(d.H, d.I) && prefill_tensor_maps(c) == 0;
  c->prefill_min_t = 0;
  if (c->tmaps_ok && gemm_at_create(*m, Tm)) {
    if ((rc = alloc_gemm_scratch(c)) != MF_OK) {
      free_ctx(c);
      return rc;
    }
    c->prefill_min_t = kPrefillMinTokens;
  }
  *out = c;
  return MF_OK;
}
}  // namespace
}  // namespace mf

using namespace mf;

extern "C" {

const char* mf_strerror(int status) {
  switch (status) {
    case MF_OK: return "ok";
    case MF_E_INVAL: return "invalid argument";
    case MF_E_BUDGET: return "static plan rejected: lower bound exceeds the budget";
    case MF_E_OOM: return "out of memory";
    case MF_E_CUDA: return "CUDA error";
    case MF_E_STATE: return "invalid state";
    case MF_E_TIMEOUT: return "a bounded device-side wait gave up";
    case MF_E_IO: return "reading the split-pack file failed";
    default: return "unknown status";
  }
}

const char* mf_last_cuda_error(void) { return g_cuda_err; }

int mf_payload_bytes(const mf_model_t* model, uint64_t* out) {
  if (!valid_model(model) || !out) return MF_E_INVAL;
  *out = canonical_payload_bytes(*model);
  return MF_OK;
}

int mf_plan(const mf_model_t* m, const mf_plan_req_t* r, mf_plan_t* out) {
  if (!valid_model(m) || !r || !out) return MF_E_INVAL;
  if (!(r->cache_pct >= 0.0 && r->cache_pct <= 100.0) || r->max_tokens < 0 || r->max_tokens > 65535) return MF_E_INVAL;
  mf_plan_t p;
  memset(&p, 0, sizeof(p));
  p.slots_per_layer = slots_for(*m, r->cache_pct);
  p.payload_bytes = canonical_payload_bytes(*m);
  p.pool_bytes = (uint64_t)m->n_layers * (uint64_t)p.slots_per_layer * p.payload_bytes;
  p.lower_bound_bytes = r->common_bytes + p.pool_bytes + r->kv_bytes;
  p.max_tokens = r->max_tokens > 0 ? r->max_tokens : 1;
  p.overhead_bytes = overhead_bytes(*m, p.slots_per_layer, p.max_tokens);
  p.footprint_bytes = p.lower_bound_bytes + p.overhead_bytes;
  p.accepted = p.lower_bound_bytes <= r->budget_bytes;
  *out = p;
  return p.accepted ? MF_OK : MF_E_BUDGET;
}

int mf_create(mf_ctx_t** out, const mf_model_t* m, const mf_plan_t* p, int device) {
  return create_ctx(out, m, p, device, true);
}

int mf_create_from_file(mf_ctx_t** out, const mf_model_t* m, const mf_plan_t* p, const char* path, int device) {
  if (!out || !path) return MF_E_INVAL;
  *out = nullptr;
  mf_ctx_t* c = nullptr;
  int rc = create_ctx(&c, m, p, device, false);
  if (rc) return rc;
  DevGuard guard(device);
  if ((rc = open_pack_file(c, path)) != MF_OK) {
    free_ctx(c);
    return rc;
  }
  c->n_put = (int64_t)c->d.L * c->d.E;  // every payload is in the file
  *out = c;
  return MF_OK;
}


int mf_pack_put(mf_ctx_t* c, int layer, int expert, const void* payload, uint64_t bytes) {
  if (!c || !payload || layer < 0 || layer >= c->d.L || expert < 0 || expert >= c->d.E) return MF_E_INVAL;
  if (!c->pack_host) return MF_E_STATE;  // a file-backed split-pack is read-only
  const Layout& l = c->d.lay;
  if (bytes != l.canonical) return MF_E_INVAL;
  const mf_model_t& m = c->model;
  uint8_t* dst = c->pack_host + ((uint64_t)layer * c->d.E + expert) * l.stride;
  memset(dst, 0, l.stride);  // padding stays zero
  const uint8_t* src = static_cast<const uint8_t*>(payload);
  const uint64_t tb_gu = (uint64_t)m.inter * (m.hidden / 32) * block_bytes(m.qtype);
  repack_tensor(src, m.inter, m.hidden, m.qtype, dst, l.rs_gu, 0, l.o_gs);
  repack_tensor(src + tb_gu, m.inter, m.hidden, m.qtype, dst, l.rs_gu, l.o_up, l.o_us);
  repack_tensor(src + 2 * tb_gu, m.hidden, m.inter, m.qtype, dst + l.d_off, l.rs_d, 0, l.o_ds);
  unsigned char* seen = &c->put_map[(size_t)layer * c->d.E + expert];
  if (__atomic_exchange_n(seen, (unsigned char)1, __ATOMIC_ACQ_REL) == 0) __atomic_fetch_add(&c->n_put, 1, __ATOMIC_ACQ_REL);
  return MF_OK;
}

int mf_load_pack(mf_ctx_t** out, const mf_model_t* m, const mf_plan_t* p, const void* const* payloads, int device) {
  if (!out || !payloads || !valid_model(m)) return MF_E_INVAL;
  *out = nullptr;
  for (int64_t i = 0; i < (int64_t)m->n_layers * m->n_experts; ++i)
    if (!payloads[i]) return MF_E_INVAL;
  mf_ctx_t* c = nullptr;
  int rc = mf_create(&c, m, p, device);
  if (rc) return rc;
  const uint64_t pb = canonical_payload_bytes(*m);
  for (int l = 0; l < m->n_layers; ++l)
    for (int e = 0; e < m->n_experts; ++e)
      if ((rc = mf_pack_put(c, l, e, payloads[(int64_t)l * m->n_experts + e], pb)) != MF_OK) {
        mf_destroy(c);
        return rc;
      }
  *out = c;
  return MF_OK;
}

int mf_moe_forward(mf_ctx_t* c, int layer, const float* x, const float* router_w, const float* logit_bias, int T,
                   float* y, int32_t* idx_out, float* w_out, void* stream) {
  if (!c || layer < 0 || layer >= c->d.L || T < 0 || T > c->d.T_max) return MF_E_INVAL;
  if (T == 0) return MF_OK;
  if (!x || !router_w || !y) return MF_E_INVAL;
  if (((uintptr_t)x | (uintptr_t)router_w) & 15) return MF_E_INVAL;  // float4 loads
  if (__atomic_load_n(&c->n_put, __ATOMIC_ACQUIRE) != (int64_t)c->d.L * c->d.E) return MF_E_STATE;
  DevGuard guard(c->device);
  if (!guard.ok) return cuda_fail(cudaSetDevice(c->device), "cudaSetDevice");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const Dev& d = c->d;
  const int S = d.S_active;

  timer_mark(c, kTRouter, 0, s);
  MF_CUDA(launch_router(d, x, router_w, logit_bias, T, layer, s));
  timer_mark(c, kTRouter, 1, s);
  if (T > 1) {  // one token per call: the router's last block resolved the slots already
    timer_mark(c, kTResolve, 0, s);
    MF_CUDA(launch_resolve(d, layer, T, s));
    timer_mark(c, kTResolve, 1, s);
  }

  const bool gemm = T > 1 && c->prefill_min_t > 0 && T >= c->prefill_min_t;

  if (T == 1 && c->ffn_fused) {  // one launch: expert FFN, with the misses materialised inside
    if (c->file) MF_CUDA(enqueue_file_reads(c, layer, 0, true, s));  // the misses, file -> staging
    timer_mark(c, kTFfn, 0, s);
    MF_CUDA(launch_ffn_single(d, layer, x, y, s));
    timer_mark(c, kTFfn, 1, s);
    if (idx_out) MF_CUDA(cudaMemcpyAsync(idx_out, d.idx, sizeof(int32_t) * d.k, cudaMemcpyDeviceToDevice, s));
    if (w_out) MF_CUDA(cudaMemcpyAsync(w_out, d.g, sizeof(float) * d.k, cudaMemcpyDeviceToDevice, s));
    return MF_OK;
  }

  long long accesses_max = (long long)T * d.k;
  if (accesses_max > d.E) accesses_max = d.E;
  const int n_waves = (int)((accesses_max + S - 1) / S);
  // Materialisation on the side stream.  One wave: its misses straight into their slots, then
  // the compute.  Several waves: wave 0 as above; wave w + 1's misses are staged while wave w
  // computes (their slots may still be read by it) and committed to the slots once it is done.
  const bool staged = n_waves > 1 && d.stage && !c->file;
  auto wave_width = [&](int w) {
    long long width = accesses_max - (long long)w * S;
    return (int)(width > S ? S : width);
  };
  MF_CUDA(cudaEventRecord(c->ev_fork[0], s));
  MF_CUDA(cudaStreamWaitEvent(c->side, c->ev_fork[0], 0));
  if (c->file) MF_CUDA(enqueue_file_reads(c, layer, 0, false, c->side));  // wave 0's misses, file -> staging
  timer_mark(c, kTMaterialize, 0, c->side);
  MF_CUDA(launch_materialize(d, layer, 0, wave_width(0), c->side, nullptr, gemm));
  timer_mark(c, kTMaterialize, 1, c->side);
  MF_CUDA(cudaEventRecord(c->ev_join[0], c->side));
  if (gemm) MF_CUDA(launch_tile_x(d, x, T, s));  // the GEMM's x tiles, while wave 0 materialises
  auto stage_next = [&](int w) -> cudaError_t {  // side stream: wave w's misses into the stage
    timer_mark(c, kTMaterialize, 0, c->side);
    cudaError_t e = launch_materialize(d, layer, w, wave_width(w), c->side, d.stage, gemm);
    timer_mark(c, kTMaterialize, 1, c->side);
    return e;
  };
  if (staged) MF_CUDA(stage_next(1));
  for (int w = 0; w < n_waves; ++w) {
    const int width = wave_width(w);
    if (w > 0) {  // side stream, once wave w - 1 has computed: wave w's misses into their slots
      MF_CUDA(cudaEventRecord(c->ev_fork[w], s));
      MF_CUDA(cudaStreamWaitEvent(c->side, c->ev_fork[w], 0));
      if (staged) {
        MF_CUDA(launch_stage_commit(d, layer, w, d.stage, c->side));
      } else {
        if (c->file) MF_CUDA(enqueue_file_reads(c, layer, w, false, c->side));
        timer_mark(c, kTMaterialize, 0, c->side);
        MF_CUDA(launch_materialize(d, layer, w, width, c->side, nullptr, gemm));
        timer_mark(c, kTMaterialize, 1, c->side);
      }
      MF_CUDA(cudaEventRecord(c->ev_join[w], c->side));
      if (staged && w + 1 < n_waves) MF_CUDA(stage_next(w + 1));  // overlaps wave w's compute
    }
    MF_CUDA(cudaStreamWaitEvent(s, c->ev_join[w], 0));  // wave w's experts are in their slots
    if (gemm) {
      timer_mark(c, kTPrefill, 0, s);
      MF_CUDA(launch_prefill_gateup(d, c->tm_gu, layer, w, s));
      MF_CUDA(launch_prefill_down(d, c->tm_d, layer, w, s));
      timer_mark(c, kTPrefill, 1, s);
      if (w == n_waves - 1) {
        timer_mark(c, kTDown, 0, s);
        MF_CUDA(launch_combine(d, T, y, s));
        timer_mark(c, kTDown, 1, s);
      }
      continue;
    }
    const bool pipe = T == 1 && c->decode_pipe;
    timer_mark(c, kTGateUp, 0, s);
    if (pipe)
      MF_CUDA(launch_gateup_single(d, layer, x, s));
    else
      MF_CUDA(launch_gateup(d, layer, w, (int)width, x, s));
    timer_mark(c, kTGateUp, 1, s);
    timer_mark(c, kTDown, 0, s);
    if (pipe)
      MF_CUDA(launch_down_single_pipe(d, layer, y, s));
    else if (T == 1)
      MF_CUDA(launch_down_single(d, layer, y, s));
    else
      MF_CUDA(launch_down_partial(d, layer, w, (int)width, s));
    if (T > 1 && w == n_waves - 1) MF_CUDA(launch_combine(d, T, y, s));
    timer_mark(c, kTDown, 1, s);
  }
  if (idx_out) MF_CUDA(cudaMemcpyAsync(idx_out, d.idx, sizeof(int32_t) * T * d.k, cudaMemcpyDeviceToDevice, s));
  if (w_out) MF_CUDA(cudaMemcpyAsync(w_out, d.g, sizeof(float) * T * d.k, cudaMemcpyDeviceToDevice, s));
  return MF_OK;
}

int mf_prefill_threshold(mf_ctx_t* c, int min_tokens) {
  if (!c || min_tokens < 0 || min_tokens == 1) return MF_E_INVAL;
  if (min_tokens > 0 && (c->d.T_max < 2 || !prefill_shape_ok(c->d.H, c->d.I))) return MF_E_INVAL;
  if (min_tokens > 0) {
    if (!c->tmaps_ok) return MF_E_CUDA;
    DevGuard guard(c->device);
    if (!guard.ok) return cuda_fail(cudaSetDevice(c->device), "cudaSetDevice");
    const int rc = alloc_gemm_scratch(c);
    if (rc) return rc;
  }
  c->prefill_min_t = min_tokens;
  return MF_OK;
}

int mf_access_order(mf_ctx_t* c, int order) {
  if (!c || (order != MF_ORDER_FIRST_OCCURRENCE && order != MF_ORDER_RESIDENT_FIRST)) return MF_E_INVAL;
  c->d.order = order;
  return MF_OK;
}

int mf_moe_forward_host(mf_ctx_t* c, int layer, const float* x, const float* router_w, const float* logit_bias, int T,
                        float* y, int32_t* idx_out, float* w_out, void* stream) {
  if (!c || layer < 0 || layer >= c->d.L || T < 0 || T > c->d.T_max) return MF_E_INVAL;
  if (T == 0) return MF_OK;
  if (!x || !router_w || !y) return MF_E_INVAL;
  DevGuard guard(c->device);
  if (!guard.ok) return cuda_fail(cudaSetDevice(c->device), "cudaSetDevice");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const Dev& d = c->d;
  // One token with pinned buffers: no copy steps.  The router reads x and the bias over the
  // CPU-GPU link (x once per block) and leaves a device copy of x for the FFN, which writes y
  // straight into the caller's buffer.
  if (T == 1 && c->ffn_fused && !c->file && !(((uintptr_t)x | (uintptr_t)router_w) & 15)) {
    void *xd = nullptr, *bd = nullptr, *yd = nullptr;
    bool pinned = cudaHostGetDevicePointer(&xd, const_cast<float*>(x), 0) == cudaSuccess &&
                  cudaHostGetDevicePointer(&yd, y, 0) == cudaSuccess &&
                  (!logit_bias || cudaHostGetDevicePointer(&bd, const_cast<float*>(logit_bias), 0) == cudaSuccess);
    if (!pinned) cudaGetLastError();  // pageable memory: not an error, the copy path below serves it
    if (pinned && !(reinterpret_cast<uintptr_t>(xd) & 15)) {
      if (__atomic_load_n(&c->n_put, __ATOMIC_ACQUIRE) != (int64_t)d.L * d.E) return MF_E_STATE;
      timer_mark(c, kTRouter, 0, s);
      MF_CUDA(launch_router(d, static_cast<const float*>(xd), router_w, static_cast<const float*>(bd), 1, layer, s,
                            c->stage_x));
      timer_mark(c, kTRouter, 1, s);
      timer_mark(c, kTFfn, 0, s);
      MF_CUDA(launch_ffn_single(d, layer, c->stage_x, static_cast<float*>(yd), s));
      timer_mark(c, kTFfn, 1, s);
      if (idx_out) MF_CUDA(cudaMemcpyAsync(idx_out, d.idx, sizeof(int32_t) * d.k, cudaMemcpyDeviceToHost, s));
      if (w_out) MF_CUDA(cudaMemcpyAsync(w_out, d.g, sizeof(float) * d.k, cudaMemcpyDeviceToHost, s));
      return MF_OK;
    }
  }
  MF_CUDA(cudaMemcpyAsync(c->stage_x, x, sizeof(float) * T * d.H, cudaMemcpyHostToDevice, s));
  if (logit_bias)
    MF_CUDA(cudaMemcpyAsync(c->stage_bias, logit_bias, sizeof(float) * T * d.E, cudaMemcpyHostToDevice, s));
  int rc = mf_moe_forward(c, layer, c->stage_x, router_w, logit_bias ? c->stage_bias : nullptr, T, c->stage_y,
                          nullptr, nullptr, stream);
  if (rc) return rc;
  MF_CUDA(cudaMemcpyAsync(y, c->stage_y, sizeof(float) * T * d.H, cudaMemcpyDeviceToHost, s));
  if (idx_out) MF_CUDA(cudaMemcpyAsync(idx_out, d.idx, sizeof(int32_t) * T * d.k, cudaMemcpyDeviceToHost, s));
  if (w_out) MF_CUDA(cudaMemcpyAsync(w_out, d.g, sizeof(float) * T * d.k, cudaMemcpyDeviceToHost, s));
  return MF_OK;
}

int mf_stats(mf_ctx_t* c, int layer, mf_stats_t* out, int reset) {
  if (!c || !out || layer < -1 || layer >= c->d.L) return MF_E_INVAL;
  DevGuard guard(c->device);
  if (!guard.ok) return cuda_fail(cudaSetDevice(c->device), "cudaSetDevice");
  MF_CUDA(cudaDeviceSynchronize());
  const int L = c->d.L;
  uint64_t* host = static_cast<uint64_t*>(malloc(sizeof(uint64_t) * 5 * L));
  if (!host) return MF_E_OOM;
  cudaError_t e = cudaMemcpy(host, c->d.stats, sizeof(uint64_t) * 5 * L, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) {
    free(host);
    return cuda_fail(e, "cudaMemcpy(stats)");
  }
  uint64_t acc[5] = {0, 0, 0, 0, 0};
  for (int l = 0; l < L; ++l)
    if (layer < 0 || l == layer)
      for (int i = 0; i < 5; ++i) acc[i] += host[l * 5 + i];
  free(host);
  out->accesses = acc[0];
  out->hits = acc[1];
  out->misses = acc[2];
  out->evictions = acc[3];
  out->bytes_materialized = acc[4];
  if (reset) {
    if (layer < 0)
      MF_CUDA(cudaMemset(c->d.stats, 0, sizeof(uint64_t) * 5 * L));
    else
      MF_CUDA(cudaMemset(c->d.stats + 5 * layer, 0, sizeof(uint64_t) * 5));
  }
  return MF_OK;
}

int mf_reset(mf_ctx_t* c, int slots_per_layer, void* stream) {
  if (!c) return MF_E_INVAL;
  if (slots_per_layer > 0 && (slots_per_layer < c->d.k || slots_per_layer > c->d.S_alloc)) return MF_E_INVAL;
  DevGuard guard(c->device);
  if (!guard.ok) return cuda_fail(cudaSetDevice(c->device), "cudaSetDevice");
  if (slots_per_layer > 0) c->d.S_active = slots_per_layer;
  MF_CUDA(launch_reset(c->d, static_cast<cudaStream_t>(stream)));
  return MF_OK;
}

int mf_trace(mf_ctx_t* c, int layer, int32_t* experts, int32_t* slots, uint8_t* hits, int cap, int* n) {
  if (!c || !n || layer < 0 || layer >= c->d.L || cap < 0) return MF_E_INVAL;
  DevGuard guard(c->device);
  if (!guard.ok) return cuda_fail(cudaSetDevice(c->device), "cudaSetDevice");
  MF_CUDA(cudaDeviceSynchronize());
  int32_t U = 0;
  MF_CUDA(cudaMemcpy(&U, c->d.tr_n + layer, sizeof(int32_t), cudaMemcpyDeviceToHost));
  *n = U;
  if (U > cap) return MF_E_INVAL;
  const size_t off = (size_t)layer * c->d.E;
  if (U > 0) {
    if (experts) MF_CUDA(cudaMemcpy(experts, c->d.tr_expert + off, sizeof(int32_t) * U, cudaMemcpyDeviceToHost));
    if (slots) MF_CUDA(cudaMemcpy(slots, c->d.tr_slot + off, sizeof(int32_t) * U, cudaMemcpyDeviceToHost));
    if (hits) MF_CUDA(cudaMemcpy(hits, c->d.tr_hit + off, U, cudaMemcpyDeviceToHost));
  }
  return MF_OK;
}

int mf_timing(mf_ctx_t* c, unsigned class_mask) {
  if (!c) return MF_E_INVAL;
  const unsigned enable = class_mask & ((1u << kTimerClasses) - 1);
  DevGuard guard(c->device);
  if (!guard.ok) return cuda_fail(cudaSetDevice(c->device), "cudaSetDevice");
  if (enable && !c->timer_ev[0]) {
    c->timer_cap = 16384;
    for (int i = 0; i < kTimerClasses; ++i) {
      c->timer_ev[i] = static_cast<cudaEvent_t*>(calloc((size_t)2 * c->timer_cap, sizeof(cudaEvent_t)));
      if (!c->timer_ev[i]) return MF_E_OOM;
      for (int j = 0; j < 2 * c->timer_cap; ++j) MF_CUDA(cudaEventCreate(&c->timer_ev[i][j]));
    }
  }
  MF_CUDA(cudaDeviceSynchronize());
  for (int i = 0; i < kTimerClasses; ++i) c->timer_n[i] = 0;
  c->timer_dropped = 0;
  c->timing = enable;
  return MF_OK;
}

int mf_timing_read(mf_ctx_t* c, double* ms, int64_t* launches) {
  if (!c || !ms || !launches) return MF_E_INVAL;
  DevGuard guard(c->device);
  if (!guard.ok) return cuda_fail(cudaSetDevice(c->device), "cudaSetDevice");
  MF_CUDA(cudaDeviceSynchronize());
  for (int i = 0; i < kTimerClasses; ++i) {
    double acc = 0.0;
    for (int j = 0; j < c->timer_n[i]; ++j) {
      float t = 0.f;
      MF_CUDA(cudaEventElapsedTime(&t, c->timer_ev[i][2 * j], c->timer_ev[i][2 * j + 1]));
      acc += t;
    }
    ms[i] = acc;
    launches[i] = c->timer_n[i];
  }
  return MF_OK;
}

int mf_wait_limit(mf_ctx_t* c, double seconds) {
  if (!c || !(seconds >= 1e-6 && seconds <= 60.0)) return MF_E_INVAL;
  c->d.wait_ns = (uint64_t)(seconds * 1e9);
  return MF_OK;
}

int mf_test_hold(mf_ctx_t* c, int hold) {
  if (!c || (hold != 0 && hold != 1)) return MF_E_INVAL;
  c->d.hold = hold;
  return MF_OK;
}

int mf_check(mf_ctx_t* c) {
  if (!c) return MF_E_INVAL;
  DevGuard guard(c->device);
  if (!guard.ok) return cuda_fail(cudaSetDevice(c->device), "cudaSetDevice");
  MF_CUDA(cudaDeviceSynchronize());
  unsigned err = 0;
  MF_CUDA(cudaMemcpy(&err, c->d.err, sizeof(err), cudaMemcpyDeviceToHost));
  const int io = pack_file_error(c);
  if (err) MF_CUDA(cudaMemset(c->d.err, 0, sizeof(unsigned)));
  if (io) {
    snprintf(g_cuda_err, sizeof(g_cuda_err), "split-pack file read: %s", strerror(io));
    return MF_E_IO;
  }
  return err ? MF_E_TIMEOUT : MF_OK;
}

void mf_destroy(mf_ctx_t* c) {
  if (!c) return;
  DevGuard guard(c->device);
  free_ctx(c);
}

}  // extern "C"
