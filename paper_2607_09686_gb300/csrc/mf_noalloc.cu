// mf_expert_ffn_noalloc: the one-token expert FFN for callers that must not allocate.
//
// It runs the same gate/up + SwiGLU and down + combine kernels as a one-token mf_moe_forward,
// but without a context: the weights are the caller's, and the scratch the kernels pass
// between each other (h, the SwiGLU activations, plus a few small index tables) lives in the
// file-scope array below instead of in a context's device allocation.
#include <atomic>
#include <cstddef>
#include <cstring>
#include <mutex>

#include "mf_internal.cuh"

namespace mf {
namespace {

constexpr int kNoAllocMaxH = kMaxTopK * 4096;  // h floats: top_k * inter <= 32768 (128 KiB)

struct NoAllocTables {
  int32_t ident[kMaxTopK];        // slot / assignment j of expert j: 0, 1, ..., 7
  int32_t asg_off[kMaxTopK + 1];  // 0, 1, ..., 8
  int32_t info[kMaxTopK][4];      // per top_k: {top_k, 1 wave, 0, 0}
  unsigned err;                   // device error word of the kernels
};

constexpr size_t kTablesOff = (size_t)kNoAllocMaxH * sizeof(float);
constexpr size_t kNoAllocBytes = kTablesOff + ((sizeof(NoAllocTables) + 255) & ~size_t(255));

// Shared by every call on this device; each GPU that loads the library keeps it until exit.
static __device__ __align__(256) unsigned char g_noalloc[kNoAllocBytes];

constexpr int kMaxDevices = 64;
std::atomic<unsigned char*> g_base[kMaxDevices];  // device address of g_noalloc, per device (set up once)
std::mutex g_setup_mu;

// Once per device, with that device current: the array's device address (host code only has a
// stand-in for the symbol) and the constant index tables.  Host threads that make their first
// call at the same time take turns (the lock); the address is published only after the tables
// have reached the device, so a first call on any stream reads complete tables.
int setup(int dev) {
  if (g_base[dev].load(std::memory_order_acquire)) return MF_OK;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  if (g_base[dev].load(std::memory_order_relaxed)) return MF_OK;
  void* p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc);
  if (e != cudaSuccess) return MF_E_CUDA;
  NoAllocTables t;
  for (int j = 0; j < kMaxTopK; ++j) {
    t.ident[j] = j;
    t.asg_off[j] = j;
    t.info[j][0] = j + 1;
    t.info[j][1] = 1;
    t.info[j][2] = 0;
    t.info[j][3] = 0;
  }
  t.asg_off[kMaxTopK] = kMaxTopK;
  t.err = 0;
  e = cudaMemcpyToSymbol(g_noalloc, &t, sizeof(t), kTablesOff, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) return MF_E_CUDA;
  if ((e = cudaDeviceSynchronize()) != cudaSuccess) return MF_E_CUDA;  // the tables have landed
  g_base[dev].store(static_cast<unsigned char*>(p), std::memory_order_release);
  return MF_OK;
}

bool valid_shape(const mf_model_t* m) {
  return m && m->hidden > 0 && m->inter > 0 && m->hidden % 32 == 0 && m->inter % 32 == 0 && m->top_k >= 1 &&
         m->top_k <= kMaxTopK && (m->qtype == MF_Q8_0 || m->qtype == MF_Q4_0) &&
         (m->qtype == MF_Q8_0 ? m->hidden / 16 : m->hidden / 32) <= 8 * 32 &&
         (m->qtype == MF_Q8_0 ? m->inter / 16 : m->inter / 32) <= 8 * 32;
}

}  // namespace
}  // namespace mf

using namespace mf;

extern "C" int mf_expert_ffn_noalloc(const mf_model_t* model, const void* experts, const float* g, const float* x,
                                     float* y, void* stream) {
  if (!valid_shape(model) || !experts || !g || !x || !y) return MF_E_INVAL;
  if ((int64_t)model->top_k * model->inter > kNoAllocMaxH) return MF_E_INVAL;  // beyond the static scratch
  if (((uintptr_t)x | (uintptr_t)experts) & 15) return MF_E_INVAL;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return MF_E_CUDA;
  int rc = setup(dev);
  if (rc) return rc;

  mf_model_t m = *model;
  m.n_layers = 1;
  m.n_experts = m.top_k;
  Dev d;
  memset(&d, 0, sizeof(d));
  d.L = 1;
  d.H = m.hidden;
  d.E = m.top_k;
  d.k = m.top_k;
  d.I = m.inter;
  d.qtype = m.qtype;
  d.S_alloc = m.top_k;
  d.S_active = m.top_k;
  d.T_max = 1;
  d.lay = make_layout(m);
  d.wait_ns = kDefaultWaitNs;
  d.pool = static_cast<uint8_t*>(const_cast<void*>(experts));  // expert j's slot at j * stride
  unsigned char* base = g_base[dev].load(std::memory_order_acquire);
  NoAllocTables* t = reinterpret_cast<NoAllocTables*>(base + kTablesOff);
  d.h = reinterpret_cast<float*>(base);
  d.uslot = t->ident;
  d.pos_slot = t->ident;
  d.asg = t->ident;
  d.asg_off = t->asg_off;
  d.info = t->info[m.top_k - 1];
  d.err = &t->err;
  d.g = const_cast<float*>(g);

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (decode_pipe_ok(d)) {
    if (launch_gateup_single(d, 0, x, s) != cudaSuccess) return MF_E_CUDA;
    if (launch_down_single_pipe(d, 0, y, s) != cudaSuccess) return MF_E_CUDA;
  } else {
    if (launch_gateup(d, 0, 0, m.top_k, x, s) != cudaSuccess) return MF_E_CUDA;
    if (launch_down_single(d, 0, y, s) != cudaSuccess) return MF_E_CUDA;
  }
  return MF_OK;
}

extern "C" int mf_expert_ffn_noalloc_check(void) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return MF_E_CUDA;
  if (!g_base[dev].load(std::memory_order_acquire)) return MF_OK;  // no call has run on this device
  if (cudaDeviceSynchronize() != cudaSuccess) return MF_E_CUDA;
  const size_t off = kTablesOff + offsetof(NoAllocTables, err);
  unsigned err = 0;
  if (cudaMemcpyFromSymbol(&err, g_noalloc, sizeof(err), off, cudaMemcpyDeviceToHost) != cudaSuccess) return MF_E_CUDA;
  if (!err) return MF_OK;
  const unsigned zero = 0;
  if (cudaMemcpyToSymbol(g_noalloc, &zero, sizeof(zero), off, cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaDeviceSynchronize() != cudaSuccess)
    return MF_E_CUDA;
  return MF_E_TIMEOUT;
}
