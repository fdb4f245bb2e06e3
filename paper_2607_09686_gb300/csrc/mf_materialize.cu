// Materialisation of missed experts: pinned host pack -> HBM slot (section "Native Serving
// Path": on a miss the runtime copies the requested expert block into an available slot).  With
// a file-backed split-pack the host first reads the wave's misses from the file into pinned
// staging (in miss order) and the same kernel copies them from there.
//
// The misses are decided on the device (slot resolve), so the copy is driven by the GPU
// itself: SMs load 16-byte vectors straight from the pinned, device-mapped pack over the
// CPU-GPU link and store them into the slot, with no host round trip.  Launched on the
// context's side stream, blocks stride over each missed payload of the wave in turn (with no
// miss every block returns at once), 8 16-byte loads in flight per thread, 1.2 MB in all: the
// link saturates at about that.  Where they go matters for the kernel computing beside them:
// an SM with long-latency host loads outstanding serves its other blocks' memory requests
// slowly.  So the dequantising GEMV kernels (many small blocks, scheduled as SMs free up) get
// the copy concentrated on one SM in eight (large blocks), while the persistent GEMM kernels
// (one block per SM with a fixed share of the work) get it spread thin over every SM.  Both
// kernels here ask
// for the largest shared-memory carveout although they use none: an SM runs blocks of one
// carveout at a time, so only then can they share SMs with a running expert-FFN kernel (which
// needs most of the shared memory) instead of holding those SMs until they finish.
//
// Calls with several waves stage the misses of wave w + 1 (one payload per miss, in miss
// order) while wave w computes: the slots they go to may still be read by wave w.  Once wave w
// is done, k_stage_commit copies the staged payloads HBM -> HBM into their slots.
#include "mf_internal.cuh"

namespace mf {
namespace {

constexpr int kUnroll = 8;
constexpr int kMatThreadsSpread = 64;  // one block per SM
constexpr int kMatThreadsDense = 512;  // one block per 8 SMs

// dst_stage: null to write each miss into its slot, else miss m of the wave goes to
// dst_stage + m * stride
__global__ void __launch_bounds__(kMatThreadsDense) k_materialize(Dev d, int layer, int wave, uint8_t* dst_stage) {
  const int n_miss = d.info[2 + wave];
  const size_t nvec = d.lay.stride / 16;  // 16-byte vectors per payload
  const size_t step = (size_t)gridDim.x * blockDim.x * kUnroll;
  for (int m = 0; m < n_miss; ++m) {
    const int u = d.miss_list[wave * d.S_active + m];
    const uint4* src = reinterpret_cast<const uint4*>(
        d.fstage ? d.fstage + (size_t)m * d.fstride  // a file-backed pack: the host staged miss m here
                 : d.pack + ((size_t)layer * d.E + d.uniq[u]) * d.lay.stride);
    uint4* dst = reinterpret_cast<uint4*>(dst_stage ? dst_stage + (size_t)m * d.lay.stride
                                                    : d.pool + ((size_t)layer * d.S_alloc + d.uslot[u]) * d.lay.stride);
    for (size_t i0 = (size_t)blockIdx.x * blockDim.x * kUnroll + threadIdx.x; i0 < nvec; i0 += step) {
      uint4 v[kUnroll];
#pragma unroll
      for (int r = 0; r < kUnroll; ++r) {  // all loads first: kUnroll transfers in flight per thread
        const size_t i = i0 + (size_t)r * blockDim.x;
        if (i < nvec) v[r] = ld_stream(src + i);
      }
#pragma unroll
      for (int r = 0; r < kUnroll; ++r) {
        const size_t i = i0 + (size_t)r * blockDim.x;
        if (i < nvec) dst[i] = v[r];
      }
    }
  }
}

// the wave's staged payloads into their slots (HBM -> HBM)
__global__ void __launch_bounds__(256) k_stage_commit(Dev d, int layer, int wave, const uint8_t* __restrict__ stage) {
  const int n_miss = d.info[2 + wave];
  const size_t nvec = d.lay.stride / 16;
  const size_t step = (size_t)gridDim.x * blockDim.x * 4;
  for (int m = 0; m < n_miss; ++m) {
    const int u = d.miss_list[wave * d.S_active + m];
    const uint4* src = reinterpret_cast<const uint4*>(stage + (size_t)m * d.lay.stride);
    uint4* dst = reinterpret_cast<uint4*>(d.pool + ((size_t)layer * d.S_alloc + d.uslot[u]) * d.lay.stride);
    for (size_t i0 = (size_t)blockIdx.x * blockDim.x * 4 + threadIdx.x; i0 < nvec; i0 += step) {
      uint4 v[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const size_t i = i0 + (size_t)r * blockDim.x;
        if (i < nvec) v[r] = src[i];
      }
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const size_t i = i0 + (size_t)r * blockDim.x;
        if (i < nvec) dst[i] = v[r];
      }
    }
  }
}

int n_sm() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

}  // namespace

cudaError_t max_shared_carveout() {
  static cudaError_t e = [] {
    cudaError_t r = cudaFuncSetAttribute(k_materialize, cudaFuncAttributePreferredSharedMemoryCarveout,
                                         cudaSharedmemCarveoutMaxShared);
    if (r == cudaSuccess)
      r = cudaFuncSetAttribute(k_stage_commit, cudaFuncAttributePreferredSharedMemoryCarveout,
                               cudaSharedmemCarveoutMaxShared);
    return r;
  }();
  return e;
}

cudaError_t launch_materialize(const Dev& d, int layer, int wave, int max_miss, cudaStream_t s, uint8_t* dst_stage,
                               bool spread) {
  if (max_miss <= 0) return cudaSuccess;
  cudaError_t e = max_shared_carveout();
  if (e != cudaSuccess) return e;
  if (spread)
    k_materialize<<<n_sm(), kMatThreadsSpread, 0, s>>>(d, layer, wave, dst_stage);
  else
    k_materialize<<<(n_sm() + 7) / 8, kMatThreadsDense, 0, s>>>(d, layer, wave, dst_stage);
  return cudaGetLastError();
}

cudaError_t launch_stage_commit(const Dev& d, int layer, int wave, const uint8_t* stage, cudaStream_t s) {
  cudaError_t e = max_shared_carveout();
  if (e != cudaSuccess) return e;
  k_stage_commit<<<2 * n_sm(), 256, 0, s>>>(d, layer, wave, stage);
  return cudaGetLastError();
}

}  // namespace mf
