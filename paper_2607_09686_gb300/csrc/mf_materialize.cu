// Materialisation of missed experts: pinned host pack -> HBM slot (section "Native Serving
// Path": on a miss the runtime copies the requested expert block into an available slot).
//
// The misses are decided on the device (slot resolve), so the copy is driven by the GPU
// itself: SMs load 16-byte vectors straight from the pinned, device-mapped pack over the
// CPU-GPU link and store them into the slot, with no host round trip.  Launched on the
// context's side stream: two blocks per SM stride over each missed payload of the wave in
// turn; with no miss every block returns at once.
#include "mf_internal.cuh"

namespace mf {
namespace {

constexpr int kUnroll = 8;

__global__ void __launch_bounds__(256) k_materialize(Dev d, int layer, int wave) {
  const int n_miss = d.info[2 + wave];
  const size_t nvec = d.lay.stride / 16;  // 16-byte vectors per payload
  const size_t step = (size_t)gridDim.x * blockDim.x * kUnroll;
  for (int m = 0; m < n_miss; ++m) {
    const int u = d.miss_list[wave * d.S_active + m];
    const uint4* src = reinterpret_cast<const uint4*>(d.pack + ((size_t)layer * d.E + d.uniq[u]) * d.lay.stride);
    uint4* dst = reinterpret_cast<uint4*>(d.pool + ((size_t)layer * d.S_alloc + d.uslot[u]) * d.lay.stride);
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

}  // namespace

cudaError_t launch_materialize(const Dev& d, int layer, int wave, int max_miss, cudaStream_t s) {
  if (max_miss <= 0) return cudaSuccess;
  static int n_sm = 0;
  if (!n_sm) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
    if (n_sm <= 0) n_sm = 1;
  }
  // two blocks per SM stream all misses of the wave; the CPU-GPU link saturates well below this
  k_materialize<<<2 * n_sm, 256, 0, s>>>(d, layer, wave);
  return cudaGetLastError();
}

}  // namespace mf
