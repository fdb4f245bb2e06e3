// Materialisation of missed experts: pinned host pack -> HBM slot (section "Native Serving
// Path": on a miss the runtime copies the requested expert block into an available slot).
//
// The misses are decided on the device (slot resolve), so the copy is driven by the GPU
// itself: SMs load 16-byte vectors straight from the pinned, device-mapped pack over the
// CPU-GPU link and store them into the slot, with no host round trip.  Launched on the
// context's side stream.  Grid (chunks, max misses of the wave); block m copies part of
// miss m of the wave, blocks past the wave's miss count exit at once.
#include "mf_internal.cuh"

namespace mf {
namespace {

constexpr int kUnroll = 8;

__global__ void __launch_bounds__(256) k_materialize(Dev d, int layer, int wave) {
  const int m = blockIdx.y;
  if (m >= d.info[2 + wave]) return;
  const int u = d.miss_list[wave * d.S_active + m];
  const int e = d.uniq[u], s = d.uslot[u];
  const uint4* src = reinterpret_cast<const uint4*>(d.pack + ((size_t)layer * d.E + e) * d.lay.stride);
  uint4* dst = reinterpret_cast<uint4*>(d.pool + ((size_t)layer * d.S_alloc + s) * d.lay.stride);
  const size_t nvec = d.lay.stride / 16;
  const size_t step = (size_t)gridDim.x * blockDim.x * kUnroll;
  for (size_t i = (size_t)blockIdx.x * blockDim.x * kUnroll + threadIdx.x; i < nvec; i += step) {
    uint4 v[kUnroll];
#pragma unroll
    for (int r = 0; r < kUnroll; ++r) {
      size_t j = i + (size_t)r * blockDim.x;
      if (j < nvec) v[r] = ld_stream(src + j);
    }
#pragma unroll
    for (int r = 0; r < kUnroll; ++r) {
      size_t j = i + (size_t)r * blockDim.x;
      if (j < nvec) dst[j] = v[r];
    }
  }
}

}  // namespace

cudaError_t launch_materialize(const Dev& d, int layer, int wave, int max_miss, cudaStream_t s) {
  if (max_miss <= 0) return cudaSuccess;
  const size_t nvec = d.lay.stride / 16;
  const size_t per_block = (size_t)256 * kUnroll;
  size_t chunks = (nvec + per_block - 1) / per_block;
  // enough blocks in flight to cover the link latency even when one expert misses
  size_t want = 4 * 152 / (size_t)max_miss;
  if (want < 64) want = 64;
  if (chunks > want) chunks = want;
  dim3 grid((unsigned)chunks, (unsigned)max_miss);
  k_materialize<<<grid, 256, 0, s>>>(d, layer, wave);
  return cudaGetLastError();
}

}  // namespace mf
