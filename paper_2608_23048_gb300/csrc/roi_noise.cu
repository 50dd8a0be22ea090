// The noise of a call, materialised: Philox-4x32-10 words and the Gumbel
// samples exactly as the mask kernels regenerate them in registers (Algorithm 1,
// Gumbel lines).  For inspecting or reproducing a sample; the mask op itself
// never stores noise.
#include "roi_launch.h"

namespace roi {
namespace {

__global__ void __launch_bounds__(256) roi_noise_kernel(NoiseParams np, int64_t E, uint32_t* words, float* g) {
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < E; i += int64_t(gridDim.x) * blockDim.x) {
    const uint32_t x = noise_word(np, np.e_base + uint64_t(i));
    if (words != nullptr) words[i] = x;
    if (g != nullptr) g[i] = gumbel_from_word(x);
  }
}

}  // namespace

int launch_noise(const NoiseParams& np, int64_t E, uint32_t* words, float* g, cudaStream_t stream) {
  int64_t blocks = (E + 255) / 256;
  const int64_t cap = int64_t(sm_count()) * 8;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  roi_noise_kernel<<<int(blocks), 256, 0, stream>>>(np, E, words, g);
  return cudaGetLastError() == cudaSuccess ? 1 : -1;
}

}  // namespace roi
