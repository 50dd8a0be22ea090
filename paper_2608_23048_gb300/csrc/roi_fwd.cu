// Forward of the RoI mask op (Sec. 4.2.2 Eq. 10-12, Algorithm 1; Eq. 5 mask
// application): per group of M logits, regenerate the Gumbel noise, form the
// perturbed keys, run the N-step relaxed top-N, write Wm = bf16(W * S), and
// optionally S and the hard Gumbel-top-N bits.
#include "roi_launch.h"
#include "roi_tiles.cuh"

namespace roi {
namespace {

constexpr int kThreads = 256;
constexpr int kTile = 4096;    // elements per tile (16 KB of logits)
constexpr int kStages = 4;

struct FwdArgs {
  const float* phi;
  const uint16_t* W;
  uint16_t* Wm;
  float* soft;
  uint32_t* hard;
  int64_t E;
  int64_t full_tiles;
  float tau, inv_tau;
  NoiseParams np;
  unsigned int* status;
};

// Perturbed keys of one group of M (M % 4 == 0) starting at call-flat index e0.
template <int M>
__device__ __forceinline__ void group_keys(const float (&ph)[M], uint64_t e0, const NoiseParams& np,
                                           float (&kap)[M]) {
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    const uint4 x = noise_block(np, np.e_base + e0 + 4 * s);
    kap[4 * s + 0] = fmaf(ph[4 * s + 0], np.inv_lam, gumbel_from_word(x.x));
    kap[4 * s + 1] = fmaf(ph[4 * s + 1], np.inv_lam, gumbel_from_word(x.y));
    kap[4 * s + 2] = fmaf(ph[4 * s + 2], np.inv_lam, gumbel_from_word(x.z));
    kap[4 * s + 3] = fmaf(ph[4 * s + 3], np.inv_lam, gumbel_from_word(x.w));
  }
}

template <int M>
__device__ __forceinline__ void load_group(const float* phi_g, const uint16_t* W_g, float (&ph)[M],
                                           float (&w)[M]) {
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    const float4 p = reinterpret_cast<const float4*>(phi_g)[s];
    ph[4 * s] = p.x, ph[4 * s + 1] = p.y, ph[4 * s + 2] = p.z, ph[4 * s + 3] = p.w;
    const uint2 q = reinterpret_cast<const uint2*>(W_g)[s];
    w[4 * s + 0] = bf16_bits_to_float(q.x & 0xffffu);
    w[4 * s + 1] = bf16_bits_to_float(q.x >> 16);
    w[4 * s + 2] = bf16_bits_to_float(q.y & 0xffffu);
    w[4 * s + 3] = bf16_bits_to_float(q.y >> 16);
  }
}

// One group, one thread.  Returns the group's hard bits.
template <int N, int M, bool TAU1>
__device__ __forceinline__ uint32_t fwd_group(const float* phi_g, const uint16_t* W_g, int64_t e0,
                                              const FwdArgs& a) {
  float ph[M], w[M], kap[M];
  load_group<M>(phi_g, W_g, ph, w);
  group_keys<M>(ph, uint64_t(e0), a.np, kap);
  const uint32_t bits = topn_bits<M>(kap, N);

  FastGroup<N, M, TAU1, false> fg;
  fg.forward(kap, a.inv_tau);
  float S[M];
#pragma unroll
  for (int l = 0; l < M; ++l) S[l] = fg.S[l];
  if (fg.flag) {
    ExactGroup<N, M> ex;
    ex.forward(kap, N, M, a.tau, S);
  }

#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    uint2 o;
    o.x = pack_bf16x2(w[4 * s] * S[4 * s], w[4 * s + 1] * S[4 * s + 1]);
    o.y = pack_bf16x2(w[4 * s + 2] * S[4 * s + 2], w[4 * s + 3] * S[4 * s + 3]);
    reinterpret_cast<uint2*>(a.Wm + e0)[s] = o;
    if (a.soft != nullptr)
      reinterpret_cast<float4*>(a.soft + e0)[s] = make_float4(S[4 * s], S[4 * s + 1], S[4 * s + 2], S[4 * s + 3]);
  }
  return bits;
}

// Combine the M-bit masks of 32 / M consecutive lanes into words and store.
template <int M>
__device__ __forceinline__ void store_hard(uint32_t* hard, int64_t e0, uint32_t bits, bool active) {
  constexpr int kLanesPerWord = 32 / M;
  const int lane = threadIdx.x & 31;
  uint32_t v = active ? bits << ((lane % kLanesPerWord) * M) : 0u;
#pragma unroll
  for (int o = 1; o < kLanesPerWord; o <<= 1) v |= __shfl_xor_sync(0xffffffffu, v, o);
  if (active && (lane % kLanesPerWord) == 0) hard[e0 >> 5] = v;
}

template <int N, int M, bool TAU1>
__global__ void __launch_bounds__(kThreads) roi_fwd_kernel(FwdArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  constexpr int kGroupsPerThread = kTile / M / kThreads;
  TileSrc<2> src;
  src.ptr[0] = reinterpret_cast<const uint8_t*>(a.phi);
  src.esize[0] = 4;
  src.ptr[1] = reinterpret_cast<const uint8_t*>(a.W);
  src.esize[1] = 2;

  const bool ok = run_tiles<kThreads, kTile, kStages, 2>(
      smem, src, a.full_tiles, a.status, [&](const uint8_t* const* stage, int64_t tile) {
        const float* sphi = reinterpret_cast<const float*>(stage[0]);
        const uint16_t* sW = reinterpret_cast<const uint16_t*>(stage[1]);
        const int64_t base = tile * kTile;
#pragma unroll
        for (int j = 0; j < kGroupsPerThread; ++j) {
          const int gi = threadIdx.x + j * kThreads;
          const uint32_t bits = fwd_group<N, M, TAU1>(sphi + gi * M, sW + gi * M, base + gi * M, a);
          if (a.hard != nullptr) store_hard<M>(a.hard, base + gi * M, bits, true);
        }
      });
  if (!ok) return;

  // ragged tail (fewer than kTile elements), last CTA, straight from global memory
  if (blockIdx.x == gridDim.x - 1) {
    const int64_t t0 = a.full_tiles * kTile;
    const int64_t tail_groups = (a.E - t0) / M;
    const int64_t rounds = (tail_groups + kThreads - 1) / kThreads;
    for (int64_t r = 0; r < rounds; ++r) {
      const int64_t gi = threadIdx.x + r * kThreads;
      const bool active = gi < tail_groups;
      uint32_t bits = 0;
      if (active) bits = fwd_group<N, M, TAU1>(a.phi + t0 + gi * M, a.W + t0 + gi * M, t0 + gi * M, a);
      if (a.hard != nullptr) store_hard<M>(a.hard, t0 + gi * M, bits, active);
    }
  }
}

// Any 1 <= N < M <= 32: one thread per group, exact log-space routine, direct
// loads; hard words are zeroed beforehand and assembled with atomicOr.
__global__ void __launch_bounds__(128) roi_fwd_generic_kernel(FwdArgs a, int N, int M) {
  const int64_t groups = a.E / M;
  for (int64_t g = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; g < groups;
       g += int64_t(gridDim.x) * blockDim.x) {
    const int64_t e0 = g * M;
    float kap[32], S[32];
    for (int l = 0; l < M; ++l) {
      const uint32_t x = noise_word(a.np, a.np.e_base + uint64_t(e0 + l));
      kap[l] = fmaf(a.phi[e0 + l], a.np.inv_lam, gumbel_from_word(x));
    }
    ExactGroup<31, 32> ex;
    ex.forward(kap, N, M, a.tau, S);
    for (int l = 0; l < M; ++l) {
      const float w = bf16_bits_to_float(a.W[e0 + l]);
      a.Wm[e0 + l] = __bfloat16_as_ushort(__float2bfloat16_rn(w * S[l]));
      if (a.soft != nullptr) a.soft[e0 + l] = S[l];
    }
    if (a.hard != nullptr) {
      const uint32_t bits = topn_bits_dyn(kap, N, M);
      for (int l = 0; l < M; ++l)
        if ((bits >> l) & 1u) {
          const int64_t e = e0 + l;
          atomicOr(&a.hard[e >> 5], 1u << (e & 31));
        }
    }
  }
}

struct LaunchCache {
  int per_sm[64] = {0};
};

template <int N, int M, bool TAU1>
int launch_tiles(const FwdArgs& a, cudaStream_t stream) {
  auto kern = roi_fwd_kernel<N, M, TAU1>;
  const size_t smem = size_t(kStages) * kTile * 6 + 8 * kStages + 8;
  static LaunchCache cache;  // per instantiation and device; racing writers store the same value
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return -1;
  if (cache.per_sm[dev] == 0) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)) != cudaSuccess)
      return -1;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, smem) != cudaSuccess) return -1;
    cache.per_sm[dev] = per_sm < 1 ? 1 : per_sm;
  }
  const int64_t cap = int64_t(sm_count()) * cache.per_sm[dev];
  const int grid = int(a.full_tiles < 1 ? 1 : (a.full_tiles < cap ? a.full_tiles : cap));
  kern<<<grid, kThreads, smem, stream>>>(a);
  return cudaGetLastError() == cudaSuccess ? 1 : -1;
}

template <int N, int M>
int launch_nm(const FwdArgs& a, cudaStream_t stream) {
  return a.tau == 1.0f ? launch_tiles<N, M, true>(a, stream) : launch_tiles<N, M, false>(a, stream);
}

}  // namespace

int launch_fwd(const FwdCall& c) {
  FwdArgs a;
  a.phi = c.phi;
  a.W = c.W;
  a.Wm = c.Wm;
  a.soft = c.soft;
  a.hard = c.hard;
  a.E = c.E;
  a.full_tiles = c.E / kTile;
  a.tau = c.tau;
  a.inv_tau = 1.0f / c.tau;
  a.np = c.np;
  a.status = c.status;
  if (c.N == 2 && c.M == 4) return launch_nm<2, 4>(a, c.stream);
  if (c.N == 4 && c.M == 8) return launch_nm<4, 8>(a, c.stream);
  if (c.N == 2 && c.M == 8) return launch_nm<2, 8>(a, c.stream);
  // generic path
  int launched = 0;
  if (c.hard != nullptr) {
    if (cudaMemsetAsync(c.hard, 0, size_t((c.E + 31) / 32) * 4, c.stream) != cudaSuccess) return -1;
  }
  const int64_t groups = c.E / c.M;
  int64_t blocks = (groups + 127) / 128;
  const int64_t cap = int64_t(sm_count()) * 16;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  roi_fwd_generic_kernel<<<int(blocks), 128, 0, c.stream>>>(a, c.N, c.M);
  launched += 1;
  return cudaGetLastError() == cudaSuccess ? launched : -1;
}

}  // namespace roi
