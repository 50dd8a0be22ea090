// Backward of the RoI mask op: regenerate the forward's noise and relaxation in
// registers, then sweep the N steps in reverse to turn dL/dS = dWm * W into
// dL/dphi (Sec. 3.2: the map from logits to the soft N-hot vector is
// differentiable; Sec. 4.2.2 Eq. 11-12).  Optionally dW = bf16(dWm * S).
#include "roi_launch.h"
#include "roi_tiles.cuh"

namespace roi {
namespace {

constexpr int kThreads = 256;
constexpr int kTile = 4096;
constexpr int kStages = 3;

struct BwdArgs {
  const float* phi;
  const uint16_t* W;
  const uint16_t* dWm;
  float* dphi;
  uint16_t* dW;
  int64_t E;
  int64_t full_tiles;
  float tau, inv_tau;
  NoiseParams np;
  unsigned int* status;
};

template <int M>
__device__ __forceinline__ void unpack4(uint2 q, float* out) {
  out[0] = bf16_bits_to_float(q.x & 0xffffu);
  out[1] = bf16_bits_to_float(q.x >> 16);
  out[2] = bf16_bits_to_float(q.y & 0xffffu);
  out[3] = bf16_bits_to_float(q.y >> 16);
}

template <int N, int M, bool TAU1>
__device__ __forceinline__ void bwd_group(const float* phi_g, const uint16_t* W_g, const uint16_t* dWm_g,
                                          int64_t e0, const BwdArgs& a) {
  float ph[M], w[M], dw[M], kap[M], c[M];
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    const float4 p = reinterpret_cast<const float4*>(phi_g)[s];
    ph[4 * s] = p.x, ph[4 * s + 1] = p.y, ph[4 * s + 2] = p.z, ph[4 * s + 3] = p.w;
    unpack4<M>(reinterpret_cast<const uint2*>(W_g)[s], w + 4 * s);
    unpack4<M>(reinterpret_cast<const uint2*>(dWm_g)[s], dw + 4 * s);
  }
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    const uint4 x = noise_block(a.np, a.np.e_base + uint64_t(e0) + 4 * s);
    kap[4 * s + 0] = fmaf(ph[4 * s + 0], a.np.inv_lam, gumbel_from_word(x.x));
    kap[4 * s + 1] = fmaf(ph[4 * s + 1], a.np.inv_lam, gumbel_from_word(x.y));
    kap[4 * s + 2] = fmaf(ph[4 * s + 2], a.np.inv_lam, gumbel_from_word(x.z));
    kap[4 * s + 3] = fmaf(ph[4 * s + 3], a.np.inv_lam, gumbel_from_word(x.w));
  }
#pragma unroll
  for (int l = 0; l < M; ++l) c[l] = dw[l] * w[l];

  FastGroup<N, M, TAU1, true> fg;
  fg.forward(kap, a.inv_tau);
  float dk[M], S[M];
  if (!fg.flag) {
    fg.backward(c, a.inv_tau, dk);
#pragma unroll
    for (int l = 0; l < M; ++l) S[l] = fg.S[l];
  } else {
    ExactGroup<N, M> ex;
    ex.forward(kap, N, M, a.tau, S);
    ex.backward(c, N, M, a.tau, dk);
  }
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    reinterpret_cast<float4*>(a.dphi + e0)[s] =
        make_float4(dk[4 * s] * a.np.inv_lam, dk[4 * s + 1] * a.np.inv_lam, dk[4 * s + 2] * a.np.inv_lam,
                    dk[4 * s + 3] * a.np.inv_lam);
    if (a.dW != nullptr) {
      uint2 o;
      o.x = pack_bf16x2(dw[4 * s] * S[4 * s], dw[4 * s + 1] * S[4 * s + 1]);
      o.y = pack_bf16x2(dw[4 * s + 2] * S[4 * s + 2], dw[4 * s + 3] * S[4 * s + 3]);
      reinterpret_cast<uint2*>(a.dW + e0)[s] = o;
    }
  }
}

template <int N, int M, bool TAU1>
__global__ void __launch_bounds__(kThreads) roi_bwd_kernel(BwdArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  constexpr int kGroupsPerThread = kTile / M / kThreads;
  TileSrc<3> src;
  src.ptr[0] = reinterpret_cast<const uint8_t*>(a.phi);
  src.esize[0] = 4;
  src.ptr[1] = reinterpret_cast<const uint8_t*>(a.W);
  src.esize[1] = 2;
  src.ptr[2] = reinterpret_cast<const uint8_t*>(a.dWm);
  src.esize[2] = 2;

  const bool ok = run_tiles<kThreads, kTile, kStages, 3>(
      smem, src, a.full_tiles, a.status, [&](const uint8_t* const* stage, int64_t tile) {
        const float* sphi = reinterpret_cast<const float*>(stage[0]);
        const uint16_t* sW = reinterpret_cast<const uint16_t*>(stage[1]);
        const uint16_t* sdW = reinterpret_cast<const uint16_t*>(stage[2]);
        const int64_t base = tile * kTile;
#pragma unroll 1
        for (int j = 0; j < kGroupsPerThread; ++j) {
          const int gi = threadIdx.x + j * kThreads;
          bwd_group<N, M, TAU1>(sphi + gi * M, sW + gi * M, sdW + gi * M, base + gi * M, a);
        }
      });
  if (!ok) return;

  if (blockIdx.x == gridDim.x - 1) {
    const int64_t t0 = a.full_tiles * kTile;
    const int64_t tail_groups = (a.E - t0) / M;
    for (int64_t gi = threadIdx.x; gi < tail_groups; gi += kThreads)
      bwd_group<N, M, TAU1>(a.phi + t0 + gi * M, a.W + t0 + gi * M, a.dWm + t0 + gi * M, t0 + gi * M, a);
  }
}

__global__ void __launch_bounds__(128) roi_bwd_generic_kernel(BwdArgs a, int N, int M) {
  const int64_t groups = a.E / M;
  for (int64_t g = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; g < groups;
       g += int64_t(gridDim.x) * blockDim.x) {
    const int64_t e0 = g * M;
    float kap[32], S[32], c[32], dk[32];
    for (int l = 0; l < M; ++l) {
      const uint32_t x = noise_word(a.np, a.np.e_base + uint64_t(e0 + l));
      kap[l] = fmaf(a.phi[e0 + l], a.np.inv_lam, gumbel_from_word(x));
      c[l] = bf16_bits_to_float(a.dWm[e0 + l]) * bf16_bits_to_float(a.W[e0 + l]);
    }
    ExactGroup<31, 32> ex;
    ex.forward(kap, N, M, a.tau, S);
    ex.backward(c, N, M, a.tau, dk);
    for (int l = 0; l < M; ++l) {
      a.dphi[e0 + l] = dk[l] * a.np.inv_lam;
      if (a.dW != nullptr)
        a.dW[e0 + l] = __bfloat16_as_ushort(__float2bfloat16_rn(bf16_bits_to_float(a.dWm[e0 + l]) * S[l]));
    }
  }
}

struct LaunchCache {
  int per_sm[64] = {0};
};

template <int N, int M, bool TAU1>
int launch_tiles(const BwdArgs& a, cudaStream_t stream) {
  auto kern = roi_bwd_kernel<N, M, TAU1>;
  const size_t smem = size_t(kStages) * kTile * 8 + 8 * kStages + 8;
  static LaunchCache cache;
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
int launch_nm(const BwdArgs& a, cudaStream_t stream) {
  return a.tau == 1.0f ? launch_tiles<N, M, true>(a, stream) : launch_tiles<N, M, false>(a, stream);
}

}  // namespace

int launch_bwd(const BwdCall& c) {
  BwdArgs a;
  a.phi = c.phi;
  a.W = c.W;
  a.dWm = c.dWm;
  a.dphi = c.dphi;
  a.dW = c.dW;
  a.E = c.E;
  a.full_tiles = c.E / kTile;
  a.tau = c.tau;
  a.inv_tau = 1.0f / c.tau;
  a.np = c.np;
  a.status = c.status;
  if (c.N == 2 && c.M == 4) return launch_nm<2, 4>(a, c.stream);
  if (c.N == 4 && c.M == 8) return launch_nm<4, 8>(a, c.stream);
  if (c.N == 2 && c.M == 8) return launch_nm<2, 8>(a, c.stream);
  const int64_t groups = c.E / c.M;
  int64_t blocks = (groups + 127) / 128;
  const int64_t cap = int64_t(sm_count()) * 16;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  roi_bwd_generic_kernel<<<int(blocks), 128, 0, c.stream>>>(a, c.N, c.M);
  return cudaGetLastError() == cudaSuccess ? 1 : -1;
}

}  // namespace roi
