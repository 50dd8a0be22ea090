// Deployment export: argtop_N(phi) per group (the lambda -> 0 limit of the
// Gumbel-top-N sampler, Sec. 4.2.3; the mode of the mask law of Eq. 8), packed
// as bits, with optional pruned weights (kept copied, pruned +0.0).
#include "roi_launch.h"

namespace roi {
namespace {

// One thread per output word (32 elements); groups that straddle two words are
// ranked by both threads, so no atomics are needed and any M <= 32 works.
__global__ void __launch_bounds__(256) roi_export_kernel(const float* __restrict__ phi, int N, int M, int64_t E,
                                                         uint32_t* __restrict__ bits,
                                                         const uint16_t* __restrict__ W,
                                                         uint16_t* __restrict__ Wp) {
  const int64_t nwords = (E + 31) / 32;
  for (int64_t wi = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; wi < nwords;
       wi += int64_t(gridDim.x) * blockDim.x) {
    const int64_t lo = wi * 32;
    const int64_t hi = lo + 32 < E ? lo + 32 : E;
    uint32_t word = 0;
    for (int64_t g = lo / M; g * M < hi; ++g) {
      float k[32];
      for (int l = 0; l < M; ++l) k[l] = phi[g * M + l];
      const uint32_t gb = topn_bits_dyn(k, N, M);
      for (int l = 0; l < M; ++l) {
        const int64_t e = g * M + l;
        if (e >= lo && e < hi && ((gb >> l) & 1u)) word |= 1u << (e - lo);
      }
    }
    bits[wi] = word;
    if (Wp != nullptr) {
      for (int64_t e = lo; e < hi; ++e) Wp[e] = ((word >> (e - lo)) & 1u) ? W[e] : uint16_t(0);
    }
  }
}

// M = 4 and M = 8: one thread per 32 elements with 16-byte loads.
template <int M>
__global__ void __launch_bounds__(256) roi_export_vec_kernel(const float* __restrict__ phi, int N, int64_t E,
                                                             uint32_t* __restrict__ bits,
                                                             const uint16_t* __restrict__ W,
                                                             uint16_t* __restrict__ Wp) {
  const int64_t nwords = E / 32;  // full words only; launcher handles E % 32 with the generic kernel
  for (int64_t wi = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; wi < nwords;
       wi += int64_t(gridDim.x) * blockDim.x) {
    const float4* p = reinterpret_cast<const float4*>(phi + wi * 32);
    uint32_t word = 0;
    if constexpr (M == 8) {
      // two groups at a time: threshold ranking, with the comparison-based
      // routine for non-finite keys and tied thresholds
#pragma unroll
      for (int gp = 0; gp < 2; ++gp) {
        float k[2][8];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const float4 v0 = p[(2 * gp + h) * 2], v1 = p[(2 * gp + h) * 2 + 1];
          k[h][0] = v0.x, k[h][1] = v0.y, k[h][2] = v0.z, k[h][3] = v0.w;
          k[h][4] = v1.x, k[h][5] = v1.y, k[h][6] = v1.z, k[h][7] = v1.w;
        }
        F2 kk[8];
#pragma unroll
        for (int l = 0; l < 8; ++l) kk[l] = f2(k[0][l], k[1][l]);
        const F2 ks = sum_of(kk);
        const uint32_t bad = vbelow(ks - ks, 0.0f);  // a non-finite key
        uint32_t b2[2];
        switch (N) {
          case 1: topn_bits8_threshold<1>(kk, b2); break;
          case 2: topn_bits8_threshold<2>(kk, b2); break;
          case 3: topn_bits8_threshold<3>(kk, b2); break;
          case 4: topn_bits8_threshold<4>(kk, b2); break;
          case 5: topn_bits8_threshold<5>(kk, b2); break;
          case 6: topn_bits8_threshold<6>(kk, b2); break;
          default: topn_bits8_threshold<7>(kk, b2); break;
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          if (((bad >> h) & 1u) || b2[h] == 0xffffffffu) b2[h] = topn_bits<8>(k[h], N);
          word |= b2[h] << ((2 * gp + h) * 8);
        }
      }
    } else {
#pragma unroll
      for (int g = 0; g < 32 / M; ++g) {
        float k[M];
#pragma unroll
        for (int s = 0; s < M / 4; ++s) {
          const float4 v = p[g * (M / 4) + s];
          k[4 * s] = v.x, k[4 * s + 1] = v.y, k[4 * s + 2] = v.z, k[4 * s + 3] = v.w;
        }
        word |= topn_bits<M>(k, N) << (g * M);
      }
    }
    bits[wi] = word;
    if (Wp != nullptr) {
      const uint4* wv = reinterpret_cast<const uint4*>(W + wi * 32);
      uint4* out = reinterpret_cast<uint4*>(Wp + wi * 32);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint4 v = wv[q];
        uint32_t* u = reinterpret_cast<uint32_t*>(&v);
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const int e = q * 8 + h * 2;
          const uint32_t keep_lo = (word >> e) & 1u, keep_hi = (word >> (e + 1)) & 1u;
          u[h] &= (keep_lo ? 0x0000ffffu : 0u) | (keep_hi ? 0xffff0000u : 0u);
        }
        out[q] = v;
      }
    }
  }
}

// Compressed 2:4 export.  A warp takes 1024 elements (256 groups) at a time; lane l
// holds groups l + 32 j (j < 8), so every load and store instruction of the warp is
// contiguous.  Per group: the two kept weights in index order (one 32-bit word) and
// the 4-bit code i0 | i1 << 2; the codes of the eight groups of a metadata word sit
// in eight consecutive lanes and are OR-combined with shuffles.
__global__ void __launch_bounds__(256) roi_export_2of4_kernel(const float* __restrict__ phi,
                                                              const uint16_t* __restrict__ W, int64_t E,
                                                              uint32_t* __restrict__ values,
                                                              uint32_t* __restrict__ meta) {
  const int lane = threadIdx.x & 31;
  const int64_t groups = E / 4;
  const int64_t chunks = (groups + 255) / 256;
  const int64_t warp = (blockIdx.x * int64_t(blockDim.x) + threadIdx.x) >> 5;
  const int64_t warps = (int64_t(gridDim.x) * blockDim.x) >> 5;
  const float4* p4 = reinterpret_cast<const float4*>(phi);
  const uint2* w2 = reinterpret_cast<const uint2*>(W);
  for (int64_t ch = warp; ch < chunks; ch += warps) {
    const int64_t g0 = ch * 256 + lane;
    float4 k[8];
    uint2 q[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t g = g0 + 32 * j;
      if (g < groups) {
        k[j] = p4[g];
        q[j] = w2[g];
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int64_t g = g0 + 32 * j;
      uint32_t code = 0;
      if (g < groups) {
        const float kk[4] = {k[j].x, k[j].y, k[j].z, k[j].w};
        const uint32_t bits = topn_bits4(kk, 2);
        // the two set bits of a 2-of-4 mask: lowest i0, then i1
        const uint32_t i0 = __ffs(bits) - 1u;
        const uint32_t i1 = __ffs(bits & (bits - 1u)) - 1u;
        code = i0 | (i1 << 2);
        auto at = [&q, j](uint32_t i) {
          const uint32_t half = i < 2 ? q[j].x : q[j].y;
          return (i & 1u) ? half >> 16 : half & 0xffffu;
        };
        values[g] = at(i0) | (at(i1) << 16);
      }
      uint32_t v = code << (4 * (lane & 7));
      v |= __shfl_xor_sync(0xffffffffu, v, 1);
      v |= __shfl_xor_sync(0xffffffffu, v, 2);
      v |= __shfl_xor_sync(0xffffffffu, v, 4);
      if ((lane & 7) == 0 && g < groups) meta[g >> 3] = v;
    }
  }
}

int grid_for(int64_t items, int threads) {
  int64_t blocks = (items + threads - 1) / threads;
  const int64_t cap = int64_t(sm_count()) * 8;
  if (blocks > cap) blocks = cap;
  return int(blocks < 1 ? 1 : blocks);
}

}  // namespace

int launch_export_compressed_2of4(const CompressCall& c) {
  const int64_t warps = (c.E / 4 + 255) / 256;
  roi_export_2of4_kernel<<<grid_for(warps * 32, 256), 256, 0, c.stream>>>(
      c.phi, c.W, c.E, reinterpret_cast<uint32_t*>(c.values), c.meta);
  return cudaGetLastError() == cudaSuccess ? 1 : -1;
}

int launch_export(const ExportCall& c) {
  int launched = 0;
  if ((c.M == 4 || c.M == 8) && c.E >= 32) {
    const int64_t full = c.E / 32;
    if (c.M == 4)
      roi_export_vec_kernel<4><<<grid_for(full, 256), 256, 0, c.stream>>>(c.phi, c.N, c.E, c.bits, c.W, c.Wp);
    else
      roi_export_vec_kernel<8><<<grid_for(full, 256), 256, 0, c.stream>>>(c.phi, c.N, c.E, c.bits, c.W, c.Wp);
    ++launched;
    if (cudaGetLastError() != cudaSuccess) return -1;
    if (c.E % 32 == 0) return launched;
    // last partial word
    const int64_t lo = full * 32;
    roi_export_kernel<<<1, 32, 0, c.stream>>>(c.phi + lo, c.N, c.M, c.E - lo, c.bits + full,
                                              c.W ? c.W + lo : nullptr, c.Wp ? c.Wp + lo : nullptr);
    ++launched;
    return cudaGetLastError() == cudaSuccess ? launched : -1;
  }
  roi_export_kernel<<<grid_for((c.E + 31) / 32, 256), 256, 0, c.stream>>>(c.phi, c.N, c.M, c.E, c.bits, c.W, c.Wp);
  ++launched;
  return cudaGetLastError() == cudaSuccess ? launched : -1;
}

}  // namespace roi
