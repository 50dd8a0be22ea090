// Backward of the RoI mask op: regenerate the forward's noise and relaxation in
// registers, then sweep the N steps in reverse to turn dL/dS = dWm * W into
// dL/dphi (Sec. 3.2: the map from logits to the soft N-hot vector is
// differentiable; Sec. 4.2.2 Eq. 11-12).  Optionally dW = bf16(dWm * S).
#include "roi_launch.h"
#include "roi_tiles.cuh"

namespace roi {
namespace {

// Launch shape per group size M: threads per CTA, pairs of groups per thread per
// tile (relaxed in lockstep on packed FP32 for M = 4, one after the other for
// M = 8), shared-memory stages, and the CTAs per SM the register budget is sized for.
template <int M>
struct Cfg {
  static constexpr int kThreads = 256;
  static constexpr int kPairs = 1;
  static constexpr int kStages = M == 4 ? 3 : 2;
  static constexpr int kMinBlocks = M == 4 ? 4 : 2;
  static constexpr int kTile = 2 * kPairs * kThreads * M;  // elements
};

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

__device__ __forceinline__ void unpack4(uint2 q, float* out) {
  out[0] = bf16_bits_to_float(q.x & 0xffffu);
  out[1] = bf16_bits_to_float(q.x >> 16);
  out[2] = bf16_bits_to_float(q.y & 0xffffu);
  out[3] = bf16_bits_to_float(q.y >> 16);
}

template <class V>
__device__ __forceinline__ float lane_of(V v, int h) {
  if constexpr (vlanes<V>() == 1) {
    return v;
  } else {
    return h == 0 ? lo(v) : hi(v);
  }
}

// L groups (one per lane of V) in lockstep: regenerate keys and relaxation,
// sweep back, write dL/dphi (and dW).
template <int N, int M, bool TAU1, class V>
__device__ __forceinline__ void bwd_groups(const float* const* phi_g, const uint16_t* const* W_g,
                                           const uint16_t* const* dWm_g, const int64_t* e0, const BwdArgs& a) {
  constexpr int L = vlanes<V>();
  V kap[M], c[M];
  {
    float ph[L][M], w[L][M], dw[L][M];
    uint32_t x[L][M];
#pragma unroll
    for (int h = 0; h < L; ++h) {
      const uint64_t q0 = (a.np.e_base + uint64_t(e0[h])) >> 2;
#pragma unroll
      for (int s = 0; s < M / 4; ++s) {
        const float4 p = reinterpret_cast<const float4*>(phi_g[h])[s];
        ph[h][4 * s] = p.x, ph[h][4 * s + 1] = p.y, ph[h][4 * s + 2] = p.z, ph[h][4 * s + 3] = p.w;
        unpack4(reinterpret_cast<const uint2*>(W_g[h])[s], w[h] + 4 * s);
        unpack4(reinterpret_cast<const uint2*>(dWm_g[h])[s], dw[h] + 4 * s);
        const uint4 q = noise_block_q(a.np, q0 + s);
        x[h][4 * s] = q.x, x[h][4 * s + 1] = q.y, x[h][4 * s + 2] = q.z, x[h][4 * s + 3] = q.w;
      }
    }
#pragma unroll
    for (int l = 0; l < M; ++l) {
      V one_plus, phv, wv, dwv;
      if constexpr (L == 1) {
        one_plus = one_plus_from_word(x[0][l]);
        phv = ph[0][l], wv = w[0][l], dwv = dw[0][l];
      } else {
        one_plus =
            f2(one_plus_from_word(x[0][l]), one_plus_from_word(x[1][l]));
        phv = f2(ph[0][l], ph[1][l]), wv = f2(w[0][l], w[1][l]), dwv = f2(dw[0][l], dw[1][l]);
      }
      const V u = vsub(one_plus, vconst<V>(__uint_as_float(0x3f7fffffu)));
      kap[l] = key_log2(phv, u, a.np.l2e_inv_lam);  // log2 units
      c[l] = vmul(dwv, wv);
    }
  }

  FastGroup<N, M, TAU1, true, V> fg;
  fg.forward(kap, a.inv_tau);
  if (a.dW != nullptr) {
    // dW = bf16(dWm * S) now, while mu is live anyway (dWm is re-read)
#pragma unroll
    for (int s = 0; s < M / 4; ++s) {
      if constexpr (L == 2) {
        // both groups' products of member l in one packed multiply
        const uint2 qa = reinterpret_cast<const uint2*>(dWm_g[0])[s];
        const uint2 qb = reinterpret_cast<const uint2*>(dWm_g[1])[s];
        const F2 p0 = f2(__uint_as_float(qa.x << 16), __uint_as_float(qb.x << 16)) * fg.soft(4 * s);
        const F2 p1 = f2(__uint_as_float(qa.x & 0xffff0000u), __uint_as_float(qb.x & 0xffff0000u)) * fg.soft(4 * s + 1);
        const F2 p2 = f2(__uint_as_float(qa.y << 16), __uint_as_float(qb.y << 16)) * fg.soft(4 * s + 2);
        const F2 p3 = f2(__uint_as_float(qa.y & 0xffff0000u), __uint_as_float(qb.y & 0xffff0000u)) * fg.soft(4 * s + 3);
        reinterpret_cast<uint2*>(a.dW + e0[0])[s] =
            make_uint2(pack_bf16x2(lo(p0), lo(p1)), pack_bf16x2(lo(p2), lo(p3)));
        reinterpret_cast<uint2*>(a.dW + e0[1])[s] =
            make_uint2(pack_bf16x2(hi(p0), hi(p1)), pack_bf16x2(hi(p2), hi(p3)));
      } else {
        float d[4];
        unpack4(reinterpret_cast<const uint2*>(dWm_g[0])[s], d);
        uint2 o;
        o.x = pack_bf16x2(__fmul_rn(d[0], fg.soft(4 * s)), __fmul_rn(d[1], fg.soft(4 * s + 1)));
        o.y = pack_bf16x2(__fmul_rn(d[2], fg.soft(4 * s + 2)), __fmul_rn(d[3], fg.soft(4 * s + 3)));
        reinterpret_cast<uint2*>(a.dW + e0[0])[s] = o;
      }
    }
  }
  V dkv[M];
  fg.backward(c, a.inv_tau, dkv);
  // dL/dphi = dL/dkappa / lambda
#pragma unroll
  for (int l = 0; l < M; ++l) dkv[l] = vmul(dkv[l], vconst<V>(a.np.inv_lam));
#pragma unroll
  for (int h = 0; h < L; ++h) {
    float dk[M];
#pragma unroll
    for (int l = 0; l < M; ++l) dk[l] = lane_of(dkv[l], h);
    if ((fg.flag >> h) & 1u) {
      float k[M], cc[M], S[M];
#pragma unroll
      for (int l = 0; l < M; ++l) {
        k[l] = lane_of(kap[l], h) * kLn2;  // natural-log keys
        cc[l] = lane_of(c[l], h);
      }
      ExactGroup<N, M> ex;
      ex.forward(k, N, M, a.tau, S);
      ex.backward(cc, N, M, a.tau, dk);
#pragma unroll
      for (int l = 0; l < M; ++l) dk[l] = __fmul_rn(dk[l], a.np.inv_lam);
      if (a.dW != nullptr) {
#pragma unroll
        for (int s = 0; s < M / 4; ++s) {
          float d[4];
          unpack4(reinterpret_cast<const uint2*>(dWm_g[h])[s], d);
          uint2 o;
          o.x = pack_bf16x2(__fmul_rn(d[0], S[4 * s]), __fmul_rn(d[1], S[4 * s + 1]));
          o.y = pack_bf16x2(__fmul_rn(d[2], S[4 * s + 2]), __fmul_rn(d[3], S[4 * s + 3]));
          reinterpret_cast<uint2*>(a.dW + e0[h])[s] = o;
        }
      }
    }
#pragma unroll
    for (int s = 0; s < M / 4; ++s)
      reinterpret_cast<float4*>(a.dphi + e0[h])[s] = make_float4(dk[4 * s], dk[4 * s + 1], dk[4 * s + 2], dk[4 * s + 3]);
  }
}

template <int N, int M, bool TAU1>
__global__ void __launch_bounds__(Cfg<M>::kThreads, Cfg<M>::kMinBlocks) roi_bwd_kernel(BwdArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  using C = Cfg<M>;
  constexpr int kT = C::kTile;
  TileSrc<3> src;
  src.ptr[0] = reinterpret_cast<const uint8_t*>(a.phi);
  src.esize[0] = 4;
  src.ptr[1] = reinterpret_cast<const uint8_t*>(a.W);
  src.esize[1] = 2;
  src.ptr[2] = reinterpret_cast<const uint8_t*>(a.dWm);
  src.esize[2] = 2;

  const bool ok = run_tiles<C::kThreads, kT, C::kStages, 3>(
      smem, src, a.full_tiles, a.status, [&](const uint8_t* const* stage, int64_t tile) {
        const float* sphi = reinterpret_cast<const float*>(stage[0]);
        const uint16_t* sW = reinterpret_cast<const uint16_t*>(stage[1]);
        const uint16_t* sdW = reinterpret_cast<const uint16_t*>(stage[2]);
        const int64_t base = tile * kT;
#pragma unroll
        for (int p = 0; p < C::kPairs; ++p) {
          const int g0 = threadIdx.x + 2 * p * C::kThreads, g1 = g0 + C::kThreads;
          const float* pp[2] = {sphi + g0 * M, sphi + g1 * M};
          const uint16_t* pw[2] = {sW + g0 * M, sW + g1 * M};
          const uint16_t* pd[2] = {sdW + g0 * M, sdW + g1 * M};
          const int64_t e0[2] = {base + g0 * M, base + g1 * M};
          if constexpr (M == 4) {
            bwd_groups<N, M, TAU1, F2>(pp, pw, pd, e0, a);
          } else {
            // M = 8: the paired step history does not fit the register file; one group at a time
#pragma unroll 1
            for (int h = 0; h < 2; ++h) bwd_groups<N, M, TAU1, float>(pp + h, pw + h, pd + h, e0 + h, a);
          }
        }
      });
  if (!ok) return;

  if (blockIdx.x == gridDim.x - 1) {
    const int64_t t0 = a.full_tiles * kT;
    const int64_t tail_groups = (a.E - t0) / M;
    for (int64_t gi = threadIdx.x; gi < tail_groups; gi += C::kThreads) {
      const float* pp[1] = {a.phi + t0 + gi * M};
      const uint16_t* pw[1] = {a.W + t0 + gi * M};
      const uint16_t* pd[1] = {a.dWm + t0 + gi * M};
      const int64_t e0[1] = {t0 + gi * M};
      bwd_groups<N, M, TAU1, float>(pp, pw, pd, e0, a);
    }
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
  using C = Cfg<M>;
  auto kern = roi_bwd_kernel<N, M, TAU1>;
  const size_t smem = tile_smem_bytes<C::kTile, C::kStages>(8);
  static LaunchCache cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return -1;
  if (cache.per_sm[dev] == 0) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem)) != cudaSuccess)
      return -1;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, C::kThreads, smem) != cudaSuccess) return -1;
    cache.per_sm[dev] = per_sm < 1 ? 1 : per_sm;
  }
  const int64_t cap = int64_t(sm_count()) * cache.per_sm[dev];
  const int grid = int(a.full_tiles < 1 ? 1 : (a.full_tiles < cap ? a.full_tiles : cap));
  kern<<<grid, C::kThreads, smem, stream>>>(a);
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
  a.full_tiles = c.E / (c.M == 8 ? Cfg<8>::kTile : Cfg<4>::kTile);
  a.tau = c.tau;
  a.inv_tau = 1.0f / c.tau;
  a.np = c.np;
  a.status = c.status;
  if (c.N == 2 && c.M == 4) return launch_nm<2, 4>(a, c.stream);
  if (c.N == 4 && c.M == 8) return launch_nm<4, 8>(a, c.stream);
  if (c.N == 2 && c.M == 8) return launch_nm<2, 8>(a, c.stream);
  if (slice_supported(c.N, c.M)) return launch_slice_bwd(c);
  const int64_t groups = c.E / c.M;
  int64_t blocks = (groups + 127) / 128;
  const int64_t cap = int64_t(sm_count()) * 16;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  roi_bwd_generic_kernel<<<int(blocks), 128, 0, c.stream>>>(a, c.N, c.M);
  return cudaGetLastError() == cudaSuccess ? 1 : -1;
}

}  // namespace roi
