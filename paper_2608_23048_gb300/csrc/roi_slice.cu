// Wide groups (M = 16, 32: the 8:16 and 16:32 patterns) on warp slices: the
// M / 4 consecutive lanes of a slice hold one group, four elements each.  Same
// method as the one-thread-per-group kernels (Sec. 4.2.2 Eq. 10-12, Algorithm 1;
// Eq. 5; backward through the relaxation), with the per-group sums, maxima and
// "sum of the other members" formed across the slice by a shuffle butterfly
// that never subtracts.  Hard ranks compare every key of the group through
// shuffles.  Groups whose exclusive sums underflow go to ExactGroup, run by the
// slice's first lane.
#include "roi_launch.h"
#include "roi_tiles.cuh"

namespace roi {
namespace {

constexpr int kThreads = 256;
constexpr int kTile = 2048;  // 512 four-element slots: two per thread
constexpr int kStagesFwd = 4;
constexpr int kStagesBwd = 3;

template <int SL>
struct Slice {
  static_assert(SL == 4 || SL == 8, "slices of 4 or 8 lanes");
  // Sum over the slice's other lanes (never total minus own) and the total,
  // identical on every lane of the slice.
  __device__ __forceinline__ static float others(float p, float& tot) {
    float oth = 0.f, acc = p;
#pragma unroll
    for (int o = 1; o < SL; o <<= 1) {
      const float sib = __shfl_xor_sync(0xffffffffu, acc, o);
      oth = __fadd_rn(oth, sib);
      acc = __fadd_rn(acc, sib);
    }
    tot = acc;
    return oth;
  }
  __device__ __forceinline__ static float total(float p) {
    float t;
    others(p, t);
    return t;
  }
  __device__ __forceinline__ static float max(float v) {
#pragma unroll
    for (int o = 1; o < SL; o <<= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
  }
  __device__ __forceinline__ static uint32_t any(uint32_t f) {
#pragma unroll
    for (int o = 1; o < SL; o <<= 1) f |= __shfl_xor_sync(0xffffffffu, f, o);
    return f;
  }
};

__device__ __forceinline__ float sum4(const float (&x)[4]) {
  return __fadd_rn(__fadd_rn(x[0], x[1]), __fadd_rn(x[2], x[3]));
}
__device__ __forceinline__ void excl4(const float (&x)[4], float oth, float (&ex)[4]) {
  const float p01 = __fadd_rn(x[0], x[1]), p23 = __fadd_rn(x[2], x[3]);
  ex[0] = __fadd_rn(__fadd_rn(x[1], p23), oth);
  ex[1] = __fadd_rn(__fadd_rn(x[0], p23), oth);
  ex[2] = __fadd_rn(__fadd_rn(p01, x[3]), oth);
  ex[3] = __fadd_rn(__fadd_rn(p01, x[2]), oth);
}
__device__ __forceinline__ float max4(const float (&x)[4]) { return fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3])); }
__device__ __forceinline__ float min4(const float (&x)[4]) { return fminf(fminf(x[0], x[1]), fminf(x[2], x[3])); }

struct SliceArgs {
  const float* phi;
  const uint16_t* W;
  const uint16_t* dWm;
  uint16_t* Wm;
  float* soft;
  uint32_t* hard;
  float* dphi;
  uint16_t* dW;
  int64_t E;
  int64_t full_tiles;
  float tau, inv_tau;
  NoiseParams np;
  unsigned int* status;
};

// Keys of one four-element slot starting at call-flat index e0, in log2 units
// (t = kappa log2 e).
__device__ __forceinline__ void slot_keys(const float* phi4, int64_t e0, const NoiseParams& np, float (&kap)[4]) {
  const float4 p = *reinterpret_cast<const float4*>(phi4);
  const uint4 x = noise_block_q(np, (np.e_base + uint64_t(e0)) >> 2);
  kap[0] = key_log2(p.x, uniform_from_word(x.x), np.l2e_inv_lam);
  kap[1] = key_log2(p.y, uniform_from_word(x.y), np.l2e_inv_lam);
  kap[2] = key_log2(p.z, uniform_from_word(x.z), np.l2e_inv_lam);
  kap[3] = key_log2(p.w, uniform_from_word(x.w), np.l2e_inv_lam);
}

// Forward relaxation of the group held by this slice; mu of every step kept if
// KEEP.  Returns the slice-uniform fallback flag.
template <int N, int M, bool TAU1, bool KEEP>
struct SliceRelax {
  static constexpr int SL = M / 4;
  float mu[KEEP ? N : 1][4];
  float S[4];
  float rt_last;

  __device__ __forceinline__ uint32_t forward(const float (&kap)[4], float inv_tau, int base_lane) {
    uint32_t flag = 0;
    float cur[4];
    if constexpr (TAU1) {
      const float kref = __shfl_sync(0xffffffffu, kap[0], base_lane);
      float e[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) e[j] = ex2_approx(__fsub_rn(kap[j], kref));
      float tot;
      Slice<SL>::others(sum4(e), tot);
      flag = (!(min4(e) >= kTinyExcl) || !(tot <= 1.0f / kTinyExcl)) ? 1u : 0u;
      const float r = rcp_approx(tot);
#pragma unroll
      for (int j = 0; j < 4; ++j) cur[j] = __fmul_rn(e[j], r);
#pragma unroll
      for (int k = 0; k < N; ++k) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if constexpr (KEEP) mu[k][j] = cur[j];
          S[j] = k == 0 ? cur[j] : __fadd_rn(S[j], cur[j]);
        }
        if (k + 1 < N) {
          float totc, o[4], v[4];
          const float oth = Slice<SL>::others(sum4(cur), totc);
          excl4(cur, oth, o);
#pragma unroll
          for (int j = 0; j < 4; ++j) v[j] = __fmul_rn(cur[j], o[j]);
          const float rt = rcp_approx(Slice<SL>::total(sum4(v)));
          if (k == N - 2) rt_last = rt;
#pragma unroll
          for (int j = 0; j < 4; ++j) cur[j] = __fmul_rn(v[j], rt);
        }
      }
    } else {
      const float kmax = Slice<SL>::max(max4(kap));
      const float sc = inv_tau;
      float d[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) d[j] = __fmul_rn(__fsub_rn(kap[j], kmax), sc);
      if (!(kmax - kmax == 0.0f)) flag = 1u;
#pragma unroll
      for (int k = 0; k < N; ++k) {
        float e[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) e[j] = ex2_approx(d[j]);
        float tot;
        const float oth = Slice<SL>::others(sum4(e), tot);
        const float r = rcp_approx(tot);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          cur[j] = __fmul_rn(e[j], r);
          if constexpr (KEEP) mu[k][j] = cur[j];
          S[j] = k == 0 ? cur[j] : __fadd_rn(S[j], cur[j]);
        }
        if (k + 1 < N) {
          float ex[4];
          excl4(e, oth, ex);
          if (!(min4(ex) >= kTinyExcl)) flag = 1u;
#pragma unroll
          for (int j = 0; j < 4; ++j) d[j] = __fmaf_rn(lg2_approx(__fmul_rn(ex[j], r)), inv_tau, d[j]);
          const float dm = Slice<SL>::max(max4(d));
#pragma unroll
          for (int j = 0; j < 4; ++j) d[j] = __fsub_rn(d[j], dm);
        }
      }
    }
    return Slice<SL>::any(flag);
  }

  // dk = dL/dkappa of this slot's elements for c = dL/dS (same sweep as FastGroup).
  __device__ __forceinline__ void backward(const float (&c)[4], float inv_tau, float (&dk)[4]) const {
    static_assert(KEEP, "needs the steps");
    float b[4], hl[4];
    {
      float cm[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) cm[j] = __fmul_rn(c[j], mu[N - 1][j]);
      const float cmu = Slice<SL>::total(sum4(cm));
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float t = __fmul_rn(inv_tau, __fsub_rn(c[j], cmu));
        b[j] = __fmul_rn(mu[N - 1][j], t);
        if constexpr (TAU1) hl[j] = __fmul_rn(__fmul_rn(mu[N - 2][j], rt_last), t);
      }
    }
#pragma unroll
    for (int k = N - 2; k >= 0; --k) {
      float cm[4], h[4], H[4];
      if (TAU1 && k == N - 2) {
#pragma unroll
        for (int j = 0; j < 4; ++j) h[j] = hl[j];
      } else {
        float om[4], tmp;
        excl4(mu[k], Slice<SL>::others(sum4(mu[k]), tmp), om);
#pragma unroll
        for (int j = 0; j < 4; ++j) h[j] = __fmul_rn(b[j], rcp_approx(om[j]));
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) cm[j] = __fmul_rn(c[j], mu[k][j]);
      const float cmu = Slice<SL>::total(sum4(cm));
      const float B = Slice<SL>::total(sum4(b));
      float tmp;
      excl4(h, Slice<SL>::others(sum4(h), tmp), H);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        b[j] = __fmaf_rn(__fmul_rn(mu[k][j], inv_tau),
                         __fsub_rn(__fadd_rn(__fsub_rn(c[j], cmu), H[j]), B), b[j]);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) dk[j] = b[j];
  }
};

// Hard bits of this slot: rank of each own key among the group's M keys.
template <int M>
__device__ __forceinline__ uint32_t slice_topn_bits(const float (&kap)[4], int N, int base_lane, int q) {
  constexpr int SL = M / 4;
  float kk[4];
  int rank[4] = {0, 0, 0, 0};
#pragma unroll
  for (int j = 0; j < 4; ++j) kk[j] = fmaxf(kap[j], -INFINITY);
#pragma unroll
  for (int qq = 0; qq < SL; ++qq) {
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      const float ko = __shfl_sync(0xffffffffu, kk[jj], base_lane + qq);
      const int io = qq * 4 + jj;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int im = q * 4 + j;
        rank[j] += io < im ? (ko >= kk[j]) : (io > im ? (ko > kk[j]) : 0);
      }
    }
  }
  uint32_t bits = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) bits |= uint32_t(rank[j] < N) << j;
  return bits;
}

// Exact fallback for the whole group, run by one lane: natural-log keys of all
// M elements from logits at phi_g (call-flat index g0).
template <int N, int M>
__device__ __forceinline__ void group_keys_all(const float* phi_g, int64_t g0, const NoiseParams& np, float (&k)[M]) {
#pragma unroll 1
  for (int s = 0; s < M / 4; ++s) {
    float k4[4];
    slot_keys(phi_g + 4 * s, g0 + 4 * s, np, k4);
#pragma unroll
    for (int j = 0; j < 4; ++j) k[4 * s + j] = k4[j] * kLn2;
  }
}

__device__ __forceinline__ uint2 pack4(const float (&w)[4], const float (&s)[4]) {
  uint2 o;
  o.x = pack_bf16x2(__fmul_rn(w[0], s[0]), __fmul_rn(w[1], s[1]));
  o.y = pack_bf16x2(__fmul_rn(w[2], s[2]), __fmul_rn(w[3], s[3]));
  return o;
}
__device__ __forceinline__ void unpack_bf16x4(uint2 q, float (&out)[4]) {
  out[0] = bf16_bits_to_float(q.x & 0xffffu);
  out[1] = bf16_bits_to_float(q.x >> 16);
  out[2] = bf16_bits_to_float(q.y & 0xffffu);
  out[3] = bf16_bits_to_float(q.y >> 16);
}

// One slot of the forward.  si: slot index within the launch's element range
// starting at `base` (call-flat); p/w: the slot's logits and weights (shared or
// global memory).  All 32 lanes of the warp must call this together.
template <int N, int M, bool TAU1>
__device__ __forceinline__ void fwd_slot(const float* p, const uint16_t* w, int64_t e0, bool active, const SliceArgs& a) {
  constexpr int SL = M / 4;
  const int lane = threadIdx.x & 31;
  const int q = lane % SL;
  const int base_lane = lane - q;
  float kap[4] = {0.f, 0.f, 0.f, 0.f};
  if (active) slot_keys(p, e0, a.np, kap);
  const uint32_t bits = slice_topn_bits<M>(kap, N, base_lane, q);
  SliceRelax<N, M, TAU1, false> rx;
  const uint32_t flag = rx.forward(kap, a.inv_tau, base_lane);
  if (active) {
    if (!flag) {
      float wv[4];
      unpack_bf16x4(*reinterpret_cast<const uint2*>(w), wv);
      *reinterpret_cast<uint2*>(a.Wm + e0) = pack4(wv, rx.S);
      if (a.soft != nullptr) *reinterpret_cast<float4*>(a.soft + e0) = make_float4(rx.S[0], rx.S[1], rx.S[2], rx.S[3]);
    } else if (q == 0) {
      float k[M], S[M];
      group_keys_all<N, M>(p, e0, a.np, k);
      ExactGroup<N, M> ex;
      ex.forward(k, N, M, a.tau, S);
#pragma unroll 1
      for (int s = 0; s < SL; ++s) {
        float wv[4], sv[4];
        unpack_bf16x4(*reinterpret_cast<const uint2*>(w + 4 * s), wv);
#pragma unroll
        for (int j = 0; j < 4; ++j) sv[j] = S[4 * s + j];
        *reinterpret_cast<uint2*>(a.Wm + e0 + 4 * s) = pack4(wv, sv);
        if (a.soft != nullptr) *reinterpret_cast<float4*>(a.soft + e0 + 4 * s) = make_float4(sv[0], sv[1], sv[2], sv[3]);
      }
    }
  }
  if (a.hard != nullptr) {
    // 8 lanes hold the 32 elements of a word
    uint32_t v = active ? bits << ((lane & 7) * 4) : 0u;
    v |= __shfl_xor_sync(0xffffffffu, v, 1);
    v |= __shfl_xor_sync(0xffffffffu, v, 2);
    v |= __shfl_xor_sync(0xffffffffu, v, 4);
    if (active && (lane & 7) == 0) a.hard[e0 >> 5] = v;
  }
}

template <int N, int M, bool TAU1>
__device__ __forceinline__ void bwd_slot(const float* p, const uint16_t* w, const uint16_t* dw, int64_t e0, bool active,
                                         const SliceArgs& a) {
  constexpr int SL = M / 4;
  const int lane = threadIdx.x & 31;
  const int q = lane % SL;
  const int base_lane = lane - q;
  float kap[4] = {0.f, 0.f, 0.f, 0.f}, c[4] = {0.f, 0.f, 0.f, 0.f};
  if (active) {
    slot_keys(p, e0, a.np, kap);
    float wv[4], dv[4];
    unpack_bf16x4(*reinterpret_cast<const uint2*>(w), wv);
    unpack_bf16x4(*reinterpret_cast<const uint2*>(dw), dv);
#pragma unroll
    for (int j = 0; j < 4; ++j) c[j] = __fmul_rn(dv[j], wv[j]);
  }
  SliceRelax<N, M, TAU1, true> rx;
  const uint32_t flag = rx.forward(kap, a.inv_tau, base_lane);
  if (active && !flag && a.dW != nullptr) {
    float dv[4];
    unpack_bf16x4(*reinterpret_cast<const uint2*>(dw), dv);
    *reinterpret_cast<uint2*>(a.dW + e0) = pack4(dv, rx.S);
  }
  float dk[4];
  rx.backward(c, a.inv_tau, dk);
  if (!active) return;
  if (!flag) {
    *reinterpret_cast<float4*>(a.dphi + e0) =
        make_float4(dk[0] * a.np.inv_lam, dk[1] * a.np.inv_lam, dk[2] * a.np.inv_lam, dk[3] * a.np.inv_lam);
  } else if (q == 0) {
    float k[M], cc[M], S[M], dkk[M];
    group_keys_all<N, M>(p, e0, a.np, k);
#pragma unroll 1
    for (int s = 0; s < SL; ++s) {
      float wv[4], dv[4];
      unpack_bf16x4(*reinterpret_cast<const uint2*>(w + 4 * s), wv);
      unpack_bf16x4(*reinterpret_cast<const uint2*>(dw + 4 * s), dv);
#pragma unroll
      for (int j = 0; j < 4; ++j) cc[4 * s + j] = __fmul_rn(dv[j], wv[j]);
    }
    ExactGroup<N, M> ex;
    ex.forward(k, N, M, a.tau, S);
    ex.backward(cc, N, M, a.tau, dkk);
#pragma unroll 1
    for (int s = 0; s < SL; ++s) {
      *reinterpret_cast<float4*>(a.dphi + e0 + 4 * s) =
          make_float4(dkk[4 * s] * a.np.inv_lam, dkk[4 * s + 1] * a.np.inv_lam, dkk[4 * s + 2] * a.np.inv_lam,
                      dkk[4 * s + 3] * a.np.inv_lam);
      if (a.dW != nullptr) {
        float dv[4], sv[4];
        unpack_bf16x4(*reinterpret_cast<const uint2*>(dw + 4 * s), dv);
#pragma unroll
        for (int j = 0; j < 4; ++j) sv[j] = S[4 * s + j];
        *reinterpret_cast<uint2*>(a.dW + e0 + 4 * s) = pack4(dv, sv);
      }
    }
  }
}

template <int N, int M, bool TAU1>
__global__ void __launch_bounds__(kThreads, 2) roi_slice_fwd_kernel(SliceArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  TileSrc<2> src;
  src.ptr[0] = reinterpret_cast<const uint8_t*>(a.phi);
  src.esize[0] = 4;
  src.ptr[1] = reinterpret_cast<const uint8_t*>(a.W);
  src.esize[1] = 2;
  const bool ok = run_tiles<kThreads, kTile, kStagesFwd, 2>(
      smem, src, a.full_tiles, a.status, [&](const uint8_t* const* stage, int64_t tile) {
        const float* sphi = reinterpret_cast<const float*>(stage[0]);
        const uint16_t* sW = reinterpret_cast<const uint16_t*>(stage[1]);
        const int64_t base = tile * kTile;
#pragma unroll 1
        for (int j = 0; j < 2; ++j) {
          const int si = threadIdx.x + j * kThreads;
          fwd_slot<N, M, TAU1>(sphi + 4 * si, sW + 4 * si, base + 4 * si, true, a);
        }
      });
  if (!ok) return;
  if (blockIdx.x == gridDim.x - 1) {
    const int64_t t0 = a.full_tiles * kTile;
    const int64_t slots = (a.E - t0) / 4;
    for (int64_t r = 0; r * kThreads < slots; ++r) {
      const int64_t si = threadIdx.x + r * kThreads;
      const bool active = si < slots;
      const int64_t off = t0 + 4 * (active ? si : 0);
      fwd_slot<N, M, TAU1>(a.phi + off, a.W + off, t0 + 4 * si, active, a);
    }
  }
}

template <int N, int M, bool TAU1>
__global__ void __launch_bounds__(kThreads, M == 32 ? 1 : 2) roi_slice_bwd_kernel(SliceArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  TileSrc<3> src;
  src.ptr[0] = reinterpret_cast<const uint8_t*>(a.phi);
  src.esize[0] = 4;
  src.ptr[1] = reinterpret_cast<const uint8_t*>(a.W);
  src.esize[1] = 2;
  src.ptr[2] = reinterpret_cast<const uint8_t*>(a.dWm);
  src.esize[2] = 2;
  const bool ok = run_tiles<kThreads, kTile, kStagesBwd, 3>(
      smem, src, a.full_tiles, a.status, [&](const uint8_t* const* stage, int64_t tile) {
        const float* sphi = reinterpret_cast<const float*>(stage[0]);
        const uint16_t* sW = reinterpret_cast<const uint16_t*>(stage[1]);
        const uint16_t* sdW = reinterpret_cast<const uint16_t*>(stage[2]);
        const int64_t base = tile * kTile;
#pragma unroll 1
        for (int j = 0; j < 2; ++j) {
          const int si = threadIdx.x + j * kThreads;
          bwd_slot<N, M, TAU1>(sphi + 4 * si, sW + 4 * si, sdW + 4 * si, base + 4 * si, true, a);
        }
      });
  if (!ok) return;
  if (blockIdx.x == gridDim.x - 1) {
    const int64_t t0 = a.full_tiles * kTile;
    const int64_t slots = (a.E - t0) / 4;
    for (int64_t r = 0; r * kThreads < slots; ++r) {
      const int64_t si = threadIdx.x + r * kThreads;
      const bool active = si < slots;
      const int64_t off = t0 + 4 * (active ? si : 0);
      bwd_slot<N, M, TAU1>(a.phi + off, a.W + off, a.dWm + off, t0 + 4 * si, active, a);
    }
  }
}

struct LaunchCache {
  int per_sm[64] = {0};
};

template <class Kern>
int launch_persistent(Kern kern, LaunchCache& cache, size_t smem, const SliceArgs& a, cudaStream_t stream) {
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

template <int N, int M, bool TAU1>
int slice_fwd(const SliceArgs& a, cudaStream_t stream) {
  static LaunchCache cache;
  return launch_persistent(roi_slice_fwd_kernel<N, M, TAU1>, cache, tile_smem_bytes<kTile, kStagesFwd>(6), a, stream);
}
template <int N, int M, bool TAU1>
int slice_bwd(const SliceArgs& a, cudaStream_t stream) {
  static LaunchCache cache;
  return launch_persistent(roi_slice_bwd_kernel<N, M, TAU1>, cache, tile_smem_bytes<kTile, kStagesBwd>(8), a, stream);
}

}  // namespace

bool slice_supported(int N, int M) { return (N == 8 && M == 16) || (N == 16 && M == 32); }

int launch_slice_fwd(const FwdCall& c) {
  SliceArgs a{};
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
  const bool t1 = c.tau == 1.0f;
  if (c.N == 8 && c.M == 16) return t1 ? slice_fwd<8, 16, true>(a, c.stream) : slice_fwd<8, 16, false>(a, c.stream);
  if (c.N == 16 && c.M == 32) return t1 ? slice_fwd<16, 32, true>(a, c.stream) : slice_fwd<16, 32, false>(a, c.stream);
  return -1;
}

int launch_slice_bwd(const BwdCall& c) {
  SliceArgs a{};
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
  const bool t1 = c.tau == 1.0f;
  if (c.N == 8 && c.M == 16) return t1 ? slice_bwd<8, 16, true>(a, c.stream) : slice_bwd<8, 16, false>(a, c.stream);
  if (c.N == 16 && c.M == 32) return t1 ? slice_bwd<16, 32, true>(a, c.stream) : slice_bwd<16, 32, false>(a, c.stream);
  return -1;
}

}  // namespace roi
