// Forward of the RoI mask op (Sec. 4.2.2 Eq. 10-12, Algorithm 1; Eq. 5 mask
// application): per group of M logits, regenerate the Gumbel noise, form the
// perturbed keys, run the N-step relaxed top-N, write Wm = bf16(W * S), and
// optionally S and the hard Gumbel-top-N bits.
#include "roi_launch.h"
#include "roi_tiles.cuh"

namespace roi {
namespace {

// Launch shape per group size M: threads per CTA, pairs of groups per thread per
// tile (the two groups of a pair are relaxed in lockstep on packed FP32, F2),
// shared-memory stages, and the CTAs per SM the register budget is sized for.
// One CTA per SM: CTAs sharing an SM progress at very different rates (the
// scheduler favours the older one) and the last ones then finish alone, so all of
// an SM's warps work through one tile ring instead.
// Tensors of one multi-tensor launch, at most (its parameter block holds them all).
constexpr int kMultiMax = 256;

template <int M>
struct Cfg {
  static constexpr int kThreads = 512;
  static constexpr int kPairs = M == 4 ? 3 : 1;
  static constexpr int kStages = 2;  // 144 KB (M = 4) or 96 KB (M = 8)
  static constexpr int kMinBlocks = 1;
  static constexpr int kTile = 2 * kPairs * kThreads * M;  // elements
  // groups out of the fast path's range, queued per warp (DeferredGroups): at most
  // 64 kPairs a tile on top of fewer than 32 left from earlier tiles
  static constexpr int kDeferCap = 32 + 64 * kPairs;
  static constexpr size_t kDeferOffset = (tile_smem_bytes<kTile, kStages>(6) + 15) & ~size_t(15);
  static constexpr size_t kSmem = kDeferOffset + size_t(kDeferCap) * 8 * (kThreads / 32);
  // multi-tensor launches: the tensors' first tiles behind the queues
  static constexpr size_t kMultiOffset = (kSmem + 15) & ~size_t(15);
  static constexpr size_t kMultiSmem = kMultiOffset + size_t(kMultiMax + 1) * 8;
};

struct FwdArgs {
  const float* phi;
  const uint16_t* W;
  uint16_t* Wm;
  float* soft;
  uint32_t* hard;
  bool st;  // straight-through: Wm = W where the hard mask is set, +0 elsewhere
  int64_t E;
  int64_t full_tiles;
  float tau, inv_tau;
  NoiseParams np;
  unsigned int* status;
};

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

// Perturbed keys of L groups (one per lane of V), in log2 units
// (t = (phi / lambda + g) log2 e), whose first elements have call-flat indices
// e0[h]; ph[h] holds each group's logits.  NARROW: the call's counters are below
// 2^32 and q0[h] holds the low word of group h's first counter.
template <int M, class V, bool NARROW>
__device__ __forceinline__ void group_keys(const float (&ph)[vlanes<V>()][M], const int64_t* e0, const uint32_t* q0,
                                           const NoiseParams& np, V (&kap)[M]) {
  constexpr int L = vlanes<V>();
  uint32_t x[L][M];
#pragma unroll
  for (int h = 0; h < L; ++h) {
#pragma unroll
    for (int s = 0; s < M / 4; ++s) {
      uint4 w;
      if constexpr (NARROW) {
        w = noise_block_lo(np, q0[h] + s);
      } else {
        w = noise_block_q(np, ((np.e_base + uint64_t(e0[h])) >> 2) + s);
      }
      x[h][4 * s] = w.x, x[h][4 * s + 1] = w.y, x[h][4 * s + 2] = w.z, x[h][4 * s + 3] = w.w;
    }
  }
#pragma unroll
  for (int l = 0; l < M; ++l) {
    V one_plus, phv;
    if constexpr (L == 1) {
      one_plus = one_plus_from_word(x[0][l]);
      phv = ph[0][l];
    } else {
      one_plus = f2(one_plus_from_word(x[0][l]), one_plus_from_word(x[1][l]));
      phv = f2(ph[0][l], ph[1][l]);
    }
    // u = (1 + k 2^-23) - (1 - 2^-24), exact (see uniform_from_word)
    const V u = vsub(one_plus, vconst<V>(__uint_as_float(0x3f7fffffu)));
    kap[l] = key_log2(phv, u, np.l2e_inv_lam);
  }
}

template <class V>
__device__ __forceinline__ float lane_of(V v, int h) {
  if constexpr (vlanes<V>() == 1) {
    return v;
  } else {
    return h == 0 ? lo(v) : hi(v);
  }
}

// L groups (one per lane of V) processed in lockstep by one thread; writes their
// outputs and returns each group's hard bits in bits[h].
// The keys of L groups from their staged logits (first half of fwd_groups).
template <int M, class V, bool NARROW = false>
__device__ __forceinline__ void fwd_keys(const float* const* phi_g, const int64_t* e0, const uint32_t* q0,
                                         const FwdArgs& a, V (&kap)[M]) {
  constexpr int L = vlanes<V>();
  float ph[L][M];
#pragma unroll
  for (int h = 0; h < L; ++h) {
#pragma unroll
    for (int s = 0; s < M / 4; ++s) {
      const float4 p = reinterpret_cast<const float4*>(phi_g[h])[s];
      ph[h][4 * s] = p.x, ph[h][4 * s + 1] = p.y, ph[h][4 * s + 2] = p.z, ph[h][4 * s + 3] = p.w;
    }
  }
  group_keys<M, V, NARROW>(ph, e0, q0, a.np, kap);
}

// Relaxation, hard bits and outputs of L groups whose keys are `kap`.
template <int N, int M, bool TAU1, class V, bool ST = false, bool DEFER = false>
__device__ __forceinline__ uint32_t fwd_finish(const V (&kap)[M], const uint16_t* const* W_g, const int64_t* e0,
                                               const FwdArgs& a, uint32_t* bits) {
  constexpr int L = vlanes<V>();
  FastGroup<N, M, TAU1, false, V> fg;
  fg.forward(kap, a.inv_tau);
  float S[L][M];
#pragma unroll
  for (int h = 0; h < L; ++h)
#pragma unroll
    for (int l = 0; l < M; ++l) S[h][l] = lane_of(fg.S[l], h);
  // ranking the log2-unit keys ranks kappa
  constexpr bool kFastTopn = (M == 4 || M == 8) && L == 2;
  if constexpr (kFastTopn) {
    // finite keys only: flagged groups are re-ranked below
    uint32_t b2[2];
    if constexpr (M == 4) {
      topn_bits4_signs(kap, N, b2);
    } else {
      topn_bits8_threshold<N>(kap, b2);
    }
    bits[0] = b2[0], bits[1] = b2[1];
    if constexpr (M == 8) {
#pragma unroll
      for (int h = 0; h < L; ++h) {
        if (bits[h] == 0xffffffffu) {  // threshold tied with another member
          float k[M];
#pragma unroll
          for (int l = 0; l < M; ++l) k[l] = lane_of(kap[l], h);
          bits[h] = topn_bits<M>(k, N);
        }
      }
    }
  } else {
#pragma unroll
    for (int h = 0; h < L; ++h) {
      float k[M];
#pragma unroll
      for (int l = 0; l < M; ++l) k[l] = lane_of(kap[l], h);
      if constexpr (M == 4) {
        bits[h] = topn_bits4(k, N);
      } else {
        bits[h] = topn_bits<M>(k, N);
      }
    }
  }
  // groups out of the fast path's range: ranked by comparison, and either relaxed
  // here by the exact routine (DEFER off) or (DEFER) left to fwd_exact_group, which
  // the caller runs for them from the deferred queue and which writes their soft
  // mask and Wm again
  if constexpr (!DEFER) {
    if (fg.flag != 0u) {
#pragma unroll
      for (int h = 0; h < L; ++h) {
        if ((fg.flag >> h) & 1u) {
          float k[M], kn[M];
#pragma unroll
          for (int l = 0; l < M; ++l) {
            k[l] = lane_of(kap[l], h);
            kn[l] = k[l] * kLn2;  // natural-log keys
          }
          if constexpr (kFastTopn) {
            if constexpr (M == 4) {
              bits[h] = topn_bits4(k, N);
            } else {
              bits[h] = topn_bits<M>(k, N);
            }
          }
          // finite keys spread beyond the fast path's float range (tau != 1: at tau = 1
          // that takes a key gap of ~69 natural-log units, and the tau = 1 kernels keep
          // their code to the exact routine)
          if (!TAU1 && all_finite(k)) {
            RobustGroup<N, M> rg;
            rg.forward(k, a.inv_tau, S[h]);
          } else {
            ExactGroup<N, M> ex;
            ex.forward(kn, N, M, a.tau, S[h]);
          }
        }
      }
    }
  } else if (kFastTopn && fg.flag != 0u) {
#pragma unroll
    for (int h = 0; h < L; ++h) {
      if ((fg.flag >> h) & 1u) {
        float k[M];
#pragma unroll
        for (int l = 0; l < M; ++l) k[l] = lane_of(kap[l], h);
        if constexpr (M == 4) {
          bits[h] = topn_bits4(k, N);
        } else {
          bits[h] = topn_bits<M>(k, N);
        }
      }
    }
  }
  // Wm = bf16(W * S); W is read here, not kept live through the relaxation
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    const float* sa = S[0] + 4 * s;
    if constexpr (ST) {
      // straight-through: the weights the hard mask keeps, +0 elsewhere
#pragma unroll
      for (int h = 0; h < L; ++h)
        reinterpret_cast<uint2*>(a.Wm + e0[h])[s] = keep4(reinterpret_cast<const uint2*>(W_g[h])[s], bits[h] >> (4 * s));
    } else if constexpr (L == 2) {
      // both groups' products of member l in one packed multiply
      const float* sb = S[1] + 4 * s;
      const uint2 qa = reinterpret_cast<const uint2*>(W_g[0])[s];
      const uint2 qb = reinterpret_cast<const uint2*>(W_g[1])[s];
      const F2 p0 = f2(__uint_as_float(qa.x << 16), __uint_as_float(qb.x << 16)) * f2(sa[0], sb[0]);
      const F2 p1 = f2(__uint_as_float(qa.x & 0xffff0000u), __uint_as_float(qb.x & 0xffff0000u)) * f2(sa[1], sb[1]);
      const F2 p2 = f2(__uint_as_float(qa.y << 16), __uint_as_float(qb.y << 16)) * f2(sa[2], sb[2]);
      const F2 p3 = f2(__uint_as_float(qa.y & 0xffff0000u), __uint_as_float(qb.y & 0xffff0000u)) * f2(sa[3], sb[3]);
      reinterpret_cast<uint2*>(a.Wm + e0[0])[s] =
          make_uint2(pack_bf16x2(lo(p0), lo(p1)), pack_bf16x2(lo(p2), lo(p3)));
      reinterpret_cast<uint2*>(a.Wm + e0[1])[s] =
          make_uint2(pack_bf16x2(hi(p0), hi(p1)), pack_bf16x2(hi(p2), hi(p3)));
    } else {
      const uint2 q = reinterpret_cast<const uint2*>(W_g[0])[s];
      const float wv[4] = {bf16_bits_to_float(q.x & 0xffffu), bf16_bits_to_float(q.x >> 16),
                           bf16_bits_to_float(q.y & 0xffffu), bf16_bits_to_float(q.y >> 16)};
      uint2 o;
      o.x = pack_bf16x2(__fmul_rn(wv[0], sa[0]), __fmul_rn(wv[1], sa[1]));
      o.y = pack_bf16x2(__fmul_rn(wv[2], sa[2]), __fmul_rn(wv[3], sa[3]));
      reinterpret_cast<uint2*>(a.Wm + e0[0])[s] = o;
    }
    if (a.soft != nullptr) {
#pragma unroll
      for (int h = 0; h < L; ++h) {
        const float* sh = S[h] + 4 * s;
        reinterpret_cast<float4*>(a.soft + e0[h])[s] = make_float4(sh[0], sh[1], sh[2], sh[3]);
      }
    }
  }
  return DEFER ? fg.flag : 0u;
}

// The exact routine for one group out of the fast path's range (first element g0,
// call-flat), from global memory: the log2-domain routine for finite keys spread
// beyond the float range (tau != 1; at tau = 1 that takes a key gap of ~69
// natural-log units and the tau = 1 kernels keep only the general routine), the
// exact one otherwise.  Writes soft and (unless straight-through) Wm.
template <int N, int M, bool TAU1, bool ST>
__device__ __forceinline__ void fwd_exact_group(int64_t g0, const FwdArgs& a) {
  if (ST && a.soft == nullptr) return;
  // the keys as the tiles' packed code forms them (the group in both halves), so they
  // equal, bit for bit, those the fast path and the masked linear's prologue see
  const float* pp[2] = {a.phi + g0, a.phi + g0};
  const int64_t e0[2] = {g0, g0};
  F2 k2[M];
  fwd_keys<M, F2>(pp, e0, nullptr, a, k2);
  float k[M], S[M];
#pragma unroll
  for (int l = 0; l < M; ++l) k[l] = lo(k2[l]);
  if (!TAU1 && all_finite(k)) {
    RobustGroup<N, M> rg;
    rg.forward(k, a.inv_tau, S);
  } else {
#pragma unroll
    for (int l = 0; l < M; ++l) k[l] *= kLn2;  // natural-log keys
    ExactGroup<N, M> ex;
    ex.forward(k, N, M, a.tau, S);
  }
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    if constexpr (!ST) {
      const uint2 q = reinterpret_cast<const uint2*>(a.W + g0)[s];
      uint2 o;
      o.x = pack_bf16x2(__fmul_rn(bf16_bits_to_float(q.x & 0xffffu), S[4 * s]),
                        __fmul_rn(bf16_bits_to_float(q.x >> 16), S[4 * s + 1]));
      o.y = pack_bf16x2(__fmul_rn(bf16_bits_to_float(q.y & 0xffffu), S[4 * s + 2]),
                        __fmul_rn(bf16_bits_to_float(q.y >> 16), S[4 * s + 3]));
      reinterpret_cast<uint2*>(a.Wm + g0)[s] = o;
    }
    if (a.soft != nullptr)
      reinterpret_cast<float4*>(a.soft + g0)[s] = make_float4(S[4 * s], S[4 * s + 1], S[4 * s + 2], S[4 * s + 3]);
  }
}

// One group straight from global memory (the ragged tail; the exact routine in place).
template <int N, int M, bool TAU1, bool ST = false>
__device__ __forceinline__ void fwd_groups(const float* const* phi_g, const uint16_t* const* W_g, const int64_t* e0,
                                           const FwdArgs& a, uint32_t* bits) {
  float kap[M];
  fwd_keys<M, float>(phi_g, e0, nullptr, a, kap);
  fwd_finish<N, M, TAU1, float, ST>(kap, W_g, e0, a, bits);
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

// The same for a tile's two groups per thread (first elements e0a, e0b; all
// lanes active).  Both masks travel in one register, the first group's in the
// low half-word and the second's in the high one; the shuffles OR the masks of
// the 16 / M lanes that fill a half-word, then one exchange between the two
// halves of each word's lane range completes the first group's word on the
// leader of the first half and the second group's word on the leader of the
// second half.
template <int M>
__device__ __forceinline__ void store_hard_pair(uint32_t* hard, int64_t e0a, int64_t e0b, uint32_t bits_a,
                                                uint32_t bits_b) {
  constexpr int kHalf = 16 / M;  // lanes per half-word
  const int lane = threadIdx.x & 31;
  const int sh = (lane % kHalf) * M;
  uint32_t v = (bits_a << sh) | (bits_b << (16 + sh));
#pragma unroll
  for (int o = 1; o < kHalf; o <<= 1) v |= __shfl_xor_sync(0xffffffffu, v, o);
  const uint32_t w = __shfl_xor_sync(0xffffffffu, v, kHalf);
  const bool upper = (lane & kHalf) != 0;
  // lower leader: {own low half, partner's low half}; upper leader: {partner's high half, own high half}
  const uint32_t word = __byte_perm(v, w, upper ? 0x3276u : 0x5410u);
  if (lane % kHalf == 0) hard[(upper ? e0b : e0a) >> 5] = word;
}

// One full tile of a tensor (local tile index `tile`), inputs staged in shared
// memory.  NARROW: the call's counters are below 2^32 (a.np.narrow).
template <int N, int M, bool TAU1, bool ST, bool NARROW, bool DEFER, class Defer, class Exact>
__device__ __forceinline__ void fwd_tile(const uint8_t* const* stage, int64_t tile, const FwdArgs& a, Defer& dg,
                                         int64_t tag, const Exact& exact) {
  using C = Cfg<M>;
  constexpr int kT = C::kTile;
  const float* sphi = reinterpret_cast<const float*>(stage[0]);
  const uint16_t* sW = reinterpret_cast<const uint16_t*>(stage[1]);
  const int64_t base = tile * kT;
  // low word of the tile's first counter (uniform); group g adds g M / 4
  const uint32_t qt = uint32_t((a.np.e_base + uint64_t(base)) >> 2);
  // pair p: groups t and t + kThreads of the p-th block of 2 kThreads groups.
  // The keys of pair p + 1 (integer-heavy: Philox, range reduction) are
  // formed before pair p is relaxed (floating-point-heavy), so the two
  // streams share the issue slots of one basic block.
  F2 kap[2][M];
  {
    const int g0 = threadIdx.x, g1 = g0 + C::kThreads;
    const float* pp[2] = {sphi + g0 * M, sphi + g1 * M};
    const int64_t e0[2] = {base + g0 * M, base + g1 * M};
    const uint32_t q0[2] = {qt + uint32_t(g0 * (M / 4)), qt + uint32_t(g1 * (M / 4))};
    fwd_keys<M, F2, NARROW>(pp, e0, q0, a, kap[0]);
  }
#pragma unroll
  for (int p = 0; p < C::kPairs; ++p) {
    if (p + 1 < C::kPairs) {
      const int g0 = threadIdx.x + 2 * (p + 1) * C::kThreads, g1 = g0 + C::kThreads;
      const float* pp[2] = {sphi + g0 * M, sphi + g1 * M};
      const int64_t e0[2] = {base + g0 * M, base + g1 * M};
      const uint32_t q0[2] = {qt + uint32_t(g0 * (M / 4)), qt + uint32_t(g1 * (M / 4))};
      fwd_keys<M, F2, NARROW>(pp, e0, q0, a, kap[(p + 1) & 1]);
    }
    const int g0 = threadIdx.x + 2 * p * C::kThreads, g1 = g0 + C::kThreads;
    const uint16_t* pw[2] = {sW + g0 * M, sW + g1 * M};
    const int64_t e0[2] = {base + g0 * M, base + g1 * M};
    uint32_t bits[2];
    const uint32_t flag = fwd_finish<N, M, TAU1, F2, ST, DEFER>(kap[p & 1], pw, e0, a, bits);
    if (a.hard != nullptr) store_hard_pair<M>(a.hard, e0[0], e0[1], bits[0], bits[1]);
    if constexpr (DEFER) {
      dg.push((flag & 1u) != 0u, tag | e0[0]);
      dg.push((flag & 2u) != 0u, tag | e0[1]);
    }
  }
  if constexpr (DEFER) dg.drain(false, exact);
}

// The ragged tail of a tensor (fewer than one tile after its full tiles), by one
// CTA, straight from global memory.
template <int N, int M, bool TAU1, bool ST>
__device__ __forceinline__ void fwd_tail(const FwdArgs& a) {
  using C = Cfg<M>;
  const int64_t t0 = a.full_tiles * C::kTile;
  const int64_t tail_groups = (a.E - t0) / M;
  const int64_t rounds = (tail_groups + C::kThreads - 1) / C::kThreads;
  for (int64_t r = 0; r < rounds; ++r) {
    const int64_t gi = threadIdx.x + r * C::kThreads;
    const bool active = gi < tail_groups;
    uint32_t bits = 0;
    if (active) {
      const float* pp[1] = {a.phi + t0 + gi * M};
      const uint16_t* pw[1] = {a.W + t0 + gi * M};
      const int64_t e0[1] = {t0 + gi * M};
      fwd_groups<N, M, TAU1, ST>(pp, pw, e0, a, &bits);
    }
    if (a.hard != nullptr) store_hard<M>(a.hard, t0 + gi * M, bits, active);
  }
}

// ST: straight-through Wm (a separate instantiation)
template <int N, int M, bool TAU1, bool ST, bool DEFER>
__global__ void __launch_bounds__(Cfg<M>::kThreads, Cfg<M>::kMinBlocks) roi_fwd_kernel(FwdArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  using C = Cfg<M>;
  TileSrc<2> src;
  src.ptr[0] = reinterpret_cast<const uint8_t*>(a.phi);
  src.esize[0] = 4;
  src.ptr[1] = reinterpret_cast<const uint8_t*>(a.W);
  src.esize[1] = 2;
  DeferredGroups<C::kDeferCap> dg;
  dg.init(smem + C::kDeferOffset);
  const auto exact = [&](int64_t g0) { fwd_exact_group<N, M, TAU1, ST>(g0, a); };
  // a batch's next tensor may start on the SMs this launch frees (no-op otherwise)
  pdl_launch_dependents();
  const bool ok = run_tiles<C::kThreads, C::kTile, C::kStages, 2>(
      smem, src, a.full_tiles, a.status,
      [&](const uint8_t* const* stage, int64_t tile) {
        // 32-bit counters for M = 4 only: at M = 8 the second copy of the tile
        // body measured slower (register allocation), so those keep one
        if constexpr (M == 4) {
          if (a.np.narrow) {
            fwd_tile<N, M, TAU1, ST, true, DEFER>(stage, tile, a, dg, 0, exact);
            return;
          }
        }
        fwd_tile<N, M, TAU1, ST, false, DEFER>(stage, tile, a, dg, 0, exact);
      });
  if constexpr (DEFER) {
    if (ok) dg.drain(true, exact);
  }
  if (ok && blockIdx.x == gridDim.x - 1) fwd_tail<N, M, TAU1, ST>(a);
  // the launch completes only after the batch's previous one (stream order)
  if (blockIdx.x == 0) pdl_wait();
}

// Multi-tensor launches: the tensors' arguments, and their first tiles in the
// concatenated tile sequence of the launch (tile0).
struct FwdItem {
  const float* phi;
  const uint16_t* W;
  uint16_t* Wm;
  float* soft;
  uint32_t* hard;
  int64_t E;
  int64_t tile0;
  NoiseParams np;
};
struct FwdMulti {
  int count;
  int64_t total_tiles;
  bool st;
  float tau, inv_tau;
  unsigned int* status;
  FwdItem it[kMultiMax];
};
static_assert(sizeof(FwdMulti) <= 32764, "kernel parameter block");
template <int M>
__device__ __forceinline__ FwdArgs multi_args(const FwdMulti& mm, int i) {
  const FwdItem& x = mm.it[i];
  FwdArgs a;
  a.phi = x.phi;
  a.W = x.W;
  a.Wm = x.Wm;
  a.soft = x.soft;
  a.hard = x.hard;
  a.st = mm.st;
  a.E = x.E;
  a.full_tiles = x.E / Cfg<M>::kTile;
  a.tau = mm.tau;
  a.inv_tau = mm.inv_tau;
  a.np = x.np;
  a.status = mm.status;
  return a;
}
// The tile kernel over many small tensors at once: the persistent CTAs walk the
// concatenation of the tensors' full tiles, finding a tile's tensor by binary
// search over tile0 (in shared memory) only when a tile leaves the current one.
// Deferred groups carry their tensor's index above bit 48; each tensor's ragged
// tail goes to one CTA after the tiles.
template <int N, int M, bool TAU1, bool ST, bool DEFER>
__global__ void __launch_bounds__(Cfg<M>::kThreads, Cfg<M>::kMinBlocks)
    roi_fwd_multi_kernel(const __grid_constant__ FwdMulti mm) {
  extern __shared__ __align__(128) uint8_t smem[];
  using C = Cfg<M>;
  const uint32_t esize[2] = {4, 2};
  constexpr int64_t kLow = (int64_t(1) << 48) - 1;
  // the tensors' first tiles, in shared memory for the searches
  int64_t* tile0 = reinterpret_cast<int64_t*>(smem + C::kMultiOffset);
  for (int i = threadIdx.x; i <= mm.count; i += C::kThreads) tile0[i] = i < mm.count ? mm.it[i].tile0 : mm.total_tiles;
  __syncthreads();
  const auto find = [&](int64_t t) {
    int lo = 0, hi = mm.count - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (tile0[mid] <= t) {
        lo = mid;
      } else {
        hi = mid - 1;
      }
    }
    return lo;
  };
  DeferredGroups<C::kDeferCap> dg;
  dg.init(smem + C::kDeferOffset);
  const auto exact = [&](int64_t e) { fwd_exact_group<N, M, TAU1, ST>(e & kLow, multi_args<M>(mm, int(e >> 48))); };
  // the current tensor of this warp's tiles (and of the copies thread 0 issues),
  // looked up again only when a tile falls outside it
  int cur = -1, src_cur = -1;
  int64_t lo = 0, hi = 0, src_lo = 0, src_hi = 0;
  FwdArgs a;
  const float* src_phi = nullptr;
  const uint16_t* src_W = nullptr;
  pdl_launch_dependents();
  const bool ok = run_tiles_src<C::kThreads, C::kTile, C::kStages, 2>(
      smem, esize, mm.total_tiles, mm.status,
      [&](int64_t t, int arr) {
        if (t < src_lo || t >= src_hi) {
          src_cur = find(t);
          src_lo = tile0[src_cur];
          src_hi = tile0[src_cur + 1];
          src_phi = mm.it[src_cur].phi;
          src_W = mm.it[src_cur].W;
        }
        const size_t off = size_t(t - src_lo) * C::kTile;
        return arr == 0 ? reinterpret_cast<const uint8_t*>(src_phi + off) : reinterpret_cast<const uint8_t*>(src_W + off);
      },
      [&](const uint8_t* const* stage, int64_t t) {
        if (t < lo || t >= hi) {
          cur = find(t);
          lo = tile0[cur];
          hi = tile0[cur + 1];
          a = multi_args<M>(mm, cur);
        }
        const int64_t local = t - lo;
        const int64_t tag = int64_t(cur) << 48;
        if constexpr (M == 4) {
          if (a.np.narrow) {
            fwd_tile<N, M, TAU1, ST, true, DEFER>(stage, local, a, dg, tag, exact);
            return;
          }
        }
        fwd_tile<N, M, TAU1, ST, false, DEFER>(stage, local, a, dg, tag, exact);
      });
  if constexpr (DEFER) {
    if (ok) dg.drain(true, exact);
  }
  if (ok) {
    for (int i = blockIdx.x; i < mm.count; i += gridDim.x) {
      const FwdArgs ai = multi_args<M>(mm, i);
      if (ai.full_tiles * C::kTile < ai.E) fwd_tail<N, M, TAU1, ST>(ai);
    }
  }
  if (blockIdx.x == 0) pdl_wait();
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
    const uint32_t bits = (a.hard != nullptr || a.st) ? topn_bits_dyn(kap, N, M) : 0u;
    for (int l = 0; l < M; ++l) {
      const float w = bf16_bits_to_float(a.W[e0 + l]);
      a.Wm[e0 + l] = a.st ? (((bits >> l) & 1u) ? a.W[e0 + l] : uint16_t(0))
                          : __bfloat16_as_ushort(__float2bfloat16_rn(w * S[l]));
      if (a.soft != nullptr) a.soft[e0 + l] = S[l];
    }
    if (a.hard != nullptr) {
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

template <int N, int M, bool TAU1, bool ST, bool DEFER>
int launch_tiles(const FwdArgs& a, cudaStream_t stream, bool pdl) {
  using C = Cfg<M>;
  auto kern = roi_fwd_kernel<N, M, TAU1, ST, DEFER>;
  const size_t smem = C::kSmem;
  static_assert(C::kSmem <= 232448, "shared memory per CTA");
  static LaunchCache cache;  // per instantiation and device; racing writers store the same value
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
  return launch_maybe_pdl(kern, grid, C::kThreads, smem, stream, pdl, a);
}

// Groups out of the fast path's range go to the exact routine in place (one thread,
// the rest of its warp waiting) or, below tau = 0.075, through the deferred queue
// (32 at a time).  At tau = 0.05 (the end of the paper's schedule) some 4-5 % of
// the groups leave the range and the queue makes the 7B-shaped 4:8 forward 2.1x
// faster; at tau >= 0.1 (under 0.2 % of them) the queue's code measured 2-9 % slower.
constexpr float kDeferBelowTau = 0.075f;

template <int N, int M, bool ST>
int launch_st(const FwdArgs& a, cudaStream_t stream, bool pdl) {
  if (a.tau == 1.0f) return launch_tiles<N, M, true, ST, false>(a, stream, pdl);
  return a.tau < kDeferBelowTau ? launch_tiles<N, M, false, ST, true>(a, stream, pdl)
                                : launch_tiles<N, M, false, ST, false>(a, stream, pdl);
}

template <int N, int M>
int launch_nm(const FwdArgs& a, cudaStream_t stream, bool pdl = false) {
  return a.st ? launch_st<N, M, true>(a, stream, pdl) : launch_st<N, M, false>(a, stream, pdl);
}

template <int N, int M, bool TAU1, bool ST, bool DEFER>
int launch_multi_kern(const FwdMulti& mm, cudaStream_t stream, bool pdl) {
  using C = Cfg<M>;
  auto kern = roi_fwd_multi_kernel<N, M, TAU1, ST, DEFER>;
  static LaunchCache cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return -1;
  if (cache.per_sm[dev] == 0) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(C::kMultiSmem)) != cudaSuccess)
      return -1;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, C::kThreads, C::kMultiSmem) != cudaSuccess)
      return -1;
    cache.per_sm[dev] = per_sm < 1 ? 1 : per_sm;
  }
  const int64_t cap = int64_t(sm_count()) * cache.per_sm[dev];
  int64_t want = mm.total_tiles > mm.count ? mm.total_tiles : mm.count;
  const int grid = int(want < 1 ? 1 : (want < cap ? want : cap));
  return launch_maybe_pdl(kern, grid, C::kThreads, C::kMultiSmem, stream, pdl, mm);
}

template <int N, int M, bool ST>
int launch_multi_st(const FwdMulti& mm, cudaStream_t stream, bool pdl) {
  if (mm.tau == 1.0f) return launch_multi_kern<N, M, true, ST, false>(mm, stream, pdl);
  return mm.tau < kDeferBelowTau ? launch_multi_kern<N, M, false, ST, true>(mm, stream, pdl)
                                 : launch_multi_kern<N, M, false, ST, false>(mm, stream, pdl);
}

// One launch over calls[0 .. count), with launch_st's choice of variant.
template <int N, int M>
int launch_multi(const FwdCall* calls, int count, bool pdl) {
  using C = Cfg<M>;
  static thread_local FwdMulti mm;
  mm.count = count;
  mm.st = calls[0].st;
  mm.tau = calls[0].tau;
  mm.inv_tau = 1.0f / calls[0].tau;
  mm.status = calls[0].status;
  int64_t tiles = 0;
  for (int i = 0; i < count; ++i) {
    const FwdCall& c = calls[i];
    FwdItem& x = mm.it[i];
    x.phi = c.phi;
    x.W = c.W;
    x.Wm = c.Wm;
    x.soft = c.soft;
    x.hard = c.hard;
    x.E = c.E;
    x.tile0 = tiles;
    x.np = c.np;
    x.np.narrow = counters_narrow(c.np, c.E);
    tiles += c.E / C::kTile;
  }
  mm.total_tiles = tiles;
  const cudaStream_t stream = calls[0].stream;
  return mm.st ? launch_multi_st<N, M, true>(mm, stream, pdl) : launch_multi_st<N, M, false>(mm, stream, pdl);
}

}  // namespace

namespace {
int launch_fwd_impl(const FwdCall& c, bool pdl) {
  FwdArgs a;
  a.phi = c.phi;
  a.W = c.W;
  a.Wm = c.Wm;
  a.soft = c.soft;
  a.hard = c.hard;
  a.st = c.st;
  a.E = c.E;
  a.full_tiles = c.E / (c.M == 8 ? Cfg<8>::kTile : Cfg<4>::kTile);
  a.tau = c.tau;
  a.inv_tau = 1.0f / c.tau;
  a.np = c.np;
  a.np.narrow = counters_narrow(c.np, c.E);
  a.status = c.status;
  if (c.N == 2 && c.M == 4) return launch_nm<2, 4>(a, c.stream, pdl);
  if (c.N == 4 && c.M == 8) return launch_nm<4, 8>(a, c.stream, pdl);
  if (c.N == 2 && c.M == 8) return launch_nm<2, 8>(a, c.stream, pdl);
  if (slice_supported(c.N, c.M)) return launch_slice_fwd(c, pdl);
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
}  // namespace

int launch_fwd(const FwdCall& c) { return launch_fwd_impl(c, false); }

// The tensors of a batch are independent (the caller checked that no output
// overlaps another range), so from the second launch on the tile kernels are
// launched with programmatic stream serialization: each may start while the
// previous one drains, and completes only after it (see roi_fwd_kernel).  Runs of
// small tensors with the same tile kernel share one multi-tensor launch
// (multi_small).
int launch_fwd_batch(const FwdCall* calls, int count) {
  int launched = 0;
  bool prev_tiled = false;
  for (int i = 0; i < count;) {
    const FwdCall& c = calls[i];
    if ((c.N == 2 && c.M == 4) || (c.N == 4 && c.M == 8) || (c.N == 2 && c.M == 8)) {
      // the run of small items from i on with the same tile kernel
      const int64_t tile = c.M == 8 ? Cfg<8>::kTile : Cfg<4>::kTile;
      int n = 0;
      while (i + n < count && n < kMultiMax && calls[i + n].N == c.N && calls[i + n].M == c.M &&
             multi_small(calls[i + n].E, tile))
        ++n;
      if (n >= multi_min_run(false)) {
        int r = -1;
        if (c.N == 2 && c.M == 4) r = launch_multi<2, 4>(calls + i, n, prev_tiled);
        if (c.N == 4 && c.M == 8) r = launch_multi<4, 8>(calls + i, n, prev_tiled);
        if (c.N == 2 && c.M == 8) r = launch_multi<2, 8>(calls + i, n, prev_tiled);
        if (r < 0) return -1;
        launched += r;
        prev_tiled = r > 0;
        i += n;
        continue;
      }
    }
    const bool tiled = (c.N == 2 && c.M == 4) || (c.N == 4 && c.M == 8) || (c.N == 2 && c.M == 8) ||
                       slice_supported(c.N, c.M);
    const int r = launch_fwd_impl(c, tiled && prev_tiled);
    if (r < 0) return -1;
    launched += r;
    prev_tiled = tiled && r > 0;
    ++i;
  }
  return launched;
}

}  // namespace roi
