// Backward of the RoI mask op: regenerate the forward's noise and relaxation in
// registers, then sweep the N steps in reverse to turn dL/dS = dWm * W into
// dL/dphi (Sec. 3.2: the map from logits to the soft N-hot vector is
// differentiable; Sec. 4.2.2 Eq. 11-12).  Optionally dW = bf16(dWm * S).
#include <type_traits>

#include "roi_launch.h"
#include "roi_tiles.cuh"

namespace roi {
namespace {

// Launch shape per group size M: threads per CTA, pairs of groups per thread per
// tile (the two groups of a pair are relaxed in lockstep on packed FP32),
// shared-memory stages, and the CTAs per SM the register budget is sized for.
// One CTA per SM (see roi_fwd.cu): M = 4 with two pairs per thread and up to 128
// registers; M = 8, whose paired sweep needs ~170 registers, with 384 threads.
template <int M>
struct Cfg {
  static constexpr int kThreads = M == 4 ? 512 : 384;
  static constexpr int kPairs = M == 4 ? 2 : 1;
  static constexpr int kStages = M == 4 ? 3 : 2;  // 192 KB (M = 4), 96 KB + 72 KB step history (M = 8)
  static constexpr int kMinBlocks = 1;
  static constexpr int kTile = 2 * kPairs * kThreads * M;  // elements
  // groups out of the fast path's range, queued per warp (DeferredGroups): at most
  // 64 kPairs a tile on top of fewer than 32 left from earlier tiles
  static constexpr int kDeferCap = 32 + 64 * kPairs;
};
// Tensors of one multi-tensor launch, at most (its parameter block holds them all).
constexpr int kMultiMaxBwd = 192;
// Byte offset of the shared-memory step history (M = 8) behind the tile ring,
// and its size: steps 0 .. N-2 of two groups (one F2 per member) per thread.
template <int M>
constexpr size_t kHistOffset = (tile_smem_bytes<Cfg<M>::kTile, Cfg<M>::kStages>(8) + 15) & ~size_t(15);
template <int N, int M>
constexpr size_t kHistBytes = M == 8 ? size_t(N - 1) * M * Cfg<M>::kThreads * sizeof(F2) : 0;
// Fused optimizer with the step history in shared memory (M = 8): each thread's
// AdamW moments (two groups, m and v) are staged behind the history by per-thread
// async copies issued when the groups start, so their latency hides behind the
// relaxation without holding registers.
template <int N, int M>
constexpr size_t kMomOffset = (kHistOffset<M> + kHistBytes<N, M> + 15) & ~size_t(15);
template <int M>
constexpr size_t kMomBytes = size_t(2) * M * 2 * sizeof(float) * Cfg<M>::kThreads;
// The deferred queues behind everything else.
template <int N, int M, bool OPT>
constexpr size_t kDeferOffset =
    (kHistBytes<N, M> == 0 ? tile_smem_bytes<Cfg<M>::kTile, Cfg<M>::kStages>(8) + 15
     : OPT                 ? kMomOffset<N, M> + kMomBytes<M> + 15
                           : kHistOffset<M> + kHistBytes<N, M> + 15) & ~size_t(15);
template <int N, int M, bool OPT>
constexpr size_t kBwdSmem = kDeferOffset<N, M, OPT> + size_t(Cfg<M>::kDeferCap) * 8 * (Cfg<M>::kThreads / 32);
// multi-tensor launches: the tensors' first tiles behind the queues
template <int N, int M, bool OPT>
constexpr size_t kBwdMultiOffset = (kBwdSmem<N, M, OPT> + 15) & ~size_t(15);
template <int N, int M, bool OPT>
constexpr size_t kBwdMultiSmem = kBwdMultiOffset<N, M, OPT> + size_t(kMultiMaxBwd + 1) * 8;

// This thread's moment slot (M = 8 fused optimizer) in the dynamic shared memory.
extern __shared__ __align__(128) uint8_t roi_bwd_smem[];
template <int N, int M>
__device__ __forceinline__ float4* moment_slot() {
  return reinterpret_cast<float4*>(roi_bwd_smem + kMomOffset<N, M>) + threadIdx.x;
}

struct BwdArgs {
  const float* phi;
  const uint16_t* W;
  const uint16_t* dWm;
  float* dphi;
  uint16_t* dW;
  const uint32_t* hard_in;  // straight-through: dW = dWm where the forward's hard bit is set
  int64_t E;
  int64_t full_tiles;
  float tau, inv_tau;
  NoiseParams np;
  unsigned int* status;
};

// The fused optimizer's arguments (read only by the OPT instantiations).
struct BwdOptArgs {
  float* phi_out;  // logits updated in place
  float* m;
  float* v;
  AdamW opt;
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

// Keys (log2 units) of L groups (one per lane of V): logits from the tile stage,
// noise regenerated four members (one Philox block) at a time.
template <int M, class V, bool NARROW = false>
__device__ __forceinline__ void bwd_keys(const float* const* phi_g, const int64_t* e0, const uint32_t* q0,
                                         const NoiseParams& np, V (&kap)[M]) {
  constexpr int L = vlanes<V>();
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    float ph[L][4];
    uint32_t x[L][4];
#pragma unroll
    for (int h = 0; h < L; ++h) {
      const float4 p = reinterpret_cast<const float4*>(phi_g[h])[s];
      ph[h][0] = p.x, ph[h][1] = p.y, ph[h][2] = p.z, ph[h][3] = p.w;
      const uint4 q = NARROW ? noise_block_lo(np, q0[h] + s)
                             : noise_block_q(np, ((np.e_base + uint64_t(e0[h])) >> 2) + s);
      x[h][0] = q.x, x[h][1] = q.y, x[h][2] = q.z, x[h][3] = q.w;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      V one_plus, phv;
      if constexpr (L == 1) {
        one_plus = one_plus_from_word(x[0][j]);
        phv = ph[0][j];
      } else {
        one_plus = f2(one_plus_from_word(x[0][j]), one_plus_from_word(x[1][j]));
        phv = f2(ph[0][j], ph[1][j]);
      }
      const V u = vsub(one_plus, vconst<V>(__uint_as_float(0x3f7fffffu)));
      kap[4 * s + j] = key_log2(phv, u, np.l2e_inv_lam);
    }
  }
}

// dL/dS = dWm * W of L groups (the rounding of Wm treated as identity).
template <int M, class V>
__device__ __forceinline__ void bwd_upstream(const uint16_t* const* W_g, const uint16_t* const* dWm_g, V (&c)[M]) {
  constexpr int L = vlanes<V>();
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    float w[L][4], dw[L][4];
#pragma unroll
    for (int h = 0; h < L; ++h) {
      unpack4(reinterpret_cast<const uint2*>(W_g[h])[s], w[h]);
      unpack4(reinterpret_cast<const uint2*>(dWm_g[h])[s], dw[h]);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if constexpr (L == 1) {
        c[4 * s + j] = vmul(dw[0][j], w[0][j]);
      } else {
        c[4 * s + j] = vmul(f2(dw[0][j], dw[1][j]), f2(w[0][j], w[1][j]));
      }
    }
  }
}

// Keys and upstream gradients together, reading each stage word once.
template <int M, class V, bool NARROW = false>
__device__ __forceinline__ void bwd_inputs(const float* const* phi_g, const uint16_t* const* W_g,
                                           const uint16_t* const* dWm_g, const int64_t* e0, const uint32_t* q0,
                                           const NoiseParams& np, V (&kap)[M], V (&c)[M]) {
  constexpr int L = vlanes<V>();
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    float ph[L][4], w[L][4], dw[L][4];
    uint32_t x[L][4];
#pragma unroll
    for (int h = 0; h < L; ++h) {
      const float4 p = reinterpret_cast<const float4*>(phi_g[h])[s];
      ph[h][0] = p.x, ph[h][1] = p.y, ph[h][2] = p.z, ph[h][3] = p.w;
      unpack4(reinterpret_cast<const uint2*>(W_g[h])[s], w[h]);
      unpack4(reinterpret_cast<const uint2*>(dWm_g[h])[s], dw[h]);
      const uint4 q = NARROW ? noise_block_lo(np, q0[h] + s)
                             : noise_block_q(np, ((np.e_base + uint64_t(e0[h])) >> 2) + s);
      x[h][0] = q.x, x[h][1] = q.y, x[h][2] = q.z, x[h][3] = q.w;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      V one_plus, phv, wv, dwv;
      if constexpr (L == 1) {
        one_plus = one_plus_from_word(x[0][j]);
        phv = ph[0][j], wv = w[0][j], dwv = dw[0][j];
      } else {
        one_plus = f2(one_plus_from_word(x[0][j]), one_plus_from_word(x[1][j]));
        phv = f2(ph[0][j], ph[1][j]), wv = f2(w[0][j], w[1][j]), dwv = f2(dw[0][j], dw[1][j]);
      }
      const V u = vsub(one_plus, vconst<V>(__uint_as_float(0x3f7fffffu)));
      kap[4 * s + j] = key_log2(phv, u, np.l2e_inv_lam);
      c[4 * s + j] = vmul(dwv, wv);
    }
  }
}

// L groups (one per lane of V) in lockstep: regenerate keys and relaxation,
// sweep back, write dL/dphi (and dW).  `hist` (shared memory, this thread's
// slot) holds steps 0 .. N-2 of the relaxation when HIST is set; otherwise the
// whole history stays in registers.  With HIST (M = 8) registers are tight:
// the keys die after the forward relaxation (a flagged group re-forms them) and
// the upstream gradients are formed only for the sweep.
template <int N, int M, bool TAU1, class V, bool HIST = false, bool ST = false, bool OPT = false,
          bool NARROW = false, bool DEFER = false>
__device__ __forceinline__ uint32_t bwd_groups(const float* const* phi_g, const uint16_t* const* W_g,
                                           const uint16_t* const* dWm_g, const int64_t* e0, const uint32_t* q0,
                                           const BwdArgs& a, const BwdOptArgs& o, V* hist = nullptr) {
  constexpr int L = vlanes<V>();
  // straight-through: the forward's hard bits of these groups, loaded now so the
  // load's latency hides behind the relaxation.  With HIST (registers tight) dW,
  // which needs nothing else, is written at once and the bits die here.
  uint32_t keep[ST ? L : 1][ST ? M / 4 : 1];
  if constexpr (ST) {
#pragma unroll
    for (int h = 0; h < L; ++h)
#pragma unroll
      for (int s = 0; s < M / 4; ++s) keep[h][s] = hard4(a.hard_in, e0[h] + 4 * s);
    if (HIST && a.dW != nullptr) {
#pragma unroll
      for (int s = 0; s < M / 4; ++s)
#pragma unroll
        for (int h = 0; h < L; ++h)
          reinterpret_cast<uint2*>(a.dW + e0[h])[s] =
              keep4(reinterpret_cast<const uint2*>(dWm_g[h])[s], keep[h][s]);
    }
  }
  // fused optimizer: the moments, fetched now for the epilogue, into registers
  // (M = 4) or into this thread's shared-memory slot `mom` (with HIST)
  constexpr bool kPrefetchMoments = OPT && !HIST;
  constexpr bool kStageMoments = OPT && HIST;
  constexpr int kT = Cfg<M>::kThreads;
  if constexpr (kStageMoments) {
    float4* mom = moment_slot<N, M>();
#pragma unroll
    for (int h = 0; h < L; ++h)
#pragma unroll
      for (int s = 0; s < M / 4; ++s) {
        cp_async16(mom + (2 * (h * (M / 4) + s)) * kT, o.m + e0[h] + 4 * s);
        cp_async16(mom + (2 * (h * (M / 4) + s) + 1) * kT, o.v + e0[h] + 4 * s);
      }
    cp_async_commit();
  }
  float4 mom_m[kPrefetchMoments ? L : 1][kPrefetchMoments ? M / 4 : 1];
  float4 mom_v[kPrefetchMoments ? L : 1][kPrefetchMoments ? M / 4 : 1];
  if constexpr (kPrefetchMoments) {
#pragma unroll
    for (int h = 0; h < L; ++h)
#pragma unroll
      for (int s = 0; s < M / 4; ++s) {
        mom_m[h][s] = reinterpret_cast<const float4*>(o.m + e0[h])[s];
        mom_v[h][s] = reinterpret_cast<const float4*>(o.v + e0[h])[s];
      }
  }
  using Steps = typename std::conditional<HIST, SmemSteps<N, M, V, Cfg<M>::kThreads>, RegSteps<N, M, V>>::type;
  FastGroup<N, M, TAU1, true, V, Steps> fg;
  if constexpr (HIST) fg.st.at = hist;
  V kap[HIST ? 1 : M], c[M], dkv[M];
  if constexpr (HIST) {
    V k[M];
    bwd_keys<M, V, NARROW>(phi_g, e0, q0, a.np, k);
    fg.forward(k, a.inv_tau);
  } else {
    bwd_inputs<M, V, NARROW>(phi_g, W_g, dWm_g, e0, q0, a.np, kap, c);
    fg.forward(kap, a.inv_tau);
  }
  if (a.dW != nullptr && !(ST && HIST)) {
    // dW = bf16(dWm * S) now, while the relaxation is live anyway (dWm is re-read);
    // straight-through: dWm where the forward's hard mask is set, +0 elsewhere
#pragma unroll
    for (int s = 0; s < M / 4; ++s) {
      if constexpr (ST) {
#pragma unroll
        for (int h = 0; h < L; ++h)
          reinterpret_cast<uint2*>(a.dW + e0[h])[s] =
              keep4(reinterpret_cast<const uint2*>(dWm_g[h])[s], keep[h][s]);
      } else if constexpr (L == 2) {
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
  if constexpr (HIST) bwd_upstream<M, V>(W_g, dWm_g, c);
  fg.backward(c, a.inv_tau, dkv);
  // dL/dphi = dL/dkappa / lambda (lambda = 1: nothing to scale, the same bits)
  if (a.np.inv_lam != 1.0f) {
#pragma unroll
    for (int l = 0; l < M; ++l) dkv[l] = vmul(dkv[l], vconst<V>(a.np.inv_lam));
  }
  if constexpr (kStageMoments) cp_async_wait_all();
#pragma unroll
  for (int h = 0; h < L; ++h) {
    float dk[M];
#pragma unroll
    for (int l = 0; l < M; ++l) dk[l] = lane_of(dkv[l], h);
    // DEFER: a group out of the fast path's range leaves its outputs (and its AdamW
    // step) to bwd_exact_group, which the caller runs for it from the deferred queue
    if (DEFER && ((fg.flag >> h) & 1u)) continue;
    if (!DEFER && ((fg.flag >> h) & 1u)) {
      // rare: the log2-domain or (non-finite keys) the exact routine in place, with HIST
      // from re-formed keys of this group (the opaque copy of the parameters keeps
      // the compiler from holding the first keys live)
      float k[M], cc[M], S[M];
      if constexpr (HIST) {
        NoiseParams np = a.np;
        asm volatile("" : "+r"(np.k0));
        bwd_keys<M, float>(phi_g + h, e0 + h, nullptr, np, k);
      } else {
#pragma unroll
        for (int l = 0; l < M; ++l) k[l] = lane_of(kap[l], h);
      }
#pragma unroll
      for (int l = 0; l < M; ++l) cc[l] = lane_of(c[l], h);
      if (!TAU1 && all_finite(k)) {
        RobustGroup<N, M> rg;  // finite keys spread beyond the fast path's float range (as roi_fwd.cu)
        rg.forward(k, a.inv_tau, S);
        rg.backward(cc, a.inv_tau, dk);
      } else {
#pragma unroll
        for (int l = 0; l < M; ++l) k[l] *= kLn2;  // natural-log keys
        ExactGroup<N, M> ex;
        ex.forward(k, N, M, a.tau, S);
        ex.backward(cc, N, M, a.tau, dk);
      }
#pragma unroll
      for (int l = 0; l < M; ++l) dk[l] = __fmul_rn(dk[l], a.np.inv_lam);
      if (!ST && a.dW != nullptr) {
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
    if constexpr (OPT) {
      // fused AdamW step on these logits (their old values are still in phi_g)
#pragma unroll
      for (int s = 0; s < M / 4; ++s) {
        const float g4[4] = {dk[4 * s], dk[4 * s + 1], dk[4 * s + 2], dk[4 * s + 3]};
        if constexpr (kPrefetchMoments) {
          adamw4(o.phi_out, o.m, o.v, e0[h] + 4 * s, reinterpret_cast<const float4*>(phi_g[h])[s], g4, o.opt,
                 mom_m[h][s], mom_v[h][s]);
        } else if constexpr (kStageMoments) {
          const float4* mom = moment_slot<N, M>();
          adamw4(o.phi_out, o.m, o.v, e0[h] + 4 * s, reinterpret_cast<const float4*>(phi_g[h])[s], g4, o.opt,
                 mom[(2 * (h * (M / 4) + s)) * kT], mom[(2 * (h * (M / 4) + s) + 1) * kT]);
        } else {
          adamw4(o.phi_out, o.m, o.v, e0[h] + 4 * s, reinterpret_cast<const float4*>(phi_g[h])[s], g4, o.opt);
        }
      }
    }
    if (!OPT || a.dphi != nullptr) {
#pragma unroll
      for (int s = 0; s < M / 4; ++s)
        reinterpret_cast<float4*>(a.dphi + e0[h])[s] = make_float4(dk[4 * s], dk[4 * s + 1], dk[4 * s + 2], dk[4 * s + 3]);
    }
  }
  return DEFER ? fg.flag : 0u;
}

// The exact routine for one group out of the fast path's range (first element g0,
// call-flat), from global memory (as fwd_exact_group): dphi, the fused AdamW step
// (the fast path left this group's logits and moments untouched) and, unless
// straight-through, dW = bf16(dWm * S).
template <int N, int M, bool TAU1, bool ST, bool OPT>
__device__ __forceinline__ void bwd_exact_group(int64_t g0, const BwdArgs& a, const BwdOptArgs& o) {
  // keys and upstream gradients as the tiles' packed code forms them (the group in
  // both halves)
  const float* pp[2] = {a.phi + g0, a.phi + g0};
  const uint16_t* pw[2] = {a.W + g0, a.W + g0};
  const uint16_t* pd[2] = {a.dWm + g0, a.dWm + g0};
  const int64_t e0[2] = {g0, g0};
  F2 k2[M], c2[M];
  bwd_keys<M, F2>(pp, e0, nullptr, a.np, k2);
  bwd_upstream<M, F2>(pw, pd, c2);
  float k[M], cc[M], S[M], dk[M];
#pragma unroll
  for (int l = 0; l < M; ++l) k[l] = lo(k2[l]), cc[l] = lo(c2[l]);
  if (!TAU1 && all_finite(k)) {
    RobustGroup<N, M> rg;
    rg.forward(k, a.inv_tau, S);
    rg.backward(cc, a.inv_tau, dk);
  } else {
#pragma unroll
    for (int l = 0; l < M; ++l) k[l] *= kLn2;  // natural-log keys
    ExactGroup<N, M> ex;
    ex.forward(k, N, M, a.tau, S);
    ex.backward(cc, N, M, a.tau, dk);
  }
#pragma unroll
  for (int l = 0; l < M; ++l) dk[l] = __fmul_rn(dk[l], a.np.inv_lam);
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    if (!ST && a.dW != nullptr) {
      float d[4];
      unpack4(reinterpret_cast<const uint2*>(a.dWm + g0)[s], d);
      uint2 w;
      w.x = pack_bf16x2(__fmul_rn(d[0], S[4 * s]), __fmul_rn(d[1], S[4 * s + 1]));
      w.y = pack_bf16x2(__fmul_rn(d[2], S[4 * s + 2]), __fmul_rn(d[3], S[4 * s + 3]));
      reinterpret_cast<uint2*>(a.dW + g0)[s] = w;
    }
    const float g4[4] = {dk[4 * s], dk[4 * s + 1], dk[4 * s + 2], dk[4 * s + 3]};
    if constexpr (OPT) adamw4(o.phi_out, o.m, o.v, g0 + 4 * s, reinterpret_cast<const float4*>(a.phi + g0)[s], g4, o.opt);
    if (!OPT || a.dphi != nullptr)
      reinterpret_cast<float4*>(a.dphi + g0)[s] = make_float4(g4[0], g4[1], g4[2], g4[3]);
  }
}

// One full tile of a tensor (local tile index `tile`), inputs staged in shared
// memory.  NARROW: the call's counters are below 2^32 (a.np.narrow).
// `tag` (the tensor's index in a multi-tensor launch, shifted to bit 48) is or-ed into
// the queued entries.
template <int N, int M, bool TAU1, bool ST, bool OPT, bool NARROW, bool DEFER, class Defer, class Exact>
__device__ __forceinline__ void bwd_tile(const uint8_t* const* stage, int64_t tile, const BwdArgs& a,
                                         const BwdOptArgs& o, uint8_t* smem, Defer& dg, int64_t tag,
                                         const Exact& exact) {
  using C = Cfg<M>;
  const float* sphi = reinterpret_cast<const float*>(stage[0]);
  const uint16_t* sW = reinterpret_cast<const uint16_t*>(stage[1]);
  const uint16_t* sdW = reinterpret_cast<const uint16_t*>(stage[2]);
  const int64_t base = tile * C::kTile;
  // low word of the tile's first counter (uniform); group g adds g M / 4
  const uint32_t qt = uint32_t((a.np.e_base + uint64_t(base)) >> 2);
#pragma unroll
  for (int p = 0; p < C::kPairs; ++p) {
    const int g0 = threadIdx.x + 2 * p * C::kThreads, g1 = g0 + C::kThreads;
    const float* pp[2] = {sphi + g0 * M, sphi + g1 * M};
    const uint16_t* pw[2] = {sW + g0 * M, sW + g1 * M};
    const uint16_t* pd[2] = {sdW + g0 * M, sdW + g1 * M};
    const int64_t e0[2] = {base + g0 * M, base + g1 * M};
    const uint32_t q0[2] = {qt + uint32_t(g0 * (M / 4)), qt + uint32_t(g1 * (M / 4))};
    uint32_t flag;
    if constexpr (M == 4) {
      flag = bwd_groups<N, M, TAU1, F2, false, ST, OPT, NARROW, DEFER>(pp, pw, pd, e0, q0, a, o);
    } else {
      // M = 8: the paired step history does not fit the register file; steps
      // 0 .. N-2 go to shared memory behind the tile ring
      F2* hist = reinterpret_cast<F2*>(smem + kHistOffset<M>) + threadIdx.x;
      flag = bwd_groups<N, M, TAU1, F2, true, ST, OPT, NARROW, DEFER>(pp, pw, pd, e0, q0, a, o, hist);
    }
    if constexpr (DEFER) {
      dg.push((flag & 1u) != 0u, tag | e0[0]);
      dg.push((flag & 2u) != 0u, tag | e0[1]);
    }
  }
  if constexpr (DEFER) dg.drain(false, exact);
}

// The ragged tail of a tensor (fewer than one tile after its full tiles), by one
// CTA, straight from global memory.
template <int N, int M, bool TAU1, bool ST, bool OPT>
__device__ __forceinline__ void bwd_tail(const BwdArgs& a, const BwdOptArgs& o) {
  using C = Cfg<M>;
  const int64_t t0 = a.full_tiles * C::kTile;
  const int64_t tail_groups = (a.E - t0) / M;
  for (int64_t gi = threadIdx.x; gi < tail_groups; gi += C::kThreads) {
    const float* pp[1] = {a.phi + t0 + gi * M};
    const uint16_t* pw[1] = {a.W + t0 + gi * M};
    const uint16_t* pd[1] = {a.dWm + t0 + gi * M};
    const int64_t e0[1] = {t0 + gi * M};
    bwd_groups<N, M, TAU1, float, false, ST, OPT>(pp, pw, pd, e0, nullptr, a, o);
  }
}

// ST: straight-through dW from the forward's hard bits; OPT: fused AdamW step on
// the logits (separate instantiations, so the plain kernel's code is not touched)
// NARROW_ONLY: launched only for calls whose counters are all below 2^32 (32-bit
// counters): every M = 4 variant, and the 4:8 tau = 1 backward fused with AdamW (at
// 4:8 the narrow plain backward spilled, 225 against 192 us per 18944 x 3584
// tensor, while the fused one gained, 386 against 418 us)
template <int N, int M, bool TAU1, bool ST, bool OPT, bool NARROW_ONLY, bool DEFER>
__global__ void __launch_bounds__(Cfg<M>::kThreads, Cfg<M>::kMinBlocks) roi_bwd_kernel(BwdArgs a, BwdOptArgs o) {
  uint8_t* smem = roi_bwd_smem;
  using C = Cfg<M>;
  TileSrc<3> src;
  src.ptr[0] = reinterpret_cast<const uint8_t*>(a.phi);
  src.esize[0] = 4;
  src.ptr[1] = reinterpret_cast<const uint8_t*>(a.W);
  src.esize[1] = 2;
  src.ptr[2] = reinterpret_cast<const uint8_t*>(a.dWm);
  src.esize[2] = 2;
  DeferredGroups<C::kDeferCap> dg;
  dg.init(smem + kDeferOffset<N, M, OPT>);
  const auto exact = [&](int64_t g0) { bwd_exact_group<N, M, TAU1, ST, OPT>(g0, a, o); };
  // a batch's next tensor may start on the SMs this launch frees (no-op otherwise)
  pdl_launch_dependents();
  const bool ok = run_tiles<C::kThreads, C::kTile, C::kStages, 3>(
      smem, src, a.full_tiles, a.status,
      [&](const uint8_t* const* stage, int64_t tile) {
        bwd_tile<N, M, TAU1, ST, OPT, NARROW_ONLY, DEFER>(stage, tile, a, o, smem, dg, 0, exact);
      });
  if constexpr (DEFER) {
    if (ok) dg.drain(true, exact);
  }
  if (ok && blockIdx.x == gridDim.x - 1) bwd_tail<N, M, TAU1, ST, OPT>(a, o);
  // the launch completes only after the batch's previous one (stream order)
  if (blockIdx.x == 0) pdl_wait();
}

// Multi-tensor launches: the tensors' arguments, and their first tiles in the
// concatenated tile sequence of the launch (tile0).
struct BwdItem {
  const float* phi;
  const uint16_t* W;
  const uint16_t* dWm;
  float* dphi;
  uint16_t* dW;
  const uint32_t* hard_in;
  float* phi_out;
  float* m;
  float* v;
  int64_t E;
  int64_t tile0;
  NoiseParams np;
};
struct BwdMulti {
  int count;
  int64_t total_tiles;
  float tau, inv_tau;
  unsigned int* status;
  AdamW opt;
  BwdItem it[kMultiMaxBwd];
};
static_assert(sizeof(BwdMulti) <= 32764, "kernel parameter block");
template <int M>
__device__ __forceinline__ BwdArgs multi_args(const BwdMulti& mm, int i) {
  const BwdItem& x = mm.it[i];
  BwdArgs a;
  a.phi = x.phi;
  a.W = x.W;
  a.dWm = x.dWm;
  a.dphi = x.dphi;
  a.dW = x.dW;
  a.hard_in = x.hard_in;
  a.E = x.E;
  a.full_tiles = x.E / Cfg<M>::kTile;
  a.tau = mm.tau;
  a.inv_tau = mm.inv_tau;
  a.np = x.np;
  a.status = mm.status;
  return a;
}
__device__ __forceinline__ BwdOptArgs multi_opt(const BwdMulti& mm, int i) {
  BwdOptArgs o;
  o.phi_out = mm.it[i].phi_out;
  o.m = mm.it[i].m;
  o.v = mm.it[i].v;
  o.opt = mm.opt;
  return o;
}
// roi_bwd_kernel over many small tensors at once, walked as roi_fwd_multi_kernel
// walks them.
template <int N, int M, bool TAU1, bool ST, bool OPT, bool NARROW_ONLY, bool DEFER>
__global__ void __launch_bounds__(Cfg<M>::kThreads, Cfg<M>::kMinBlocks)
    roi_bwd_multi_kernel(const __grid_constant__ BwdMulti mm) {
  uint8_t* smem = roi_bwd_smem;
  using C = Cfg<M>;
  const uint32_t esize[3] = {4, 2, 2};
  constexpr int64_t kLow = (int64_t(1) << 48) - 1;
  int64_t* tile0 = reinterpret_cast<int64_t*>(smem + kBwdMultiOffset<N, M, OPT>);
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
  dg.init(smem + kDeferOffset<N, M, OPT>);
  const auto exact = [&](int64_t e) {
    const int i = int(e >> 48);
    bwd_exact_group<N, M, TAU1, ST, OPT>(e & kLow, multi_args<M>(mm, i), multi_opt(mm, i));
  };
  int cur = -1, src_cur = -1;
  int64_t lo = 0, hi = 0, src_lo = 0, src_hi = 0;
  BwdArgs a;
  BwdOptArgs o;
  const uint8_t* src_ptr[3] = {nullptr, nullptr, nullptr};
  pdl_launch_dependents();
  const bool ok = run_tiles_src<C::kThreads, C::kTile, C::kStages, 3>(
      smem, esize, mm.total_tiles, mm.status,
      [&](int64_t t, int arr) {
        if (t < src_lo || t >= src_hi) {
          src_cur = find(t);
          src_lo = tile0[src_cur];
          src_hi = tile0[src_cur + 1];
          src_ptr[0] = reinterpret_cast<const uint8_t*>(mm.it[src_cur].phi);
          src_ptr[1] = reinterpret_cast<const uint8_t*>(mm.it[src_cur].W);
          src_ptr[2] = reinterpret_cast<const uint8_t*>(mm.it[src_cur].dWm);
        }
        return src_ptr[arr] + size_t(t - src_lo) * C::kTile * esize[arr];
      },
      [&](const uint8_t* const* stage, int64_t t) {
        if (t < lo || t >= hi) {
          cur = find(t);
          lo = tile0[cur];
          hi = tile0[cur + 1];
          a = multi_args<M>(mm, cur);
          o = multi_opt(mm, cur);
        }
        bwd_tile<N, M, TAU1, ST, OPT, NARROW_ONLY, DEFER>(stage, t - lo, a, o, smem, dg, int64_t(cur) << 48, exact);
      });
  if constexpr (DEFER) {
    if (ok) dg.drain(true, exact);
  }
  if (ok) {
    for (int i = blockIdx.x; i < mm.count; i += gridDim.x) {
      const BwdArgs ai = multi_args<M>(mm, i);
      if (ai.full_tiles * C::kTile < ai.E) bwd_tail<N, M, TAU1, ST, OPT>(ai, multi_opt(mm, i));
    }
  }
  if (blockIdx.x == 0) pdl_wait();
}

__global__ void __launch_bounds__(128) roi_bwd_generic_kernel(BwdArgs a, BwdOptArgs o, int N, int M) {
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
      const int64_t e = e0 + l;
      const float g = dk[l] * a.np.inv_lam;
      if (a.dphi != nullptr) a.dphi[e] = g;
      if (o.phi_out != nullptr) {
        float ph = a.phi[e], mm = o.m[e], vv = o.v[e];
        adamw_elem(ph, g, mm, vv, o.opt);
        o.phi_out[e] = ph;
        o.m[e] = mm;
        o.v[e] = vv;
      }
      if (a.dW != nullptr) {
        if (a.hard_in != nullptr) {
          a.dW[e] = ((a.hard_in[e >> 5] >> (e & 31)) & 1u) ? a.dWm[e] : uint16_t(0);
        } else {
          a.dW[e] = __bfloat16_as_ushort(__float2bfloat16_rn(bf16_bits_to_float(a.dWm[e]) * S[l]));
        }
      }
    }
  }
}

struct LaunchCache {
  int per_sm[64] = {0};
};

template <int N, int M, bool TAU1, bool ST, bool OPT, bool NARROW_ONLY, bool DEFER>
int launch_tiles(const BwdArgs& a, const BwdOptArgs& o, cudaStream_t stream, bool pdl = false) {
  using C = Cfg<M>;
  auto kern = roi_bwd_kernel<N, M, TAU1, ST, OPT, NARROW_ONLY, DEFER>;
  const size_t smem = kBwdSmem<N, M, OPT>;
  static_assert(kBwdSmem<N, M, OPT> <= 232448, "shared memory per CTA");
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
  return launch_maybe_pdl(kern, grid, C::kThreads, smem, stream, pdl, a, o);
}

// Groups out of the fast path's range: the exact routine in place, or through the
// deferred queue (32 at a time) for every 2:4 backward (measured 2.7 % faster at
// tau = 1 on the 7B-shaped set) and for the others below tau = 0.075 (at tau = 0.05
// some 4-5 % of the groups leave the range and the queue makes the 7B-shaped 4:8
// backward 3.5x faster; at tau = 0.5 the 4:8 queue code measured 3 % slower).
constexpr float kDeferBelowTau = 0.075f;

template <int N, int M, bool ST, bool OPT, bool NARROW_ONLY = false>
int launch_tau(const BwdArgs& a, const BwdOptArgs& o, cudaStream_t stream, bool pdl) {
  if (a.tau == 1.0f) return launch_tiles<N, M, true, ST, OPT, NARROW_ONLY, M == 4>(a, o, stream, pdl);
  if constexpr (M == 4) {
    return launch_tiles<N, M, false, ST, OPT, NARROW_ONLY, true>(a, o, stream, pdl);
  } else {
    return a.tau < kDeferBelowTau ? launch_tiles<N, M, false, ST, OPT, NARROW_ONLY, true>(a, o, stream, pdl)
                                  : launch_tiles<N, M, false, ST, OPT, NARROW_ONLY, false>(a, o, stream, pdl);
  }
}

template <int N, int M>
int launch_nm(const BwdArgs& a, const BwdOptArgs& o, cudaStream_t stream, bool pdl = false) {
  if constexpr (N == 4 && M == 8) {
    if (a.tau == 1.0f && a.np.narrow && o.phi_out != nullptr)
      return launch_tiles<N, M, true, false, true, true, false>(a, o, stream, pdl);
  }
  if constexpr (M == 4) {
    if (a.np.narrow) {
      if (o.phi_out != nullptr) return launch_tau<N, M, false, true, true>(a, o, stream, pdl);
      if (a.hard_in != nullptr && a.dW != nullptr) return launch_tau<N, M, true, false, true>(a, o, stream, pdl);
      return launch_tau<N, M, false, false, true>(a, o, stream, pdl);
    }
  }
  if (o.phi_out != nullptr) return launch_tau<N, M, false, true>(a, o, stream, pdl);
  if (a.hard_in != nullptr && a.dW != nullptr) return launch_tau<N, M, true, false>(a, o, stream, pdl);
  return launch_tau<N, M, false, false>(a, o, stream, pdl);
}

template <int N, int M, bool TAU1, bool ST, bool OPT, bool NARROW_ONLY, bool DEFER>
int launch_multi_kern(const BwdMulti& mm, cudaStream_t stream, bool pdl) {
  using C = Cfg<M>;
  auto kern = roi_bwd_multi_kernel<N, M, TAU1, ST, OPT, NARROW_ONLY, DEFER>;
  constexpr size_t smem = kBwdMultiSmem<N, M, OPT>;
  static_assert(smem <= 232448, "shared memory per CTA");
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
  const int64_t want = mm.total_tiles > mm.count ? mm.total_tiles : mm.count;
  const int grid = int(want < 1 ? 1 : (want < cap ? want : cap));
  return launch_maybe_pdl(kern, grid, C::kThreads, smem, stream, pdl, mm);
}

template <int N, int M, bool ST, bool OPT, bool NARROW_ONLY = false>
int launch_multi_tau(const BwdMulti& mm, cudaStream_t stream, bool pdl) {
  if (mm.tau == 1.0f) return launch_multi_kern<N, M, true, ST, OPT, NARROW_ONLY, M == 4>(mm, stream, pdl);
  if constexpr (M == 4) {
    return launch_multi_kern<N, M, false, ST, OPT, NARROW_ONLY, true>(mm, stream, pdl);
  } else {
    return mm.tau < kDeferBelowTau ? launch_multi_kern<N, M, false, ST, OPT, NARROW_ONLY, true>(mm, stream, pdl)
                                   : launch_multi_kern<N, M, false, ST, OPT, NARROW_ONLY, false>(mm, stream, pdl);
  }
}

// The backward variant a call needs, in launch_nm's order: 2 fused AdamW,
// 1 straight-through dW, 0 plain.
int bwd_kind(const BwdCall& c) { return c.phi_out != nullptr ? 2 : (c.hard_in != nullptr && c.dW != nullptr ? 1 : 0); }

// One launch over calls[0 .. count): one kind, one counter width, with launch_nm's
// choice of variant.
template <int N, int M>
int launch_multi(const BwdCall* calls, int count, bool pdl) {
  using C = Cfg<M>;
  static thread_local BwdMulti mm;
  mm.count = count;
  mm.tau = calls[0].tau;
  mm.inv_tau = 1.0f / calls[0].tau;
  mm.status = calls[0].status;
  mm.opt = calls[0].opt;
  int64_t tiles = 0;
  for (int i = 0; i < count; ++i) {
    const BwdCall& c = calls[i];
    BwdItem& x = mm.it[i];
    x.phi = c.phi;
    x.W = c.W;
    x.dWm = c.dWm;
    x.dphi = c.dphi;
    x.dW = c.dW;
    x.hard_in = c.hard_in;
    x.phi_out = c.phi_out;
    x.m = c.m;
    x.v = c.v;
    x.E = c.E;
    x.tile0 = tiles;
    x.np = c.np;
    x.np.narrow = counters_narrow(c.np, c.E);
    tiles += c.E / C::kTile;
  }
  mm.total_tiles = tiles;
  const cudaStream_t stream = calls[0].stream;
  const int kind = bwd_kind(calls[0]);
  const bool narrow = mm.it[0].np.narrow;
  if constexpr (N == 4 && M == 8) {
    if (mm.tau == 1.0f && narrow && kind == 2)
      return launch_multi_kern<N, M, true, false, true, true, false>(mm, stream, pdl);
  }
  if constexpr (M == 4) {
    if (narrow) {
      if (kind == 2) return launch_multi_tau<N, M, false, true, true>(mm, stream, pdl);
      if (kind == 1) return launch_multi_tau<N, M, true, false, true>(mm, stream, pdl);
      return launch_multi_tau<N, M, false, false, true>(mm, stream, pdl);
    }
  }
  if (kind == 2) return launch_multi_tau<N, M, false, true>(mm, stream, pdl);
  if (kind == 1) return launch_multi_tau<N, M, true, false>(mm, stream, pdl);
  return launch_multi_tau<N, M, false, false>(mm, stream, pdl);
}

}  // namespace

namespace {
int launch_bwd_impl(const BwdCall& c, bool pdl) {
  BwdArgs a;
  a.phi = c.phi;
  a.W = c.W;
  a.dWm = c.dWm;
  a.dphi = c.dphi;
  a.dW = c.dW;
  a.hard_in = c.hard_in;
  BwdOptArgs o;
  o.phi_out = c.phi_out;
  o.m = c.m;
  o.v = c.v;
  o.opt = c.opt;
  a.E = c.E;
  a.full_tiles = c.E / (c.M == 8 ? Cfg<8>::kTile : Cfg<4>::kTile);
  a.tau = c.tau;
  a.inv_tau = 1.0f / c.tau;
  a.np = c.np;
  a.np.narrow = counters_narrow(c.np, c.E);
  a.status = c.status;
  if (c.N == 2 && c.M == 4) return launch_nm<2, 4>(a, o, c.stream, pdl);
  if (c.N == 4 && c.M == 8) return launch_nm<4, 8>(a, o, c.stream, pdl);
  if (c.N == 2 && c.M == 8) return launch_nm<2, 8>(a, o, c.stream, pdl);
  if (slice_supported(c.N, c.M)) return launch_slice_bwd(c, pdl);
  const int64_t groups = c.E / c.M;
  int64_t blocks = (groups + 127) / 128;
  const int64_t cap = int64_t(sm_count()) * 16;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  roi_bwd_generic_kernel<<<int(blocks), 128, 0, c.stream>>>(a, o, c.N, c.M);
  return cudaGetLastError() == cudaSuccess ? 1 : -1;
}
}  // namespace

int launch_bwd(const BwdCall& c) { return launch_bwd_impl(c, false); }

// As launch_fwd_batch: the tensors are independent, so from the second launch on
// the tile kernels (plain or fused with AdamW) are launched with programmatic
// stream serialization, and runs of small tensors with the same tile kernel share
// one multi-tensor launch.
int launch_bwd_batch(const BwdCall* calls, int count) {
  int launched = 0;
  bool prev_tiled = false;
  for (int i = 0; i < count;) {
    const BwdCall& c = calls[i];
    if ((c.N == 2 && c.M == 4) || (c.N == 4 && c.M == 8) || (c.N == 2 && c.M == 8)) {
      // the run of small items from i on with the same tile kernel
      const int64_t tile = c.M == 8 ? Cfg<8>::kTile : Cfg<4>::kTile;
      const int kind = bwd_kind(c);
      const bool narrow = counters_narrow(c.np, c.E);
      int n = 0;
      while (i + n < count && n < kMultiMaxBwd && calls[i + n].N == c.N && calls[i + n].M == c.M &&
             bwd_kind(calls[i + n]) == kind && counters_narrow(calls[i + n].np, calls[i + n].E) == narrow &&
             multi_small(calls[i + n].E, tile))
        ++n;
      if (n >= multi_min_run(kind == 0 && c.tau >= kDeferBelowTau)) {
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
    const int r = launch_bwd_impl(c, tiled && prev_tiled);
    if (r < 0) return -1;
    launched += r;
    prev_tiled = tiled && r > 0;
    ++i;
  }
  return launched;
}

}  // namespace roi
