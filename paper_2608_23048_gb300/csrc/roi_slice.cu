// Wide groups (M = 16, 32: the 8:16 and 16:32 patterns) on warp slices: the
// SL = M / 4 consecutive lanes of a slice hold one group, four members each.  Same method as the
// one-thread-per-group kernels (Sec. 4.2.2 Eq. 10-12, Algorithm 1; Eq. 5;
// backward through the relaxation), with the per-group sums, maxima and "sum of
// the other members" formed across the slice by a shuffle butterfly that never
// subtracts.  A thread holds the slots t and t + 256 of a tile; where registers
// allow, the two groups of those slots are relaxed in lockstep on packed FP32
// (V = F2, one group per half), otherwise one after the other (V = float).
// Groups whose keys leave the fast path's range are queued by the slice's first
// lane (DeferredGroups) and handled 32 at a time, one per lane, by WideRobustGroup
// (ExactGroup for non-finite keys).
#include "roi_launch.h"
#include "roi_tiles.cuh"

namespace roi {
namespace {

constexpr int kThreads = 256;
constexpr int kTile = 2048;  // 512 four-member slots: slots t and t + 256 per thread
constexpr int kStagesFwd = 4;
// backward ring stages: two at 8:16, whose two CTAs per SM also hold their step
// histories in shared memory, three at 16:32 (one CTA per SM)
template <int M>
constexpr int kStagesBwd = M == 16 ? 2 : 3;
// Both directions relax the two slots of a thread in lockstep on packed FP32; the
// backward keeps its step history in shared memory behind the tile ring.  CTAs per
// SM the registers are sized for (measured on the 3B-shaped set, tau = 0.2):
// forward two; backward two at 8:16 (128 registers) and one at 16:32, whose paired
// sixteen steps take 255 registers (at two CTAs it spills: 86.4 against 65.3 ms).
template <int M>
constexpr bool kPairedFwd = true;
template <int M>
constexpr bool kPairedBwd = true;
constexpr int kMinBlocksFwd = 2;
template <int M>
constexpr int kMinBlocksBwd = M == 32 ? 1 : 2;
// The backward's step history: steps 0 .. N-2 of one slot, or of the two slots of
// a pair (four floats or F2 a step), per thread, thread-strided so a warp touches
// consecutive words; the last step stays in registers.  Behind it, per step, the
// sum of mu over the slice's other lanes, which the sweep needs for 1 - mu.
template <int M>
constexpr size_t kSliceHistOffset = (tile_smem_bytes<kTile, kStagesBwd<M>>(8) + 15) & ~size_t(15);
template <int M>
constexpr bool kReloadHist = M == 16;
// Deferred exact-routine groups (DeferredGroups): a warp queues at most 64 / SL
// groups per tile (or per round of the ragged tail) and drains once 32 are queued.
constexpr int kDeferCap = 48;
// The kernels queue flagged groups (DeferredGroups) and run the exact routine for
// them 32 at a time.  Measured on the 3B-shaped set: at tau = 0.2 (no group flagged)
// the 16:32 step takes 87.3 ms with the queue against 94.3 ms with the exact routine
// in place; at tau = 0.05 (~4 % flagged) 8:16 takes 52.8 ms against 2424 ms and
// 16:32 135 ms against 14.7 s.
constexpr size_t kDeferBytes = size_t(kDeferCap) * 8 * (kThreads / 32);
constexpr size_t kFwdDeferOffset = (tile_smem_bytes<kTile, kStagesFwd>(6) + 15) & ~size_t(15);
template <int N, int M>
constexpr size_t kSliceHistBytes = size_t(N - 1) * 5 * (kPairedBwd<M> ? 8 : 4) * kThreads;
template <int N, int M>
constexpr size_t kSliceDeferOffset = (kSliceHistOffset<M> + kSliceHistBytes<N, M> + 15) & ~size_t(15);

__device__ __forceinline__ float shfl_xor(float v, int o) { return __shfl_xor_sync(0xffffffffu, v, o); }
__device__ __forceinline__ F2 shfl_xor(F2 v, int o) {
  return f2(__shfl_xor_sync(0xffffffffu, lo(v), o), __shfl_xor_sync(0xffffffffu, hi(v), o));
}
__device__ __forceinline__ float shfl_idx(float v, int src) { return __shfl_sync(0xffffffffu, v, src); }
__device__ __forceinline__ F2 shfl_idx(F2 v, int src) {
  return f2(__shfl_sync(0xffffffffu, lo(v), src), __shfl_sync(0xffffffffu, hi(v), src));
}

template <int SL, class V>
struct Slice {
  static_assert(SL == 4 || SL == 8, "slices of 4 or 8 lanes");
  // Sum over the slice's other lanes (never total minus own) and the total,
  // identical on every lane of the slice.
  __device__ __forceinline__ static V others(V p, V& tot) {
    V oth = shfl_xor(p, 1), acc = vadd(p, oth);
#pragma unroll
    for (int o = 2; o < SL; o <<= 1) {
      const V sib = shfl_xor(acc, o);
      oth = vadd(oth, sib);
      acc = vadd(acc, sib);
    }
    tot = acc;
    return oth;
  }
  __device__ __forceinline__ static V total(V p) {
    V t;
    others(p, t);
    return t;
  }
  __device__ __forceinline__ static V max(V v) {
#pragma unroll
    for (int o = 1; o < SL; o <<= 1) v = vmax(v, shfl_xor(v, o));
    return v;
  }
  __device__ __forceinline__ static uint32_t any(uint32_t f) {
#pragma unroll
    for (int o = 1; o < SL; o <<= 1) f |= __shfl_xor_sync(0xffffffffu, f, o);
    return f;
  }
};

template <class V>
__device__ __forceinline__ V sum4(const V (&x)[4]) {
  return vadd(vadd(x[0], x[1]), vadd(x[2], x[3]));
}
template <class V>
__device__ __forceinline__ void excl4(const V (&x)[4], V oth, V (&ex)[4]) {
  const V p01 = vadd(x[0], x[1]), p23 = vadd(x[2], x[3]);
  ex[0] = vadd(vadd(x[1], p23), oth);
  ex[1] = vadd(vadd(x[0], p23), oth);
  ex[2] = vadd(vadd(p01, x[3]), oth);
  ex[3] = vadd(vadd(p01, x[2]), oth);
}
template <class V>
__device__ __forceinline__ V max4(const V (&x)[4]) {
  return vmax(vmax(x[0], x[1]), vmax(x[2], x[3]));
}
template <class V>
__device__ __forceinline__ V min4(const V (&x)[4]) {
  return vmin(vmin(x[0], x[1]), vmin(x[2], x[3]));
}
template <class V>
__device__ __forceinline__ float lane_of(V v, int h) {
  if constexpr (vlanes<V>() == 1) {
    return v;
  } else {
    return h == 0 ? lo(v) : hi(v);
  }
}

struct SliceArgs {
  const float* phi;
  const uint16_t* W;
  const uint16_t* dWm;
  uint16_t* Wm;
  float* soft;
  uint32_t* hard;
  float* dphi;
  uint16_t* dW;
  bool st;                  // straight-through forward: Wm = W where the hard mask is set
  const uint32_t* hard_in;  // straight-through backward: dW = dWm where the forward's bit is set
  float* phi_out;           // fused AdamW: logits updated in place
  float* m;
  float* v;
  AdamW opt;
  int64_t E;
  int64_t full_tiles;
  float tau, inv_tau;
  NoiseParams np;
  unsigned int* status;
};

// Dynamic shared memory of the backward kernel (tile ring, then the step history).
extern __shared__ __align__(128) uint8_t roi_slice_smem[];

// Keys (log2 units, t = kappa log2 e) of L four-member slots (one per lane of V)
// whose first elements have call-flat indices e0[h].
template <class V>
__device__ __forceinline__ void slot_keys(const float* const* p4, const int64_t* e0, const NoiseParams& np,
                                          V (&kap)[4]) {
  constexpr int L = vlanes<V>();
  float ph[L][4];
  uint32_t x[L][4];
#pragma unroll
  for (int h = 0; h < L; ++h) {
    const float4 p = *reinterpret_cast<const float4*>(p4[h]);
    ph[h][0] = p.x, ph[h][1] = p.y, ph[h][2] = p.z, ph[h][3] = p.w;
    const uint4 q = noise_block_q(np, (np.e_base + uint64_t(e0[h])) >> 2);
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
    kap[j] = key_log2(phv, u, np.l2e_inv_lam);
  }
}

// Forward relaxation of the group(s) held by this slice; mu of every step kept
// if KEEP.  forward() returns the fallback flags (bit h: lane h of V), uniform
// over the slice.
constexpr float kTinyTotal = 7.52316384526264e-37f;  // 2^-120

template <int N, int M, bool TAU1, bool KEEP, class V>
struct SliceRelax {
  static constexpr int SL = M / 4;
  // KEEP: mu of the last step in registers, of steps 0 .. N-2 in shared memory
  // at hist[(4 k + j) kThreads] (V = float)
  V mu_last[4];
  V* hist;
  V S[4];
  V rt_last;
  __device__ __forceinline__ void put(int k, int j, V v) {
    if (k == N - 1) {
      mu_last[j] = v;
    } else {
      hist[(4 * k + j) * kThreads] = v;
    }
  }
  __device__ __forceinline__ V get(int k, int j) const { return k == N - 1 ? mu_last[j] : hist[(4 * k + j) * kThreads]; }
  // the other lanes' sum of mu of step k < N - 1, kept by forward() for the sweep
  __device__ __forceinline__ void put_oth(int k, V v) { hist[(4 * (N - 1) + k) * kThreads] = v; }
  __device__ __forceinline__ V get_oth(int k) const { return hist[(4 * (N - 1) + k) * kThreads]; }
  __device__ __forceinline__ void get4(int k, V (&m)[4]) const {
#pragma unroll
    for (int j = 0; j < 4; ++j) m[j] = get(k, j);
  }
  // S_j: accumulated by forward() without KEEP; with KEEP summed from the history
  // on demand (in forward()'s order), which only the backward's optional dW asks for.
  __device__ __forceinline__ V soft(int j) const {
    if constexpr (!KEEP) {
      return S[j];
    } else {
      V t = get(0, j);
#pragma unroll
      for (int k = 1; k < N; ++k) t = vadd(t, get(k, j));
      return t;
    }
  }

  __device__ __forceinline__ uint32_t forward(const V (&kap)[4], float inv_tau, int base_lane) {
    uint32_t flag = 0;
    V cur[4];
    if constexpr (TAU1) {
      // weights relative to the slice's first key; a member more than 100 log2
      // units from it (or a non-finite key) sends the group to the exact routine
      const V kref = shfl_idx(kap[0], base_lane);
      V e[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) e[j] = vmap(vsub(kap[j], kref), ex2_approx);
      V tot;
      Slice<SL, V>::others(sum4(e), tot);
      flag = vbelow(min4(e), kTinyExcl) | vbelow(vsub(vconst<V>(1.0f / kTinyExcl), tot), 0.0f);
      const V r = vmap(tot, rcp_approx);
#pragma unroll
      for (int j = 0; j < 4; ++j) cur[j] = vmul(e[j], r);
#pragma unroll
      for (int k = 0; k < N; ++k) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if constexpr (KEEP) put(k, j, cur[j]);
          if constexpr (!KEEP) S[j] = k == 0 ? cur[j] : vadd(S[j], cur[j]);
        }
        if (k + 1 < N) {
          V totc, o[4], v[4];
          const V oth = Slice<SL, V>::others(sum4(cur), totc);
          if constexpr (KEEP) put_oth(k, oth);
          excl4(cur, oth, o);
#pragma unroll
          for (int j = 0; j < 4; ++j) v[j] = vmul(cur[j], o[j]);
          const V rt = vmap(Slice<SL, V>::total(sum4(v)), rcp_approx);
          if (k == N - 2) rt_last = rt;
#pragma unroll
          for (int j = 0; j < 4; ++j) cur[j] = vmul(v[j], rt);
        }
      }
    } else {
      const V kmax = Slice<SL, V>::max(max4(kap));
      const V sc = vconst<V>(inv_tau);
      V d[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) d[j] = vmul(vsub(kap[j], kmax), sc);
      flag = vbelow(vsub(kmax, kmax), 0.0f);  // non-finite maximum
#pragma unroll
      for (int k = 0; k < N; ++k) {
        V e[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) e[j] = vmap(d[j], ex2_approx);
        V tot;
        const V oth = Slice<SL, V>::others(sum4(e), tot);
        const V r = vmap(tot, rcp_approx);
        if constexpr (KEEP) {
          if (k + 1 < N) put_oth(k, vmul(oth, r));
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          cur[j] = vmul(e[j], r);
          if constexpr (KEEP) put(k, j, cur[j]);
          if constexpr (!KEEP) S[j] = k == 0 ? cur[j] : vadd(S[j], cur[j]);
        }
        if (k + 1 < N) {
          // d_l += log2(1 - mu_l) / tau, the offsets first renormalised by log2 of the
          // total (so sum 2^d = 1, every offset <= 0 and the largest >= -log2 M): the
          // total comes from the butterfly above, so no maximum over the slice is
          // needed on the step's critical path.  A group whose exclusive sums drop
          // below 2^-100 of the total, or whose total drops below 2^-120 (offsets that
          // fell too far in one step, possible only for tau well below 0.05), goes
          // to the exact routine.
          V ex[4], om[4];
          excl4(e, oth, ex);
#pragma unroll
          for (int j = 0; j < 4; ++j) om[j] = vmul(ex[j], r);
          flag |= vbelow(min4(om), kTinyExcl) | vbelow(tot, kTinyTotal);
          const V lz = vmap(tot, lg2_approx);
#pragma unroll
          for (int j = 0; j < 4; ++j) d[j] = vfma(vmap(om[j], lg2_approx), sc, vsub(d[j], lz));
        }
      }
    }
    return Slice<SL, V>::any(flag);
  }

  // dk = dL/dkappa of this slot's members for c = dL/dS (the sweep of FastGroup).
  __device__ __forceinline__ void backward(const V (&c)[4], float inv_tau, V (&dk)[4]) const {
    static_assert(KEEP, "needs the steps");
    const V itau = vconst<V>(inv_tau);
    V b[4], hl[4];
    {
      V cm[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) cm[j] = vmul(c[j], mu_last[j]);
      const V cmu = Slice<SL, V>::total(sum4(cm));
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        V t = vsub(c[j], cmu);
        if constexpr (!TAU1) t = vmul(itau, t);
        b[j] = vmul(mu_last[j], t);
        if constexpr (TAU1) hl[j] = vmul(vmul(get(N - 2, j), rt_last), t);
      }
    }
#pragma unroll
    for (int k = N - 2; k >= 0; --k) {
      V cm[4], h[4], H[4], mk[4];
      get4(k, mk);
      if (TAU1 && k == N - 2) {
#pragma unroll
        for (int j = 0; j < 4; ++j) h[j] = hl[j];
      } else {
        V om[4];
        excl4(mk, get_oth(k), om);
#pragma unroll
        for (int j = 0; j < 4; ++j) h[j] = vmul(b[j], vmap(om[j], rcp_approx));
      }
      // c_l - <c, mu> + H_l - B as (c_l + H_l) - K, K = <c, mu> + B = sum of (c mu + b)
#pragma unroll
      for (int j = 0; j < 4; ++j) cm[j] = vfma(c[j], mk[j], b[j]);
      const V K = Slice<SL, V>::total(sum4(cm));
      V tmp;
      excl4(h, Slice<SL, V>::others(sum4(h), tmp), H);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const V mu_j = TAU1 ? mk[j] : vmul(mk[j], itau);
        b[j] = vfma(mu_j, vsub(vadd(c[j], H[j]), K), b[j]);
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) dk[j] = b[j];
  }
};

// Hard bits of a slot: rank of each own key among the group's M keys.
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

// Compare-exchange keeping x[a] >= x[b].
__device__ __forceinline__ void ce_desc(float (&x)[4], int a, int b) {
  const float u = x[a], v = x[b];
  x[a] = fmaxf(u, v);
  x[b] = fminf(u, v);
}
// Sorts a bitonic run of four descending.
__device__ __forceinline__ void bitonic4_desc(float (&x)[4]) {
  ce_desc(x, 0, 2), ce_desc(x, 1, 3), ce_desc(x, 0, 1), ce_desc(x, 2, 3);
}
// One bitonic merge step across lanes: with this lane's four keys sorted
// descending and the partner lane's (lane ^ o) too, the lane keeps the larger
// (upper = false) or smaller (upper = true) element of each pair (i, partner's
// 3 - i); the result is a bitonic run, sorted again in the lane.
__device__ __forceinline__ void merge_across(float (&x)[4], int o, bool upper) {
  float p[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) p[i] = __shfl_xor_sync(0xffffffffu, x[3 - i], o);
#pragma unroll
  for (int i = 0; i < 4; ++i) x[i] = upper ? fminf(x[i], p[i]) : fmaxf(x[i], p[i]);
  bitonic4_desc(x);
}

// Hard bits of a slot for N = M / 2 (the two patterns of these kernels) from the
// group's N-th largest key.  Each lane sorts its four keys; bitonic merges across
// lanes sort each half of the slice (M / 2 keys over SL / 2 lanes); the top M / 2
// of the group are then the larger elements of the pairs (i-th of the first half,
// i-th from the end of the second half), so their minimum is the threshold.  A
// member is kept iff its key is at least the threshold.  Returns false (bits
// unusable) if the slice's keys are not all finite or the threshold is tied, so
// that more than N members pass: the caller ranks such groups by comparison.
template <int N, int M>
__device__ __forceinline__ bool slice_topn_threshold(const float (&kap)[4], int q, uint32_t& bits) {
  static_assert(2 * N == M, "threshold selection needs N = M / 2");
  constexpr int SL = M / 4;
  float x[4] = {kap[0], kap[1], kap[2], kap[3]};
  ce_desc(x, 0, 1), ce_desc(x, 2, 3), ce_desc(x, 0, 2), ce_desc(x, 1, 3), ce_desc(x, 1, 2);
  // sorted runs of 8 over lane pairs
  merge_across(x, 1, (q & 1) != 0);
  if constexpr (SL == 8) {
    // sorted runs of 16 over lane quads: the larger / smaller 8 of the two runs of
    // 8 go to the quad's lower / upper lane pair (each lane's four sorted), and a
    // merge within each pair orders them
    merge_across(x, 3, (q & 2) != 0);
    merge_across(x, 1, (q & 1) != 0);
  }
  // pairs (i, M/2 - 1 - i) across the two halves: lane q pairs with lane SL - 1 - q
  float m = INFINITY;
#pragma unroll
  for (int i = 0; i < 4; ++i) m = fminf(m, fmaxf(x[i], __shfl_xor_sync(0xffffffffu, x[3 - i], SL - 1)));
#pragma unroll
  for (int o = 1; o < SL / 2; o <<= 1) m = fminf(m, __shfl_xor_sync(0xffffffffu, m, o));
  bits = 0;
  float fin = 0.0f;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    bits |= uint32_t(kap[j] >= m) << j;
    fin += kap[j] - kap[j];  // 0 for finite keys, NaN otherwise
  }
  int cnt = __popc(bits) + (fin == 0.0f ? 0 : 64);
#pragma unroll
  for (int o = 1; o < SL; o <<= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  return cnt == N;
}

// Hard bits of L slots (one per lane of V): the threshold selection, and for a
// group it cannot settle (a tie at the threshold, a non-finite key) comparison
// ranking, run by the whole warp when any of its slots needs it.
template <int N, int M, class V>
__device__ __forceinline__ void slot_topn(const V (&kap)[4], int base_lane, int q, uint32_t (&bits)[vlanes<V>()]) {
#pragma unroll
  for (int h = 0; h < vlanes<V>(); ++h) {
    float k[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) k[j] = lane_of(kap[j], h);
    const bool ok = slice_topn_threshold<N, M>(k, q, bits[h]);
    if (__any_sync(0xffffffffu, !ok)) {
      const uint32_t b = slice_topn_bits<M>(k, N, base_lane, q);
      if (!ok) bits[h] = b;
    }
  }
}

// The keys of all M elements of one group, in log2 units, from logits at phi_g
// (call-flat index g0), by one lane.
template <int N, int M>
__device__ __forceinline__ void group_keys_all(const float* phi_g, int64_t g0, const NoiseParams& np, float (&k)[M]) {
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    const float* p[1] = {phi_g + 4 * s};
    const int64_t e[1] = {g0 + 4 * s};
    float k4[4];
    slot_keys<float>(p, e, np, k4);
#pragma unroll
    for (int j = 0; j < 4; ++j) k[4 * s + j] = k4[j];
  }
}
// The exact relaxation of one group with keys t (log2 units): WideRobustGroup for
// finite keys, ExactGroup (natural-log keys) otherwise; soft mask S and, with c,
// dk = dL/dkappa.
template <int N, int M, bool BWD>
__device__ __forceinline__ void exact_relax(float (&t)[M], const float (&c)[M], const SliceArgs& a, float (&S)[M],
                                            float (&dk)[M]) {
  if (all_finite(t)) {
    WideRobustGroup<N, M> rg;
    rg.forward(t, a.inv_tau, S);
    if constexpr (BWD) rg.backward(c, a.inv_tau, dk);
  } else {
#pragma unroll
    for (int l = 0; l < M; ++l) t[l] *= kLn2;  // natural-log keys
    ExactGroup<N, M> ex;
    ex.forward(t, N, M, a.tau, S);
    if constexpr (BWD) ex.backward(c, N, M, a.tau, dk);
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

// The exact routine for one group (first element g0, call-flat), from global
// memory: the forward's outputs (Wm unless straight-through, soft).
template <int N, int M>
__device__ __forceinline__ void exact_group_fwd(int64_t g0, const SliceArgs& a) {
  if (a.soft == nullptr && a.st) return;
  float k[M], S[M], unused[M];
  group_keys_all<N, M>(a.phi + g0, g0, a.np, k);
  exact_relax<N, M, false>(k, k, a, S, unused);
#pragma unroll 1
  for (int s = 0; s < M / 4; ++s) {
    float wv[4], sv[4];
    unpack_bf16x4(*reinterpret_cast<const uint2*>(a.W + g0 + 4 * s), wv);
#pragma unroll
    for (int j = 0; j < 4; ++j) sv[j] = S[4 * s + j];
    if (!a.st) *reinterpret_cast<uint2*>(a.Wm + g0 + 4 * s) = pack4(wv, sv);
    if (a.soft != nullptr) *reinterpret_cast<float4*>(a.soft + g0 + 4 * s) = make_float4(sv[0], sv[1], sv[2], sv[3]);
  }
}
// The backward's outputs of one group: dphi, the fused AdamW step, dW unless the
// straight-through variant (which wrote it with the fast path).  The group's logits
// are untouched until here (the fast path skips its AdamW step).
template <int N, int M>
__device__ __forceinline__ void exact_group_bwd(int64_t g0, const SliceArgs& a) {
  float k[M], cc[M], S[M], dkk[M];
  group_keys_all<N, M>(a.phi + g0, g0, a.np, k);
#pragma unroll 1
  for (int s = 0; s < M / 4; ++s) {
    float wv[4], dv[4];
    unpack_bf16x4(*reinterpret_cast<const uint2*>(a.W + g0 + 4 * s), wv);
    unpack_bf16x4(*reinterpret_cast<const uint2*>(a.dWm + g0 + 4 * s), dv);
#pragma unroll
    for (int j = 0; j < 4; ++j) cc[4 * s + j] = __fmul_rn(dv[j], wv[j]);
  }
  exact_relax<N, M, true>(k, cc, a, S, dkk);
#pragma unroll 1
  for (int s = 0; s < M / 4; ++s) {
    const int64_t e = g0 + 4 * s;
    const float g4[4] = {__fmul_rn(dkk[4 * s], a.np.inv_lam), __fmul_rn(dkk[4 * s + 1], a.np.inv_lam),
                         __fmul_rn(dkk[4 * s + 2], a.np.inv_lam), __fmul_rn(dkk[4 * s + 3], a.np.inv_lam)};
    if (a.dphi != nullptr) *reinterpret_cast<float4*>(a.dphi + e) = make_float4(g4[0], g4[1], g4[2], g4[3]);
    if (a.phi_out != nullptr) adamw4(a.phi_out, a.m, a.v, e, *reinterpret_cast<const float4*>(a.phi + e), g4, a.opt);
    if (a.dW != nullptr && a.hard_in == nullptr) {
      float dv[4], sv[4];
      unpack_bf16x4(*reinterpret_cast<const uint2*>(a.dWm + e), dv);
#pragma unroll
      for (int j = 0; j < 4; ++j) sv[j] = S[4 * s + j];
      *reinterpret_cast<uint2*>(a.dW + e) = pack4(dv, sv);
    }
  }
}

// Forward of L slots (one per lane of V; p/w: each slot's logits and weights in
// shared or global memory, e0: call-flat index of its first element).  All 32
// lanes of the warp call this together; inactive slots (ragged tail, V = float
// only) take part in the shuffles with zero keys.  Returns each slot's hard bits.
template <int N, int M, bool TAU1, class V>
__device__ __forceinline__ void fwd_slots(const float* const* p, const uint16_t* const* w, const int64_t* e0,
                                          bool active, const SliceArgs& a, uint32_t (&bits)[vlanes<V>()],
                                          uint32_t& defer) {
  constexpr int SL = M / 4;
  constexpr int L = vlanes<V>();
  const int lane = threadIdx.x & 31;
  const int q = lane % SL;
  const int base_lane = lane - q;
  V kap[4];
  if (active) {
    slot_keys<V>(p, e0, a.np, kap);
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) kap[j] = vconst<V>(0.0f);
  }
  slot_topn<N, M, V>(kap, base_lane, q, bits);
  SliceRelax<N, M, TAU1, false, V> rx;
  const uint32_t flag = rx.forward(kap, a.inv_tau, base_lane);
  // groups out of the fast path's range: queued by their first lane for the exact
  // routine, which writes their outputs
  defer = active && q == 0 ? flag : 0u;
  if (!active) return;
#pragma unroll
  for (int h = 0; h < L; ++h) {
    // straight-through: every slot keeps the weights its hard bits select
    if (a.st) *reinterpret_cast<uint2*>(a.Wm + e0[h]) = keep4(*reinterpret_cast<const uint2*>(w[h]), bits[h]);
    if (!((flag >> h) & 1u)) {
      float wv[4], sv[4];
      unpack_bf16x4(*reinterpret_cast<const uint2*>(w[h]), wv);
#pragma unroll
      for (int j = 0; j < 4; ++j) sv[j] = lane_of(rx.S[j], h);
      if (!a.st) *reinterpret_cast<uint2*>(a.Wm + e0[h]) = pack4(wv, sv);
      if (a.soft != nullptr) *reinterpret_cast<float4*>(a.soft + e0[h]) = make_float4(sv[0], sv[1], sv[2], sv[3]);
    }
  }
}

// Backward of L slots (as fwd_slots).
template <int N, int M, bool TAU1, class V>
__device__ __forceinline__ void bwd_slots(const float* const* p, const uint16_t* const* w, const uint16_t* const* dw,
                                          const int64_t* e0, bool active, const SliceArgs& a, uint32_t& defer) {
  constexpr int SL = M / 4;
  constexpr int L = vlanes<V>();
  const int lane = threadIdx.x & 31;
  const int q = lane % SL;
  const int base_lane = lane - q;
  V kap[4], c[4];
  if (active) {
    slot_keys<V>(p, e0, a.np, kap);
    float wv[L][4], dv[L][4];
#pragma unroll
    for (int h = 0; h < L; ++h) {
      unpack_bf16x4(*reinterpret_cast<const uint2*>(w[h]), wv[h]);
      unpack_bf16x4(*reinterpret_cast<const uint2*>(dw[h]), dv[h]);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if constexpr (L == 1) {
        c[j] = vmul(dv[0][j], wv[0][j]);
      } else {
        c[j] = vmul(f2(dv[0][j], dv[1][j]), f2(wv[0][j], wv[1][j]));
      }
    }
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) kap[j] = c[j] = vconst<V>(0.0f);
  }
  SliceRelax<N, M, TAU1, true, V> rx;
  rx.hist = reinterpret_cast<V*>(roi_slice_smem + kSliceHistOffset<M>) + threadIdx.x;
  const uint32_t flag = rx.forward(kap, a.inv_tau, base_lane);
  defer = active && q == 0 ? flag : 0u;
  if (active && a.dW != nullptr) {
#pragma unroll
    for (int h = 0; h < L; ++h) {
      if (a.hard_in != nullptr) {
        // straight-through: dWm where the forward's hard mask is set
        *reinterpret_cast<uint2*>(a.dW + e0[h]) = keep4(*reinterpret_cast<const uint2*>(dw[h]), hard4(a.hard_in, e0[h]));
      } else if (!((flag >> h) & 1u)) {
        float dv[4], sv[4];
        unpack_bf16x4(*reinterpret_cast<const uint2*>(dw[h]), dv);
#pragma unroll
        for (int j = 0; j < 4; ++j) sv[j] = lane_of(rx.soft(j), h);
        *reinterpret_cast<uint2*>(a.dW + e0[h]) = pack4(dv, sv);
      }
    }
  }
  V dk[4];
  // 8:16: the sweep re-reads the step history from shared memory (a compiler memory
  // barrier here keeps the forward's values from being carried in registers, which
  // spills at two CTAs per SM); 16:32 runs one CTA per SM and keeps them in registers.
  if constexpr (kReloadHist<M>) asm volatile("" ::: "memory");
  rx.backward(c, a.inv_tau, dk);
  if (!active) return;
  if (a.np.inv_lam != 1.0f) {  // lambda = 1: nothing to scale, the same bits
#pragma unroll
    for (int j = 0; j < 4; ++j) dk[j] = vmul(dk[j], vconst<V>(a.np.inv_lam));
  }
#pragma unroll
  for (int h = 0; h < L; ++h) {
    if (!((flag >> h) & 1u)) {
      const float g4[4] = {lane_of(dk[0], h), lane_of(dk[1], h), lane_of(dk[2], h), lane_of(dk[3], h)};
      if (a.dphi != nullptr) *reinterpret_cast<float4*>(a.dphi + e0[h]) = make_float4(g4[0], g4[1], g4[2], g4[3]);
      if (a.phi_out != nullptr) adamw4(a.phi_out, a.m, a.v, e0[h], *reinterpret_cast<const float4*>(p[h]), g4, a.opt);
    }
  }
}

// Hard words of one slot per lane (8 lanes fill a word).
__device__ __forceinline__ void store_hard_slot(uint32_t* hard, int64_t e0, uint32_t bits, bool active) {
  const int lane = threadIdx.x & 31;
  uint32_t v = active ? bits << ((lane & 7) * 4) : 0u;
  v |= __shfl_xor_sync(0xffffffffu, v, 1);
  v |= __shfl_xor_sync(0xffffffffu, v, 2);
  v |= __shfl_xor_sync(0xffffffffu, v, 4);
  if (active && (lane & 7) == 0) hard[e0 >> 5] = v;
}
// The same for the two slots of a thread (first elements e0a, e0b; all lanes
// active): both masks travel in one register, the first slot's in the low
// half-word; after the shuffles within each 4-lane half, one exchange between
// the halves completes the first slot's word on lane 0 of the 8 and the second
// slot's word on lane 4.
__device__ __forceinline__ void store_hard_slot_pair(uint32_t* hard, int64_t e0a, int64_t e0b, uint32_t bits_a,
                                                     uint32_t bits_b) {
  const int lane = threadIdx.x & 31;
  const int sh = (lane & 3) * 4;
  uint32_t v = (bits_a << sh) | (bits_b << (16 + sh));
  v |= __shfl_xor_sync(0xffffffffu, v, 1);
  v |= __shfl_xor_sync(0xffffffffu, v, 2);
  const uint32_t o = __shfl_xor_sync(0xffffffffu, v, 4);
  const bool upper = (lane & 4) != 0;
  const uint32_t word = __byte_perm(v, o, upper ? 0x3276u : 0x5410u);
  if ((lane & 3) == 0) hard[(upper ? e0b : e0a) >> 5] = word;
}

template <int N, int M, bool TAU1>
__global__ void __launch_bounds__(kThreads, kMinBlocksFwd) roi_slice_fwd_kernel(SliceArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  TileSrc<2> src;
  src.ptr[0] = reinterpret_cast<const uint8_t*>(a.phi);
  src.esize[0] = 4;
  src.ptr[1] = reinterpret_cast<const uint8_t*>(a.W);
  src.esize[1] = 2;
  DeferredGroups<kDeferCap> dg;
  dg.init(reinterpret_cast<int64_t*>(smem + kFwdDeferOffset));
  const auto exact = [&](int64_t g0) { exact_group_fwd<N, M>(g0, a); };
  // a batch's next tensor may start on the SMs this launch frees (no-op otherwise)
  pdl_launch_dependents();
  const bool ok = run_tiles<kThreads, kTile, kStagesFwd, 2>(
      smem, src, a.full_tiles, a.status, [&](const uint8_t* const* stage, int64_t tile) {
        const float* sphi = reinterpret_cast<const float*>(stage[0]);
        const uint16_t* sW = reinterpret_cast<const uint16_t*>(stage[1]);
        const int64_t base = tile * kTile;
        const int s0 = threadIdx.x, s1 = threadIdx.x + kThreads;
        const float* pp[2] = {sphi + 4 * s0, sphi + 4 * s1};
        const uint16_t* pw[2] = {sW + 4 * s0, sW + 4 * s1};
        const int64_t e0[2] = {base + 4 * s0, base + 4 * s1};
        uint32_t bits[2], defer[2];
        if constexpr (kPairedFwd<M>) {
          uint32_t d2;
          fwd_slots<N, M, TAU1, F2>(pp, pw, e0, true, a, bits, d2);
          defer[0] = d2 & 1u, defer[1] = d2 >> 1;
        } else {
#pragma unroll 1
          for (int j = 0; j < 2; ++j) {
            uint32_t b1[1];
            fwd_slots<N, M, TAU1, float>(pp + j, pw + j, e0 + j, true, a, b1, defer[j]);
            bits[j] = b1[0];
          }
        }
        if (a.hard != nullptr) store_hard_slot_pair(a.hard, e0[0], e0[1], bits[0], bits[1]);
        dg.push(defer[0] != 0u, e0[0]);
        dg.push(defer[1] != 0u, e0[1]);
        dg.drain(false, exact);
      });
  if (ok && blockIdx.x == gridDim.x - 1) {
    const int64_t t0 = a.full_tiles * kTile;
    const int64_t slots = (a.E - t0) / 4;
    for (int64_t r = 0; r * kThreads < slots; ++r) {
      const int64_t si = threadIdx.x + r * kThreads;
      const bool active = si < slots;
      const int64_t off = t0 + 4 * (active ? si : 0);
      const float* pp[1] = {a.phi + off};
      const uint16_t* pw[1] = {a.W + off};
      const int64_t e0[1] = {t0 + 4 * si};
      uint32_t bits[1], defer;
      fwd_slots<N, M, TAU1, float>(pp, pw, e0, active, a, bits, defer);
      if (a.hard != nullptr) store_hard_slot(a.hard, e0[0], bits[0], active);
      dg.push(defer != 0u, e0[0]);
      dg.drain(false, exact);
    }
  }
  if (ok) dg.drain(true, exact);
  // the launch completes only after the batch's previous one (stream order)
  if (blockIdx.x == 0) pdl_wait();
}

template <int N, int M, bool TAU1>
__global__ void __launch_bounds__(kThreads, kMinBlocksBwd<M>) roi_slice_bwd_kernel(SliceArgs a) {
  uint8_t* smem = roi_slice_smem;
  TileSrc<3> src;
  src.ptr[0] = reinterpret_cast<const uint8_t*>(a.phi);
  src.esize[0] = 4;
  src.ptr[1] = reinterpret_cast<const uint8_t*>(a.W);
  src.esize[1] = 2;
  src.ptr[2] = reinterpret_cast<const uint8_t*>(a.dWm);
  src.esize[2] = 2;
  DeferredGroups<kDeferCap> dg;
  dg.init(reinterpret_cast<int64_t*>(smem + kSliceDeferOffset<N, M>));
  const auto exact = [&](int64_t g0) { exact_group_bwd<N, M>(g0, a); };
  pdl_launch_dependents();
  const bool ok = run_tiles<kThreads, kTile, kStagesBwd<M>, 3>(
      smem, src, a.full_tiles, a.status, [&](const uint8_t* const* stage, int64_t tile) {
        const float* sphi = reinterpret_cast<const float*>(stage[0]);
        const uint16_t* sW = reinterpret_cast<const uint16_t*>(stage[1]);
        const uint16_t* sdW = reinterpret_cast<const uint16_t*>(stage[2]);
        const int64_t base = tile * kTile;
        const int s0 = threadIdx.x, s1 = threadIdx.x + kThreads;
        const float* pp[2] = {sphi + 4 * s0, sphi + 4 * s1};
        const uint16_t* pw[2] = {sW + 4 * s0, sW + 4 * s1};
        const uint16_t* pd[2] = {sdW + 4 * s0, sdW + 4 * s1};
        const int64_t e0[2] = {base + 4 * s0, base + 4 * s1};
        uint32_t defer[2];
        if constexpr (kPairedBwd<M>) {
          uint32_t d2;
          bwd_slots<N, M, TAU1, F2>(pp, pw, pd, e0, true, a, d2);
          defer[0] = d2 & 1u, defer[1] = d2 >> 1;
        } else {
#pragma unroll 1
          for (int j = 0; j < 2; ++j)
            bwd_slots<N, M, TAU1, float>(pp + j, pw + j, pd + j, e0 + j, true, a, defer[j]);
        }
        dg.push(defer[0] != 0u, e0[0]);
        dg.push(defer[1] != 0u, e0[1]);
        dg.drain(false, exact);
      });
  if (ok && blockIdx.x == gridDim.x - 1) {
    const int64_t t0 = a.full_tiles * kTile;
    const int64_t slots = (a.E - t0) / 4;
    for (int64_t r = 0; r * kThreads < slots; ++r) {
      const int64_t si = threadIdx.x + r * kThreads;
      const bool active = si < slots;
      const int64_t off = t0 + 4 * (active ? si : 0);
      const float* pp[1] = {a.phi + off};
      const uint16_t* pw[1] = {a.W + off};
      const uint16_t* pd[1] = {a.dWm + off};
      const int64_t e0[1] = {t0 + 4 * si};
      uint32_t defer;
      bwd_slots<N, M, TAU1, float>(pp, pw, pd, e0, active, a, defer);
      dg.push(defer != 0u, e0[0]);
      dg.drain(false, exact);
    }
  }
  if (ok) dg.drain(true, exact);
  if (blockIdx.x == 0) pdl_wait();
}

struct LaunchCache {
  int per_sm[64] = {0};
};

template <class Kern>
int launch_persistent(Kern kern, LaunchCache& cache, size_t smem, const SliceArgs& a, cudaStream_t stream,
                      bool pdl) {
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
  return launch_maybe_pdl(kern, grid, kThreads, smem, stream, pdl, a);
}

template <int N, int M, bool TAU1>
int slice_fwd(const SliceArgs& a, cudaStream_t stream, bool pdl) {
  static LaunchCache cache;
  return launch_persistent(roi_slice_fwd_kernel<N, M, TAU1>, cache, kFwdDeferOffset + kDeferBytes, a, stream, pdl);
}
template <int N, int M, bool TAU1>
int slice_bwd(const SliceArgs& a, cudaStream_t stream, bool pdl) {
  static LaunchCache cache;
  constexpr size_t smem = kSliceDeferOffset<N, M> + kDeferBytes;
  static_assert(smem <= 232448, "shared memory per CTA");
  return launch_persistent(roi_slice_bwd_kernel<N, M, TAU1>, cache, smem, a, stream, pdl);
}

template <int N, int M>
int slice_fwd_nm(const SliceArgs& a, cudaStream_t stream, bool pdl) {
  return a.tau == 1.0f ? slice_fwd<N, M, true>(a, stream, pdl) : slice_fwd<N, M, false>(a, stream, pdl);
}
template <int N, int M>
int slice_bwd_nm(const SliceArgs& a, cudaStream_t stream, bool pdl) {
  return a.tau == 1.0f ? slice_bwd<N, M, true>(a, stream, pdl) : slice_bwd<N, M, false>(a, stream, pdl);
}

}  // namespace

bool slice_supported(int N, int M) { return (N == 8 && M == 16) || (N == 16 && M == 32); }

int launch_slice_fwd(const FwdCall& c, bool pdl) {
  SliceArgs a{};
  a.phi = c.phi;
  a.W = c.W;
  a.Wm = c.Wm;
  a.soft = c.soft;
  a.hard = c.hard;
  a.st = c.st;
  a.E = c.E;
  a.full_tiles = c.E / kTile;
  a.tau = c.tau;
  a.inv_tau = 1.0f / c.tau;
  a.np = c.np;
  a.status = c.status;
  if (c.N == 8 && c.M == 16) return slice_fwd_nm<8, 16>(a, c.stream, pdl);
  if (c.N == 16 && c.M == 32) return slice_fwd_nm<16, 32>(a, c.stream, pdl);
  return -1;
}

int launch_slice_bwd(const BwdCall& c, bool pdl) {
  SliceArgs a{};
  a.phi = c.phi;
  a.W = c.W;
  a.dWm = c.dWm;
  a.dphi = c.dphi;
  a.dW = c.dW;
  a.hard_in = c.hard_in;
  a.phi_out = c.phi_out;
  a.m = c.m;
  a.v = c.v;
  a.opt = c.opt;
  a.E = c.E;
  a.full_tiles = c.E / kTile;
  a.tau = c.tau;
  a.inv_tau = 1.0f / c.tau;
  a.np = c.np;
  a.status = c.status;
  if (c.N == 8 && c.M == 16) return slice_bwd_nm<8, 16>(a, c.stream, pdl);
  if (c.N == 16 && c.M == 32) return slice_bwd_nm<16, 32>(a, c.stream, pdl);
  return -1;
}

}  // namespace roi
