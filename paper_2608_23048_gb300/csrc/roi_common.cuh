// Device building blocks of the RoI mask op (sm_103a).
//
// Paper: "Reservoir of Importance: Learning Semi-Structured Sparsity with
// Differentiable Subset Sampling".  What is computed per group of M weights:
//   kappa = phi / lambda + g, g = -log(-log u)          (Sec. 4.2.2 Eq. 10, Sec. 4.2.3)
//   alpha(1) = kappa; mu(k) = softmax(alpha(k) / tau);
//   alpha(k+1) = alpha(k) + log(1 - mu(k))               (Sec. 4.2.2 Eq. 11-12, Algorithm 1)
//   S = sum_k mu(k); hard = Gumbel-top-N of kappa        (Sec. 3.2)
// and the reverse-mode derivative of S with respect to kappa.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include "roi_vec.cuh"

namespace roi {

// ---------------------------------------------------------------------------
// small helpers
// ---------------------------------------------------------------------------
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
// Exclusive sums below this value mean all other members of a group are more
// than ~69 natural-log units below the top key: exp() of them no longer fits the
// fast path's float range and the group is recomputed by the exact routine.
constexpr float kTinyExcl = 7.888609052210118e-31f;  // 2^-100

// The device status record (defined in roi_api.cu, one per device, passed to the
// kernels by address): word 0 holds the status bits, words 2-3 (a 64-bit value,
// 8-byte aligned) the wall-time limit in ns of a wait for a stage of a copy ring.
// kStatusTimeout is set in word 0 when a kernel gave up such a wait.
constexpr unsigned int kStatusTimeout = 1u;
constexpr int kStatusLimitWord = 2;

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float bf16_bits_to_float(uint32_t bits16) {
  return __uint_as_float(bits16 << 16);
}
// Straight-through variant: the four bf16 weights of q where the low four bits of
// `keep` are set (bit j: element j), +0 elsewhere.
__device__ __forceinline__ uint2 keep4(uint2 q, uint32_t keep) {
  const uint32_t m0 = ((keep & 1u) ? 0x0000ffffu : 0u) | ((keep & 2u) ? 0xffff0000u : 0u);
  const uint32_t m1 = ((keep & 4u) ? 0x0000ffffu : 0u) | ((keep & 8u) ? 0xffff0000u : 0u);
  return make_uint2(q.x & m0, q.y & m1);
}
// The hard-mask bits of elements e .. e + 3 (e % 4 == 0) from the flat word array.
__device__ __forceinline__ uint32_t hard4(const uint32_t* hard, int64_t e) {
  return (hard[e >> 5] >> (uint32_t(e) & 31u)) & 0xfu;
}
// One AdamW step on a logit (decoupled weight decay, bias-corrected moments):
//   phi <- phi (1 - lr wd); m <- b1 m + (1 - b1) g; v <- b2 v + (1 - b2) g^2;
//   phi <- phi - (step m) / (sqrt(v) r + eps),  step = lr / (1 - b1^t), r = 1 / sqrt(1 - b2^t).
// Explicitly rounded operations, correctly rounded divide and square root.
struct AdamW {
  float b1, omb1, b2, omb2, eps, decay, step, r;  // decay = 1 - lr wd, omb_i = 1 - b_i
};
__device__ __forceinline__ void adamw_elem(float& phi, float g, float& m, float& v, const AdamW& o) {
  phi = __fmul_rn(phi, o.decay);
  m = __fadd_rn(__fmul_rn(o.b1, m), __fmul_rn(o.omb1, g));
  v = __fadd_rn(__fmul_rn(o.b2, v), __fmul_rn(o.omb2, __fmul_rn(g, g)));
  const float den = __fadd_rn(__fmul_rn(__fsqrt_rn(v), o.r), o.eps);
  phi = __fsub_rn(phi, __fdiv_rn(__fmul_rn(o.step, m), den));
}
// The step for four consecutive logits at `e` (16-byte aligned): old logits phi4
// (from the tile stage or global memory), gradients g, moments mm, vv; the new
// logits and moments are stored.
__device__ __forceinline__ void adamw4(float* phi_out, float* m, float* v, int64_t e, float4 phi4,
                                       const float (&g)[4], const AdamW& o, float4 mm, float4 vv) {
  adamw_elem(phi4.x, g[0], mm.x, vv.x, o);
  adamw_elem(phi4.y, g[1], mm.y, vv.y, o);
  adamw_elem(phi4.z, g[2], mm.z, vv.z, o);
  adamw_elem(phi4.w, g[3], mm.w, vv.w, o);
  *reinterpret_cast<float4*>(phi_out + e) = phi4;
  *reinterpret_cast<float4*>(m + e) = mm;
  *reinterpret_cast<float4*>(v + e) = vv;
}
// ... loading the moments here.
__device__ __forceinline__ void adamw4(float* phi_out, float* m, float* v, int64_t e, float4 phi4,
                                       const float (&g)[4], const AdamW& o) {
  adamw4(phi_out, m, v, e, phi4, g, o, *reinterpret_cast<const float4*>(m + e),
         *reinterpret_cast<const float4*>(v + e));
}

// Two floats -> two bf16 (round to nearest even), packed low|high.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// ---------------------------------------------------------------------------
// noise: Philox-4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11, Philox family)
// ---------------------------------------------------------------------------
constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    // one 32x32 -> 64-bit product per multiplier gives both (hi, lo) words
    const uint64_t p0 = uint64_t(kPhiloxM0) * c.x;
    const uint64_t p1 = uint64_t(kPhiloxM1) * c.z;
    const uint32_t hi0 = uint32_t(p0 >> 32), lo0 = uint32_t(p0);
    const uint32_t hi1 = uint32_t(p1 >> 32), lo1 = uint32_t(p1);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    k0 += kPhiloxW0;
    k1 += kPhiloxW1;
  }
  return c;
}

struct NoiseParams {
  uint32_t k0, k1;       // seed words
  uint32_t step, tensor_id;
  float inv_lam;         // 1 / lambda
  float l2e_inv_lam;     // log2(e) / lambda: keys in log2 units, t = phi log2(e) / lambda - log2(E)
  uint64_t e_base;       // row_offset * cols: flat index of this call's element 0
  // every counter of the call is below 2^32 (e_base + E <= 2^34): the tile kernels
  // then form the counter's low word in 32-bit arithmetic and its high word is 0
  bool narrow = false;
};

// The four noise words of block q (elements 4q .. 4q+3).
__device__ __forceinline__ uint4 noise_block_q(const NoiseParams& np, uint64_t q) {
  return philox4x32_10(make_uint4(uint32_t(q), uint32_t(q >> 32), np.step, np.tensor_id), np.k0, np.k1);
}
// Block q of a call whose counters are all below 2^32 (the same words as
// noise_block_q(np, q)); the high word is the constant 0, so the first two rounds
// take their other inputs (step, tensor id, key) from kernel parameters.
__device__ __forceinline__ uint4 noise_block_lo(const NoiseParams& np, uint32_t q) {
  return philox4x32_10(make_uint4(q, 0u, np.step, np.tensor_id), np.k0, np.k1);
}
// Four consecutive noise words for elements e4 .. e4+3 (e4 % 4 == 0).
__device__ __forceinline__ uint4 noise_block(const NoiseParams& np, uint64_t e4) {
  return noise_block_q(np, e4 >> 2);
}
// The word of a single element (any e).
__device__ __forceinline__ uint32_t noise_word(const NoiseParams& np, uint64_t e) {
  const uint4 w = noise_block(np, e & ~uint64_t(3));
  const uint32_t s = uint32_t(e & 3);
  return s == 0 ? w.x : s == 1 ? w.y : s == 2 ? w.z : w.w;
}

// The bits of 1 + k 2^-23 with k = x >> 9: (x >> 9) | 0x3f800000 is one funnel
// shift of the 64-bit pair {127 : x} right by 9 (127 << 23 == 0x3f800000).
__device__ __forceinline__ float one_plus_from_word(uint32_t x) {
  return __uint_as_float(__funnelshift_r(x, 127u, 9));
}
// u = ((x >> 9) + 1/2) * 2^-23, exactly: (1 + k 2^-23) - (1 - 2^-24) is exact
// by Sterbenz's lemma and equals (2k + 1) 2^-24.
__device__ __forceinline__ float uniform_from_word(uint32_t x) {
  return __fsub_rn(one_plus_from_word(x), __uint_as_float(0x3f7fffffu));
}

// E = -ln(u) for u in [2^-24, 1) with a small relative error everywhere,
// including u -> 1 where E -> 0 (the hardware log2 has an absolute error floor
// there).  Method: u = 2^e m with m in [sqrt(1/2), sqrt(2)), split exactly from
// the float's bits (subtracting the bits of sqrt(1/2) makes the exponent field
// round log2 u to the nearest integer at the sqrt(2) boundaries), so
// ln u = e ln2 + ln m; ln m = 2 atanh(s), s = (m - 1) / (m + 1), |s| < 0.172,
// 2 atanh(s) = 2s + (2/3)s^3 + (2/5)s^5 + (2/7)s^7 + (2/9)s^9 + O(s^11)
// (truncation below 2^-28 relative).  m - 1 is exact (Sterbenz).  In t = -2s,
// formed with one reciprocal as (m - 1) / (-(m + 1) / 2) (the halving folded into
// the fma that forms the denominator), -ln m = t + t^3/12 + t^5/80 + t^7/448 +
// t^9/2304: the leading term is added last and exactly in a fused multiply-add,
// with no separate negation or doubling.
__device__ __forceinline__ int rounded_exponent(float x) {
  return int(__float_as_uint(x) - 0x3f3504f3u) >> 23;  // 0x3f3504f3: sqrt(1/2)
}
template <class V>
__device__ __forceinline__ V neg_log_unit(V u) {
  // m = u 2^-e (the exponent field moved by e) and e as a float (the integer
  // added into the mantissa of 1.5 * 2^23)
  const V m = vmap(u, [](float x) { return __uint_as_float(__float_as_uint(x) - (uint32_t(rounded_exponent(x)) << 23)); });
  const V ef = vsub(vmap(u, [](float x) { return __int_as_float(rounded_exponent(x) + 0x4B400000); }),
                    vconst<V>(12582912.0f));
  const V one = vconst<V>(1.0f);
  const V f = vsub(m, one);
  const V t = vmul(f, vmap(vfma(m, vconst<V>(-0.5f), vconst<V>(-0.5f)), rcp_approx));
  const V t2 = vmul(t, t);
  V q = vfma(t2, vconst<V>(1.0f / 2304.0f), vconst<V>(1.0f / 448.0f));
  q = vfma(t2, q, vconst<V>(1.0f / 80.0f));
  q = vfma(t2, q, vconst<V>(1.0f / 12.0f));
  const V nlnm = vfma(vmul(t, t2), q, t);  // -ln m
  return vfma(ef, vconst<V>(-kLn2), nlnm);
}

// log2 of E = -ln u.  The keys the fast kernels rank and relax are kept in log2
// units, t = kappa log2(e) = phi log2(e) / lambda - log2(E) (Eq. 10 with
// g = -ln E), so exp2 of key differences needs no further scaling.  The outer
// log only needs absolute accuracy (it enters the key additively) and uses the
// hardware log2.
template <class V>
__device__ __forceinline__ V log2_neg_log_unit(V u) {
  return vmap(neg_log_unit(u), lg2_approx);
}
// Key in log2 units from the logit and the uniform.
template <class V>
__device__ __forceinline__ V key_log2(V phi, V u, float l2e_inv_lam) {
  return vsub(vmul(phi, vconst<V>(l2e_inv_lam)), log2_neg_log_unit(u));
}
// Gumbel(0,1) sample g = -log(-log u) (Algorithm 1) in natural units.
template <class V>
__device__ __forceinline__ V gumbel_from_u(V u) {
  return vmul(log2_neg_log_unit(u), vconst<V>(-kLn2));
}
__device__ __forceinline__ float gumbel_from_word(uint32_t x) {
  return gumbel_from_u(uniform_from_word(x));
}

// ---------------------------------------------------------------------------
// hard top-N of one group: bit l set iff key l is among the N largest
// (NaN ranks as -inf, equal keys: lower index first)
// ---------------------------------------------------------------------------
template <int M>
__device__ __forceinline__ uint32_t topn_bits(const float (&kap)[M], int N) {
  float k[M];
  int rank[M];
#pragma unroll
  for (int l = 0; l < M; ++l) {
    k[l] = fmaxf(kap[l], -INFINITY);  // NaN -> -inf
    rank[l] = 0;
  }
#pragma unroll
  for (int l = 1; l < M; ++l) {
#pragma unroll
    for (int i = 0; i < l; ++i) {
      const int t = k[i] >= k[l];  // i beats l (i has the lower index)
      rank[l] += t;
      rank[i] += 1 - t;
    }
  }
  uint32_t bits = 0;
#pragma unroll
  for (int l = 0; l < M; ++l) bits |= uint32_t(rank[l] < N) << l;
  return bits;
}

// M = 4: l is selected iff it beats at least 4 - N of the other three keys.
__device__ __forceinline__ uint32_t topn_bits4(const float (&kap)[4], int N) {
  const float k0 = fmaxf(kap[0], -INFINITY), k1 = fmaxf(kap[1], -INFINITY);
  const float k2 = fmaxf(kap[2], -INFINITY), k3 = fmaxf(kap[3], -INFINITY);
  // tij: i beats j (i < j, ties to the lower index)
  const bool t01 = k0 >= k1, t02 = k0 >= k2, t03 = k0 >= k3;
  const bool t12 = k1 >= k2, t13 = k1 >= k3, t23 = k2 >= k3;
  const bool w0[3] = {t01, t02, t03}, w1[3] = {!t01, t12, t13};
  const bool w2[3] = {!t02, !t12, t23}, w3[3] = {!t03, !t13, !t23};
  auto pick = [N](const bool (&w)[3]) -> uint32_t {
    if (N == 2) return uint32_t((w[0] & w[1]) | (w[0] & w[2]) | (w[1] & w[2]));
    if (N == 1) return uint32_t(w[0] & w[1] & w[2]);
    return uint32_t(w[0] | w[1] | w[2]);
  };
  return pick(w0) | (pick(w1) << 1) | (pick(w2) << 2) | (pick(w3) << 3);
}

// M = 4, two groups at once (one per lane of F2), for groups whose four keys are
// all finite: the sign bit of k_i - k_j is set iff k_i < k_j, i.e. iff j outranks
// i (equal keys give +0, so the lower index wins, as above).  The six pairwise
// differences of both groups take six packed subtractions; each member's
// selection is then one 3-input logic function of its three signs (majority for
// N = 2, AND for N = 1, OR for N = 3).  Differences are exact in sign: no
// flush-to-zero, and x - y == 0 only for x == y.
__device__ __forceinline__ void topn_bits4_signs(const F2 (&k)[4], int N, uint32_t (&bits)[2]) {
  const F2 d01 = k[0] - k[1], d02 = k[0] - k[2], d03 = k[0] - k[3];
  const F2 d12 = k[1] - k[2], d13 = k[1] - k[3], d23 = k[2] - k[3];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    auto sg = [h](F2 d) { return __float_as_uint(h == 0 ? lo(d) : hi(d)); };
    const uint32_t s01 = sg(d01), s02 = sg(d02), s03 = sg(d03), s12 = sg(d12), s13 = sg(d13), s23 = sg(d23);
    // member l wins against j < l when s_jl is set, against j > l when s_lj is clear
    uint32_t w0, w1, w2, w3;
    if (N == 2) {
      auto maj = [](uint32_t a, uint32_t b, uint32_t c) { return (a & b) | (a & c) | (b & c); };
      w0 = ~maj(s01, s02, s03);
      w1 = maj(s01, ~s12, ~s13);
      w2 = maj(s02, s12, ~s23);
      w3 = maj(s03, s13, s23);
    } else if (N == 1) {
      w0 = ~(s01 | s02 | s03);
      w1 = s01 & ~s12 & ~s13;
      w2 = s02 & s12 & ~s23;
      w3 = s03 & s13 & s23;
    } else {
      w0 = ~(s01 & s02 & s03);
      w1 = s01 | ~s12 | ~s13;
      w2 = s02 | s12 | ~s23;
      w3 = s03 | s13 | s23;
    }
    bits[h] = (w0 >> 31) | ((w1 >> 31) << 1) | ((w2 >> 31) << 2) | ((w3 >> 31) << 3);
  }
}

// Three-input maximum / minimum (one instruction on sm_100 and later).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// M = 8, two groups at once, for groups whose keys are all finite: member l is
// selected iff its key is at least the group's N-th largest key, read off the
// sign bit of the packed difference.  The N-th largest comes from the two sorted
// halves: with a_1 >= .. >= a_4 and b_1 >= .. >= b_4 (five compare-exchanges
// each), the N-th largest of all eight is the largest min(a_i, b_j) over
// i + j = N (a_0 = b_0 = +inf): some such pair lies within the top N, and of
// any such pair one member lies outside the top N - 1.  When the threshold is
// tied with another member more than N members pass; such a group gets
// 0xffffffff and the caller re-ranks it with topn_bits<8>.
template <int N>
__device__ __forceinline__ void topn_bits8_threshold(const F2 (&k)[8], uint32_t (&bits)[2]) {
  static_assert(N >= 1 && N < 8, "1 <= N < 8");
  float thr[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    float s[8];
#pragma unroll
    for (int l = 0; l < 8; ++l) s[l] = h == 0 ? lo(k[l]) : hi(k[l]);
    // descending: after a compare-exchange (a, b), s[a] >= s[b]
    auto ce = [&s](int a, int b) {
      const float x = s[a], y = s[b];
      s[a] = fmaxf(x, y);
      s[b] = fminf(x, y);
    };
    ce(0, 1), ce(2, 3), ce(0, 2), ce(1, 3), ce(1, 2);  // s[0..3] = a_1..a_4
    ce(4, 5), ce(6, 7), ce(4, 6), ce(5, 7), ce(5, 6);  // s[4..7] = b_1..b_4
    float c[5];
    int nc = 0;
#pragma unroll
    for (int i = 0; i <= N; ++i) {
      const int j = N - i;
      if (i > 4 || j > 4) continue;
      c[nc++] = i == 0 ? s[3 + j] : j == 0 ? s[i - 1] : fminf(s[i - 1], s[3 + j]);
    }
    float t = c[0];
    int q = 1;
#pragma unroll
    for (; q + 1 < nc; q += 2) t = fmax3(t, c[q], c[q + 1]);
    if (q < nc) t = fmaxf(t, c[q]);
    thr[h] = t;
  }
  const F2 t = f2(thr[0], thr[1]);
  uint32_t sg[2][8];
#pragma unroll
  for (int l = 0; l < 8; ++l) {
    const F2 d = k[l] - t;  // >= 0 (sign bit clear) iff member l passes
    sg[0][l] = __float_as_uint(lo(d));
    sg[1][l] = __float_as_uint(hi(d));
  }
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    // the sign bytes of members 0-3 and 4-7 into two words; their four top bits
    // (7, 15, 23, 31) land in bits 28-31 of the product with 2^21 + 2^14 + 2^7 + 1
    const uint32_t a = __byte_perm(__byte_perm(sg[h][0], sg[h][1], 0x0073u), __byte_perm(sg[h][2], sg[h][3], 0x0073u), 0x5410u);
    const uint32_t b = __byte_perm(__byte_perm(sg[h][4], sg[h][5], 0x0073u), __byte_perm(sg[h][6], sg[h][7], 0x0073u), 0x5410u);
    const uint32_t pa = ((~a & 0x80808080u) * 0x00204081u) >> 28;
    const uint32_t pb = ((~b & 0x80808080u) * 0x00204081u) >> 28;
    const uint32_t v = pa | (pb << 4);
    bits[h] = __popc(v) == N ? v : 0xffffffffu;
  }
}

// Runtime-M version for the generic path (M <= 32).
__device__ __forceinline__ uint32_t topn_bits_dyn(const float* kap, int N, int M) {
  uint32_t bits = 0;
  for (int l = 0; l < M; ++l) {
    const float kl = fmaxf(kap[l], -INFINITY);
    int rank = 0;
    for (int i = 0; i < M; ++i) {
      const float ki = fmaxf(kap[i], -INFINITY);
      rank += (i < l) ? (ki >= kl) : (i > l ? (ki > kl) : 0);
    }
    bits |= uint32_t(rank < N) << l;
  }
  return bits;
}

// ---------------------------------------------------------------------------
// Exact log-space relaxation of one group (fp32, accurate expf/logf).
// Follows the recursion literally: z = alpha / tau, mu = exp(z - LSE z),
// log(1 - mu_l) = LSE_{i != l} z_i - LSE z (no clamp).  The backward uses the
// bounded form d l_i / d z_l = [l != i] exp(z_l - LSE_{j != i} z_j) - mu_l.
// Used for groups the fast path flags, for ragged tails and for N:M patterns
// without a specialised kernel.  NMAX x MMAX bounds the (runtime) N x M.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float lse_excluding(const float* z, int M, int skip) {
  float m = -INFINITY;
  for (int i = 0; i < M; ++i)
    if (i != skip) m = fmaxf(m, z[i]);
  if (m == -INFINITY) return -INFINITY;  // every member -inf
  if (m == INFINITY) return INFINITY;     // a +inf member
  float s = 0.f;
  for (int i = 0; i < M; ++i)
    if (i != skip) s = __fadd_rn(s, expf(__fsub_rn(z[i], m)));
  return __fadd_rn(m, logf(s));
}

template <int NMAX, int MMAX>
struct ExactGroup {
  float zh[NMAX][MMAX];  // z at every step (history for the backward)

  // Forward: fills S[0..M).  kap: perturbed keys.
  __device__ __forceinline__ void forward(const float* kap, int N, int M, float tau, float* S) {
    float z[MMAX];
    for (int l = 0; l < M; ++l) {
      z[l] = __fdiv_rn(kap[l], tau);
      S[l] = 0.f;
    }
    for (int k = 0; k < N; ++k) {
      for (int l = 0; l < M; ++l) zh[k][l] = z[l];
      const float lt = lse_excluding(z, M, -1);
      for (int l = 0; l < M; ++l) S[l] = __fadd_rn(S[l], expf(__fsub_rn(z[l], lt)));
      if (k + 1 < N) {
        float zn[MMAX];
        float zmax = -INFINITY;
        for (int l = 0; l < M; ++l) {
          zn[l] = __fadd_rn(z[l], __fdiv_rn(__fsub_rn(lse_excluding(z, M, l), lt), tau));
          zmax = fmaxf(zmax, zn[l]);
        }
        // shift so the largest key is 0 (softmax and log(1 - mu) are shift-invariant):
        // keeps the rounding of the keys that matter small over many steps
        if (zmax > -INFINITY && zmax < INFINITY) {
          for (int l = 0; l < M; ++l) z[l] = __fsub_rn(zn[l], zmax);
        } else {
          for (int l = 0; l < M; ++l) z[l] = zn[l];
        }
      }
    }
  }

  // Backward after forward(): dk = dL/dkappa for c = dL/dS.
  __device__ __forceinline__ void backward(const float* c, int N, int M, float tau, float* dk) {
    float b[MMAX];
    for (int l = 0; l < M; ++l) b[l] = 0.f;
    for (int k = N - 1; k >= 0; --k) {
      const float* z = zh[k];
      const float lt = lse_excluding(z, M, -1);
      float mu[MMAX], gz[MMAX];
      float cmu = 0.f, B = 0.f;
      for (int l = 0; l < M; ++l) {
        mu[l] = expf(z[l] - lt);
        cmu += c[l] * mu[l];
        B += b[l];
      }
      for (int l = 0; l < M; ++l) gz[l] = mu[l] * (c[l] - cmu) - mu[l] * B;
      if (k + 1 < N) {
        for (int i = 0; i < M; ++i) {
          if (b[i] == 0.f) continue;
          const float li = lse_excluding(z, M, i);
          for (int l = 0; l < M; ++l)
            if (l != i) gz[l] += b[i] * expf(z[l] - li);
        }
      }
      for (int l = 0; l < M; ++l) b[l] += gz[l] / tau;
    }
    for (int l = 0; l < M; ++l) dk[l] = b[l];
  }
};

// ---------------------------------------------------------------------------
// Log2-domain relaxation of one group whose keys are finite but spread beyond
// the fast path's float range (compile-time N, M; the fast kernels' fallback).
// The same recursion as ExactGroup, in log2 units z = t / tau (t: keys in log2
// units), with the hardware exp2 / log2: every log-sum-exp, and every exclusive
// one (over all members but l), is formed against its own maximum, so no sum
// underflows whatever the spread; O(M^2) exponentials per step.  mu and the
// softmax-without-i weights nu do not depend on the base, so the backward below
// is ExactGroup's (the oracle's bounded form) and returns dL/dkappa as it does.
// ---------------------------------------------------------------------------
template <int M>
__device__ __forceinline__ void lse2_excluding_each(const float (&x)[M], float (&out)[M]) {
  float pre[M], suf[M];  // maxima of the members before / after l
  pre[0] = -INFINITY;
#pragma unroll
  for (int l = 1; l < M; ++l) pre[l] = fmaxf(pre[l - 1], x[l - 1]);
  suf[M - 1] = -INFINITY;
#pragma unroll
  for (int l = M - 2; l >= 0; --l) suf[l] = fmaxf(suf[l + 1], x[l + 1]);
#pragma unroll
  for (int l = 0; l < M; ++l) {
    const float m = fmaxf(pre[l], suf[l]);
    float s = 0.0f;
#pragma unroll
    for (int i = 0; i < M; ++i)
      if (i != l) s = __fadd_rn(s, ex2_approx(__fsub_rn(x[i], m)));
    out[l] = __fadd_rn(m, lg2_approx(s));
  }
}

template <int N, int M>
struct RobustGroup {
  float zh[N][M];  // z entering each step, shifted so its maximum is 0

  // mu = softmax of z (log2 units); returns log2 of the normaliser against max 0
  static __device__ __forceinline__ float softmax2(const float (&z)[M], float (&mu)[M]) {
    float s = 0.0f;
#pragma unroll
    for (int l = 0; l < M; ++l) {
      mu[l] = ex2_approx(z[l]);
      s = __fadd_rn(s, mu[l]);
    }
    const float r = rcp_approx(s);
#pragma unroll
    for (int l = 0; l < M; ++l) mu[l] = __fmul_rn(mu[l], r);
    return lg2_approx(s);
  }

  // t: the keys in log2 units (t = kappa log2 e), all finite.  Fills S.
  __device__ __forceinline__ void forward(const float (&t)[M], float inv_tau, float (&S)[M]) {
    float z[M], zmax = -INFINITY;
#pragma unroll
    for (int l = 0; l < M; ++l) {
      z[l] = __fmul_rn(t[l], inv_tau);
      zmax = fmaxf(zmax, z[l]);
      S[l] = 0.0f;
    }
#pragma unroll
    for (int k = 0; k < N; ++k) {
#pragma unroll
      for (int l = 0; l < M; ++l) {
        z[l] = __fsub_rn(z[l], zmax);
        zh[k][l] = z[l];
      }
      float mu[M];
      const float lz = softmax2(z, mu);
#pragma unroll
      for (int l = 0; l < M; ++l) S[l] = __fadd_rn(S[l], mu[l]);
      if (k + 1 < N) {
        // z_l += log2(1 - mu_l) / tau, log2(1 - mu_l) = LSE2 over the others - LSE2 of all
        float lx[M];
        lse2_excluding_each(z, lx);
        zmax = -INFINITY;
#pragma unroll
        for (int l = 0; l < M; ++l) {
          z[l] = __fmaf_rn(__fsub_rn(lx[l], lz), inv_tau, z[l]);
          zmax = fmaxf(zmax, z[l]);
        }
      }
    }
  }

  // After forward(): dk = dL/dkappa for c = dL/dS.
  __device__ __forceinline__ void backward(const float (&c)[M], float inv_tau, float (&dk)[M]) const {
    float b[M];
#pragma unroll
    for (int l = 0; l < M; ++l) b[l] = 0.0f;
#pragma unroll
    for (int k = N - 1; k >= 0; --k) {
      const float(&z)[M] = zh[k];
      float mu[M], gz[M];
      softmax2(z, mu);
      float cmu = 0.0f, B = 0.0f;
#pragma unroll
      for (int l = 0; l < M; ++l) {
        cmu = __fmaf_rn(c[l], mu[l], cmu);
        B = __fadd_rn(B, b[l]);
      }
#pragma unroll
      for (int l = 0; l < M; ++l) gz[l] = __fmul_rn(mu[l], __fsub_rn(__fsub_rn(c[l], cmu), B));
      if (k + 1 < N) {
        // (J^T b)_l adds sum over i != l of b_i nu(-i)_l, nu(-i)_l = 2^(z_l - LSE2 over j != i)
        float lx[M];
        lse2_excluding_each(z, lx);
#pragma unroll
        for (int i = 0; i < M; ++i)
#pragma unroll
          for (int l = 0; l < M; ++l)
            if (l != i) gz[l] = __fmaf_rn(b[i], ex2_approx(__fsub_rn(z[l], lx[i])), gz[l]);
      }
#pragma unroll
      for (int l = 0; l < M; ++l) b[l] = __fmaf_rn(gz[l], inv_tau, b[l]);
    }
#pragma unroll
    for (int l = 0; l < M; ++l) dk[l] = b[l];
  }
};

// ---------------------------------------------------------------------------
// The log2-domain relaxation of RobustGroup in O(M) per step, for the wide groups
// of the warp-slice kernels (M = 16, 32), finite keys.  With m1 the largest z,
// a its (first) index and m2 the largest of the others, every exclusive sum over
// j != l is formed against m1 for l != a (it contains 2^0 from member a, so it
// cannot underflow) and against m2 for l = a; the sums use prefix and suffix sums,
// no subtraction.  The backward's sum over i != l of b_i 2^(z_l - LSE_{j != i} z_j)
// splits the same way: for i != a, 2^(m1 - LSE_{j != i}) lies in [1/M, 1] and the
// terms are 2^(z_l - m1) times an exclusive sum; the i = a term is formed directly.
// Members stay in registers; the step history goes to local memory.
// ---------------------------------------------------------------------------
template <int M>
struct Top2 {
  float m1, m2;
  int a;
  __device__ __forceinline__ explicit Top2(const float (&z)[M]) {
    m1 = -INFINITY, m2 = -INFINITY, a = 0;
#pragma unroll
    for (int l = 0; l < M; ++l) {
      if (z[l] > m1) {
        m2 = m1, m1 = z[l], a = l;
      } else {
        m2 = fmaxf(m2, z[l]);
      }
    }
  }
};
// out[l] = sum over j != l of x[j] (prefix plus suffix sums)
template <int M>
__device__ __forceinline__ void exclusive_sums_scalar(const float (&x)[M], float (&out)[M]) {
  float pre = 0.0f;
#pragma unroll
  for (int l = 0; l < M; ++l) {
    out[l] = pre;
    pre = __fadd_rn(pre, x[l]);
  }
  float suf = 0.0f;
#pragma unroll
  for (int l = M - 1; l >= 0; --l) {
    out[l] = __fadd_rn(out[l], suf);
    suf = __fadd_rn(suf, x[l]);
  }
}

template <int N, int M>
struct WideRobustGroup {
  float zh[N][M];  // z entering each step

  // LSE2 over j != l for every l, and LSE2 over all (returned), of z with top-2 `t`;
  // e[l] = 2^(z_l - m1).
  static __device__ __forceinline__ float lse2_all_and_excluding(const float (&z)[M], const Top2<M>& t,
                                                                 float (&e)[M], float (&lx)[M]) {
    float s1 = 0.0f;
#pragma unroll
    for (int l = 0; l < M; ++l) {
      e[l] = ex2_approx(__fsub_rn(z[l], t.m1));
      s1 = __fadd_rn(s1, e[l]);
    }
    float ex[M];
    exclusive_sums_scalar(e, ex);
    float s2 = 0.0f;  // sum over j != a of 2^(z_j - m2)
#pragma unroll
    for (int l = 0; l < M; ++l) {
      lx[l] = __fadd_rn(t.m1, lg2_approx(ex[l]));
      s2 = __fadd_rn(s2, l == t.a ? 0.0f : ex2_approx(__fsub_rn(z[l], t.m2)));
    }
    float lxa = __fadd_rn(t.m2, lg2_approx(s2));
#pragma unroll
    for (int l = 0; l < M; ++l)
      if (l == t.a) lx[l] = lxa;
    return __fadd_rn(t.m1, lg2_approx(s1));
  }

  // t: the keys in log2 units, all finite.  Fills S.
  __device__ __forceinline__ void forward(const float (&t)[M], float inv_tau, float (&S)[M]) {
    float z[M];
#pragma unroll
    for (int l = 0; l < M; ++l) {
      z[l] = __fmul_rn(t[l], inv_tau);
      S[l] = 0.0f;
    }
#pragma unroll 1
    for (int k = 0; k < N; ++k) {
      const Top2<M> top(z);
#pragma unroll
      for (int l = 0; l < M; ++l) {
        z[l] = __fsub_rn(z[l], top.m1);  // shift: the largest is 0
        zh[k][l] = z[l];
      }
      const Top2<M> t0{z};
      float e[M], lx[M];
      const float lz = lse2_all_and_excluding(z, t0, e, lx);
      float s1 = 0.0f;
#pragma unroll
      for (int l = 0; l < M; ++l) s1 = __fadd_rn(s1, e[l]);
      const float r = rcp_approx(s1);
#pragma unroll
      for (int l = 0; l < M; ++l) S[l] = __fadd_rn(S[l], __fmul_rn(e[l], r));
      if (k + 1 < N) {
#pragma unroll
        for (int l = 0; l < M; ++l) z[l] = __fmaf_rn(__fsub_rn(lx[l], lz), inv_tau, z[l]);
      }
    }
  }

  // After forward(): dk = dL/dkappa for c = dL/dS.
  __device__ __forceinline__ void backward(const float (&c)[M], float inv_tau, float (&dk)[M]) const {
    float b[M];
#pragma unroll
    for (int l = 0; l < M; ++l) b[l] = 0.0f;
#pragma unroll 1
    for (int k = N - 1; k >= 0; --k) {
      float z[M];
#pragma unroll
      for (int l = 0; l < M; ++l) z[l] = zh[k][l];
      const Top2<M> t(z);
      float e[M], lx[M];
      const float lz = lse2_all_and_excluding(z, t, e, lx);
      float mu[M], gz[M];
      float cmu = 0.0f, B = 0.0f;
#pragma unroll
      for (int l = 0; l < M; ++l) {
        mu[l] = ex2_approx(__fsub_rn(z[l], lz));
        cmu = __fmaf_rn(c[l], mu[l], cmu);
        B = __fadd_rn(B, b[l]);
      }
#pragma unroll
      for (int l = 0; l < M; ++l) gz[l] = __fmul_rn(mu[l], __fsub_rn(__fsub_rn(c[l], cmu), B));
      if (k + 1 < N) {
        // (J^T b)_l adds sum over i != l of b_i 2^(z_l - lx_i)
        float w[M], wx[M];
#pragma unroll
        for (int i = 0; i < M; ++i) w[i] = i == t.a ? 0.0f : __fmul_rn(b[i], ex2_approx(__fsub_rn(t.m1, lx[i])));
        exclusive_sums_scalar(w, wx);
        float ba = 0.0f, lxa = 0.0f;
#pragma unroll
        for (int i = 0; i < M; ++i)
          if (i == t.a) ba = b[i], lxa = lx[i];
#pragma unroll
        for (int l = 0; l < M; ++l) {
          float add = __fmul_rn(e[l], wx[l]);
          if (l != t.a) add = __fmaf_rn(ba, ex2_approx(__fsub_rn(z[l], lxa)), add);
          gz[l] = __fadd_rn(gz[l], add);
        }
      }
#pragma unroll
      for (int l = 0; l < M; ++l) b[l] = __fmaf_rn(gz[l], inv_tau, b[l]);
    }
#pragma unroll
    for (int l = 0; l < M; ++l) dk[l] = b[l];
  }
};

// True if every key of a group is finite.
template <int M>
__device__ __forceinline__ bool all_finite(const float (&k)[M]) {
  float s = 0.0f;
#pragma unroll
  for (int l = 0; l < M; ++l) s += k[l] - k[l];  // 0 for finite keys, NaN otherwise
  return s == 0.0f;
}

// ---------------------------------------------------------------------------
// Groups the fast path leaves to an exact routine, deferred: each warp queues their
// first element indices in its own CAP entries of shared memory and, once 32 are
// queued (checked between tiles) or at the end of its work, handles them one per
// lane.  The exact routines then run on every lane of the warp, and their code sits
// outside the fast path's loop body instead of inside it.  All 32 lanes call
// push() and drain() together; `n` is the same on every lane.
// ---------------------------------------------------------------------------
template <int CAP>
struct DeferredGroups {
  uint32_t base;  // shared-memory address of this warp's entries
  int n;

  __device__ __forceinline__ void init(const void* entries) {
    base = static_cast<uint32_t>(__cvta_generic_to_shared(entries)) + (threadIdx.x >> 5) * CAP * 8;
    n = 0;
  }
  // Queues g for the lanes with `want` (at most CAP - n of them in all).
  __device__ __forceinline__ void push(bool want, int64_t g) {
    const uint32_t m = __ballot_sync(0xffffffffu, want);
    if (want) {
      const uint32_t at = base + 8u * uint32_t(n + __popc(m & ((1u << (threadIdx.x & 31)) - 1u)));
      asm volatile("st.shared.u64 [%0], %1;" ::"r"(at), "l"(g) : "memory");
    }
    n += __popc(m);
  }
  // Handles queued groups 32 at a time (all of them if `all`), fn(g) on one lane each.
  template <class Fn>
  __device__ __forceinline__ void drain(bool all, Fn&& fn) {
    if (n < 32 && !(all && n > 0)) return;
    __syncwarp();
    const int lane = threadIdx.x & 31;
    do {
      const int k = n < 32 ? n : 32;
      if (lane < k) {
        int64_t g;
        asm volatile("ld.shared.u64 %0, [%1];" : "=l"(g) : "r"(base + 8u * uint32_t(n - k + lane)) : "memory");
        fn(g);
      }
      n -= k;
      __syncwarp();
    } while (n >= 32 || (all && n > 0));
  }
};

// ---------------------------------------------------------------------------
// Fast register-resident relaxation of one group (V = float) or of two groups in
// lockstep (V = F2, one per half), M <= 8, held by one thread.
//
// State: per step the normalised weights mu(k) and, for k < N, the exact
// complements om(k) = 1 - mu(k), each formed as a sum of the other members
// (never as 1 - mu, so no cancellation).
//  - tau == 1 (TAU1): w -> w (1 - mu) needs no transcendental: the next step's
//    softmax is mu' = mu om / sum(mu om).
//  - otherwise keys are kept as log2 offsets d from the group maximum:
//    d += log2(om) / tau, renormalised to max 0 each step.
// The relaxation is a fixed sequence of explicitly rounded operations; the
// backward kernel recomputes it from the same keys and agrees with the forward's
// S to within fp32 rounding (packed products may be fused into FMAs by the
// compiler, see roi_vec.cuh).  The fallback decision depends only on sums of
// exp2 outputs and is therefore the same in both kernels.
// `flag` (one bit per lane) is raised when a key is not finite and, depending on
// tau, when a key lies more than 100 log2 units from the first one (tau = 1) or
// an exclusive sum drops below 2^-100 (a key gap of ~69 natural-log units); the
// caller then recomputes that group with ExactGroup (and re-ranks it with the
// comparison-based top-N, which orders NaN as -inf).
// ---------------------------------------------------------------------------
template <int M, class V>
__device__ __forceinline__ void exclusive_sums(const V (&x)[M], V (&ex)[M]) {
  static_assert(M == 4 || M == 8, "tree exclusive sums for M = 4, 8");
  if constexpr (M == 4) {
    const V p01 = vadd(x[0], x[1]), p23 = vadd(x[2], x[3]);
    ex[0] = vadd(x[1], p23);
    ex[1] = vadd(x[0], p23);
    ex[2] = vadd(p01, x[3]);
    ex[3] = vadd(p01, x[2]);
  } else {
    // pair sums, then each pair's exclusive sum (the other three pairs), then the partner
    const V p01 = vadd(x[0], x[1]), p23 = vadd(x[2], x[3]), p45 = vadd(x[4], x[5]), p67 = vadd(x[6], x[7]);
    const V q0 = vadd(p01, p23), q1 = vadd(p45, p67);
    const V e01 = vadd(p23, q1), e23 = vadd(p01, q1), e45 = vadd(q0, p67), e67 = vadd(q0, p45);
    ex[0] = vadd(x[1], e01);
    ex[1] = vadd(x[0], e01);
    ex[2] = vadd(x[3], e23);
    ex[3] = vadd(x[2], e23);
    ex[4] = vadd(x[5], e45);
    ex[5] = vadd(x[4], e45);
    ex[6] = vadd(x[7], e67);
    ex[7] = vadd(x[6], e67);
  }
}

template <int M, class V>
__device__ __forceinline__ V sum_of(const V (&x)[M]) {
  if constexpr (M == 4) {
    return vadd(vadd(x[0], x[1]), vadd(x[2], x[3]));
  } else {
    return vadd(vadd(vadd(x[0], x[1]), vadd(x[2], x[3])), vadd(vadd(x[4], x[5]), vadd(x[6], x[7])));
  }
}

template <int M, class V>
__device__ __forceinline__ V max_of(const V (&x)[M]) {
  V m = x[0];
#pragma unroll
  for (int l = 1; l < M; ++l) m = vmax(m, x[l]);
  return m;
}

template <int M, class V>
__device__ __forceinline__ V min_of(const V (&x)[M]) {
  V m = x[0];
#pragma unroll
  for (int l = 1; l < M; ++l) m = vmin(m, x[l]);
  return m;
}

// Step history mu(k), k = 0 .. N-1, of a relaxation kept for the backward sweep:
// in registers ...
template <int N, int M, class V>
struct RegSteps {
  static constexpr bool kSmem = false;
  V mu[N][M];
  __device__ __forceinline__ void put(int k, int l, V v) { mu[k][l] = v; }
  __device__ __forceinline__ V get(int k, int l) const { return mu[k][l]; }
};
// ... or steps 0 .. N-2 in shared memory and the last one in registers.  Slot
// (k, l) of a thread is at[(k M + l) STRIDE]; with `at` = base + threadIdx.x and
// STRIDE = threads per CTA a warp touches consecutive words.
template <int N, int M, class V, int STRIDE>
struct SmemSteps {
  static constexpr bool kSmem = true;
  V* at;
  V last[M];
  __device__ __forceinline__ void put(int k, int l, V v) {
    if (k == N - 1) {
      last[l] = v;
    } else {
      at[(k * M + l) * STRIDE] = v;
    }
  }
  __device__ __forceinline__ V get(int k, int l) const {
    return k == N - 1 ? last[l] : at[(k * M + l) * STRIDE];
  }
};

template <int N, int M, bool TAU1, bool KEEP, class V = float,
          class Steps = RegSteps<KEEP ? N : 1, KEEP ? M : 1, V>>
struct FastGroup {
  // KEEP: store mu of every step for a backward sweep.  S is then not
  // accumulated: soft() re-sums it from the history on demand (in the order
  // forward() accumulates it), which only the backward's optional dW asks for.
  static constexpr bool kSumS = !KEEP;
  Steps st;
  V S[kSumS ? M : 1];
  V rt_last;  // tau = 1, KEEP: 1 / sum(mu om) of step N-2 (mu(N-1) = mu(N-2) om rt_last)
  uint32_t flag;

  // S_l of a KEEP run, summed exactly as forward() accumulates it.
  __device__ __forceinline__ V soft(int l) const {
    if constexpr (kSumS) {
      return S[l];
    } else {
      V s = st.get(0, l);
#pragma unroll
      for (int k = 1; k < N; ++k) s = vadd(s, st.get(k, l));
      return s;
    }
  }

  // kap: the keys in log2 units (t = kappa log2 e).
  __device__ __forceinline__ void forward(const V (&kap)[M], float inv_tau) {
    V cur[M];
    flag = 0;
    if constexpr (TAU1) {
      // Weights relative to the group's first key (any reference works: they are
      // normalised next).  A group with a key more than 100 (log2 units, ~69
      // natural) from the first one, or with a non-finite key, goes to the exact
      // routine: the squared offsets are summed on the FMA pipe and compared once.
      // (a non-finite first key makes every offset non-finite, so it is caught too)
      V e[M], x[M];
      e[0] = vconst<V>(1.0f);
#pragma unroll
      for (int l = 1; l < M; ++l) {
        x[l] = vsub(kap[l], kap[0]);
        e[l] = vmap(x[l], ex2_approx);
      }
      V sq = vmul(x[1], x[1]);
#pragma unroll
      for (int l = 2; l < M; ++l) sq = vfma(x[l], x[l], sq);
      flag = vbelow(vsub(vconst<V>(1.0e4f), sq), 0.0f);
      const V tot = sum_of(e);
      const V r = vmap(tot, rcp_approx);
#pragma unroll
      for (int l = 0; l < M; ++l) cur[l] = vmul(e[l], r);
#pragma unroll
      for (int k = 0; k < N; ++k) {
        // without KEEP the last step is added into S as it is formed (one fma)
        if (KEEP || k == 0 || k + 1 < N) {
#pragma unroll
          for (int l = 0; l < M; ++l) {
            if constexpr (KEEP) st.put(k, l, cur[l]);
            if constexpr (kSumS) S[l] = k == 0 ? cur[l] : vadd(S[l], cur[l]);
          }
        }
        if (k + 1 < N) {
          V o[M], v[M];
          exclusive_sums(cur, o);
#pragma unroll
          for (int l = 0; l < M; ++l) v[l] = vmul(cur[l], o[l]);
          const V rt = vmap(sum_of(v), rcp_approx);
          if constexpr (KEEP) {
            if (k == N - 2) rt_last = rt;
          }
          if (!KEEP && k + 2 == N) {
#pragma unroll
            for (int l = 0; l < M; ++l) S[l] = vfma(v[l], rt, S[l]);
          } else {
#pragma unroll
            for (int l = 0; l < M; ++l) cur[l] = vmul(v[l], rt);
          }
        }
      }
    } else {
      const V kmax = max_of(kap);
      const V sc = vconst<V>(inv_tau);
      const V itau = vconst<V>(inv_tau);
      V d[M];
#pragma unroll
      for (int l = 0; l < M; ++l) d[l] = vmul(vsub(kap[l], kmax), sc);
      const V ksum = sum_of(kap);
      flag = vbelow(vsub(ksum, ksum), 0.0f);  // a non-finite key (or a sum beyond the float range)
      V tmin = vconst<V>(1.0f);
#pragma unroll
      for (int k = 0; k < N; ++k) {
        V e[M];
#pragma unroll
        for (int l = 0; l < M; ++l) e[l] = vmap(d[l], ex2_approx);
        const V tot = sum_of(e);
        if (M >= 8 && k > 0) tmin = vmin(tmin, tot);
        const V r = vmap(tot, rcp_approx);
        if (!KEEP && k > 0 && k + 1 == N) {
          // last step without KEEP: added into S as it is formed (one fma)
#pragma unroll
          for (int l = 0; l < M; ++l) S[l] = vfma(e[l], r, S[l]);
        } else {
#pragma unroll
          for (int l = 0; l < M; ++l) {
            cur[l] = vmul(e[l], r);
            if constexpr (KEEP) st.put(k, l, cur[l]);
            if constexpr (kSumS) S[l] = k == 0 ? cur[l] : vadd(S[l], cur[l]);
          }
        }
        if (k + 1 < N) {
          // d_l += log2(1 - mu_l) / tau.  A group whose exclusive sums fall below 2^-100
          // of the total goes to the exact routine.  M = 8: the offsets are first
          // renormalised by log2 of the total (so sum 2^d = 1 and every offset <= 0)
          // instead of by their maximum after the update (seven comparisons per step;
          // 1.5B-shaped 4:8 at tau = 0.5 2 % faster, the 2:4 step 1 % slower), and a
          // total below 2^-120 (offsets that fell too far in one step) is flagged too.
          V ex[M];
          exclusive_sums(e, ex);
          if constexpr (M >= 8) {
            flag |= vbelow(vmul(min_of(ex), r), kTinyExcl);
            const V lz = vmap(tot, lg2_approx);
#pragma unroll
            for (int l = 0; l < M; ++l) d[l] = vfma(vmap(vmul(ex[l], r), lg2_approx), itau, vsub(d[l], lz));
          } else {
            flag |= vbelow(min_of(ex), kTinyExcl);
#pragma unroll
            for (int l = 0; l < M; ++l) d[l] = vfma(vmap(vmul(ex[l], r), lg2_approx), itau, d[l]);
            const V dm = max_of(d);
#pragma unroll
            for (int l = 0; l < M; ++l) d[l] = vsub(d[l], dm);
          }
        }
      }
      if constexpr (M >= 8) flag |= vbelow(tmin, 7.52316384526264e-37f);  // 2^-120
    }
  }

  // Reverse sweep (requires KEEP): dk = dL/dkappa for c = dL/dS.
  //   abar_l = b_l + (mu_l / tau) (c_l - <c, mu> + H_l - B),
  //   H_l = sum_{i != l} b_i / om_i,  B = sum_i b_i,
  // with om_i = 1 - mu_i formed as the sum of the other members' mu.  REUSE (tau = 1):
  // the update reads c mu + b from the K terms (one operation less per member and
  // step, one more array live).
  template <bool REUSE = true>
  __device__ __forceinline__ void backward(const V (&c)[M], float inv_tau, V (&dk)[M]) const {
    static_assert(KEEP, "backward needs the stored steps");
    const V itau = vconst<V>(inv_tau);
    V b[M], hl[M];
    {
      V cm[M];
#pragma unroll
      for (int l = 0; l < M; ++l) cm[l] = vmul(c[l], st.get(N - 1, l));
      const V cmu = sum_of(cm);
#pragma unroll
      for (int l = 0; l < M; ++l) {
        V t = vsub(c[l], cmu);
        if constexpr (!TAU1) t = vmul(itau, t);
        b[l] = vmul(st.get(N - 1, l), t);
        // tau = 1: b / om(N-2) = mu(N-2) rt_last (c - <c, mu(N-1)>), no division
        if constexpr (TAU1 && N >= 2) hl[l] = vmul(vmul(st.get(N - 2, l), rt_last), t);
      }
    }
    auto sweep = [&](int k) {
      V mk[M], cm[M], h[M], H[M];
#pragma unroll
      for (int l = 0; l < M; ++l) mk[l] = st.get(k, l);
      if (!TAU1 || k != N - 2) {
        V om[M];
        exclusive_sums(mk, om);
#pragma unroll
        for (int l = 0; l < M; ++l) h[l] = vmul(b[l], vmap(om[l], rcp_approx));
      } else {
#pragma unroll
        for (int l = 0; l < M; ++l) h[l] = hl[l];
      }
      // c_l - <c, mu> + H_l - B as (c_l + H_l) - K, K = <c, mu> + B = sum of (c mu + b)
#pragma unroll
      for (int l = 0; l < M; ++l) cm[l] = vfma(c[l], mk[l], b[l]);
      const V K = sum_of(cm);
      exclusive_sums(h, H);
#pragma unroll
      for (int l = 0; l < M; ++l) {
        if constexpr (TAU1 && REUSE) {
          // b + mu (c + H - K) = (c mu + b) + mu (H - K), and c mu + b is cm
          b[l] = vfma(mk[l], vsub(H[l], K), cm[l]);
        } else if constexpr (TAU1) {
          b[l] = vfma(mk[l], vsub(vadd(c[l], H[l]), K), b[l]);
        } else {
          b[l] = vfma(vmul(mk[l], itau), vsub(vadd(c[l], H[l]), K), b[l]);
        }
      }
    };
#pragma unroll
    for (int k = N - 2; k >= 0; --k) sweep(k);
#pragma unroll
    for (int l = 0; l < M; ++l) dk[l] = b[l];
  }
};

// ---------------------------------------------------------------------------
// bounded waits and bulk copies (TMA, 1-D)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
// Programmatic dependent launch: let the stream's next launch start early / wait
// for the previous launch to complete (both no-ops for an ordinary launch).
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Non-blocking test of phase `parity` of `bar`.
__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Waits for phase `parity` of `bar` for at most ~2 s of wall time (the fixed limit
// of the waits that drain a CTA's own copies before it exits).
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (global_timer_ns() - t0 > 2000000000ull) return false;
  }
}
// Waits for a stage of a copy ring, for at most the limit in the status record
// (read only when the stage has not landed yet, through the read-only cache: the
// host changes it only between launches; 2 s unless the caller set another one).
// A limit of 0 gives up at once, whether the stage has landed or not (the tests'
// deterministic way onto the timeout path).  `lim` comes from ring_wait_limit(),
// read once per kernel.
__device__ __forceinline__ uint64_t ring_wait_limit(const unsigned int* status) {
  return __ldg(reinterpret_cast<const unsigned long long*>(status + kStatusLimitWord));
}
__device__ __forceinline__ bool mbar_wait_ring(uint64_t* bar, uint32_t parity, uint64_t lim) {
  if (mbar_test_wait(bar, parity)) return lim != 0;
  if (lim == 0) return false;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (global_timer_ns() - t0 > lim) return false;
  }
}
// Global -> shared bulk copy completing on `bar` (bytes % 16 == 0, both 16-B aligned).
__device__ __forceinline__ void bulk_g2s(void* dst_smem, const void* src_gmem, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst_smem)),
      "l"(src_gmem), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// Per-thread 16-byte global -> shared copy (cp.async, L2 only); the issuing
// thread waits for its own copies with cp_async_wait_all before reading them.
__device__ __forceinline__ void cp_async16(void* dst_smem, const void* src_gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst_smem)), "l"(src_gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

}  // namespace roi
