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

// Bit set in the device status word (defined in roi_api.cu, passed to the
// kernels by address) when a kernel gave up waiting for its own bulk copies.
constexpr unsigned int kStatusTimeout = 1u;

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
    const uint32_t hi0 = __umulhi(kPhiloxM0, c.x), lo0 = kPhiloxM0 * c.x;
    const uint32_t hi1 = __umulhi(kPhiloxM1, c.z), lo1 = kPhiloxM1 * c.z;
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
  uint64_t e_base;       // row_offset * cols: flat index of this call's element 0
};

// Four consecutive noise words for elements e4 .. e4+3 (e4 % 4 == 0).
__device__ __forceinline__ uint4 noise_block(const NoiseParams& np, uint64_t e4) {
  const uint64_t q = e4 >> 2;
  return philox4x32_10(make_uint4(uint32_t(q), uint32_t(q >> 32), np.step, np.tensor_id),
                       np.k0, np.k1);
}
// The word of a single element (any e).
__device__ __forceinline__ uint32_t noise_word(const NoiseParams& np, uint64_t e) {
  const uint4 w = noise_block(np, e & ~uint64_t(3));
  const uint32_t s = uint32_t(e & 3);
  return s == 0 ? w.x : s == 1 ? w.y : s == 2 ? w.z : w.w;
}

// u = ((x >> 9) + 1/2) * 2^-23, exactly: (1 + k 2^-23) - (1 - 2^-24) is exact
// by Sterbenz's lemma and equals (2k + 1) 2^-24.
__device__ __forceinline__ float uniform_from_word(uint32_t x) {
  return __uint_as_float(0x3f800000u | (x >> 9)) - __uint_as_float(0x3f7fffffu);
}

// Gumbel(0,1) sample from a word: -log(-log u) (Algorithm 1), accurate logf.
__device__ __forceinline__ float gumbel_from_word(uint32_t x) {
  const float u = uniform_from_word(x);
  return -logf(-logf(u));
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
  if (m == -INFINITY) return -INFINITY;
  float s = 0.f;
  for (int i = 0; i < M; ++i)
    if (i != skip) s += expf(z[i] - m);
  return m + logf(s);
}

template <int NMAX, int MMAX>
struct ExactGroup {
  float zh[NMAX][MMAX];  // z at every step (history for the backward)

  // Forward: fills S[0..M).  kap: perturbed keys.
  __device__ __forceinline__ void forward(const float* kap, int N, int M, float tau, float* S) {
    float z[MMAX];
    for (int l = 0; l < M; ++l) {
      z[l] = kap[l] / tau;
      S[l] = 0.f;
    }
    for (int k = 0; k < N; ++k) {
      for (int l = 0; l < M; ++l) zh[k][l] = z[l];
      const float lt = lse_excluding(z, M, -1);
      for (int l = 0; l < M; ++l) S[l] += expf(z[l] - lt);
      if (k + 1 < N) {
        float zn[MMAX];
        for (int l = 0; l < M; ++l) zn[l] = z[l] + (lse_excluding(z, M, l) - lt) / tau;
        for (int l = 0; l < M; ++l) z[l] = zn[l];
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
// Fast register-resident relaxation of one group held by one thread (M <= 8).
//
// State: per step the normalised weights mu(k) and, for k < N, the exact
// complements om(k) = 1 - mu(k), each formed as a sum of the other members
// (never as 1 - mu, so no cancellation).
//  - tau == 1 (TAU1): w -> w (1 - mu) needs no transcendental: the next step's
//    softmax is mu' = mu om / sum(mu om).
//  - otherwise keys are kept as log2 offsets d from the group maximum:
//    d += log2(om) / tau, renormalised to max 0 each step.
// `flag` is raised when an exclusive sum drops below 2^-100 (a key gap of ~69
// natural-log units); the caller then recomputes the group with ExactGroup.
// ---------------------------------------------------------------------------
template <int M>
__device__ __forceinline__ void exclusive_sums(const float (&x)[M], float (&ex)[M]) {
  static_assert(M == 4 || M == 8, "tree exclusive sums for M = 4, 8");
  if constexpr (M == 4) {
    const float p01 = x[0] + x[1], p23 = x[2] + x[3];
    ex[0] = x[1] + p23;
    ex[1] = x[0] + p23;
    ex[2] = p01 + x[3];
    ex[3] = p01 + x[2];
  } else {
    const float p01 = x[0] + x[1], p23 = x[2] + x[3], p45 = x[4] + x[5], p67 = x[6] + x[7];
    const float q0 = p01 + p23, q1 = p45 + p67;
    ex[0] = (x[1] + p23) + q1;
    ex[1] = (x[0] + p23) + q1;
    ex[2] = (p01 + x[3]) + q1;
    ex[3] = (p01 + x[2]) + q1;
    ex[4] = (x[5] + p67) + q0;
    ex[5] = (x[4] + p67) + q0;
    ex[6] = (p45 + x[7]) + q0;
    ex[7] = (p45 + x[6]) + q0;
  }
}

template <int M>
__device__ __forceinline__ float sum_of(const float (&x)[M]) {
  if constexpr (M == 4) {
    return (x[0] + x[1]) + (x[2] + x[3]);
  } else {
    return ((x[0] + x[1]) + (x[2] + x[3])) + ((x[4] + x[5]) + (x[6] + x[7]));
  }
}

template <int M>
__device__ __forceinline__ float max_of(const float (&x)[M]) {
  float m = x[0];
#pragma unroll
  for (int l = 1; l < M; ++l) m = fmaxf(m, x[l]);
  return m;
}

template <int M>
__device__ __forceinline__ float min_of(const float (&x)[M]) {
  float m = x[0];
#pragma unroll
  for (int l = 1; l < M; ++l) m = fminf(m, x[l]);
  return m;
}

template <int N, int M, bool TAU1, bool KEEP>
struct FastGroup {
  // KEEP: store mu / om of every step for a backward sweep.
  float mu[KEEP ? N : 1][M];
  float om[(KEEP && N > 1) ? N - 1 : 1][M];
  float S[M];
  bool flag;

  __device__ __forceinline__ void forward(const float (&kap)[M], float inv_tau) {
    const float kmax = max_of(kap);
    float cur[M];
#pragma unroll
    for (int l = 0; l < M; ++l) S[l] = 0.f;
    flag = false;
    if constexpr (TAU1) {
      float e[M];
#pragma unroll
      for (int l = 0; l < M; ++l) e[l] = ex2_approx((kap[l] - kmax) * kLog2e);
      flag = !(min_of(e) >= kTinyExcl);  // also catches NaN
      const float r = rcp_approx(sum_of(e));
#pragma unroll
      for (int l = 0; l < M; ++l) cur[l] = e[l] * r;
#pragma unroll
      for (int k = 0; k < N; ++k) {
#pragma unroll
        for (int l = 0; l < M; ++l) {
          S[l] += cur[l];
          if constexpr (KEEP) mu[k][l] = cur[l];
        }
        if (k + 1 < N) {
          float o[M], v[M];
          exclusive_sums(cur, o);
#pragma unroll
          for (int l = 0; l < M; ++l) {
            if constexpr (KEEP) om[k < N - 1 ? k : 0][l] = o[l];
            v[l] = cur[l] * o[l];
          }
          const float rt = rcp_approx(sum_of(v));
#pragma unroll
          for (int l = 0; l < M; ++l) cur[l] = v[l] * rt;
        }
      }
    } else {
      const float sc = inv_tau * kLog2e;
      float d[M];
#pragma unroll
      for (int l = 0; l < M; ++l) d[l] = (kap[l] - kmax) * sc;
      if (!(kmax > -INFINITY && kmax < INFINITY)) flag = true;
#pragma unroll
      for (int k = 0; k < N; ++k) {
        float e[M];
#pragma unroll
        for (int l = 0; l < M; ++l) e[l] = ex2_approx(d[l]);
        const float r = rcp_approx(sum_of(e));
#pragma unroll
        for (int l = 0; l < M; ++l) {
          cur[l] = e[l] * r;
          S[l] += cur[l];
          if constexpr (KEEP) mu[k][l] = cur[l];
        }
        if (k + 1 < N) {
          float ex[M];
          exclusive_sums(e, ex);
          flag |= !(min_of(ex) >= kTinyExcl);
#pragma unroll
          for (int l = 0; l < M; ++l) {
            const float o = ex[l] * r;
            if constexpr (KEEP) om[k < N - 1 ? k : 0][l] = o;
            d[l] += lg2_approx(o) * inv_tau;
          }
          const float dm = max_of(d);
#pragma unroll
          for (int l = 0; l < M; ++l) d[l] -= dm;
        }
      }
    }
  }

  // Reverse sweep (requires KEEP): dk = dL/dkappa for c = dL/dS.
  //   abar_l = b_l + (mu_l / tau) (c_l - <c, mu> + H_l - B),
  //   H_l = sum_{i != l} b_i / om_i,  B = sum_i b_i.
  __device__ __forceinline__ void backward(const float (&c)[M], float inv_tau, float (&dk)[M]) const {
    static_assert(KEEP, "backward needs the stored steps");
    float b[M];
    {
      float cm[M];
#pragma unroll
      for (int l = 0; l < M; ++l) cm[l] = c[l] * mu[N - 1][l];
      const float cmu = sum_of(cm);
#pragma unroll
      for (int l = 0; l < M; ++l) b[l] = mu[N - 1][l] * inv_tau * (c[l] - cmu);
    }
#pragma unroll
    for (int k = N - 2; k >= 0; --k) {
      float cm[M], h[M], H[M];
#pragma unroll
      for (int l = 0; l < M; ++l) {
        cm[l] = c[l] * mu[k][l];
        h[l] = b[l] * rcp_approx(om[k][l]);
      }
      const float cmu = sum_of(cm);
      const float B = sum_of(b);
      exclusive_sums(h, H);
#pragma unroll
      for (int l = 0; l < M; ++l) b[l] += mu[k][l] * inv_tau * (((c[l] - cmu) + H[l]) - B);
    }
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
// Waits for phase `parity` of `bar` for at most ~2 s of wall time.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (global_timer_ns() - t0 > 2000000000ull) return false;
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

}  // namespace roi
