// Masked linear forward: Y[t, r] = sum_k X[t, k] Wm[r, k] with
// Wm = bf16(W * S) (Eq. 5, the layer's product with the relaxed mask of
// Sec. 4.2.2 Eq. 10-12), where the mask is formed in the GEMM's prologue and
// handed to the tensor cores through shared memory: Wm never reaches global
// memory, and W and the logits are read once.
//
// One CTA owns 128 weight rows (the MMA's M, one TMEM lane per row) and every
// token (the MMA's N <= 256, one TMEM column per token), and walks K in chunks
// of 32 through a ring of four shared-memory stages.  A producer warp (one
// elected lane) stages each chunk's logits, weights and tokens with tiled TMA
// loads (2-D tensor maps, out-of-range rows and columns zero-filled) and, once
// every compute thread has arrived on the stage's `ready` mbarrier, issues two
// tcgen05.mma (K = 16 each) of the A tile against the token tile, commits them
// to the stage's `mma` mbarrier and refills the stage when they are done.  The
// compute warps never wait for each other: each thread relaxes one pair of
// groups per chunk from shared memory (the same keys, noise and rounding as
// roi_mask_fwd, so Wm is bit-identical to its output), writes their bf16
// products into the chunk's A tile and arrives.  Layers with few row blocks
// split K across CTAs, which write fp32 partials; a second launch, dependent on
// the first (programmatic dependent launch: it is scheduled while the GEMM drains
// and reads once the GEMM has completed), adds them in split order across the
// whole GPU, so Y does not depend on timing.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "roi_launch.h"
#include "roi_tc.cuh"

namespace roi {
namespace {

constexpr int kRows = 128;                      // weight rows per CTA (MMA M)
constexpr int kBK = 32;                         // K elements per chunk
constexpr int kStages = 4;
constexpr uint32_t kLBO = 128;                  // A tile: core matrices adjacent along K
constexpr uint32_t kSBO = (kBK / 8) * 128;      // A tile: adjacent 8-row groups (512 B)
constexpr uint32_t kTileA = kRows * kBK * 2;    // 8 KB
constexpr uint32_t kTilePhi = kRows * kBK * 4;  // 16 KB, [128][32] fp32 (one TMA box)
constexpr uint32_t kTileW = kRows * kBK * 2;    // 8 KB, [128][32] bf16 (one TMA box)
#ifndef ROI_LIN_MIN_CHUNKS
#define ROI_LIN_MIN_CHUNKS 4
#endif
constexpr int kMinChunksPerSplit = ROI_LIN_MIN_CHUNKS;  // K chunks per split, at least

template <int M>
struct LinCfg {
  // one pair of groups per thread per chunk: 128 rows x 32 / M groups / 2
  static constexpr int kThreads = kRows * kBK / M / 2;  // 512 (M = 4), 256 (M = 8)
};

struct LinArgs {
  float* Y;               // [T, rows]
  float* part;            // [splits, T, rows] (splits > 1)
  int64_t T, rows, cols;
  int T_pad;              // T rounded up to 16 (the MMA's N)
  int splits, nchunks;
  uint32_t tmem_cols;
  float tau, inv_tau;
  NoiseParams np;
  unsigned int* status;
};

// Shared-memory layout (bytes from the 1024-aligned dynamic base), per stage:
// the A tile (core-matrix layout, LBO 128, SBO 512), the token tile (four TMA
// boxes of 8 K-columns x T_pad rows, so core matrix (row group i, K group j) sits
// at j * 16 T_pad + 128 i), and the staged logits and weights ([128][32]
// row-major TMA boxes); then the mbarriers.
struct LinSmem {
  uint32_t a, x, phi, w, full, ready, mma, misc, total, tile_x;
};
__host__ __device__ inline LinSmem lin_smem(int T_pad) {
  LinSmem s;
  s.tile_x = uint32_t(T_pad) * kBK * 2;
  s.a = 0;
  s.x = s.a + kStages * kTileA;
  s.phi = s.x + ((kStages * s.tile_x + 1023) & ~1023u);
  s.w = s.phi + kStages * kTilePhi;
  s.full = s.w + kStages * kTileW;
  s.ready = s.full + kStages * 8;
  s.mma = s.ready + kStages * 8;
  s.misc = s.mma + kStages * 8;
  s.total = s.misc + 16;
  return s;
}

template <class V>
__device__ __forceinline__ float lane_of(V v, int h) {
  if constexpr (vlanes<V>() == 1) {
    return v;
  } else {
    return h == 0 ? lo(v) : hi(v);
  }
}

// This thread's pair in a chunk: groups (r, gk) and (r + 64, gk), the lanes of a
// warp on consecutive groups of a row (conflict-free reads of the staged tiles).
template <int M>
__device__ __forceinline__ void pair_coords(int& r, int& gk) {
  constexpr int kPerRow = kBK / M;  // groups per chunk row: 8 (M = 4), 4 (M = 8)
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  gk = lane % kPerRow;
  r = w * (32 / kPerRow) + lane / kPerRow;  // 0 .. 63
}

// One thread: the TMA loads of chunk kc into `stage` (logits, weights, and the
// token tile as four boxes of 8 K-columns), all completing on full[stage].
__device__ __forceinline__ void issue_chunk(const CUtensorMap* tm_phi, const CUtensorMap* tm_w,
                                            const CUtensorMap* tm_x, uint8_t* smem, const LinSmem& L, int stage,
                                            int row0, int kc) {
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + L.full) + stage;
  mbar_arrive_expect_tx(bar, kTilePhi + kTileW + L.tile_x);
  const int k0 = kc * kBK;
  tma_load_2d(smem + L.phi + stage * kTilePhi, tm_phi, k0, row0, bar);
  tma_load_2d(smem + L.w + stage * kTileW, tm_w, k0, row0, bar);
  uint8_t* sx = smem + L.x + stage * L.tile_x;
#pragma unroll
  for (int j = 0; j < kBK / 8; ++j) tma_load_2d(sx + j * (L.tile_x / 4), tm_x, k0 + 8 * j, 0, bar);
}

// Relax this thread's pair of chunk kc from the staged logits and write
// bf16(W * S) into the chunk's A tile (core-matrix layout).
template <int N, int M, bool TAU1>
__device__ __forceinline__ void chunk_masked_weights(const LinArgs& a, uint8_t* smem, const LinSmem& L, int stage,
                                                     int64_t row0, int kc) {
  int r, gk;
  pair_coords<M>(r, gk);
  const float* sphi = reinterpret_cast<const float*>(smem + L.phi + stage * kTilePhi);
  const uint16_t* sw = reinterpret_cast<const uint16_t*>(smem + L.w + stage * kTileW);
  const int64_t k = int64_t(kc) * kBK + gk * M;
  int64_t e0[2];
  float ph[2][M];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    e0[h] = (row0 + r + 64 * h) * a.cols + k;
#pragma unroll
    for (int s = 0; s < M / 4; ++s) {
      const float4 p = *reinterpret_cast<const float4*>(sphi + (r + 64 * h) * kBK + gk * M + 4 * s);
      ph[h][4 * s] = p.x, ph[h][4 * s + 1] = p.y, ph[h][4 * s + 2] = p.z, ph[h][4 * s + 3] = p.w;
    }
  }
  // keys in log2 units, as the mask forward forms them
  F2 kap[M];
  {
    uint32_t x[2][M];
    // every counter of the call below 2^32: the counter's low word in 32-bit
    // arithmetic and a zero high word (as the mask kernels; rows past the last may
    // wrap, but their outputs are never stored)
    if (a.np.narrow) {
      const uint32_t qk = uint32_t(a.np.e_base >> 2) + uint32_t(k >> 2);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const uint32_t q0 = qk + uint32_t(row0 + r + 64 * h) * uint32_t(a.cols >> 2);
#pragma unroll
        for (int s = 0; s < M / 4; ++s) {
          const uint4 w = noise_block_lo(a.np, q0 + s);
          x[h][4 * s] = w.x, x[h][4 * s + 1] = w.y, x[h][4 * s + 2] = w.z, x[h][4 * s + 3] = w.w;
        }
      }
    } else {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const uint64_t q0 = (a.np.e_base + uint64_t(e0[h])) >> 2;
#pragma unroll
        for (int s = 0; s < M / 4; ++s) {
          const uint4 w = noise_block_q(a.np, q0 + s);
          x[h][4 * s] = w.x, x[h][4 * s + 1] = w.y, x[h][4 * s + 2] = w.z, x[h][4 * s + 3] = w.w;
        }
      }
    }
#pragma unroll
    for (int l = 0; l < M; ++l) {
      const F2 one_plus = f2(one_plus_from_word(x[0][l]), one_plus_from_word(x[1][l]));
      const F2 u = vsub(one_plus, vconst<F2>(__uint_as_float(0x3f7fffffu)));
      kap[l] = key_log2(f2(ph[0][l], ph[1][l]), u, a.np.l2e_inv_lam);
    }
  }
  FastGroup<N, M, TAU1, false, F2> fg;
  fg.forward(kap, a.inv_tau);
  float S[2][M];
#pragma unroll
  for (int h = 0; h < 2; ++h)
#pragma unroll
    for (int l = 0; l < M; ++l) S[h][l] = lane_of(fg.S[l], h);
  if (fg.flag != 0u) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      if ((fg.flag >> h) & 1u) {
        // the mask forward's fallback, so Wm stays its bit for bit
        float k[M], kn[M];
#pragma unroll
        for (int l = 0; l < M; ++l) {
          k[l] = lane_of(kap[l], h);
          kn[l] = k[l] * kLn2;  // natural-log keys
        }
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
  // both groups' products of member l in one packed multiply (as the mask forward)
  uint8_t* sa = smem + L.a + stage * kTileA;
#pragma unroll
  for (int s = 0; s < M / 4; ++s) {
    const uint2 qa = *reinterpret_cast<const uint2*>(sw + r * kBK + gk * M + 4 * s);
    const uint2 qb = *reinterpret_cast<const uint2*>(sw + (r + 64) * kBK + gk * M + 4 * s);
    const float* xa = S[0] + 4 * s;
    const float* xb = S[1] + 4 * s;
    const F2 p0 = f2(__uint_as_float(qa.x << 16), __uint_as_float(qb.x << 16)) * f2(xa[0], xb[0]);
    const F2 p1 = f2(__uint_as_float(qa.x & 0xffff0000u), __uint_as_float(qb.x & 0xffff0000u)) * f2(xa[1], xb[1]);
    const F2 p2 = f2(__uint_as_float(qa.y << 16), __uint_as_float(qb.y << 16)) * f2(xa[2], xb[2]);
    const F2 p3 = f2(__uint_as_float(qa.y & 0xffff0000u), __uint_as_float(qb.y & 0xffff0000u)) * f2(xa[3], xb[3]);
    const int kl = gk * M + 4 * s;  // K offset within the chunk (multiple of 4)
    const uint32_t base = uint32_t(kl >> 3) * kLBO + uint32_t(kl & 7) * 2;
    const int ra = r, rb = r + 64;
    *reinterpret_cast<uint2*>(sa + uint32_t(ra >> 3) * kSBO + uint32_t(ra & 7) * 16 + base) =
        make_uint2(pack_bf16x2(lo(p0), lo(p1)), pack_bf16x2(lo(p2), lo(p3)));
    *reinterpret_cast<uint2*>(sa + uint32_t(rb >> 3) * kSBO + uint32_t(rb & 7) * 16 + base) =
        make_uint2(pack_bf16x2(hi(p0), hi(p1)), pack_bf16x2(hi(p2), hi(p3)));
  }
}

template <int N, int M, bool TAU1>
__global__ void __launch_bounds__(LinCfg<M>::kThreads + 32, 1)
    roi_masked_linear_kernel(const __grid_constant__ CUtensorMap tm_phi, const __grid_constant__ CUtensorMap tm_w,
                             const __grid_constant__ CUtensorMap tm_x, LinArgs a) {
  using C = LinCfg<M>;
  constexpr int kComputeWarps = C::kThreads / 32;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const LinSmem L = lin_smem(a.T_pad);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.full);    // TMA of a stage landed
  uint64_t* ready = reinterpret_cast<uint64_t*>(smem + L.ready);  // every compute thread wrote its A part
  uint64_t* mma = reinterpret_cast<uint64_t*>(smem + L.mma);      // the stage's MMAs completed
  uint32_t* misc = reinterpret_cast<uint32_t*>(smem + L.misc);    // [0] TMEM base, [2] ok
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool producer = warp == kComputeWarps;  // TMA and MMA issue (one elected lane)
  // the split-K reduction launch may be scheduled now (it waits for this grid)
  pdl_launch_dependents();

  const int rb = blockIdx.x / a.splits, sp = blockIdx.x % a.splits;
  const int row0 = rb * kRows;
  const int base = a.nchunks / a.splits, rem = a.nchunks % a.splits;
  const int c_begin = sp * base + (sp < rem ? sp : rem);
  const int nc = base + (sp < rem ? 1 : 0);

  if (tid == 0) {
#pragma unroll
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(ready + s, C::kThreads);
      mbar_init(mma + s, 1);
    }
    misc[2] = 1u;
    fence_mbar_init();
  }
  if (warp == 0) tc_alloc(misc, a.tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = misc[0];

  bool ok = true;
  const uint64_t lim = ring_wait_limit(a.status);
  // producer lane: chunks whose TMA fill was issued, and whose MMAs were committed
  int issued = 0, committed = 0;
  if (producer) {
    if (lane == 0) {
      const uint32_t idesc = tc_idesc_bf16_f32(kRows, a.T_pad);
      const uint32_t lbo_x = L.tile_x / 4, sbo_x = 128;
      for (int c = 0; c < kStages && c < nc; ++c) {
        issue_chunk(&tm_phi, &tm_w, &tm_x, smem, L, c, row0, c_begin + c);
        issued = c + 1;
      }
      uint32_t phase = 0;  // parity of the current pass over the stages
      int s = 0;
      for (int c = 0; c < nc && ok; ++c) {
        ok = mbar_wait_ring(ready + s, phase, lim);
        if (!ok) break;
        tc_fence_after();
        const uint32_t sa = smem_addr(smem + L.a + s * kTileA);
        const uint32_t sx = smem_addr(smem + L.x + s * L.tile_x);
#pragma unroll
        for (int j = 0; j < kBK / 16; ++j) {
          tc_mma_bf16(tmem, tc_smem_desc(sa + j * 2 * kLBO, kLBO, kSBO),
                      tc_smem_desc(sx + j * 2 * lbo_x, lbo_x, sbo_x), idesc, c > 0 || j > 0);
        }
        tc_commit(mma + s);
        committed = c + 1;
        if (c + kStages < nc) {
          // refill this stage once its MMAs are done (its staged logits and
          // weights were consumed before `ready` completed)
          ok = mbar_wait_ring(mma + s, phase, lim);
          if (ok) {
            issue_chunk(&tm_phi, &tm_w, &tm_x, smem, L, s, row0, c_begin + c + kStages);
            issued = c + kStages + 1;
          }
        }
        if (s == kStages - 1) {
          s = 0;
          phase ^= 1u;
        } else {
          ++s;
        }
      }
      if (!ok) misc[2] = 0u;
    }
  } else {
    uint32_t phase = 0;
    int s = 0;
    for (int c = 0; c < nc; ++c) {
      if (ok) ok = mbar_wait_ring(full + s, phase, lim);
      if (!ok) break;
      chunk_masked_weights<N, M, TAU1>(a, smem, L, s, row0, c_begin + c);
      fence_proxy_async_smem();
      mbar_arrive(ready + s);
      if (s == kStages - 1) {
        s = 0;
        phase ^= 1u;
      } else {
        ++s;
      }
    }
    // the last chunk's commit covers every MMA issued before it (the previous
    // completion of that stage preceded the refill this thread already saw)
    if (nc > 0 && ok) ok = mbar_wait_ring(mma + (nc - 1) % kStages, uint32_t((nc - 1) / kStages) & 1u, lim);
  }
  if (!ok) misc[2] = 0u;
  __syncthreads();
  ok = misc[2] != 0u;
  if (!ok && producer && lane == 0) {
    // a wait gave up: before this CTA releases its shared memory and TMEM, let the
    // TMA fills it issued land (the last fill of each stage; fills of a stage
    // complete in order) and the MMAs it committed finish (a commit tracks every
    // earlier MMA of this thread), with the fixed bounded wait
    for (int c = issued > kStages ? issued - kStages : 0; c < issued; ++c)
      mbar_wait_bounded(full + c % kStages, uint32_t(c / kStages) & 1u);
    if (committed > 0) mbar_wait_bounded(mma + (committed - 1) % kStages, uint32_t((committed - 1) / kStages) & 1u);
  }
  if (!ok) __syncthreads();
  tc_fence_after();
  if (!ok && tid == 0) atomicOr(a.status, kStatusTimeout);

  // epilogue (compute warps): warp w reads TMEM lanes 32 (w % 4) .. + 31 (weight
  // rows), 16 token columns at a time, blocks split among the warps of a quarter
  constexpr int kQuarters = 4, kPerQuarter = kComputeWarps / kQuarters;
  const int quarter = warp % kQuarters, slot = warp / kQuarters;
  const int64_t row = int64_t(row0) + quarter * 32 + lane;
  float* dst = a.splits > 1 ? a.part + int64_t(sp) * a.T * a.rows : a.Y;
  if (ok && !producer) {
    for (int b = slot; b < a.T_pad / 16; b += kPerQuarter) {
      uint32_t v[16];
      tc_ld16(tmem + (uint32_t(quarter * 32) << 16) + uint32_t(b * 16), v);
      if (row < a.rows) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int64_t t = int64_t(b) * 16 + j;
          if (t < a.T) dst[t * a.rows + row] = __uint_as_float(v[j]);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tc_dealloc(tmem, a.tmem_cols);
}

// Split K: Y = the splits' fp32 partials ([splits][n] after one another) added in
// split order, four consecutive outputs per thread when n % 4 == 0 (part and Y are
// 16-byte aligned), the loads of up to eight splits in flight.
__global__ void __launch_bounds__(256) roi_linear_reduce_kernel(const float* part, float* Y, int splits, int64_t n) {
  pdl_wait();  // the partials of the GEMM launched before
  const int64_t stride = int64_t(gridDim.x) * blockDim.x;
  if ((n & 3) == 0) {
    const int64_t n4 = n / 4;
    const float4* p = reinterpret_cast<const float4*>(part);
    for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n4; i += stride) {
      float4 acc = __ldcs(p + i);
      for (int q0 = 1; q0 < splits; q0 += 8) {
        float4 v[8];
#pragma unroll
        for (int j = 0; j < 8; ++j)
          if (q0 + j < splits) v[j] = __ldcs(p + (q0 + j) * n4 + i);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (q0 + j < splits) {
            acc.x = __fadd_rn(acc.x, v[j].x);
            acc.y = __fadd_rn(acc.y, v[j].y);
            acc.z = __fadd_rn(acc.z, v[j].z);
            acc.w = __fadd_rn(acc.w, v[j].w);
          }
        }
      }
      reinterpret_cast<float4*>(Y)[i] = acc;
    }
  } else {
    for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n; i += stride) {
      float acc = __ldcs(part + i);
      for (int q = 1; q < splits; ++q) acc = __fadd_rn(acc, __ldcs(part + q * n + i));
      Y[i] = acc;
    }
  }
}

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link
// dependency on the driver library).
PFN_cuTensorMapEncodeTiled_v12000 encode_tiled() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// A 2-D row-major tensor of dim1 rows x dim0 elements, box of box1 rows x box0
// elements, no swizzle, out-of-range elements read as zero.
bool make_map(CUtensorMap* m, CUtensorMapDataType dt, uint32_t esize, const void* base, uint64_t dim0,
              uint64_t dim1, uint32_t box0, uint32_t box1) {
  auto fn = encode_tiled();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {dim0, dim1};
  const cuuint64_t strides[1] = {dim0 * esize};
  const cuuint32_t box[2] = {box0, box1};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

template <int N, int M>
int launch_nm(const LinearCall& c, const LinArgs& a) {
  CUtensorMap tm_phi, tm_w, tm_x;
  if (!make_map(&tm_phi, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, c.phi, uint64_t(c.cols), uint64_t(c.rows), kBK, kRows) ||
      !make_map(&tm_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, c.W, uint64_t(c.cols), uint64_t(c.rows), kBK, kRows) ||
      !make_map(&tm_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, c.X, uint64_t(c.cols), uint64_t(c.T), 8,
                uint32_t(a.T_pad)))
    return -1;
  const LinSmem L = lin_smem(a.T_pad);
  const size_t smem = size_t(L.total) + 1024;  // + alignment slack
  auto kern = a.tau == 1.0f ? roi_masked_linear_kernel<N, M, true> : roi_masked_linear_kernel<N, M, false>;
  // the shared-memory limit is set once per device and kernel, to the largest size
  static int set_to[2][64] = {{0}};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return -1;
  int& cur = set_to[a.tau == 1.0f ? 1 : 0][dev];
  if (cur < int(smem)) {
    const int want = int(lin_smem(256).total) + 1024;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, want) != cudaSuccess) return -1;
    cur = want;
  }
  const int64_t row_blocks = (a.rows + kRows - 1) / kRows;
  kern<<<int(row_blocks * a.splits), LinCfg<M>::kThreads + 32, smem, c.stream>>>(tm_phi, tm_w, tm_x, a);
  if (cudaGetLastError() != cudaSuccess) return -1;
  if (a.splits == 1) return 1;
  const int64_t n = a.T * a.rows;
  const int64_t items = (n & 3) == 0 ? n / 4 : n;
  int64_t blocks = (items + 255) / 256;
  const int64_t cap = int64_t(sm_count()) * 8;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  if (launch_maybe_pdl(roi_linear_reduce_kernel, int(blocks), 256, 0, c.stream, true, a.part, a.Y, a.splits, n) < 0)
    return -1;
  return 2;
}

}  // namespace

int linear_splits(int64_t T, int64_t rows, int64_t cols) {
  const int64_t row_blocks = (rows + kRows - 1) / kRows;
  const int64_t nchunks = (cols + kBK - 1) / kBK;
  int64_t s = (sm_count() + row_blocks / 2) / row_blocks;
  const int64_t cap = nchunks / kMinChunksPerSplit;
  if (s > cap) s = cap;
  if (s < 1) s = 1;
  (void)T;
  return int(s);
}

size_t linear_workspace_bytes(int64_t T, int64_t rows, int64_t cols) {
  const int s = linear_splits(T, rows, cols);
  if (s <= 1) return 0;
  return size_t(s) * size_t(T) * size_t(rows) * 4;
}

bool linear_supported(int N, int M) { return (N == 2 && M == 4) || (N == 4 && M == 8) || (N == 2 && M == 8); }

int launch_masked_linear(const LinearCall& c) {
  LinArgs a;
  a.Y = c.Y;
  a.T = c.T;
  a.rows = c.rows;
  a.cols = c.cols;
  a.T_pad = int((c.T + 15) / 16 * 16);
  uint32_t cols_t = 32;
  while (cols_t < uint32_t(a.T_pad)) cols_t <<= 1;
  a.tmem_cols = cols_t;
  a.nchunks = int((c.cols + kBK - 1) / kBK);
  a.tau = c.tau;
  a.inv_tau = 1.0f / c.tau;
  a.np = c.np;
  a.np.narrow = counters_narrow(c.np, c.rows * c.cols);
  a.status = c.status;
  // split K only as far as the caller's workspace holds the partials
  int splits = linear_splits(c.T, c.rows, c.cols);
  const size_t per_split = size_t(c.T) * size_t(c.rows) * 4;
  while (splits > 1 && (c.workspace == nullptr || size_t(splits) * per_split > c.workspace_bytes)) --splits;
  a.splits = splits;
  a.part = splits > 1 ? reinterpret_cast<float*>(c.workspace) : nullptr;
  int r = -1;
  if (c.N == 2 && c.M == 4) r = launch_nm<2, 4>(c, a);
  else if (c.N == 4 && c.M == 8) r = launch_nm<4, 8>(c, a);
  else if (c.N == 2 && c.M == 8) r = launch_nm<2, 8>(c, a);
  return r;
}

}  // namespace roi
