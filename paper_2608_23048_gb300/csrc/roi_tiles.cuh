// Persistent tile pipeline: each CTA walks tiles blockIdx.x, blockIdx.x + grid, ...
// of TILE contiguous elements.  The inputs of upcoming tiles are staged into a
// ring of shared-memory stages with 1-D bulk copies (TMA) that complete on one
// mbarrier per stage.  Warps never wait for each other: each warp waits (bounded)
// for its stage to land, computes from shared memory, stores its outputs straight
// to global memory, then counts itself out of the stage; the last warp out issues
// the copies that refill the stage with the tile STAGES ahead.
#pragma once

#include "roi_common.cuh"

namespace roi {

template <int NARR>
struct TileSrc {
  const uint8_t* ptr[NARR];  // global base of each input array
  uint32_t esize[NARR];      // bytes per element of each input array
};

// Shared memory needed by run_tiles: the stages, then per stage one mbarrier,
// one "warps done" counter and one "fills issued" counter.
template <int TILE, int STAGES>
constexpr size_t tile_smem_bytes(uint32_t bytes_per_element) {
  return ((size_t(STAGES) * TILE * bytes_per_element + 7) & ~size_t(7)) + size_t(STAGES) * 16;
}

// Runs `compute(stage_ptrs, tile)` for every tile of this CTA among tiles
// 0 .. full_tiles - 1; `src_of(tile, a)` gives the global address of input array
// a's part of the tile (TILE * esize[a] contiguous bytes, 16-byte aligned).
// Returns false if a wait timed out (status recorded, copies drained).
template <int THREADS, int TILE, int STAGES, int NARR, class SrcOf, class Compute>
__device__ __forceinline__ bool run_tiles_src(uint8_t* smem, const uint32_t (&esize)[NARR], int64_t full_tiles,
                                              unsigned int* status, SrcOf&& src_of, Compute&& compute) {
  constexpr int kWarps = THREADS / 32;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  size_t arr_off[NARR];
  size_t off = 0;
  uint32_t stage_bytes = 0;
#pragma unroll
  for (int a = 0; a < NARR; ++a) {
    arr_off[a] = off;
    off += size_t(STAGES) * TILE * esize[a];
    stage_bytes += TILE * esize[a];
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + ((off + 7) & ~size_t(7)));
  uint32_t* done = reinterpret_cast<uint32_t*>(bars + STAGES);   // warps finished with the current fill
  uint32_t* fills = done + STAGES;                                // fills issued per stage

  const int64_t first = blockIdx.x;
  const int64_t stride = gridDim.x;
  const int64_t my_tiles = first < full_tiles ? (full_tiles - first + stride - 1) / stride : 0;

  // fill stage s with tile t
  auto issue = [&](int s, int64_t t) {
    fills[s] += 1;
    mbar_arrive_expect_tx(&bars[s], stage_bytes);
#pragma unroll
    for (int a = 0; a < NARR; ++a) {
      const uint32_t es = esize[a];
      bulk_g2s(smem + arr_off[a] + size_t(s) * TILE * es, src_of(t, a), TILE * es, &bars[s]);
    }
  };

  if (tid == 0) {
#pragma unroll
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&bars[s], 1);
      done[s] = 0;
      fills[s] = 0;
    }
    fence_mbar_init();
    for (int i = 0; i < STAGES && i < my_tiles; ++i) issue(i, first + i * stride);
  }
  __syncthreads();

  const uint64_t lim = ring_wait_limit(status);
  // stage index and mbarrier phase advance incrementally (no 64-bit division)
  int s = 0;
  uint32_t parity = 0;
  int64_t tile = first;
  for (int64_t i = 0; i < my_tiles; ++i, tile += stride) {
    if (!mbar_wait_ring(&bars[s], parity, lim)) {
      if (lane == 0) {
        atomicOr(status, kStatusTimeout);
        // let copies still in flight land before the CTA's shared memory is released
        for (int q = 0; q < STAGES; ++q) {
          const uint32_t n = *reinterpret_cast<volatile uint32_t*>(&fills[q]);
          if (n > 0) mbar_wait_bounded(&bars[q], (n - 1) & 1u);
        }
      }
      __syncwarp();
      return false;
    }
    const uint8_t* stage[NARR];
#pragma unroll
    for (int a = 0; a < NARR; ++a) stage[a] = smem + arr_off[a] + size_t(s) * TILE * esize[a];
    compute(stage, tile);
    __syncwarp();
    if (lane == 0) {
      __threadfence_block();
      if (atomicAdd(&done[s], 1u) == kWarps - 1) {
        // every warp is done reading this fill: refill it with the tile STAGES ahead
        done[s] = 0;
        if (i + STAGES < my_tiles) {
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          issue(s, tile + STAGES * stride);
        }
      }
    }
    if (++s == STAGES) {
      s = 0;
      parity ^= 1u;
    }
  }
  return true;
}

// One tensor per input array: tile t of array a starts at ptr[a] + t * TILE * esize[a].
template <int THREADS, int TILE, int STAGES, int NARR, class Compute>
__device__ __forceinline__ bool run_tiles(uint8_t* smem, const TileSrc<NARR>& src, int64_t full_tiles,
                                          unsigned int* status, Compute&& compute) {
  return run_tiles_src<THREADS, TILE, STAGES, NARR>(
      smem, src.esize, full_tiles, status,
      [&](int64_t t, int a) { return src.ptr[a] + size_t(t) * TILE * src.esize[a]; }, compute);
}

}  // namespace roi
