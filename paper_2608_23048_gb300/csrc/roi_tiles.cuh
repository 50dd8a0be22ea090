// Persistent tile pipeline: each CTA walks tiles blockIdx.x, blockIdx.x + grid, ...
// of TILE contiguous elements.  One thread stages the inputs of upcoming tiles
// into a ring of shared-memory stages with 1-D bulk copies (TMA) that complete
// on one mbarrier per stage; all threads wait (bounded), compute from shared
// memory and store their outputs straight to global memory (coalesced).
#pragma once

#include "roi_common.cuh"

namespace roi {

template <int NARR>
struct TileSrc {
  const uint8_t* ptr[NARR];  // global base of each input array
  uint32_t esize[NARR];      // bytes per element of each input array
};

template <int TILE, int STAGES, int NARR>
struct TileSmem {
  static constexpr size_t bars_offset(const uint32_t (&es)[NARR]) {
    size_t off = 0;
    for (int a = 0; a < NARR; ++a) off += size_t(STAGES) * TILE * es[a];
    return off;
  }
};

// Runs `compute(stage_ptrs, tile)` for every full tile of this CTA.  Returns
// false if a wait timed out (status recorded, copies drained).
template <int THREADS, int TILE, int STAGES, int NARR, class Compute>
__device__ __forceinline__ bool run_tiles(uint8_t* smem, const TileSrc<NARR>& src, int64_t full_tiles,
                                          unsigned int* status, Compute&& compute) {
  const int tid = threadIdx.x;
  size_t arr_off[NARR];
  size_t off = 0;
  uint32_t stage_bytes = 0;
#pragma unroll
  for (int a = 0; a < NARR; ++a) {
    arr_off[a] = off;
    off += size_t(STAGES) * TILE * src.esize[a];
    stage_bytes += TILE * src.esize[a];
  }
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + ((off + 7) & ~size_t(7)));

  const int64_t first = blockIdx.x;
  const int64_t stride = gridDim.x;
  const int64_t my_tiles = first < full_tiles ? (full_tiles - first + stride - 1) / stride : 0;

  if (tid == 0) {
#pragma unroll
    for (int s = 0; s < STAGES; ++s) mbar_init(&bars[s], 1);
    fence_mbar_init();
  }
  __syncthreads();

  auto issue = [&](int64_t i) {
    const int s = int(i % STAGES);
    const int64_t t = first + i * stride;
    mbar_arrive_expect_tx(&bars[s], stage_bytes);
#pragma unroll
    for (int a = 0; a < NARR; ++a) {
      const uint32_t es = src.esize[a];
      bulk_g2s(smem + arr_off[a] + size_t(s) * TILE * es, src.ptr[a] + size_t(t) * TILE * es, TILE * es,
               &bars[s]);
    }
  };

  int64_t issued = 0;
  if (tid == 0) {
    for (; issued < my_tiles && issued < STAGES; ++issued) issue(issued);
  }

  for (int64_t i = 0; i < my_tiles; ++i) {
    const int s = int(i % STAGES);
    const uint32_t parity = uint32_t((i / STAGES) & 1);
    const bool timed_out = !mbar_wait_bounded(&bars[s], parity);
    if (!timed_out) {
      const uint8_t* stage[NARR];
#pragma unroll
      for (int a = 0; a < NARR; ++a) stage[a] = smem + arr_off[a] + size_t(s) * TILE * src.esize[a];
      compute(stage, first + i * stride);
    }
    if (__syncthreads_or(timed_out)) {
      if (tid == 0) {
        atomicOr(status, kStatusTimeout);
        // let copies still in flight land before the CTA's shared memory is released
        for (int64_t j = i; j < issued; ++j)
          mbar_wait_bounded(&bars[int(j % STAGES)], uint32_t((j / STAGES) & 1));
      }
      __syncthreads();
      return false;
    }
    if (tid == 0 && issued < my_tiles) {
      issue(issued);
      ++issued;
    }
  }
  return true;
}

}  // namespace roi
