// Host-side launch interface between the C ABI (roi_api.cu) and the kernels.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "roi_common.cuh"

namespace roi {

// Every Philox counter (e_base + e) / 4 of a call of E elements is below 2^32
// (its flat element indices stay below 2^34).
inline bool counters_narrow(const NoiseParams& np, int64_t E) {
  const uint64_t lim = uint64_t(1) << 34;
  return np.e_base <= lim && uint64_t(E) <= lim - np.e_base;
}

struct FwdCall {
  const float* phi;
  const uint16_t* W;
  uint16_t* Wm;
  float* soft;      // nullable
  uint32_t* hard;   // nullable
  bool st;          // straight-through: Wm = W where the hard mask is set, +0 elsewhere
  int64_t E;        // rows * cols
  int N, M;
  float tau;
  NoiseParams np;
  unsigned int* status;
  cudaStream_t stream;
};

struct BwdCall {
  const float* phi;
  const uint16_t* W;
  const uint16_t* dWm;
  float* dphi;
  uint16_t* dW;     // nullable
  const uint32_t* hard_in;  // nullable; straight-through: dW = dWm where set, +0 elsewhere
  float* phi_out;   // nullable; fused AdamW: the logits updated in place (== phi)
  float* m;         // AdamW first and second moments (with phi_out)
  float* v;
  AdamW opt;
  int64_t E;
  int N, M;
  float tau;
  NoiseParams np;
  unsigned int* status;
  cudaStream_t stream;
};

struct ExportCall {
  const float* phi;
  uint32_t* bits;
  const uint16_t* W;  // nullable
  uint16_t* Wp;       // nullable
  int64_t E;
  int N, M;
  cudaStream_t stream;
};

struct CompressCall {
  const float* phi;
  const uint16_t* W;
  uint16_t* values;  // [E / 2]
  uint32_t* meta;    // [E / 32]
  int64_t E;         // multiple of 32
  cudaStream_t stream;
};

struct LinearCall {
  const uint16_t* X;    // [T, cols] bf16
  const float* phi;     // [rows, cols]
  const uint16_t* W;    // [rows, cols] bf16
  float* Y;             // [T, rows]
  void* workspace;      // nullable: split-K partials and tickets
  size_t workspace_bytes;
  int64_t T, rows, cols;
  int N, M;
  float tau;
  NoiseParams np;
  unsigned int* status;
  cudaStream_t stream;
};

// Each returns the number of kernels launched (>= 0) or -1 after a CUDA error.
int launch_fwd(const FwdCall& c);
int launch_bwd(const BwdCall& c);
// Many independent tensors on one stream: one launch per tensor, or per run of
// small tensors (multi_small), the tile kernels chained by programmatic dependent
// launch so each may start while the previous one drains (stream order is kept:
// each completes after its predecessor).
int launch_fwd_batch(const FwdCall* calls, int count);
int launch_bwd_batch(const BwdCall* calls, int count);
int launch_export(const ExportCall& c);
int launch_export_compressed_2of4(const CompressCall& c);
// Warp-slice kernels for M = 16, 32 (roi_slice.cu).
bool slice_supported(int N, int M);
int launch_slice_fwd(const FwdCall& c, bool pdl = false);
int launch_slice_bwd(const BwdCall& c, bool pdl = false);
int launch_noise(const NoiseParams& np, int64_t E, uint32_t* words, float* g, cudaStream_t stream);

// Masked linear forward on the tensor cores (roi_linear.cu).
bool linear_supported(int N, int M);
int linear_splits(int64_t T, int64_t rows, int64_t cols);
size_t linear_workspace_bytes(int64_t T, int64_t rows, int64_t cols);
int launch_masked_linear(const LinearCall& c);

// Launches kern<<<grid, threads, smem, stream>>>(args...), with programmatic stream
// serialization allowed when `pdl` (the kernel then may start before the stream's
// previous kernel has finished).  Returns 1, or -1 after a CUDA error.
template <class... KArgs, class... Args>
int launch_maybe_pdl(void (*kern)(KArgs...), int grid, int threads, size_t smem, cudaStream_t stream, bool pdl,
                     const Args&... args) {
  if (!pdl) {
    kern<<<grid, threads, smem, stream>>>(args...);
    return cudaGetLastError() == cudaSuccess ? 1 : -1;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(grid));
  cfg.blockDim = dim3(unsigned(threads));
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...) == cudaSuccess ? 1 : -1;
}

// Streaming multiprocessors of the current device (cached).
int sm_count();

// Batched calls: a run of consecutive items with the same tile kernel, each of
// them small (fewer than kMultiTilesPerSm full tiles per SM), goes to one
// multi-tensor launch when it holds at least multi_min_run items.  One launch per
// small tensor spends much of its time on fixed costs (ring fill and drain, the
// ragged tail, the gap to the next launch).  A larger tensor keeps a launch of its
// own: the multi-tensor kernels hold the current tensor's arguments in registers
// rather than in the constant bank, and measured 4-7 % slower on 18944 x 3584
// tensors.  That per-tile cost also decides the run lengths: the plain backward
// gains from runs of 2 (the q, k, v, o tensors of a 7B-shaped layer), while the
// forward and the backward fused with AdamW lost on those runs (7B-shaped 2:4 step,
// forward 11.72 -> 11.80 ms, fused backward 28.8 -> 29.0 ms) and gain only over long
// ones.  So does the plain backward where many groups go through the deferred
// queue (tau below the deferral threshold): each drained group reads its tensor's
// arguments from the parameter block by a per-lane index (tau = 0.05, 1.5B-shaped
// 4:8 backward 7.01 -> 7.24 ms with short runs shared).  A fwd + bwd step over a
// Qwen2.5-shaped layer set went from 1.90 to 1.57 ms (0.5B-shaped, 2:4: one launch
// per direction), 8.92 to 8.78 ms (1.5B-shaped, 4:8) and 24.31 to 24.19 ms
// (7B-shaped, 2:4).
constexpr int64_t kMultiTilesPerSm = 12;
inline int multi_min_run(bool short_runs_pay) { return short_runs_pay ? 2 : 8; }
inline bool multi_small(int64_t E, int64_t tile) { return E / tile < kMultiTilesPerSm * sm_count(); }

}  // namespace roi
