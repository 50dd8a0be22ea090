// C ABI of libroi (see include/roi.h): host-side validation, then one launch.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <vector>
#include <cstdint>
#include <cstring>

#include "roi.h"
#include "roi_launch.h"

namespace roi {

// The device status record: word 0 the status bits (kStatusTimeout), words 2-3
// the ring-wait limit in ns (2 s).  One per device; the kernels get its address.
__device__ __align__(16) unsigned int g_roi_device_status[4] = {0u, 0u, 2000000000u, 0u};

namespace {

std::atomic<uint64_t> g_launches{0};

unsigned int* status_word() {
  // Device address of this module's status word on the current device.
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_roi_device_status) != cudaSuccess) return nullptr;
  return static_cast<unsigned int*>(p);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct Range {
  const void* p;
  uint64_t bytes;
};

bool overlaps(const Range& a, const Range& b) {
  if (a.p == nullptr || b.p == nullptr || a.bytes == 0 || b.bytes == 0) return false;
  const uintptr_t a0 = reinterpret_cast<uintptr_t>(a.p), b0 = reinterpret_cast<uintptr_t>(b.p);
  return a0 < b0 + b.bytes && b0 < a0 + a.bytes;
}

// Outputs must not overlap inputs or each other.
template <int NI, int NO>
bool any_alias(const Range (&in)[NI], const Range (&out)[NO]) {
  for (int o = 0; o < NO; ++o) {
    for (int i = 0; i < NI; ++i)
      if (overlaps(out[o], in[i])) return true;
    for (int p = o + 1; p < NO; ++p)
      if (overlaps(out[o], out[p])) return true;
  }
  return false;
}

bool finite_positive(float x) { return std::isfinite(x) && x > 0.0f; }

// Across a batch: true if an output range overlaps any other range (input or
// output).  Sort by start; a range overlaps an earlier one iff it starts before
// the largest end seen so far (of outputs, for an input; of all, for an output).
struct Tagged {
  uintptr_t lo, hi;
  bool out;
};
bool batch_alias(std::vector<Tagged>& r) {
  std::sort(r.begin(), r.end(), [](const Tagged& a, const Tagged& b) { return a.lo < b.lo; });
  uintptr_t end_all = 0, end_out = 0;
  for (const Tagged& x : r) {
    if (x.out ? x.lo < end_all : x.lo < end_out) return true;
    end_all = std::max(end_all, x.hi);
    if (x.out) end_out = std::max(end_out, x.hi);
  }
  return false;
}
void add_range(std::vector<Tagged>& r, const void* p, uint64_t bytes, bool out) {
  if (p == nullptr || bytes == 0) return;
  const uintptr_t lo = reinterpret_cast<uintptr_t>(p);
  r.push_back({lo, lo + uintptr_t(bytes), out});
}

roi_status check_common(int N, int M, float tau, int64_t rows, int64_t cols) {
  if (!(N >= 1 && N < M && M <= 32)) return ROI_ERR_NM;
  if (rows < 0 || cols <= 0 || cols % M != 0) return ROI_ERR_SHAPE;
  if (rows > 0 && cols > INT64_MAX / 64 / rows) return ROI_ERR_SHAPE;
  if (!finite_positive(tau)) return ROI_ERR_TAU;
  return ROI_OK;
}

NoiseParams make_noise(const roi_noise_state& st, int64_t cols) {
  NoiseParams np;
  np.k0 = static_cast<uint32_t>(st.seed & 0xffffffffu);
  np.k1 = static_cast<uint32_t>(st.seed >> 32);
  np.step = st.step;
  np.tensor_id = st.tensor_id;
  np.inv_lam = 1.0f / st.lambda;
  np.l2e_inv_lam = static_cast<float>(1.4426950408889634 / static_cast<double>(st.lambda));
  np.e_base = static_cast<uint64_t>(st.row_offset) * static_cast<uint64_t>(cols);
  return np;
}

roi_status finish(int launched) {
  if (launched < 0) return ROI_ERR_CUDA;
  g_launches.fetch_add(static_cast<uint64_t>(launched), std::memory_order_relaxed);
  return ROI_OK;
}

}  // namespace

int sm_count() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  if (cache[dev] == 0) {
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    cache[dev] = n > 0 ? n : 1;
  }
  return cache[dev];
}

}  // namespace roi

using namespace roi;

extern "C" {

static roi_status mask_fwd(const float* logits, const roi_bf16* W, int N, int M, float tau, const roi_noise_state* st,
                           int64_t rows, int64_t cols, roi_bf16* out_Wm, float* out_soft, uint32_t* out_hard,
                           bool straight_through, void* stream) {
  if (st == nullptr) return ROI_ERR_NULL;
  roi_status s = check_common(N, M, tau, rows, cols);
  if (s != ROI_OK) return s;
  if (st->row_offset < 0) return ROI_ERR_SHAPE;
  if (!finite_positive(st->lambda)) return ROI_ERR_TAU;
  if (rows == 0) return ROI_OK;  // nothing is read or written; pointers may be NULL
  if (logits == nullptr || W == nullptr || out_Wm == nullptr) return ROI_ERR_NULL;
  if (!aligned16(logits) || !aligned16(W) || !aligned16(out_Wm) || !aligned16(out_soft) || !aligned16(out_hard))
    return ROI_ERR_ALIGN;
  const int64_t E = rows * cols;
  const Range in[2] = {{logits, uint64_t(E) * 4}, {W, uint64_t(E) * 2}};
  const Range out[3] = {{out_Wm, uint64_t(E) * 2}, {out_soft, uint64_t(E) * 4}, {out_hard, uint64_t((E + 31) / 32) * 4}};
  if (any_alias(in, out)) return ROI_ERR_ALIAS;
  if (E == 0) return ROI_OK;
  FwdCall c;
  c.phi = logits;
  c.W = W;
  c.Wm = out_Wm;
  c.soft = out_soft;
  c.hard = out_hard;
  c.st = straight_through;
  c.E = E;
  c.N = N;
  c.M = M;
  c.tau = tau;
  c.np = make_noise(*st, cols);
  c.status = status_word();
  if (c.status == nullptr) return ROI_ERR_CUDA;
  c.stream = static_cast<cudaStream_t>(stream);
  return finish(launch_fwd(c));
}

static roi_status fwd_batch(const roi_fwd_item* items, int count, int N, int M, float tau, bool straight_through,
                            void* stream) {
  if (count < 0) return ROI_ERR_SHAPE;
  if (count > 0 && items == nullptr) return ROI_ERR_NULL;
  roi_status s = check_common(N, M, tau, 0, M);
  if (s != ROI_OK) return s;
  std::vector<Tagged> ranges;
  ranges.reserve(size_t(count) * 5);
  for (int i = 0; i < count; ++i) {
    const roi_fwd_item& it = items[i];
    s = check_common(N, M, tau, it.rows, it.cols);
    if (s != ROI_OK) return s;
    if (it.st.row_offset < 0) return ROI_ERR_SHAPE;
    if (!finite_positive(it.st.lambda)) return ROI_ERR_TAU;
    if (it.rows == 0) continue;
    if (it.logits == nullptr || it.W == nullptr || it.out_Wm == nullptr) return ROI_ERR_NULL;
    if (!aligned16(it.logits) || !aligned16(it.W) || !aligned16(it.out_Wm) || !aligned16(it.out_soft) ||
        !aligned16(it.out_hard))
      return ROI_ERR_ALIGN;
    const int64_t E = it.rows * it.cols;
    add_range(ranges, it.logits, uint64_t(E) * 4, false);
    add_range(ranges, it.W, uint64_t(E) * 2, false);
    add_range(ranges, it.out_Wm, uint64_t(E) * 2, true);
    add_range(ranges, it.out_soft, uint64_t(E) * 4, true);
    add_range(ranges, it.out_hard, uint64_t((E + 31) / 32) * 4, true);
  }
  if (batch_alias(ranges)) return ROI_ERR_ALIAS;
  if (ranges.empty()) return ROI_OK;  // only empty items: nothing is read or written
  unsigned int* status = status_word();
  if (status == nullptr) return ROI_ERR_CUDA;
  std::vector<FwdCall> calls;
  calls.reserve(size_t(count));
  for (int i = 0; i < count; ++i) {
    const roi_fwd_item& it = items[i];
    if (it.rows == 0) continue;
    FwdCall c;
    c.phi = it.logits;
    c.W = it.W;
    c.Wm = it.out_Wm;
    c.soft = it.out_soft;
    c.hard = it.out_hard;
    c.st = straight_through;
    c.E = it.rows * it.cols;
    c.N = N;
    c.M = M;
    c.tau = tau;
    c.np = make_noise(it.st, it.cols);
    c.status = status;
    c.stream = static_cast<cudaStream_t>(stream);
    calls.push_back(c);
  }
  return finish(launch_fwd_batch(calls.data(), int(calls.size())));
}

roi_status roi_mask_fwd_batch(const roi_fwd_item* items, int count, int N, int M, float tau, void* stream) {
  return fwd_batch(items, count, N, M, tau, false, stream);
}

roi_status roi_mask_fwd_st_batch(const roi_fwd_item* items, int count, int N, int M, float tau, void* stream) {
  return fwd_batch(items, count, N, M, tau, true, stream);
}

roi_status roi_mask_bwd_st_batch(const roi_bwd_st_item* items, int count, int N, int M, float tau, void* stream) {
  if (count < 0) return ROI_ERR_SHAPE;
  if (count > 0 && items == nullptr) return ROI_ERR_NULL;
  roi_status s = check_common(N, M, tau, 0, M);
  if (s != ROI_OK) return s;
  std::vector<Tagged> ranges;
  ranges.reserve(size_t(count) * 6);
  for (int i = 0; i < count; ++i) {
    const roi_bwd_st_item& it = items[i];
    s = check_common(N, M, tau, it.rows, it.cols);
    if (s != ROI_OK) return s;
    if (it.st.row_offset < 0) return ROI_ERR_SHAPE;
    if (!finite_positive(it.st.lambda)) return ROI_ERR_TAU;
    if (it.rows == 0) continue;
    if (it.logits == nullptr || it.W == nullptr || it.dWm == nullptr || it.out_dlogits == nullptr ||
        (it.out_dW != nullptr && it.hard == nullptr))
      return ROI_ERR_NULL;
    if (!aligned16(it.logits) || !aligned16(it.W) || !aligned16(it.dWm) || !aligned16(it.hard) ||
        !aligned16(it.out_dlogits) || !aligned16(it.out_dW))
      return ROI_ERR_ALIGN;
    const int64_t E = it.rows * it.cols;
    add_range(ranges, it.logits, uint64_t(E) * 4, false);
    add_range(ranges, it.W, uint64_t(E) * 2, false);
    add_range(ranges, it.dWm, uint64_t(E) * 2, false);
    add_range(ranges, it.hard, uint64_t((E + 31) / 32) * 4, false);
    add_range(ranges, it.out_dlogits, uint64_t(E) * 4, true);
    add_range(ranges, it.out_dW, uint64_t(E) * 2, true);
  }
  if (batch_alias(ranges)) return ROI_ERR_ALIAS;
  if (ranges.empty()) return ROI_OK;
  unsigned int* status = status_word();
  if (status == nullptr) return ROI_ERR_CUDA;
  std::vector<BwdCall> calls;
  calls.reserve(size_t(count));
  for (int i = 0; i < count; ++i) {
    const roi_bwd_st_item& it = items[i];
    if (it.rows == 0) continue;
    BwdCall c{};
    c.phi = it.logits;
    c.W = it.W;
    c.dWm = it.dWm;
    c.dphi = it.out_dlogits;
    c.dW = it.out_dW;
    c.hard_in = it.out_dW != nullptr ? it.hard : nullptr;
    c.E = it.rows * it.cols;
    c.N = N;
    c.M = M;
    c.tau = tau;
    c.np = make_noise(it.st, it.cols);
    c.status = status;
    c.stream = static_cast<cudaStream_t>(stream);
    calls.push_back(c);
  }
  return finish(launch_bwd_batch(calls.data(), int(calls.size())));
}

roi_status roi_mask_bwd_batch(const roi_bwd_item* items, int count, int N, int M, float tau, void* stream) {
  if (count < 0) return ROI_ERR_SHAPE;
  if (count > 0 && items == nullptr) return ROI_ERR_NULL;
  roi_status s = check_common(N, M, tau, 0, M);
  if (s != ROI_OK) return s;
  std::vector<Tagged> ranges;
  ranges.reserve(size_t(count) * 5);
  for (int i = 0; i < count; ++i) {
    const roi_bwd_item& it = items[i];
    s = check_common(N, M, tau, it.rows, it.cols);
    if (s != ROI_OK) return s;
    if (it.st.row_offset < 0) return ROI_ERR_SHAPE;
    if (!finite_positive(it.st.lambda)) return ROI_ERR_TAU;
    if (it.rows == 0) continue;
    if (it.logits == nullptr || it.W == nullptr || it.dWm == nullptr || it.out_dlogits == nullptr)
      return ROI_ERR_NULL;
    if (!aligned16(it.logits) || !aligned16(it.W) || !aligned16(it.dWm) || !aligned16(it.out_dlogits) ||
        !aligned16(it.out_dW))
      return ROI_ERR_ALIGN;
    const int64_t E = it.rows * it.cols;
    add_range(ranges, it.logits, uint64_t(E) * 4, false);
    add_range(ranges, it.W, uint64_t(E) * 2, false);
    add_range(ranges, it.dWm, uint64_t(E) * 2, false);
    add_range(ranges, it.out_dlogits, uint64_t(E) * 4, true);
    add_range(ranges, it.out_dW, uint64_t(E) * 2, true);
  }
  if (batch_alias(ranges)) return ROI_ERR_ALIAS;
  if (ranges.empty()) return ROI_OK;  // only empty items: nothing is read or written
  unsigned int* status = status_word();
  if (status == nullptr) return ROI_ERR_CUDA;
  std::vector<BwdCall> calls;
  calls.reserve(size_t(count));
  for (int i = 0; i < count; ++i) {
    const roi_bwd_item& it = items[i];
    if (it.rows == 0) continue;
    BwdCall c{};
    c.phi = it.logits;
    c.W = it.W;
    c.dWm = it.dWm;
    c.dphi = it.out_dlogits;
    c.dW = it.out_dW;
    c.E = it.rows * it.cols;
    c.N = N;
    c.M = M;
    c.tau = tau;
    c.np = make_noise(it.st, it.cols);
    c.status = status;
    c.stream = static_cast<cudaStream_t>(stream);
    calls.push_back(c);
  }
  return finish(launch_bwd_batch(calls.data(), int(calls.size())));
}

roi_status roi_mask_fwd_ex(const float* logits, const roi_bf16* W, int N, int M, float tau,
                           const roi_noise_state* st, int64_t rows, int64_t cols, roi_bf16* out_Wm,
                           float* out_soft, uint32_t* out_hard, void* stream) {
  return mask_fwd(logits, W, N, M, tau, st, rows, cols, out_Wm, out_soft, out_hard, false, stream);
}

roi_status roi_mask_fwd_st(const float* logits, const roi_bf16* W, int N, int M, float tau,
                           const roi_noise_state* st, int64_t rows, int64_t cols, roi_bf16* out_Wm,
                           float* out_soft, uint32_t* out_hard, void* stream) {
  return mask_fwd(logits, W, N, M, tau, st, rows, cols, out_Wm, out_soft, out_hard, true, stream);
}

roi_status roi_mask_fwd(const float* logits, const roi_bf16* W, int N, int M, float tau, uint64_t seed,
                        uint32_t step, int64_t rows, int64_t cols, roi_bf16* out_Wm, float* out_soft,
                        uint32_t* out_hard, void* stream) {
  roi_noise_state st;
  st.seed = seed;
  st.step = step;
  st.tensor_id = 0;
  st.lambda = 1.0f;
  st.row_offset = 0;
  return roi_mask_fwd_ex(logits, W, N, M, tau, &st, rows, cols, out_Wm, out_soft, out_hard, stream);
}

// The fused optimizer of roi_mask_bwd_adamw: logits updated in place, moments m, v.
struct FusedAdamW {
  float* phi;
  float* m;
  float* v;
  AdamW opt;
};

static roi_status mask_bwd(const float* logits, const roi_bf16* W, const roi_noise_state* st, int N, int M,
                           const roi_bf16* dWm, const uint32_t* hard, float tau, int64_t rows, int64_t cols,
                           float* out_dlogits, roi_bf16* out_dW, const FusedAdamW* fo, void* stream) {
  if (st == nullptr) return ROI_ERR_NULL;
  roi_status s = check_common(N, M, tau, rows, cols);
  if (s != ROI_OK) return s;
  if (st->row_offset < 0) return ROI_ERR_SHAPE;
  if (!finite_positive(st->lambda)) return ROI_ERR_TAU;
  if (rows == 0) return ROI_OK;
  if (logits == nullptr || W == nullptr || dWm == nullptr || (out_dlogits == nullptr && fo == nullptr))
    return ROI_ERR_NULL;
  if (fo != nullptr && (fo->m == nullptr || fo->v == nullptr)) return ROI_ERR_NULL;
  if (!aligned16(logits) || !aligned16(W) || !aligned16(dWm) || !aligned16(out_dlogits) || !aligned16(out_dW))
    return ROI_ERR_ALIGN;
  if (fo != nullptr && (!aligned16(fo->m) || !aligned16(fo->v))) return ROI_ERR_ALIGN;
  const int64_t E = rows * cols;
  // with the fused optimizer the logits are updated in place: they count as an
  // output for the overlap check against every other tensor (but not themselves)
  const Range in[4] = {{fo ? nullptr : logits, uint64_t(E) * 4}, {W, uint64_t(E) * 2}, {dWm, uint64_t(E) * 2},
                       {hard, uint64_t((E + 31) / 32) * 4}};
  const Range out[5] = {{out_dlogits, uint64_t(E) * 4}, {out_dW, uint64_t(E) * 2},
                        {fo ? logits : nullptr, uint64_t(E) * 4}, {fo ? fo->m : nullptr, uint64_t(E) * 4},
                        {fo ? fo->v : nullptr, uint64_t(E) * 4}};
  if (any_alias(in, out)) return ROI_ERR_ALIAS;
  if (E == 0) return ROI_OK;
  BwdCall c;
  c.phi = logits;
  c.W = W;
  c.dWm = dWm;
  c.dphi = out_dlogits;
  c.dW = out_dW;
  c.hard_in = hard;
  c.phi_out = fo ? fo->phi : nullptr;
  c.m = fo ? fo->m : nullptr;
  c.v = fo ? fo->v : nullptr;
  c.opt = fo ? fo->opt : AdamW{};
  c.E = E;
  c.N = N;
  c.M = M;
  c.tau = tau;
  c.np = make_noise(*st, cols);
  c.status = status_word();
  if (c.status == nullptr) return ROI_ERR_CUDA;
  c.stream = static_cast<cudaStream_t>(stream);
  return finish(launch_bwd(c));
}

roi_status roi_mask_bwd(const float* logits, const roi_bf16* W, const roi_noise_state* st, int N, int M,
                        const roi_bf16* dWm, float tau, int64_t rows, int64_t cols, float* out_dlogits,
                        roi_bf16* out_dW, void* stream) {
  return mask_bwd(logits, W, st, N, M, dWm, nullptr, tau, rows, cols, out_dlogits, out_dW, nullptr, stream);
}

roi_status roi_mask_bwd_st(const float* logits, const roi_bf16* W, const roi_noise_state* st, int N, int M,
                           const roi_bf16* dWm, const uint32_t* hard, float tau, int64_t rows, int64_t cols,
                           float* out_dlogits, roi_bf16* out_dW, void* stream) {
  if (out_dW != nullptr && hard == nullptr && rows > 0) return ROI_ERR_NULL;
  if (!aligned16(hard)) return ROI_ERR_ALIGN;
  return mask_bwd(logits, W, st, N, M, dWm, out_dW != nullptr ? hard : nullptr, tau, rows, cols, out_dlogits,
                  out_dW, nullptr, stream);
}

// Checks the optimizer settings and forms the step's constants, rounded to float
// as the float32 statement of the step forms them.
static roi_status adamw_constants(const roi_adamw* opt, AdamW* out) {
  if (opt == nullptr) return ROI_ERR_NULL;
  const bool ok = std::isfinite(opt->lr) && opt->lr >= 0.0f && opt->beta1 >= 0.0f && opt->beta1 < 1.0f &&
                  opt->beta2 >= 0.0f && opt->beta2 < 1.0f && finite_positive(opt->eps) &&
                  std::isfinite(opt->weight_decay) && opt->weight_decay >= 0.0f && opt->t >= 1;
  if (!ok) return ROI_ERR_OPT;
  out->b1 = opt->beta1;
  out->omb1 = 1.0f - opt->beta1;
  out->b2 = opt->beta2;
  out->omb2 = 1.0f - opt->beta2;
  out->eps = opt->eps;
  out->decay = 1.0f - opt->lr * opt->weight_decay;
  const double t = static_cast<double>(opt->t);
  out->step = static_cast<float>(static_cast<double>(opt->lr) / (1.0 - std::pow(static_cast<double>(opt->beta1), t)));
  out->r = static_cast<float>(1.0 / std::sqrt(1.0 - std::pow(static_cast<double>(opt->beta2), t)));
  return ROI_OK;
}

roi_status roi_mask_bwd_adamw(float* logits, const roi_bf16* W, const roi_noise_state* st, int N, int M,
                              const roi_bf16* dWm, float tau, int64_t rows, int64_t cols, float* m, float* v,
                              const roi_adamw* opt, float* out_dlogits, roi_bf16* out_dW, void* stream) {
  FusedAdamW fo;
  const roi_status s = adamw_constants(opt, &fo.opt);
  if (s != ROI_OK) return s;
  fo.phi = logits;
  fo.m = m;
  fo.v = v;
  return mask_bwd(logits, W, st, N, M, dWm, nullptr, tau, rows, cols, out_dlogits, out_dW, &fo, stream);
}

roi_status roi_mask_bwd_adamw_batch(const roi_adamw_item* items, int count, int N, int M, float tau,
                                    const roi_adamw* opt, void* stream) {
  if (count < 0) return ROI_ERR_SHAPE;
  if (count > 0 && items == nullptr) return ROI_ERR_NULL;
  AdamW k;
  roi_status s = adamw_constants(opt, &k);
  if (s != ROI_OK) return s;
  s = check_common(N, M, tau, 0, M);
  if (s != ROI_OK) return s;
  std::vector<Tagged> ranges;
  ranges.reserve(size_t(count) * 7);
  for (int i = 0; i < count; ++i) {
    const roi_adamw_item& it = items[i];
    s = check_common(N, M, tau, it.rows, it.cols);
    if (s != ROI_OK) return s;
    if (it.st.row_offset < 0) return ROI_ERR_SHAPE;
    if (!finite_positive(it.st.lambda)) return ROI_ERR_TAU;
    if (it.rows == 0) continue;
    if (it.logits == nullptr || it.W == nullptr || it.dWm == nullptr || it.m == nullptr || it.v == nullptr)
      return ROI_ERR_NULL;
    if (!aligned16(it.logits) || !aligned16(it.W) || !aligned16(it.dWm) || !aligned16(it.m) || !aligned16(it.v) ||
        !aligned16(it.out_dlogits) || !aligned16(it.out_dW))
      return ROI_ERR_ALIGN;
    const int64_t E = it.rows * it.cols;
    add_range(ranges, it.W, uint64_t(E) * 2, false);
    add_range(ranges, it.dWm, uint64_t(E) * 2, false);
    add_range(ranges, it.logits, uint64_t(E) * 4, true);  // read and written
    add_range(ranges, it.m, uint64_t(E) * 4, true);
    add_range(ranges, it.v, uint64_t(E) * 4, true);
    add_range(ranges, it.out_dlogits, uint64_t(E) * 4, true);
    add_range(ranges, it.out_dW, uint64_t(E) * 2, true);
  }
  if (batch_alias(ranges)) return ROI_ERR_ALIAS;
  if (ranges.empty()) return ROI_OK;
  unsigned int* status = status_word();
  if (status == nullptr) return ROI_ERR_CUDA;
  std::vector<BwdCall> calls;
  calls.reserve(size_t(count));
  for (int i = 0; i < count; ++i) {
    const roi_adamw_item& it = items[i];
    if (it.rows == 0) continue;
    BwdCall c{};
    c.phi = it.logits;
    c.W = it.W;
    c.dWm = it.dWm;
    c.dphi = it.out_dlogits;
    c.dW = it.out_dW;
    c.phi_out = it.logits;
    c.m = it.m;
    c.v = it.v;
    c.opt = k;
    c.E = it.rows * it.cols;
    c.N = N;
    c.M = M;
    c.tau = tau;
    c.np = make_noise(it.st, it.cols);
    c.status = status;
    c.stream = static_cast<cudaStream_t>(stream);
    calls.push_back(c);
  }
  return finish(launch_bwd_batch(calls.data(), int(calls.size())));
}

float roi_anneal(float init, float end, uint32_t t, uint32_t T_anneal) {
  if (T_anneal == 0) return end;
  const double x = static_cast<double>(init) *
                   std::pow(static_cast<double>(end) / static_cast<double>(init),
                            static_cast<double>(t) / static_cast<double>(T_anneal));
  return static_cast<float>(x > static_cast<double>(end) ? x : static_cast<double>(end));
}

roi_status roi_export_compressed_2of4(const float* logits, const roi_bf16* W, int64_t rows, int64_t cols,
                                      roi_bf16* out_values, uint32_t* out_meta, void* stream) {
  roi_status s = check_common(2, 4, 1.0f, rows, cols);
  if (s != ROI_OK) return s;
  if ((rows * cols) % 32 != 0) return ROI_ERR_SHAPE;
  if (rows == 0) return ROI_OK;
  if (logits == nullptr || W == nullptr || out_values == nullptr || out_meta == nullptr) return ROI_ERR_NULL;
  if (!aligned16(logits) || !aligned16(W) || !aligned16(out_values) || !aligned16(out_meta)) return ROI_ERR_ALIGN;
  const int64_t E = rows * cols;
  const Range in[2] = {{logits, uint64_t(E) * 4}, {W, uint64_t(E) * 2}};
  const Range out[2] = {{out_values, uint64_t(E)}, {out_meta, uint64_t(E / 32) * 4}};
  if (any_alias(in, out)) return ROI_ERR_ALIAS;
  CompressCall c;
  c.phi = logits;
  c.W = W;
  c.values = out_values;
  c.meta = out_meta;
  c.E = E;
  c.stream = static_cast<cudaStream_t>(stream);
  return finish(launch_export_compressed_2of4(c));
}

roi_status roi_hard_mask_export(const float* logits, int N, int M, int64_t rows, int64_t cols, uint32_t* out_bits,
                                const roi_bf16* W, roi_bf16* out_Wpruned, void* stream) {
  roi_status s = check_common(N, M, 1.0f, rows, cols);
  if (s != ROI_OK) return s;
  if (rows == 0) return ROI_OK;
  if (logits == nullptr || out_bits == nullptr) return ROI_ERR_NULL;
  if ((W == nullptr) != (out_Wpruned == nullptr)) return ROI_ERR_NULL;
  if (!aligned16(logits) || !aligned16(out_bits) || !aligned16(W) || !aligned16(out_Wpruned)) return ROI_ERR_ALIGN;
  const int64_t E = rows * cols;
  const Range in[2] = {{logits, uint64_t(E) * 4}, {W, uint64_t(E) * 2}};
  const Range out[2] = {{out_bits, uint64_t((E + 31) / 32) * 4}, {out_Wpruned, uint64_t(E) * 2}};
  if (any_alias(in, out)) return ROI_ERR_ALIAS;
  if (E == 0) return ROI_OK;
  ExportCall c;
  c.phi = logits;
  c.bits = out_bits;
  c.W = W;
  c.Wp = out_Wpruned;
  c.E = E;
  c.N = N;
  c.M = M;
  c.stream = static_cast<cudaStream_t>(stream);
  return finish(launch_export(c));
}

size_t roi_masked_linear_workspace_size(int64_t T, int64_t rows, int64_t cols) {
  if (T <= 0 || T > 256 || rows <= 0 || cols <= 0 || cols > INT64_MAX / 64 / rows) return 0;
  return linear_workspace_bytes(T, rows, cols);
}

}  // extern "C"

namespace roi {
namespace {

// Split-K scratch of roi_masked_linear_fwd_noalloc: one static array per device,
// ROI_LINEAR_SCRATCH_BYTES long.
static __device__ __align__(256) unsigned char g_linear_scratch[ROI_LINEAR_SCRATCH_BYTES];

// The array's device address on the current device, looked up once per device
// (nullptr if the lookup fails or the address is not 256-byte aligned).
void* linear_scratch() {
  static std::atomic<void*> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  void* p = cache[dev].load(std::memory_order_acquire);
  if (p == nullptr) {
    if (cudaGetSymbolAddress(&p, g_linear_scratch) != cudaSuccess || p == nullptr ||
        (reinterpret_cast<uintptr_t>(p) & 255u) != 0)
      return nullptr;
    cache[dev].store(p, std::memory_order_release);
  }
  return p;
}

}  // namespace
}  // namespace roi

extern "C" {

roi_status roi_masked_linear_fwd(const roi_bf16* X, const float* logits, const roi_bf16* W, int N, int M, float tau,
                                 const roi_noise_state* st, int64_t T, int64_t rows, int64_t cols, float* out_Y,
                                 void* workspace, size_t workspace_bytes, void* stream) {
  if (st == nullptr) return ROI_ERR_NULL;
  roi_status s = check_common(N, M, tau, rows, cols);
  if (s != ROI_OK) return s;
  if (!linear_supported(N, M)) return ROI_ERR_NM;
  if (st->row_offset < 0 || T < 0 || T > 256 || cols % 8 != 0) return ROI_ERR_SHAPE;
  if (!finite_positive(st->lambda)) return ROI_ERR_TAU;
  if (rows == 0 || T == 0) return ROI_OK;  // nothing is read or written; pointers may be NULL
  if (X == nullptr || logits == nullptr || W == nullptr || out_Y == nullptr) return ROI_ERR_NULL;
  if (!aligned16(X) || !aligned16(logits) || !aligned16(W) || !aligned16(out_Y) || !aligned16(workspace))
    return ROI_ERR_ALIGN;
  const int64_t E = rows * cols;
  const Range in[3] = {{X, uint64_t(T * cols) * 2}, {logits, uint64_t(E) * 4}, {W, uint64_t(E) * 2}};
  const Range out[2] = {{out_Y, uint64_t(T * rows) * 4}, {workspace, workspace == nullptr ? 0 : uint64_t(workspace_bytes)}};
  if (any_alias(in, out)) return ROI_ERR_ALIAS;
  LinearCall c;
  c.X = X;
  c.phi = logits;
  c.W = W;
  c.Y = out_Y;
  c.workspace = workspace;
  c.workspace_bytes = workspace == nullptr ? 0 : workspace_bytes;
  c.T = T;
  c.rows = rows;
  c.cols = cols;
  c.N = N;
  c.M = M;
  c.tau = tau;
  c.np = make_noise(*st, cols);
  c.status = status_word();
  if (c.status == nullptr) return ROI_ERR_CUDA;
  c.stream = static_cast<cudaStream_t>(stream);
  return finish(launch_masked_linear(c));
}

roi_status roi_masked_linear_fwd_noalloc(const roi_bf16* X, const float* logits, const roi_bf16* W, int N, int M,
                                         float tau, const roi_noise_state* st, int64_t T, int64_t rows, int64_t cols,
                                         float* out_Y, void* stream) {
  const size_t need = roi_masked_linear_workspace_size(T, rows, cols);
  if (need > size_t(ROI_LINEAR_SCRATCH_BYTES)) return ROI_ERR_SHAPE;
  void* ws = nullptr;
  if (need > 0) {
    ws = linear_scratch();
    if (ws == nullptr) return ROI_ERR_CUDA;
  }
  return roi_masked_linear_fwd(X, logits, W, N, M, tau, st, T, rows, cols, out_Y, ws, need, stream);
}

static roi_status noise_call(const roi_noise_state* st, int64_t rows, int64_t cols, uint32_t* words, float* g,
                             void* stream) {
  if (st == nullptr) return ROI_ERR_NULL;
  if (rows < 0 || cols <= 0 || (rows > 0 && cols > INT64_MAX / 64 / rows) || st->row_offset < 0) return ROI_ERR_SHAPE;
  if (rows == 0) return ROI_OK;
  if (words == nullptr && g == nullptr) return ROI_ERR_NULL;
  if (!aligned16(words) || !aligned16(g)) return ROI_ERR_ALIGN;
  const int64_t E = rows * cols;
  return finish(launch_noise(make_noise(*st, cols), E, words, g, static_cast<cudaStream_t>(stream)));
}

roi_status roi_noise_words(const roi_noise_state* st, int64_t rows, int64_t cols, uint32_t* out_words, void* stream) {
  if (out_words == nullptr && rows > 0) return ROI_ERR_NULL;
  return noise_call(st, rows, cols, out_words, nullptr, stream);
}

roi_status roi_gumbel_noise(const roi_noise_state* st, int64_t rows, int64_t cols, float* out_g, void* stream) {
  if (out_g == nullptr && rows > 0) return ROI_ERR_NULL;
  return noise_call(st, rows, cols, nullptr, out_g, stream);
}

roi_status roi_set_ring_wait_limit_ns(uint64_t ns) {
  if (cudaMemcpyToSymbol(g_roi_device_status, &ns, sizeof(ns), kStatusLimitWord * sizeof(unsigned int)) !=
      cudaSuccess)
    return ROI_ERR_CUDA;
  return ROI_OK;
}

roi_status roi_device_status(void* stream) {
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return ROI_ERR_CUDA;
  unsigned int v = 0;
  if (cudaMemcpyFromSymbol(&v, g_roi_device_status, sizeof(v)) != cudaSuccess) return ROI_ERR_CUDA;
  if (v != 0) {
    const unsigned int zero = 0;
    cudaMemcpyToSymbol(g_roi_device_status, &zero, sizeof(zero));
    return ROI_ERR_TIMEOUT;
  }
  return ROI_OK;
}

const char* roi_status_string(roi_status s) {
  switch (s) {
    case ROI_OK: return "ok";
    case ROI_ERR_NULL: return "a required pointer is NULL (or W / out_Wpruned given without the other)";
    case ROI_ERR_SHAPE: return "bad shape: rows < 0, cols <= 0, cols % M != 0, size overflow or row_offset < 0";
    case ROI_ERR_NM: return "need 1 <= N < M <= 32";
    case ROI_ERR_TAU: return "tau and lambda must be finite and > 0";
    case ROI_ERR_ALIGN: return "tensor pointers must be 16-byte aligned";
    case ROI_ERR_ALIAS: return "an output overlaps an input or another output";
    case ROI_ERR_CUDA: return "CUDA error while launching";
    case ROI_ERR_TIMEOUT: return "a kernel gave up waiting on its own copies";
    case ROI_ERR_OPT: return "bad optimizer settings: need lr, weight_decay >= 0 finite, 0 <= beta < 1, eps > 0, t >= 1";
  }
  return "unknown status";
}

uint64_t roi_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

}  // extern "C"
