/*
 * roi.h - C ABI of the RoI mask-learning library (libroi.so, sm_103a).
 *
 * "Reservoir of Importance" learns a semi-structured N:M sparsity mask by
 * giving every weight one logit phi and sampling N of the M weights of each
 * group without replacement (weighted reservoir sampling, Sec. 3.1 Eq. 1;
 * Gumbel-top-K, Sec. 3.2).  Training uses the differentiable relaxation of
 * Sec. 3.2 Eq. 3-4 / Sec. 4.2.2 Eq. 11-12 / Algorithm 1:
 *
 *     kappa    = phi / lambda + g,  g = -log(-log u),  u ~ U(0,1)   (Eq. 10, Sec. 4.2.3)
 *     alpha(1) = kappa
 *     mu(k)    = softmax(alpha(k) / tau)                              (Eq. 12)
 *     alpha(k+1) = alpha(k) + log(1 - mu(k))                          (Eq. 11)
 *     S        = sum_{k=1..N} mu(k)          (soft N-hot mask)
 *     Wm       = W (.) S                     (masked weights, Eq. 5)
 *
 * Conventions shared by every call
 *  - Tensors are row-major [rows, cols] (nn.Linear layout [out, in]); a group is
 *    M contiguous elements along cols, so cols % M == 0.  Flat element index
 *    e = (row_offset + r) * cols + c.
 *  - bfloat16 tensors are passed as their 16-bit patterns (roi_bf16).
 *  - Every tensor pointer is caller-owned DEVICE memory, 16-byte aligned, and
 *    must not alias any other tensor of the same call.  The library allocates
 *    no memory.  With rows == 0 nothing is read or written and tensor pointers
 *    may be NULL.
 *  - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *    stream).  Arguments are validated on the host before anything is
 *    launched; on any non-OK return nothing was launched and nothing written.
 *  - Noise: u comes from Philox-4x32-10 (Salmon et al., SC'11) with
 *    key = (seed & 0xffffffff, seed >> 32) and
 *    counter = (q & 0xffffffff, q >> 32, step, tensor_id), q = e >> 2; element e
 *    takes output word e & 3 as x and u = ((x >> 9) + 0.5) * 2^-23.  Noise is
 *    a pure function of (seed, step, tensor_id, e): it is regenerated, never
 *    stored, so the backward call reproduces the forward's sample exactly and a
 *    row-sliced call (row_offset) reproduces the unsliced one.
 *  - Hard mask: flat bit array of ceil(rows*cols/32) uint32 words; bit b of word
 *    w is element 32*w + b (bits past the last element are 0).  It is the
 *    Gumbel-top-N of the same keys: the N largest kappa of each group, NaN
 *    ranked as -inf, equal keys resolved towards the lower index.
 */
#ifndef ROI_H_
#define ROI_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t roi_bf16; /* bfloat16 bit pattern */

typedef enum {
    ROI_OK = 0,
    ROI_ERR_NULL = 1,      /* a required pointer is NULL                                */
    ROI_ERR_SHAPE = 2,     /* rows < 0, cols <= 0, cols % M != 0, or row_offset < 0      */
    ROI_ERR_NM = 3,        /* not 1 <= N < M <= 32                                       */
    ROI_ERR_TAU = 4,       /* tau or lambda not finite or not > 0                        */
    ROI_ERR_ALIGN = 5,     /* a tensor pointer is not 16-byte aligned                    */
    ROI_ERR_ALIAS = 6,     /* an output overlaps an input or another output              */
    ROI_ERR_CUDA = 7,      /* launch failed (cudaGetLastError after the launch)          */
    ROI_ERR_TIMEOUT = 8,   /* a kernel gave up waiting on its own copies (see below)     */
    ROI_ERR_OPT = 9        /* bad optimizer settings (roi_mask_bwd_adamw)                */
} roi_status;

/* Noise state of one call (Sec. 4.2.3 sampling temperature included).
 *  seed, step, tensor_id: Philox key and counter words (see above); tensor_id
 *    keeps layers that share (seed, step) from sharing noise.
 *  lambda: sampling temperature, > 0; Gumbel-top-N runs on phi / lambda.
 *  row_offset: index of this call's first row within the full tensor, >= 0. */
typedef struct {
    uint64_t seed;
    uint32_t step;
    uint32_t tensor_id;
    float lambda;
    int64_t row_offset;
} roi_noise_state;

/* Forward of the mask op (Sec. 4.2.2 relaxation; Eq. 5 mask application;
 * Algorithm 1).  Short form: lambda = 1, tensor_id = 0, row_offset = 0.
 *  logits  [rows, cols] float32          phi
 *  W       [rows, cols] bf16             frozen weights
 *  N, M    keep N of every M (1 <= N < M <= 32, cols % M == 0)
 *  tau     relaxation temperature, finite, > 0
 *  out_Wm  [rows, cols] bf16             bf16_rne(float(W) * S), product in fp32
 *  out_soft[rows, cols] float32, nullable  S
 *  out_hard[ceil(rows*cols/32)] uint32, nullable  Gumbel-top-N hard mask
 *  stream  cudaStream_t                                                    */
roi_status roi_mask_fwd(const float* logits, const roi_bf16* W, int N, int M, float tau,
                        uint64_t seed, uint32_t step, int64_t rows, int64_t cols,
                        roi_bf16* out_Wm, float* out_soft, uint32_t* out_hard, void* stream);

/* Forward, full noise state (st is read on the host during the call). */
roi_status roi_mask_fwd_ex(const float* logits, const roi_bf16* W, int N, int M, float tau,
                           const roi_noise_state* st, int64_t rows, int64_t cols,
                           roi_bf16* out_Wm, float* out_soft, uint32_t* out_hard, void* stream);

/* Many tensors in one call: the same results, bit for bit, as roi_mask_fwd_ex /
 * roi_mask_bwd for each item in turn, with one (N, M, tau) and one stream for all.
 * Each item is validated as the single call would be; in addition no output may
 * overlap any input or output of any item (ROI_ERR_ALIAS), so the items are
 * independent.  That lets the library chain their launches with programmatic
 * dependent launch (for (N, M) = (2, 4), (4, 8), (2, 8), (8, 16), (16, 32)): a tensor's kernel may start
 * on the SMs that the previous one frees as it drains, hiding the launch gap and
 * the ragged last wave of small tensors, while each launch still completes after
 * its predecessor, so the work queued after the call sees every item done.  For
 * (2, 4), (4, 8) and (2, 8), runs of consecutive items small enough that each would
 * give an SM fewer than 12 tiles of work share one launch (runs of at least 8 items;
 * 2 for roi_mask_bwd_batch at tau >= 0.075).  Items with rows == 0 are skipped.
 * `items` is host memory, read during the call. */
typedef struct {
    const float* logits;  /* [rows, cols] */
    const roi_bf16* W;    /* [rows, cols] */
    roi_bf16* out_Wm;     /* [rows, cols] */
    float* out_soft;      /* nullable, [rows, cols] */
    uint32_t* out_hard;   /* nullable, [ceil(rows*cols/32)] */
    int64_t rows, cols;
    roi_noise_state st;
} roi_fwd_item;
typedef struct {
    const float* logits;  /* [rows, cols] */
    const roi_bf16* W;    /* [rows, cols] */
    const roi_bf16* dWm;  /* [rows, cols] */
    float* out_dlogits;   /* [rows, cols], overwritten */
    roi_bf16* out_dW;     /* nullable, [rows, cols] */
    int64_t rows, cols;
    roi_noise_state st;
} roi_bwd_item;
roi_status roi_mask_fwd_batch(const roi_fwd_item* items, int count, int N, int M, float tau, void* stream);
roi_status roi_mask_bwd_batch(const roi_bwd_item* items, int count, int N, int M, float tau, void* stream);

/* Backward of the mask op: turns the upstream gradient of the masked weights
 * into logit gradients through the relaxation (Sec. 3.2: the map from logits
 * to the soft N-hot vector is differentiable).  The noise is regenerated from
 * st, so st must equal the forward's.
 *  dL/dS       = float(dWm) * float(W)   (rounding of Wm passes the gradient)
 *  out_dlogits [rows, cols] float32      dL/dphi = (dL/dkappa) / lambda; OVERWRITTEN
 *  out_dW      [rows, cols] bf16, nullable  bf16_rne(float(dWm) * S)          */
roi_status roi_mask_bwd(const float* logits, const roi_bf16* W, const roi_noise_state* st,
                        int N, int M, const roi_bf16* dWm, float tau, int64_t rows, int64_t cols,
                        float* out_dlogits, roi_bf16* out_dW, void* stream);

/* Straight-through Gumbel-top-N variant (Appendix, "Comparison with
 * Straight-Through Gumbel-Top-K": the forward applies the discrete mask, the
 * backward propagates through the continuous relaxation).
 *  roi_mask_fwd_st: as roi_mask_fwd_ex, except out_Wm copies the bf16 bits of W
 *    where the hard mask (Gumbel-top-N of the keys, as out_hard) is set and
 *    writes +0 elsewhere.  out_soft, when given, is the relaxation's S.
 *  roi_mask_bwd_st: as roi_mask_bwd (out_dlogits identical: dL/dS = dWm * W
 *    through the relaxation), except out_dW = dWm where the forward's hard mask
 *    is set, +0 elsewhere, the gradient of the forward's product W * hard.
 *    hard: the forward's out_hard words ([ceil(rows*cols/32)] uint32, same
 *    noise state); required when out_dW is given, read only then. */
roi_status roi_mask_fwd_st(const float* logits, const roi_bf16* W, int N, int M, float tau,
                           const roi_noise_state* st, int64_t rows, int64_t cols,
                           roi_bf16* out_Wm, float* out_soft, uint32_t* out_hard, void* stream);
roi_status roi_mask_bwd_st(const float* logits, const roi_bf16* W, const roi_noise_state* st,
                           int N, int M, const roi_bf16* dWm, const uint32_t* hard, float tau,
                           int64_t rows, int64_t cols, float* out_dlogits, roi_bf16* out_dW,
                           void* stream);

/* Settings of one AdamW step on the logits (the paper's optimizer, hyper-parameter
 * table: beta1 = 0.9, beta2 = 0.95, weight decay 0.05, lr 1e-3 decaying to 1e-4).
 *  lr, weight_decay: finite, >= 0; beta1, beta2 in [0, 1); eps > 0 (1e-8);
 *  t: 1-based count of steps taken, this one included (bias correction). */
typedef struct {
    float lr;
    float beta1;
    float beta2;
    float eps;
    float weight_decay;
    uint32_t t;
} roi_adamw;

/* Backward fused with the logits' optimizer step: the logit gradient g of
 * roi_mask_bwd is formed in registers and used at once for one AdamW step
 * (decoupled weight decay):
 *     phi <- phi (1 - lr wd);  m <- b1 m + (1 - b1) g;  v <- b2 v + (1 - b2) g^2;
 *     phi <- phi - (step m) / (sqrt(v) r + eps),
 *     step = lr / (1 - b1^t),  r = 1 / sqrt(1 - b2^t)   (scalars, on the host in double)
 * in float32, every operation rounded (divide and square root correctly rounded).
 * Unlike the other calls, logits is read AND written: it holds phi_t on entry
 * and phi_{t+1} on return (elements not shared with any other tensor).
 *  m, v         [rows, cols] float32, the optimizer moments, updated in place
 *  out_dlogits  nullable: the gradient g as well
 *  out_dW       nullable: bf16_rne(float(dWm) * S), as roi_mask_bwd
 * The step needs the gradient of this mask op alone (one use of phi per step;
 * a data-parallel run reduces gradients first and uses roi_mask_bwd instead).
 * ROI_ERR_OPT for settings outside the ranges above. */
roi_status roi_mask_bwd_adamw(float* logits, const roi_bf16* W, const roi_noise_state* st, int N, int M,
                              const roi_bf16* dWm, float tau, int64_t rows, int64_t cols,
                              float* m, float* v, const roi_adamw* opt,
                              float* out_dlogits, roi_bf16* out_dW, void* stream);

/* roi_mask_bwd_adamw for many tensors in one call (one optimizer step, one
 * (N, M, tau), one stream): the same results, bit for bit, as the single call per
 * item, with the launches chained as in roi_mask_bwd_batch.  Each item is
 * validated as the single call; no output (logits, m, v, gradient, dW) may
 * overlap any other range of any item (ROI_ERR_ALIAS). */
typedef struct {
    float* logits;        /* [rows, cols], phi_t on entry, phi_{t+1} on return */
    const roi_bf16* W;    /* [rows, cols] */
    const roi_bf16* dWm;  /* [rows, cols] */
    float* m;             /* [rows, cols], updated */
    float* v;             /* [rows, cols], updated */
    float* out_dlogits;   /* nullable, [rows, cols] */
    roi_bf16* out_dW;     /* nullable, [rows, cols] */
    int64_t rows, cols;
    roi_noise_state st;
} roi_adamw_item;
roi_status roi_mask_bwd_adamw_batch(const roi_adamw_item* items, int count, int N, int M, float tau,
                                    const roi_adamw* opt, void* stream);

/* Exponential annealing of tau and lambda (Sec. 4.2.3, Eq. 13), on the host:
 *     x_t = max(x_end, x_init (x_end / x_init)^(t / T_anneal))
 * (the paper: tau 1.0 -> 0.05, lambda 1.0 -> 0.002, T_anneal = 1500).
 * init, end > 0; T_anneal == 0 gives end. */
float roi_anneal(float init, float end, uint32_t t, uint32_t T_anneal);

/* The straight-through pair for many tensors in one call (items as for
 * roi_mask_fwd_batch; for the backward, each item adds the forward's hard bits,
 * needed when out_dW is given): the same results, bit for bit, as the single
 * straight-through calls per item, launches chained as in roi_mask_fwd_batch. */
typedef struct {
    const float* logits;  /* [rows, cols] */
    const roi_bf16* W;    /* [rows, cols] */
    const roi_bf16* dWm;  /* [rows, cols] */
    const uint32_t* hard; /* the forward's out_hard; nullable when out_dW is NULL */
    float* out_dlogits;   /* [rows, cols], overwritten */
    roi_bf16* out_dW;     /* nullable, [rows, cols] */
    int64_t rows, cols;
    roi_noise_state st;
} roi_bwd_st_item;
roi_status roi_mask_fwd_st_batch(const roi_fwd_item* items, int count, int N, int M, float tau, void* stream);
roi_status roi_mask_bwd_st_batch(const roi_bwd_st_item* items, int count, int N, int M, float tau, void* stream);

/* Compressed 2:4 export for semi-structured sparse inference (the deployment the
 * paper targets, Sec. 1 and the Throughput appendix; it gives no format, so this
 * is the library's): the deployment mask argtop_2(phi) of every group of four
 * (as roi_hard_mask_export with N = 2, M = 4) and
 *  out_values [rows, cols/2] bf16   the two kept weights of each group, in index order
 *  out_meta   [rows*cols/32] uint32 per group the in-group indices i0 < i1 as the
 *             4-bit code i0 | i1 << 2; group g (row-major) in bits 4*(g%8) ..
 *             4*(g%8)+3 of word g/8.  This is the content of the sparse tensor
 *             cores' 2-bit index metadata without their hardware interleave.
 * cols % 4 == 0 and rows*cols % 32 == 0 (else ROI_ERR_SHAPE). */
roi_status roi_export_compressed_2of4(const float* logits, const roi_bf16* W, int64_t rows, int64_t cols,
                                      roi_bf16* out_values, uint32_t* out_meta, void* stream);

/* Masked linear forward: the layer's product with the masked weights (Eq. 5),
 *     Y[t, r] = sum_c X[t, c] Wm[r, c],   Wm = bf16_rne(float(W) * S),
 * where S is the relaxed mask of roi_mask_fwd_ex for the same (logits, W, N, M,
 * tau, st), bit for bit, formed in the prologue of a tensor-core GEMM: Wm is
 * never written to memory and the logits and W are read once.  The sum runs in
 * float32 on the tensor cores (products of bf16 exact, accumulation order the
 * hardware's), Y is float32.  If a kernel of the call gives up a wait
 * (roi_device_status then returns ROI_ERR_TIMEOUT), out_Y is undefined: the
 * split-K reduction still adds whatever partials the workspace holds.
 *  X             [T, cols] bf16, the layer's input tokens; 1 <= T <= 256
 *  out_Y         [T, rows] float32
 *  workspace     nullable caller-owned device memory for split-K partials
 *                (roi_masked_linear_workspace_size bytes; with less, or NULL,
 *                K is split less or not at all: same result, fewer CTAs).  The
 *                partials are added in a fixed order, so Y does not depend on
 *                the run.  Must not overlap the other tensors.
 * Supported (N, M): (2, 4), (4, 8), (2, 8) (else ROI_ERR_NM); cols % 8 == 0
 * and T <= 256 (else ROI_ERR_SHAPE).  With T == 0 or rows == 0 nothing is
 * read or written. */
roi_status roi_masked_linear_fwd(const roi_bf16* X, const float* logits, const roi_bf16* W, int N, int M,
                                 float tau, const roi_noise_state* st, int64_t T, int64_t rows, int64_t cols,
                                 float* out_Y, void* workspace, size_t workspace_bytes, void* stream);
/* Workspace bytes that let roi_masked_linear_fwd split K as far as it wants on
 * the current device (0: no split; also 0 for shapes the call rejects). */
size_t roi_masked_linear_workspace_size(int64_t T, int64_t rows, int64_t cols);

/* roi_masked_linear_fwd without a caller workspace.  The paper has no
 * counterpart: this is the library's own convenience for callers that have no
 * device allocator at hand.  The split-K partials go to one static device array
 * of ROI_LINEAR_SCRATCH_BYTES (16 MiB) per device instead, so the call allocates
 * nothing; arguments, results and errors are those of roi_masked_linear_fwd with
 * a workspace of roi_masked_linear_workspace_size bytes, except:
 *  - a call that needs more scratch than ROI_LINEAR_SCRATCH_BYTES returns
 *    ROI_ERR_SHAPE (e.g. a 3584 x 18944 layer at 256 tokens needs 18.4 MB on a
 *    152-SM GPU; pass a workspace to roi_masked_linear_fwd for those);
 *  - the array is shared by every call on the device and keeps the last call's
 *    partials; calls that overlap in time (other streams, other threads) race on
 *    it and must be serialised by the caller;
 *  - the first call on a device looks the array up (cudaGetSymbolAddress); when
 *    calls are to be recorded by stream capture, make one call before it.
 * Loading the library reserves the array on every device where its device code
 * is loaded, whether or not this call is ever made: ROI_LINEAR_SCRATCH_BYTES of
 * device memory per device until the process exits.  After a wait times out
 * (ROI_ERR_TIMEOUT) out_Y is undefined, and here its partials may be stale ones
 * of an earlier, unrelated call. */
#define ROI_LINEAR_SCRATCH_BYTES (16u << 20)
roi_status roi_masked_linear_fwd_noalloc(const roi_bf16* X, const float* logits, const roi_bf16* W, int N, int M,
                                         float tau, const roi_noise_state* st, int64_t T, int64_t rows, int64_t cols,
                                         float* out_Y, void* stream);

/* Deployment mask (Sec. 4.2.3 anneals lambda towards 0; the limit of
 * Gumbel-top-N is the deterministic top-N of phi, which is also the most
 * probable subset of Eq. 8): argtop_N(phi) per group, NaN ranked as -inf,
 * equal logits resolved towards the lower index.
 *  out_bits    [ceil(rows*cols/32)] uint32  (layout as out_hard)
 *  W, out_Wpruned  nullable together: kept weights copied bit-exactly, pruned
 *                  weights written as +0.0                                   */
roi_status roi_hard_mask_export(const float* logits, int N, int M, int64_t rows, int64_t cols,
                                uint32_t* out_bits, const roi_bf16* W, roi_bf16* out_Wpruned,
                                void* stream);

/* The noise of a call, materialised (for inspecting or reproducing a sample; the
 * mask calls never store it).  st->lambda is ignored; st->row_offset applies.
 *  roi_noise_words: out_words[rows*cols] uint32, the Philox word x_e of element e.
 *  roi_gumbel_noise: out_g[rows*cols] float32, g_e = -log(-log u_e) exactly as the
 *    mask kernels form it (Algorithm 1, Gumbel lines): -log u through a range
 *    reduction and the 2 atanh series (relative error about 2e-7), the outer log
 *    through the hardware log2 (absolute error about 1e-7). */
roi_status roi_noise_words(const roi_noise_state* st, int64_t rows, int64_t cols, uint32_t* out_words,
                           void* stream);
roi_status roi_gumbel_noise(const roi_noise_state* st, int64_t rows, int64_t cols, float* out_g, void* stream);

/* Device-side status.  The kernels wait on their own asynchronous copies with
 * a time limit (2 s unless roi_set_ring_wait_limit_ns set another); a kernel
 * that gives up records it in a status word and returns early, after its copies
 * in flight have landed (the outputs of that call are then undefined).  This call
 * synchronises `stream`, returns ROI_ERR_TIMEOUT if the word is set (and
 * clears it), ROI_ERR_CUDA on a CUDA error, else ROI_OK.
 * The word is one per device, shared by every stream, thread and call on it:
 * the return codes of the launching calls never see a timeout, and a timeout in
 * one caller's work is reported to whichever thread calls roi_device_status
 * first on that device (and cleared for the others). */
roi_status roi_device_status(void* stream);

/* Wall-time limit of a kernel's wait for a stage of its copy ring (the staged
 * tiles of logits and weights) on the current device, in ns; default
 * 2,000,000,000.  With 0 every such wait gives up at once, whether its stage has
 * landed or not; the tests use that to run the timeout path on valid copies.  The waits
 * with which a kernel that gave up drains its own copies in flight keep the fixed
 * 2 s limit.  Applies to kernels launched after the call returns (it is a
 * synchronous copy to device memory); ROI_ERR_CUDA if that copy fails. */
roi_status roi_set_ring_wait_limit_ns(uint64_t ns);

/* Static description of a status code. */
const char* roi_status_string(roi_status s);

/* Number of kernel launches the library has issued since load (host counter,
 * for benchmarking). */
uint64_t roi_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* ROI_H_ */
