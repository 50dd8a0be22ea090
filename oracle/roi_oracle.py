"""Plain CPU oracle for the RoI mask-learning hot path.

TEST INFRASTRUCTURE ONLY.  This module is the slow, obviously-correct statement
of what the GPU library computes.  Only ``tests/``, ``__graft_entry__.smoke()``
and the ``cpu_baseline`` / reference legs of ``bench.py`` may import it; the
product path (``paper_2608_23048_gb300`` and its CUDA library) never does, and the
two share no code.

Paper: "Reservoir of Importance: Learning Semi-Structured Sparsity with
Differentiable Subset Sampling" (RoI).  Every function below names the passage it
follows.  Arithmetic is float64 by default; ``dtype=np.float32`` runs the same
steps with every intermediate rounded to float32 ("the oracle run in fp32"):
+, -, *, / are IEEE float32 operations and exp / log are evaluated in float64 and
rounded once to float32 (i.e. correctly rounded elementary functions).

Data layout (the same contract the library implements):
  * logits phi: float32 [rows, cols]; groups are M contiguous elements along cols
    (cols % M == 0), i.e. consecutive M-chunks of the row-major flat array.
  * W, dWm, Wm, dW: bfloat16 carried as raw uint16 bit patterns (numpy has no
    bfloat16 type).
  * hard mask: flat bit array, uint32 words, bit b of word w = element 32*w + b.

Readings of the paper taken here:
  * Algorithm 1's candidate loop runs over the M members of a group and its
    output S has M entries; the number of relaxation steps is N (the paper's K).
  * lambda enters as kappa = phi / lambda + g (Sec. 4.2.3, Gumbel-top-K on the
    scaled logits phi / lambda); tau divides the adjusted keys in every softmax.
  * log(1 - mu_j) is taken exactly, as LSE_{i != j}(z_i) - LSE_i(z_i) with
    z = alpha / tau; no epsilon clamp.
  * U(0,1) comes from Philox-4x32-10 word x as u = ((x >> 9) + 1/2) * 2^-23.
  * Hard top-N: NaN keys rank as -inf; equal keys: lower index wins.
  * Masked weight: the product W * S is rounded to float32, then to bfloat16 with
    round-to-nearest-even.
"""
from __future__ import annotations

import numpy as np

from .philox import noise_words


# --------------------------------------------------------------------------
# precision policy
# --------------------------------------------------------------------------
class _Arith:
    """float64, or float32 with correctly rounded exp/log."""

    def __init__(self, dtype):
        self.dt = np.dtype(dtype)
        if self.dt not in (np.dtype(np.float64), np.dtype(np.float32)):
            raise ValueError("oracle dtype must be float64 or float32")

    def cast(self, x):
        return np.asarray(x, dtype=np.float64).astype(self.dt) if self.dt == np.float32 \
            else np.asarray(x, dtype=np.float64)

    def exp(self, x):
        with np.errstate(over="ignore", under="ignore"):
            return np.exp(np.asarray(x, dtype=np.float64)).astype(self.dt)

    def log(self, x):
        with np.errstate(divide="ignore", invalid="ignore"):
            return np.log(np.asarray(x, dtype=np.float64)).astype(self.dt)


def _lse(ar: _Arith, z: np.ndarray, axis: int = -1) -> np.ndarray:
    """log-sum-exp along ``axis``: m + log(sum exp(z - m)), m = max (NaN propagates)."""
    m = np.max(z, axis=axis, keepdims=True)
    finite_m = np.where(np.isfinite(m), m, ar.cast(0.0))
    with np.errstate(invalid="ignore"):
        s = np.sum(ar.exp(z - finite_m), axis=axis, keepdims=True, dtype=ar.dt)
    out = finite_m + ar.log(s)
    # all -inf -> -inf; a +inf member -> +inf
    out = np.where(np.isneginf(m), m, out)
    out = np.where(np.isposinf(m), m, out)
    return np.squeeze(out, axis=axis)


def _lse_excluding_each(ar: _Arith, z: np.ndarray) -> np.ndarray:
    """[G, M] -> [G, M]: entry j is LSE over the group's members i != j."""
    G, M = z.shape
    zz = np.broadcast_to(z[:, None, :], (G, M, M)).copy()
    idx = np.arange(M)
    zz[:, idx, idx] = -np.inf
    return _lse(ar, zz, axis=-1)


# --------------------------------------------------------------------------
# noise (Algorithm 1, Gumbel lines; Sec. 3.2 Eq. 2; Sec. 4.2.2 Eq. 10)
# --------------------------------------------------------------------------
def uniform_from_word(x: np.ndarray) -> np.ndarray:
    """u = ((x >> 9) + 1/2) * 2^-23, exactly; u lies in the open interval (0, 1)."""
    k = (np.asarray(x, dtype=np.uint32) >> np.uint32(9)).astype(np.float64)
    return (2.0 * k + 1.0) * 2.0 ** -24


def gumbel_from_uniform(u: np.ndarray, dtype=np.float64) -> np.ndarray:
    """g = -log(-log u), Algorithm 1 (Gumbel noise line)."""
    ar = _Arith(dtype)
    e = -ar.log(ar.cast(u))
    return -ar.log(e)


def element_indices(rows: int, cols: int, row_offset: int = 0) -> np.ndarray:
    """Tensor-global flat element index e = (row_offset + r) * cols + c."""
    return np.arange(rows * cols, dtype=np.uint64) + np.uint64(row_offset * cols)


def gumbel_noise(seed: int, step: int, tensor_id: int, rows: int, cols: int,
                 row_offset: int = 0, dtype=np.float64) -> np.ndarray:
    """Gumbel noise for every element of a [rows, cols] tensor (flat)."""
    x = noise_words(seed, step, tensor_id, element_indices(rows, cols, row_offset))
    return gumbel_from_uniform(uniform_from_word(x), dtype)


def perturbed_keys(phi: np.ndarray, g: np.ndarray, lam: float = 1.0, dtype=np.float64):
    """kappa = phi / lambda + g  (Eq. 10 on the scaled logits of Sec. 4.2.3)."""
    ar = _Arith(dtype)
    return ar.cast(ar.cast(phi) / ar.cast(lam)) + ar.cast(g)


# --------------------------------------------------------------------------
# relaxed top-N (Sec. 3.2 Eq. 3-4; Sec. 4.2.2 Eq. 11-12; Algorithm 1)
# --------------------------------------------------------------------------
def relaxed_topn(kappa: np.ndarray, N: int, tau: float, dtype=np.float64,
                 return_history: bool = False):
    """Soft N-hot vector S = sum_k mu^(k) for every group (rows of ``kappa``).

    alpha^(1) = kappa; for k = 1..N: mu^(k) = softmax(alpha^(k) / tau),
    alpha^(k+1) = alpha^(k) + log(1 - mu^(k)).  The last update is not needed
    and is not formed.
    """
    ar = _Arith(dtype)
    alpha = ar.cast(kappa)
    tau = ar.cast(tau)
    S = np.zeros_like(alpha)
    hist = []
    for k in range(N):
        z = alpha / tau
        L = _lse(ar, z)[:, None]
        mu = ar.exp(z - L)
        S = S + mu
        hist.append((z, mu))
        if k + 1 < N:
            ell = _lse_excluding_each(ar, z) - L      # log(1 - mu), exactly
            alpha = alpha + ell
    return (S, hist) if return_history else S


def relaxed_topn_backward(hist, c: np.ndarray, tau: float, dtype=np.float64):
    """Reverse-mode derivative of S w.r.t. kappa, contracted with c = dL/dS.

    Hand-derived from the recursion of ``relaxed_topn``.  With z = alpha / tau,
    mu = softmax(z), l_i = LSE_{j != i} z_j - LSE_j z_j:
        d mu_i / d z_l = mu_i (delta_il - mu_l)
        d l_i  / d z_l = [l != i] nu^(-i)_l - mu_l,
        nu^(-i)_l = exp(z_l - LSE_{j != i} z_j)   (softmax with i removed).
    Sweeping k = N..1 with b = dL/d alpha^(k+1) (zero at k = N):
        abar = b + (1/tau) [ mu (c - <c, mu>) + J^T b ],
        (J^T b)_l = sum_{i != l} b_i nu^(-i)_l - mu_l sum_i b_i.
    Returns dL/d kappa.
    """
    ar = _Arith(dtype)
    c = ar.cast(c)
    tau = ar.cast(tau)
    b = np.zeros_like(c)
    for z, mu in reversed(hist):
        cmu = np.sum(c * mu, axis=-1, keepdims=True, dtype=ar.dt)
        gz = mu * (c - cmu)
        lse_ex = _lse_excluding_each(ar, z)                       # [G, M] over i
        G, M = z.shape
        nu = ar.exp(z[:, None, :] - lse_ex[:, :, None])           # [G, i, l]
        idx = np.arange(M)
        nu[:, idx, idx] = 0.0
        jtb = np.einsum("gi,gil->gl", b, nu) - mu * np.sum(b, axis=-1, keepdims=True,
                                                           dtype=ar.dt)
        gz = gz + ar.cast(jtb)
        b = b + gz / tau
    return b


# --------------------------------------------------------------------------
# hard top-N (Sec. 3.2, Gumbel-top-K; Sec. 4.1 N-hot masks)
# --------------------------------------------------------------------------
def hard_topn(keys: np.ndarray, N: int) -> np.ndarray:
    """Boolean N-hot mask of the N largest keys per group (rows of ``keys``).

    NaN ranks as -inf; among equal keys the lower index wins.
    """
    k = np.where(np.isnan(keys), -np.inf, keys).astype(np.float64)
    order = np.argsort(-k, axis=-1, kind="stable")
    mask = np.zeros(k.shape, dtype=bool)
    np.put_along_axis(mask, order[:, :N], True, axis=-1)
    return mask


def topn_key_gap(keys: np.ndarray, N: int) -> np.ndarray:
    """Per group: (N-th largest key) - ((N+1)-th largest key), in float64."""
    k = np.sort(np.where(np.isnan(keys), -np.inf, keys).astype(np.float64), axis=-1)[:, ::-1]
    with np.errstate(invalid="ignore"):
        return k[:, N - 1] - k[:, N]


def pack_bits(mask_flat: np.ndarray) -> np.ndarray:
    """Flat boolean mask -> uint32 words; bit b of word w is element 32*w + b."""
    m = np.asarray(mask_flat, dtype=bool).ravel()
    nw = (m.size + 31) // 32
    padded = np.zeros(nw * 32, dtype=np.uint64)
    padded[: m.size] = m
    weights = np.uint64(1) << np.arange(32, dtype=np.uint64)
    return (padded.reshape(nw, 32) * weights).sum(axis=1).astype(np.uint32)


def unpack_bits(words: np.ndarray, n: int) -> np.ndarray:
    w = np.asarray(words, dtype=np.uint32).astype(np.uint64)
    bits = (w[:, None] >> np.arange(32, dtype=np.uint64)) & np.uint64(1)
    return bits.ravel()[:n].astype(bool)


# --------------------------------------------------------------------------
# bfloat16 (storage type of W, dWm, Wm, dW)
# --------------------------------------------------------------------------
def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def f32_to_bf16_rne(x: np.ndarray) -> np.ndarray:
    """float32 -> bfloat16 bits, round to nearest, ties to even; NaN stays NaN."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    b = x.view(np.uint32).astype(np.uint64)
    lsb = (b >> np.uint64(16)) & np.uint64(1)
    r = ((b + np.uint64(0x7FFF) + lsb) >> np.uint64(16)).astype(np.uint16)
    nan = np.isnan(x)
    r[nan] = ((b[nan] >> np.uint64(16)) | np.uint64(0x40)).astype(np.uint16)
    return r


def bf16_product(a_bits: np.ndarray, s: np.ndarray) -> np.ndarray:
    """bf16(RN_f32(float(a) * s)): the masked-weight product (Eq. 5, W (.) M)."""
    with np.errstate(over="ignore", invalid="ignore"):
        p = (bf16_to_f32(a_bits).astype(np.float64) * np.asarray(s, dtype=np.float64))
    return f32_to_bf16_rne(p.astype(np.float32))


# --------------------------------------------------------------------------
# the three library calls
# --------------------------------------------------------------------------
def _grouped(a: np.ndarray, M: int) -> np.ndarray:
    return np.asarray(a).reshape(-1, M)


def _check(rows, cols, N, M):
    if not (1 <= N < M <= 32):
        raise ValueError("need 1 <= N < M <= 32")
    if cols % M or rows < 0 or cols <= 0:
        raise ValueError("cols must be a positive multiple of M")


def mask_fwd(logits, W_bits, N, M, tau, seed, step, tensor_id=0, lam=1.0,
             row_offset=0, dtype=np.float64):
    """Forward of the mask op for one [rows, cols] tensor.

    Returns a dict with the perturbed keys, the soft mask S (Sec. 4.2.2), the hard
    N-hot mask (Gumbel-top-N of the same keys), its packed bits, and the masked
    weights Wm = bf16(W * S) (Eq. 5 with the relaxed mask).
    """
    logits = np.asarray(logits, dtype=np.float32)
    rows, cols = logits.shape
    _check(rows, cols, N, M)
    g = gumbel_noise(seed, step, tensor_id, rows, cols, row_offset, dtype)
    kappa = perturbed_keys(logits.ravel(), g, lam, dtype)
    kg = _grouped(kappa, M)
    S = relaxed_topn(kg, N, tau, dtype)
    hard = hard_topn(kg, N)
    Wm = bf16_product(np.asarray(W_bits).ravel(), S.ravel())
    return {
        "keys": kappa.reshape(rows, cols),
        "soft": S.reshape(rows, cols),
        "hard": hard.reshape(rows, cols),
        "hard_bits": pack_bits(hard.ravel()),
        "Wm": Wm.reshape(rows, cols),
    }


def mask_bwd(logits, W_bits, dWm_bits, N, M, tau, seed, step, tensor_id=0, lam=1.0,
             row_offset=0, dtype=np.float64):
    """Backward of the mask op: dL/dphi from dL/dWm, with the noise regenerated.

    dL/dS = dWm * W (the derivative of Wm = W * S with respect to S, rounding of Wm
    treated as identity); dL/dphi = (dL/dkappa) / lambda; dW = bf16(dWm * S).
    """
    ar = _Arith(dtype)
    logits = np.asarray(logits, dtype=np.float32)
    rows, cols = logits.shape
    _check(rows, cols, N, M)
    g = gumbel_noise(seed, step, tensor_id, rows, cols, row_offset, dtype)
    kappa = perturbed_keys(logits.ravel(), g, lam, dtype)
    S, hist = relaxed_topn(_grouped(kappa, M), N, tau, dtype, return_history=True)
    c = ar.cast(bf16_to_f32(np.asarray(dWm_bits).ravel())) * ar.cast(bf16_to_f32(np.asarray(W_bits).ravel()))
    dkappa = relaxed_topn_backward(hist, _grouped(c, M), tau, dtype)
    dphi = dkappa / ar.cast(lam)
    dW = bf16_product(np.asarray(dWm_bits).ravel(), S.ravel())
    return {
        "dlogits": dphi.reshape(rows, cols),
        "dW": dW.reshape(rows, cols),
        "soft": S.reshape(rows, cols),
    }


def hard_mask_export(logits, N, M, W_bits=None):
    """Deployment mask: argtop_N(phi) per group, i.e. the lambda -> 0 limit of the
    Gumbel-top-N sampler (Sec. 4.2.3 anneals lambda towards 0) and the most probable
    subset of Eq. 8.  Optional pruned weights: kept entries copied, pruned set to +0.
    """
    logits = np.asarray(logits, dtype=np.float32)
    rows, cols = logits.shape
    _check(rows, cols, N, M)
    hard = hard_topn(_grouped(logits.ravel(), M), N).ravel()
    out = {"hard": hard.reshape(rows, cols), "hard_bits": pack_bits(hard)}
    if W_bits is not None:
        wb = np.asarray(W_bits, dtype=np.uint16).ravel()
        out["W_pruned"] = np.where(hard, wb, np.uint16(0)).reshape(rows, cols)
    return out


def mask_fwd_st(logits, W_bits, N, M, tau, seed, step, tensor_id=0, lam=1.0,
                row_offset=0, dtype=np.float64):
    """Forward of the straight-through Gumbel-top-N variant (Appendix, "Comparison
    with Straight-Through Gumbel-Top-K"): the forward applies the discrete mask,
    argtop_N of the Gumbel-perturbed keys, so Wm = W where the hard mask is set and
    +0 elsewhere (the bf16 bits of W copied); S is still formed (the backward runs
    through it) and is returned like the soft forward's."""
    out = mask_fwd(logits, W_bits, N, M, tau, seed, step, tensor_id, lam, row_offset, dtype)
    wb = np.asarray(W_bits, dtype=np.uint16).reshape(out["hard"].shape)
    out["Wm"] = np.where(out["hard"], wb, np.uint16(0))
    return out


def mask_bwd_st(logits, W_bits, dWm_bits, hard_bits, N, M, tau, seed, step, tensor_id=0,
                lam=1.0, row_offset=0, dtype=np.float64):
    """Backward of the straight-through variant (same appendix): the logit gradient
    passes through the continuous relaxation exactly as in the soft method
    (dL/dS = dWm * W), while the weight gradient follows the forward's actual
    product W * hard: dW = dWm where the forward's hard mask is set, +0 elsewhere.
    `hard_bits` are the forward's packed hard-mask words."""
    out = mask_bwd(logits, W_bits, dWm_bits, N, M, tau, seed, step, tensor_id, lam, row_offset, dtype)
    rows, cols = np.asarray(logits).shape
    hard = unpack_bits(np.asarray(hard_bits, dtype=np.uint32), rows * cols).reshape(rows, cols)
    db = np.asarray(dWm_bits, dtype=np.uint16).reshape(rows, cols)
    out["dW"] = np.where(hard, db, np.uint16(0))
    return out


def export_compressed_2of4(logits, W_bits):
    """2:4 deployment export in compressed form (the semi-structured layout that
    sparse tensor cores consume, Sec. 1 and the Throughput appendix): per group of
    four, the deployment mask argtop_2(phi) (ties: lower index) selects two
    members, and
      * values[g] = the two kept weights, in index order  -> bf16 [rows, cols/2]
      * meta: the two in-group indices i0 < i1 as a 4-bit code i0 | i1 << 2, eight
        groups per uint32 word, group g in bits 4*(g % 8) .. 4*(g % 8) + 3 of word
        g // 8 (groups in row-major order)              -> uint32 [rows*cols/32]
    """
    logits = np.asarray(logits, dtype=np.float32)
    rows, cols = logits.shape
    _check(rows, cols, 2, 4)
    if (rows * cols) % 32:
        raise ValueError("rows * cols must be a multiple of 32 (eight groups per metadata word)")
    hard = hard_topn(_grouped(logits.ravel(), 4), 2)                 # [G, 4] bool
    G = hard.shape[0]
    wb = np.asarray(W_bits, dtype=np.uint16).reshape(G, 4)
    values = np.empty((G, 2), dtype=np.uint16)
    codes = np.empty(G, dtype=np.uint32)
    for g in range(G):                                               # plain loop: obviously correct
        idx = [j for j in range(4) if hard[g, j]]
        values[g] = wb[g, idx]
        codes[g] = idx[0] | (idx[1] << 2)
    meta = np.zeros(G // 8, dtype=np.uint32)
    for g in range(G):
        meta[g // 8] |= codes[g] << np.uint32(4 * (g % 8))
    return {"values": values.reshape(rows, cols // 2), "meta": meta, "hard": hard.reshape(rows, cols)}


def decompress_2of4(values, meta, rows, cols):
    """Inverse of export_compressed_2of4's layout: dense bf16 bits with the kept
    values at their indices and +0 elsewhere."""
    G = rows * cols // 4
    v = np.asarray(values, dtype=np.uint16).reshape(G, 2)
    m = np.asarray(meta, dtype=np.uint32)
    dense = np.zeros((G, 4), dtype=np.uint16)
    for g in range(G):
        code = (int(m[g // 8]) >> (4 * (g % 8))) & 0xF
        dense[g, code & 3] = v[g, 0]
        dense[g, code >> 2] = v[g, 1]
    return dense.reshape(rows, cols)


def anneal(init: float, end: float, t, T_anneal: float):
    """Exponential annealing of tau and lambda (Sec. 4.2.3, Eq. 13):
    x_t = max(x_end, x_init * (x_end / x_init) ** (t / T_anneal))."""
    t = np.asarray(t, dtype=np.float64)
    return np.maximum(end, init * (end / init) ** (t / T_anneal))


def adamw_step(phi, g, m, v, lr, beta1, beta2, eps, weight_decay, t, dtype=np.float64):
    """One AdamW step on the logits (decoupled weight decay; the optimizer and its
    hyper-parameters of Sec. 5.1 and the hyper-parameter table: beta1 = 0.9,
    beta2 = 0.95, weight decay 0.05), written out from its definition, in the
    order the definition states it:
        phi   <- phi * (1 - lr * weight_decay)          (decoupled weight decay)
        m     <- beta1 m + (1 - beta1) g
        v     <- beta2 v + (1 - beta2) g^2
        m_hat  = m / (1 - beta1^t),   v_hat = v / (1 - beta2^t)
        phi   <- phi - lr * m_hat / (sqrt(v_hat) + eps)
    t is the 1-based step count; the bias-correction denominators 1 - beta^t are
    scalars formed in float64.  Returns (phi, m, v)."""
    ar = _Arith(dtype)
    phi, g, m, v = (ar.cast(np.asarray(x, dtype=np.float64)) for x in (phi, g, m, v))
    c = lambda x: ar.cast(np.float64(x))
    phi = phi * (c(1.0) - c(lr) * c(weight_decay))
    m = c(beta1) * m + (c(1.0) - c(beta1)) * g
    v = c(beta2) * v + (c(1.0) - c(beta2)) * (g * g)
    m_hat = m / c(1.0 - beta1 ** t)
    v_hat = v / c(1.0 - beta2 ** t)
    phi = phi - c(lr) * m_hat / (ar.cast(np.sqrt(v_hat)) + c(eps))
    return phi, m, v


def masked_linear_fwd(X_bits, logits, W_bits, N, M, tau, seed, step, tensor_id=0, lam=1.0,
                      row_offset=0, dtype=np.float64):
    """The layer's product with the masked weights (Eq. 5: the linear layer uses
    W (.) S in place of W): Y[t, r] = sum_c X[t, c] * Wm[r, c], where Wm is
    mask_fwd's bfloat16 Wm for the same arguments.  X is bfloat16 [T, cols]; the
    sum of the decoded values is taken in float64 (a plain matrix product; the
    products of two bfloat16 values are exact there).

    Returns Y [T, rows] (float64), the Wm bits it used, and |X| |Wm|^T, the
    scale of the rounding error of any other evaluation order."""
    f = mask_fwd(logits, W_bits, N, M, tau, seed, step, tensor_id, lam, row_offset, dtype)
    Wm = bf16_to_f32(f["Wm"]).astype(np.float64)
    X = bf16_to_f32(np.asarray(X_bits)).astype(np.float64)
    return {"Y": X @ Wm.T, "Wm": f["Wm"], "abs": np.abs(X) @ np.abs(Wm).T}
