"""Comparison rules between the CUDA library and the oracle.

Floating outputs (the paper fixes no precision; the library computes in fp32):
the outputs are smooth functions of the scaled keys z = kappa / tau, and each side
rounds kappa to fp32 on its own (half an ulp for phi / lambda + g, up to ~1.5 ulp
for the two logs of the Gumbel transform).  That input error,
    eps_z = 4 * 2^-24 * (max_group |kappa| + 1) / tau,
is carried through N softmax steps, so the allowed difference is
    soft S   : (1e-5 + 2 N eps_z) * max(|y|, max_group |y|)
    dlogits  : (1e-5 + 8 N eps_z) * max(max_group |y|, max_group |c| / (tau lambda)),
with c = dWm * W the upstream gradient of S (the backward sums terms of size
|c| / tau, so their rounding is relative to that scale, not to a small result).
At tau = 1 the second term is below 1e-5 and the rule is the plain 1e-5 relative
bound.  The relaxation at tau < 1 with many steps can amplify rounding from step to
step, so on extreme inputs (key gaps of tens of z-units competing over 8-16 steps)
no fp32 evaluation meets a bound linear in N: the float32 oracle itself reaches
several times it.  The input's own conditioning is therefore measured as the float32
oracle's deviation from the float64 one, dev32, element by element, and the
allowance becomes bound + 4 |dev32| against the float64 oracle (the truth) and
bound + 5 |dev32| against the float32 oracle.  On the configs' inputs dev32 is far
below the bound, so the bound governs.  bf16 outputs Wm = bf16(W * S) and dW = bf16(dWm * S): bit-exact against the
library's own S (the rounding is fully defined), and against the oracle within one
bf16 ulp beyond what the S tolerance already allows (|W| * tol_S).  Hard masks:
bit-exact, except groups whose N-th and (N+1)-th float64 keys differ by less than
1e-6 (counted).
"""
import numpy as np

U = 2.0 ** -24


def eps_z(kappa64, M, tau):
    k = np.abs(np.asarray(kappa64, dtype=np.float64)).reshape(-1, M)
    k = np.where(np.isfinite(k), k, 0.0)
    return 4 * U * (k.max(axis=1, keepdims=True) + 1.0) / tau


def soft_tolerance(want, kappa64, N, M, tau):
    w = np.asarray(want, dtype=np.float64).reshape(-1, M)
    scale = np.maximum(np.abs(w), np.abs(w).max(axis=1, keepdims=True))
    return (1e-5 + 2 * N * eps_z(kappa64, M, tau)) * scale


def soft_violations(got, want, kappa64, N, M, tau, extra=None):
    g = np.asarray(got, dtype=np.float64).reshape(-1, M)
    w = np.asarray(want, dtype=np.float64).reshape(-1, M)
    tol = soft_tolerance(want, kappa64, N, M, tau)
    if extra is not None:
        tol = tol + np.abs(np.asarray(extra, dtype=np.float64)).reshape(-1, M)
    bad = ~(np.abs(g - w) <= tol)
    return int(bad.sum()), float(np.max(np.abs(g - w) / np.maximum(tol, 1e-300)))


def dlogit_tolerance(want, c, kappa64, N, M, tau, lam=1.0, extra=None):
    """Allowed |got - want| of the logit gradients, per element ([groups, M])."""
    w = np.asarray(want, dtype=np.float64).reshape(-1, M)
    cs = np.abs(np.asarray(c, dtype=np.float64)).reshape(-1, M).max(axis=1, keepdims=True) / (tau * lam)
    scale = np.maximum(np.abs(w).max(axis=1, keepdims=True), cs)
    tol = (1e-5 + 8 * N * eps_z(kappa64, M, tau)) * scale
    if extra is not None:
        tol = tol + np.abs(np.asarray(extra, dtype=np.float64)).reshape(-1, M)
    return np.broadcast_to(tol, w.shape)


def dlogit_violations(got, want, c, kappa64, N, M, tau, lam=1.0, extra=None):
    g = np.asarray(got, dtype=np.float64).reshape(-1, M)
    w = np.asarray(want, dtype=np.float64).reshape(-1, M)
    tol = dlogit_tolerance(want, c, kappa64, N, M, tau, lam, extra)
    bad = ~(np.abs(g - w) <= tol)
    return int(bad.sum()), float(np.max(np.abs(g - w) / np.maximum(tol, 1e-300)))


def adamw_tolerance(phi0, g, m0, v0, tol_g, lr, beta1, beta2, eps, wd, t):
    """Allowed |got - want| of (phi, m, v) after one AdamW step, for a float32
    evaluation in any arrangement of the same definition (decoupled decay, moments,
    bias corrections, lr * m_hat / (sqrt(v_hat) + eps)) whose gradient lies within
    tol_g of the float64 gradient g, against the float64 step on g.

    Gradient error, carried to first order (a factor 2 covers the curvature, since
    tol_g / |g| is ~1e-5):
        dm = (1 - b1) tol_g,   dv = (1 - b2) (2 |g| tol_g + tol_g^2),
        A = m_hat / D, D = sqrt(v_hat) + eps,
        dA = |dm_hat| / D + |m_hat| dsq / (D (D - dsq)),
        dsq = min(sqrt(dv_hat), dv_hat / (2 sqrt(v_hat)))   (sqrt is 1/2-Hoelder),
    and float32 rounding: each of the step's roughly ten operations rounds once
    (relative 2^-24), so 16 u of the magnitudes involved (|phi|, lr |A|, |m|, |v|).
    Returns (tol_phi, tol_m, tol_v)."""
    u = 2.0 ** -24
    phi0, g, m0, v0, tol_g = (np.asarray(x, dtype=np.float64) for x in (phi0, g, m0, v0, tol_g))
    bc1, bc2 = 1.0 - beta1 ** t, 1.0 - beta2 ** t
    m = beta1 * m0 + (1 - beta1) * g
    v = beta2 * v0 + (1 - beta2) * g * g
    dm = (1 - beta1) * tol_g + 16 * u * (np.abs(m) + beta1 * np.abs(m0) + (1 - beta1) * np.abs(g))
    dv = (1 - beta2) * (2 * np.abs(g) * tol_g + tol_g ** 2) + 16 * u * (v + beta2 * v0 + (1 - beta2) * g * g)
    m_hat, v_hat = m / bc1, v / bc2
    sq = np.sqrt(v_hat)
    D = sq + eps
    dv_hat = dv / bc2
    with np.errstate(divide="ignore", invalid="ignore"):
        dsq = np.minimum(np.sqrt(dv_hat), np.where(sq > 0, dv_hat / (2 * sq), np.inf))
        A = m_hat / D
        dA = np.abs(dm / bc1) / D + np.abs(m_hat) * dsq / (D * (D - dsq))
    # beyond half of D the first-order bound no longer holds: no allowance (such an
    # input is too ill-conditioned for this comparison and fails it)
    dA = np.where(dsq <= 0.5 * D, dA, 0.0)
    tol_phi = 2 * lr * dA + 16 * u * (np.abs(phi0) + lr * np.abs(A))
    return tol_phi, 2 * dm, 2 * dv


def plain_relative(got, want, c=None, M=4, tau=1.0, lam=1.0):
    """max |x - y| / group scale (the bare 1e-5 rule), for reporting."""
    g = np.asarray(got, dtype=np.float64).reshape(-1, M)
    w = np.asarray(want, dtype=np.float64).reshape(-1, M)
    scale = np.abs(w).max(axis=1, keepdims=True)
    if c is not None:
        scale = np.maximum(scale, np.abs(np.asarray(c, dtype=np.float64)).reshape(-1, M).max(axis=1, keepdims=True)
                           / (tau * lam))
    scale = np.maximum(scale, 1e-300)
    return float(np.max(np.abs(g - w) / scale))


def bf16_violations(got_bits, want_bits, extra=None):
    """Count entries more than one bf16 ulp (+ `extra`, absolute) apart (uint16 bit patterns)."""
    from oracle.roi_oracle import bf16_to_f32
    g = bf16_to_f32(np.asarray(got_bits).ravel()).astype(np.float64)
    w = bf16_to_f32(np.asarray(want_bits).ravel()).astype(np.float64)
    both_nan = np.isnan(g) & np.isnan(w)
    m = np.maximum(np.abs(g), np.abs(w))
    with np.errstate(divide="ignore"):
        ulp = np.where(m > 0, 2.0 ** (np.floor(np.log2(np.where(m > 0, m, 1.0))) - 7), 2.0 ** -133)
    ulp = np.maximum(ulp, 2.0 ** -133)
    if extra is not None:
        ulp = ulp + np.asarray(extra, dtype=np.float64).ravel()
    bad = ~(np.abs(g - w) <= ulp) & ~both_nan
    return int(bad.sum())


def hard_mismatches(got_words, want_words, kappa64, N, M, E):
    """(mismatching groups outside the near-tie band, near-tie groups)."""
    from oracle.roi_oracle import topn_key_gap, unpack_bits
    g = unpack_bits(np.asarray(got_words).view(np.uint32), E).reshape(-1, M)
    w = unpack_bits(np.asarray(want_words).view(np.uint32), E).reshape(-1, M)
    gap = topn_key_gap(np.asarray(kappa64, dtype=np.float64).reshape(-1, M), N)
    near = gap < 1e-6
    diff = np.any(g != w, axis=1)
    return int(np.sum(diff & ~near)), int(np.sum(near))
