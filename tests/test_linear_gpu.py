"""Parity of the fused masked linear forward (roi_masked_linear_fwd: the relaxed
mask formed in the prologue of a tensor-core GEMM) with the CPU oracle.

Tolerance, from the arithmetic: the products of two bfloat16 values are exact in
float32; the tensor cores and the split-K reduction add them in float32 in their
own order, at most K * 2^-23 * sum_k |x_k wm_k| away from the exact sum; and the
library's Wm may differ from the float64 oracle's by one bf16 ulp (at most
2^-7 |wm|) where S lies within the soft-mask tolerance of a rounding boundary, a
rare event, of which at most four are allowed per dot product.
"""
import numpy as np
import pytest

import workloads as WL
from oracle import roi_oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def roi():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2608_23048_gb300 import _build
    _build.build()
    import paper_2608_23048_gb300 as roi
    return roi


def _u16(t):
    import torch
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def gpu_linear(roi, X, phi, W, N, M, tau, st, workspace=True):
    import torch
    dev = torch.device("cuda")
    T, rows = X.shape[0], phi.shape[0]
    Xd, phid, Wd = X.to(dev), phi.to(dev), W.to(dev)
    Y = torch.full((T, rows), float("nan"), dtype=torch.float32, device=dev)
    ws = None
    if workspace:
        nb = roi.roi_masked_linear_workspace_size(T, rows, phi.shape[1])
        ws = torch.empty(max(nb, 16), dtype=torch.uint8, device=dev)
    roi.roi_masked_linear_fwd(Xd, phid, Wd, N, M, tau, st, Y, ws)
    roi.roi_device_status()
    return Y.cpu().numpy().astype(np.float64)


def linear_tolerance(Xb, Wm_bits, cols):
    x = np.abs(O.bf16_to_f32(Xb).astype(np.float64))
    w = np.abs(O.bf16_to_f32(Wm_bits).astype(np.float64))
    absum = x @ w.T
    maxterm = x.max(axis=1)[:, None] * w.max(axis=1)[None, :]  # bounds max_k |x_k wm_k|
    return cols * 2.0 ** -23 * absum + 4 * 2.0 ** -7 * maxterm, cols * 2.0 ** -23 * absum


def check(Y, Xb, ph, Wb, N, M, tau, seed, step, tid=0, lam=1.0, row_offset=0):
    o = O.masked_linear_fwd(Xb, ph, Wb, N, M, tau, seed, step, tid, lam, row_offset)
    tol, _ = linear_tolerance(Xb, o["Wm"], ph.shape[1])
    err = np.abs(Y - o["Y"])
    assert np.all(np.isfinite(Y))
    assert np.all(err <= tol), f"max excess {np.max(err - tol)}"
    return o


LIN_CASES = [
    # rows, cols, T, N, M, tau, logits
    (128, 64, 16, 2, 4, 1.0, "normal"),     # one row block, two K chunks
    (200, 520, 17, 2, 4, 1.0, "logw"),      # ragged rows and K tail, T not a multiple of 16
    (256, 256, 256, 2, 4, 0.5, "normal"),   # the MMA's largest N
    (130, 96, 1, 4, 8, 1.0, "normal"),      # one token; ragged second row block
    (128, 2048, 64, 4, 8, 0.3, "logw"),
    (64, 1000, 40, 2, 8, 1.0, "normal"),    # fewer rows than one block
    (384, 4096, 48, 2, 4, 1.0, "logw"),     # split K (three row blocks, long K)
    (130, 4096, 3, 2, 4, 1.0, "normal"),    # split K with T * rows not a multiple of 4
]


@pytest.mark.parametrize("rows,cols,T,N,M,tau,kind", LIN_CASES)
def test_masked_linear_parity(roi, rows, cols, T, N, M, tau, kind):
    W, phi, _ = WL.make_inputs(rows, cols, kind, rows + cols + M)
    X = WL.make_tokens(T, cols, rows + T)
    st = roi.NoiseState(987654321, 3, 5, 1.0, 0)
    Y = gpu_linear(roi, X, phi, W, N, M, tau, st)
    check(Y, WL.bf16_bits(X), phi.numpy(), WL.bf16_bits(W), N, M, tau, 987654321, 3, 5)


def test_noise_state_lambda_and_row_offset(roi):
    W, phi, _ = WL.make_inputs(136, 128, "normal", 5)
    X = WL.make_tokens(24, 128, 5)
    st = roi.NoiseState(11, 7, 2, 0.6, 1000)
    Y = gpu_linear(roi, X, phi, W, 2, 4, 1.0, st)
    check(Y, WL.bf16_bits(X), phi.numpy(), WL.bf16_bits(W), 2, 4, 1.0, 11, 7, 2, 0.6, 1000)


@pytest.mark.parametrize("N,M,tau", [(2, 4, 1.0), (4, 8, 1.0), (4, 8, 0.4)])
def test_wide_key_gaps_take_exact_path(roi, N, M, tau):
    """Outlier logits (+-100) send their groups to the exact routine in the prologue."""
    import torch
    W, phi, _ = WL.make_inputs(128, 256, "normal", 9)
    g = torch.Generator().manual_seed(78)
    shift = torch.randint(0, 16, phi.shape, generator=g)
    phi = (phi + 100.0 * (shift == 0).float() - 100.0 * (shift == 1).float()).contiguous()
    X = WL.make_tokens(32, 256, 9)
    st = roi.NoiseState(4, 1, 0, 1.0, 0)
    Y = gpu_linear(roi, X, phi, W, N, M, tau, st)
    check(Y, WL.bf16_bits(X), phi.numpy(), WL.bf16_bits(W), N, M, tau, 4, 1)


@pytest.mark.parametrize("N,M,tau", [(2, 4, 1.0), (4, 8, 0.5)])
def test_nonfinite_logits(roi, N, M, tau):
    """NaN or +inf logits make their group's Wm NaN (as in the mask forward), so the
    rows holding them come out NaN for every token; a -inf member only gets zero
    weight; every other output matches the oracle."""
    import torch
    rows, cols, T = 200, 256, 24
    W, phi, _ = WL.make_inputs(rows, cols, "normal", 41)
    phi = phi.clone()
    phi[3, 5] = float("nan")
    phi[7, 100] = float("inf")
    phi[150, 33] = float("-inf")
    phi[199, 255] = float("nan")        # last row of the ragged second row block
    X = WL.make_tokens(T, cols, 41)
    st = roi.NoiseState(6, 1, 0, 1.0, 0)
    Y = gpu_linear(roi, X, phi, W, N, M, tau, st)
    with np.errstate(invalid="ignore"):
        o = O.masked_linear_fwd(WL.bf16_bits(X), phi.numpy(), WL.bf16_bits(W), N, M, tau, 6, 1)
    bad = np.isnan(o["Y"])
    assert bad[:, 3].all() and bad[:, 7].all() and bad[:, 199].all() and not bad[:, 150].any()
    assert np.array_equal(np.isnan(Y), bad)
    Wm = O.bf16_to_f32(o["Wm"]).astype(np.float64)
    fin = ~np.isnan(Wm).any(axis=1)
    tol, _ = linear_tolerance(WL.bf16_bits(X)[:, :], o["Wm"][fin], cols)
    assert np.all(np.abs(Y[:, fin] - o["Y"][:, fin]) <= tol)


def test_prologue_wm_is_the_mask_forward(roi):
    """The fused product equals X times the Wm that roi_mask_fwd_ex writes, up to
    the float32 accumulation alone (no bf16 difference allowed): the prologue forms
    the same keys, noise and rounding."""
    import torch
    rows, cols, T = 256, 1024, 32
    W, phi, _ = WL.make_inputs(rows, cols, "logw", 21)
    X = WL.make_tokens(T, cols, 21)
    # outlier logits (about one in eight shifted by +-100): groups for both fallbacks
    g = torch.Generator().manual_seed(21)
    shift = torch.randint(0, 16, phi.shape, generator=g)
    wide = (phi + 100.0 * (shift == 0).float() - 100.0 * (shift == 1).float()).contiguous()
    for N, M, tau, ph in ((2, 4, 1.0, phi), (4, 8, 1.0, phi), (2, 8, 0.7, phi), (2, 4, 0.3, wide),
                          (4, 8, 0.5, wide), (2, 4, 1.0, wide)):
        phi = ph
        st = roi.NoiseState(5, 9, 1, 1.0, 0)
        Y = gpu_linear(roi, X, phi, W, N, M, tau, st)
        Wm = torch.empty(rows, cols, dtype=torch.bfloat16, device="cuda")
        roi.roi_mask_fwd_ex(phi.cuda(), W.cuda(), N, M, tau, st, Wm)
        wm_bits = _u16(Wm)
        want = O.bf16_to_f32(WL.bf16_bits(X)).astype(np.float64) @ O.bf16_to_f32(wm_bits).astype(np.float64).T
        _, acc = linear_tolerance(WL.bf16_bits(X), wm_bits, cols)
        assert np.all(np.abs(Y - want) <= acc + 1e-30)


def test_split_k_is_deterministic(roi):
    """Long K over one row block: the workspace lets K split across CTAs; two runs
    agree bit for bit, and the unsplit call (no workspace) agrees up to order."""
    import torch
    rows, cols, T = 128, 8192, 64
    W, phi, _ = WL.make_inputs(rows, cols, "normal", 31)
    X = WL.make_tokens(T, cols, 31)
    st = roi.NoiseState(8, 2, 0, 1.0, 0)
    assert roi.roi_masked_linear_workspace_size(T, rows, cols) > 0
    Y1 = gpu_linear(roi, X, phi, W, 2, 4, 1.0, st)
    Y2 = gpu_linear(roi, X, phi, W, 2, 4, 1.0, st)
    Y0 = gpu_linear(roi, X, phi, W, 2, 4, 1.0, st, workspace=False)
    assert np.array_equal(Y1, Y2)
    o = check(Y1, WL.bf16_bits(X), phi.numpy(), WL.bf16_bits(W), 2, 4, 1.0, 8, 2)
    _, acc = linear_tolerance(WL.bf16_bits(X), o["Wm"], cols)
    assert np.all(np.abs(Y1 - Y0) <= 2 * acc)
    check(Y0, WL.bf16_bits(X), phi.numpy(), WL.bf16_bits(W), 2, 4, 1.0, 8, 2)


def test_empty_calls_touch_nothing(roi):
    import torch
    W, phi, _ = WL.make_inputs(128, 64, "normal", 1)
    X = torch.empty(0, 64, dtype=torch.bfloat16, device="cuda")
    Y = torch.empty(0, 128, dtype=torch.float32, device="cuda")
    roi.roi_masked_linear_fwd(X, phi.cuda(), W.cuda(), 2, 4, 1.0, roi.NoiseState(0, 0, 0, 1.0, 0), Y)
    roi.roi_device_status()


@pytest.mark.parametrize("proj", ["gate", "down"])
@pytest.mark.parametrize("N,M", [(2, 4), (4, 8)])
def test_full_size_projection_sampled(roi, proj, N, M):
    """7B-shaped gate_proj (18944 x 3584, no K split) and down_proj (3584 x 18944,
    K split) at 256 tokens, the configuration the benchmark times: sampled output
    rows against the oracle (noise keyed through row_offset)."""
    import torch
    rows, cols = WL.LAYER_SETS["qwen2.5-7b"].shape(proj)
    seed = WL.tensor_seed(0, WL.PROJS.index(proj))
    dev = torch.device("cuda")
    W, phi, _ = WL.make_inputs(rows, cols, "normal", seed, device=dev)
    X = WL.make_tokens(256, cols, seed, device=dev)
    st = roi.NoiseState(0, 17, WL.PROJS.index(proj), 1.0, 0)
    nb = roi.roi_masked_linear_workspace_size(256, rows, cols)
    ws = torch.empty(max(nb, 16), dtype=torch.uint8, device=dev)
    Y = torch.empty(256, rows, dtype=torch.float32, device=dev)
    roi.roi_masked_linear_fwd(X, phi, W, N, M, 1.0, st, Y, ws)
    roi.roi_device_status()
    assert torch.all(torch.isfinite(Y))
    rng = np.random.default_rng(1)
    sample = sorted(set([0, 127, 128, rows - 1] + rng.integers(0, rows, 8).tolist()))
    Xb = WL.bf16_bits(X)
    phc, Wc = phi.cpu(), W.cpu()
    Yc = Y.cpu().numpy().astype(np.float64)
    for r in sample:
        o = O.masked_linear_fwd(Xb, phc[r:r + 1].numpy(), WL.bf16_bits(Wc[r:r + 1]), N, M, 1.0, 0, 17,
                                WL.PROJS.index(proj), 1.0, r)
        tol, _ = linear_tolerance(Xb, o["Wm"], cols)
        assert np.all(np.abs(Yc[:, r:r + 1] - o["Y"]) <= tol), (proj, r)
