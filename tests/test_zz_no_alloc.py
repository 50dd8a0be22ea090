"""roi_masked_linear_fwd_noalloc (split-K scratch in the library's static device
array) against roi_masked_linear_fwd with a caller workspace: two calls in a row
of different shapes, each bit-identical to the workspace call (the second runs
with the first's partials still in the array), and the size limit.  Collected
last; it passes alone and after the other tests."""
import numpy as np
import pytest

import workloads as WL

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


def _run(roi, rows, cols, T, N, M, tau, seed, noalloc):
    import torch
    dev = torch.device("cuda")
    W, phi, _ = WL.make_inputs(rows, cols, "normal", seed, device=dev)
    X = WL.make_tokens(T, cols, seed, device=dev)
    st = roi.NoiseState(seed, 2, 1, 1.0, 0)
    Y = torch.full((T, rows), float("nan"), dtype=torch.float32, device=dev)
    if noalloc:
        roi.roi_masked_linear_fwd_noalloc(X, phi, W, N, M, tau, st, Y)
    else:
        nb = roi.roi_masked_linear_workspace_size(T, rows, cols)
        ws = torch.empty(max(nb, 16), dtype=torch.uint8, device=dev)
        roi.roi_masked_linear_fwd(X, phi, W, N, M, tau, st, Y, ws)
    roi.roi_device_status()
    return Y.cpu().numpy()


def test_noalloc_matches_workspace_call_two_in_a_row(roi):
    shapes = [(384, 4096, 48, 2, 4, 1.0, 3), (128, 8192, 64, 4, 8, 0.5, 4)]
    assert all(roi.roi_masked_linear_workspace_size(T, r, c) > 0 for r, c, T, *_ in shapes)
    got = [_run(roi, *sh, noalloc=True) for sh in shapes]        # two no-alloc calls in a row
    want = [_run(roi, *sh, noalloc=False) for sh in shapes]
    for g, w in zip(got, want):
        assert np.all(np.isfinite(g))
        assert np.array_equal(g, w)


def test_noalloc_back_to_back_on_one_stream(roi):
    """Both no-alloc calls queued on one stream with no synchronisation between
    them, so the second call's GEMM follows the first call's split-K reduction on
    the shared array directly; one synchronisation after both.  Each result equals
    the workspace call's, bit for bit."""
    import torch
    dev = torch.device("cuda")
    shapes = [(384, 4096, 48, 2, 4, 1.0, 3), (128, 8192, 64, 4, 8, 0.5, 4)]
    want = [_run(roi, *sh, noalloc=False) for sh in shapes]
    stream = torch.cuda.Stream(device=dev)
    outs = []
    inputs = []
    for rows, cols, T, N, M, tau, seed in shapes:
        W, phi, _ = WL.make_inputs(rows, cols, "normal", seed, device=dev)
        X = WL.make_tokens(T, cols, seed, device=dev)
        inputs.append((X, phi, W))
        outs.append(torch.full((T, rows), float("nan"), dtype=torch.float32, device=dev))
    torch.cuda.synchronize()
    for (rows, cols, T, N, M, tau, seed), (X, phi, W), Y in zip(shapes, inputs, outs):
        roi.roi_masked_linear_fwd_noalloc(X, phi, W, N, M, tau, roi.NoiseState(seed, 2, 1, 1.0, 0), Y,
                                          stream=stream)
    roi.roi_device_status(stream)
    for g, w in zip(outs, want):
        assert np.array_equal(g.cpu().numpy(), w)


def test_noalloc_rejects_scratch_beyond_the_limit(roi):
    import torch
    rows, cols, T = 3584, 18944, 256
    need = roi.roi_masked_linear_workspace_size(T, rows, cols)
    if need <= 16 << 20:
        pytest.skip(f"this GPU needs only {need} B of scratch for the shape")
    L = roi.lib()
    st = roi.NoiseState(0, 0, 0, 1.0, 0)
    dev = torch.device("cuda")
    X = torch.zeros(T, cols, dtype=torch.bfloat16, device=dev)
    phi = torch.zeros(rows, cols, dtype=torch.float32, device=dev)
    W = torch.zeros(rows, cols, dtype=torch.bfloat16, device=dev)
    Y = torch.zeros(T, rows, dtype=torch.float32, device=dev)
    import ctypes
    s = L.roi_masked_linear_fwd_noalloc(ctypes.c_void_p(X.data_ptr()), ctypes.c_void_p(phi.data_ptr()),
                                        ctypes.c_void_p(W.data_ptr()), 2, 4, 1.0, ctypes.byref(st), T, rows, cols,
                                        ctypes.c_void_p(Y.data_ptr()), None)
    assert s == 2  # ROI_ERR_SHAPE, nothing launched
    assert torch.all(Y == 0)
