"""The timeout path of the kernels' bounded waits, run on valid copies.

roi_set_ring_wait_limit_ns(0) makes every wait of a kernel for a stage of its copy
ring give up at once (landed or not), so each CTA gives up at its first tile, with
its first copies possibly still in flight.  The kernel must then set
ROI_ERR_TIMEOUT in the device status, let its own copies in flight land (those
drain waits keep their fixed limit), and return.  With the limit restored, the
next calls on the same CUDA context run normally: their outputs equal, bit for
bit, those of the same calls made before the timeout, and match the oracle on
sampled rows.  Every copy here is valid and every wait bounded: nothing faults or
hangs the GPU.
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


def _expect_timeout(roi, launch):
    """Runs `launch` with the ring-wait limit at 0; the device status must report
    the timeout (and is cleared by reading it)."""
    roi.roi_device_status()  # start from a clear status word
    roi.roi_set_ring_wait_limit_ns(0)
    try:
        launch()
        with pytest.raises(roi.RoiError) as err:
            roi.roi_device_status()
        assert err.value.status == 8, str(err.value)  # ROI_ERR_TIMEOUT
    finally:
        roi.roi_set_ring_wait_limit_ns(roi.ROI_DEFAULT_RING_WAIT_NS)
    roi.roi_device_status()  # cleared, and the context still works


@pytest.mark.parametrize("N,M,tau", [(2, 4, 1.0), (4, 8, 1.0), (4, 8, 0.5), (8, 16, 0.2), (16, 32, 0.2)])
def test_mask_kernels_time_out_then_recover(roi, N, M, tau):
    import torch
    dev = torch.device("cuda")
    rows, cols = 1024, 4096          # hundreds of tiles: every CTA starts on an empty ring
    W, phi, dWm = WL.make_inputs(rows, cols, "normal", 55, device=dev)
    st = roi.NoiseState(5, 3, 1, 1.0, 0)

    def run():
        Wm = torch.empty_like(W)
        hard = torch.empty(roi.hard_words(rows, cols), dtype=torch.int32, device=dev)
        dphi = torch.empty_like(phi)
        roi.roi_mask_fwd_ex(phi, W, N, M, tau, st, Wm, None, hard)
        roi.roi_mask_bwd(phi, W, st, N, M, dWm, tau, dphi, None)
        return Wm, hard, dphi

    before = run()
    roi.roi_device_status()
    _expect_timeout(roi, run)
    after = run()
    roi.roi_device_status()
    for a, b in zip(before, after):
        assert torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16 else a.view(torch.int32),
                           b.view(torch.int16) if b.dtype == torch.bfloat16 else b.view(torch.int32))
    # two rows of the recovered run against the oracle (hard mask outside near ties)
    Wm, hard, dphi = after
    for r in (0, rows - 1):
        ph = phi[r:r + 1].cpu().numpy()
        ref = O.mask_fwd(ph, WL.bf16_bits(W[r:r + 1]), N, M, tau, 5, 3, tensor_id=1, row_offset=r)
        got = hard[r * cols // 32:(r + 1) * cols // 32].cpu().numpy().view(np.uint32)
        g = O.unpack_bits(got, cols).reshape(-1, M)
        w = ref["hard"].reshape(-1, M)
        near = O.topn_key_gap(ref["keys"].reshape(-1, M), N) < 1e-6
        assert not np.any(np.any(g != w, axis=1) & ~near)


def test_multi_tensor_launches_time_out_then_recover(roi):
    """Batched calls over small tensors (one multi-tensor launch per direction, the
    CTAs walking every tensor's tiles): a wait that gives up ends the launch the same
    way, and the next batch on the context gives the first batch's bits."""
    import torch
    dev = torch.device("cuda")
    shapes = [(256, 4096), (64, 1024), (300, 2048), (37, 1000), (8, 512), (128, 896), (5, 64), (90, 3584)]
    ts = []
    for k, (rows, cols) in enumerate(shapes):
        W, phi, dWm = WL.make_inputs(rows, cols, "normal", 60 + k, device=dev)
        ts.append((phi, W, dWm, roi.NoiseState(7, 2, k, 1.0, 0), rows, cols))

    def run():
        out = []
        for phi, W, dWm, st, rows, cols in ts:
            out.append((torch.empty_like(W), torch.empty(roi.hard_words(rows, cols), dtype=torch.int32, device=dev),
                        torch.empty_like(phi)))
        roi.roi_mask_fwd_batch([(phi, W, st, o[0], None, o[1]) for (phi, W, dWm, st, r, c), o in zip(ts, out)],
                               2, 4, 1.0)
        roi.roi_mask_bwd_batch([(phi, W, st, dWm, o[2], None) for (phi, W, dWm, st, r, c), o in zip(ts, out)],
                               2, 4, 1.0)
        return out

    before = run()
    roi.roi_device_status()
    launches = roi.roi_launch_count()
    _expect_timeout(roi, run)
    assert roi.roi_launch_count() - launches == 2  # one launch per direction
    after = run()
    roi.roi_device_status()
    for x, y in zip(before, after):
        assert torch.equal(x[0].view(torch.int16), y[0].view(torch.int16))
        assert torch.equal(x[1], y[1])
        assert torch.equal(x[2].view(torch.int32), y[2].view(torch.int32))


def test_masked_linear_times_out_drains_then_recovers(roi):
    """The tensor-core masked linear: on a wait that gives up, the CTA waits for the
    TMA fills and MMAs it issued before releasing shared memory and TMEM."""
    import torch
    dev = torch.device("cuda")
    rows, cols, T = 384, 8192, 64
    W, phi, _ = WL.make_inputs(rows, cols, "normal", 56, device=dev)
    X = WL.make_tokens(T, cols, 56, device=dev)
    st = roi.NoiseState(6, 1, 2, 1.0, 0)
    nb = roi.roi_masked_linear_workspace_size(T, rows, cols)
    ws = torch.empty(max(nb, 16), dtype=torch.uint8, device=dev)

    def run():
        Y = torch.full((T, rows), float("nan"), dtype=torch.float32, device=dev)
        roi.roi_masked_linear_fwd(X, phi, W, 2, 4, 1.0, st, Y, ws)
        return Y

    before = run()
    roi.roi_device_status()
    _expect_timeout(roi, run)
    after = run()
    roi.roi_device_status()
    assert torch.all(torch.isfinite(after))
    assert torch.equal(before.view(torch.int32), after.view(torch.int32))
