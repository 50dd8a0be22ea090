"""Batched calls (roi_mask_fwd_batch / roi_mask_bwd_batch): many tensors per call,
their launches chained by programmatic dependent launch (runs of small tensors
sharing one multi-tensor launch), must give, bit for bit, what the single-tensor
calls give, and match the oracle.  Sets mix tensors with and
without full tiles, ragged tails,
per-item noise states (seed, step, tensor_id, lambda, row_offset), optional outputs,
empty items, 300 items, and an (N, M) without a tile kernel (no chaining)."""
import numpy as np
import pytest

import workloads as WL
from oracle import roi_oracle as O
import _compare as C

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


def make_set(shapes, seed0):
    import torch
    dev = torch.device("cuda")
    out = []
    for k, (rows, cols) in enumerate(shapes):
        W, phi, dWm = WL.make_inputs(rows, cols, "normal" if k % 2 else "logw", seed0 + k)
        st = (seed0 * 7 + k, 3 + k % 5, k, [1.0, 0.7, 1.3][k % 3], (k * 37) % 11)
        out.append({"W": W.to(dev), "phi": phi.to(dev), "dWm": dWm.to(dev), "st": st, "rows": rows, "cols": cols})
    return out


def outputs(roi, t, soft, hard, dW):
    import torch
    rows, cols = t["rows"], t["cols"]
    return {"Wm": torch.full((rows, cols), -1, dtype=torch.int16, device="cuda").view(torch.bfloat16),
            "soft": torch.full((rows, cols), float("nan"), device="cuda") if soft else None,
            "hard": torch.full((roi.hard_words(rows, cols),), -1, dtype=torch.int32, device="cuda") if hard else None,
            "dphi": torch.full((rows, cols), float("nan"), device="cuda"),
            "dW": torch.full((rows, cols), -1, dtype=torch.int16, device="cuda").view(torch.bfloat16) if dW else None}


def run_single(roi, ts, N, M, tau, flags):
    res = []
    for t, (soft, hard, dW) in zip(ts, flags):
        o = outputs(roi, t, soft, hard, dW)
        roi.roi_mask_fwd_ex(t["phi"], t["W"], N, M, tau, t["st"], o["Wm"], o["soft"], o["hard"])
        roi.roi_mask_bwd(t["phi"], t["W"], t["st"], N, M, t["dWm"], tau, o["dphi"], o["dW"])
        res.append(o)
    roi.roi_device_status()
    return res


def run_batch(roi, ts, N, M, tau, flags):
    res = [outputs(roi, t, *f) for t, f in zip(ts, flags)]
    roi.roi_mask_fwd_batch([(t["phi"], t["W"], t["st"], o["Wm"], o["soft"], o["hard"]) for t, o in zip(ts, res)],
                           N, M, tau)
    roi.roi_mask_bwd_batch([(t["phi"], t["W"], t["st"], t["dWm"], o["dphi"], o["dW"]) for t, o in zip(ts, res)],
                           N, M, tau)
    roi.roi_device_status()
    return res


def assert_same(a, b):
    import torch
    for k in a:
        if a[k] is None:
            assert b[k] is None
            continue
        x, y = a[k], b[k]
        if x.dtype == torch.bfloat16:
            x, y = x.view(torch.int16), y.view(torch.int16)
        assert torch.equal(x, y) if x.dtype != torch.float32 else torch.equal(x.view(torch.int32), y.view(torch.int32)), k


# shapes: tails of every size, tensors smaller than one tile, large ones spanning many tiles
SHAPES = [(37, 1000), (3, 64), (64, 3584), (512, 256), (1, 32), (129, 2048), (8, 8), (300, 520), (16, 24576)]


# tau = 0.05: many groups leave the fast path's range and go through the deferred
# queues, whose entries name their tensor in a launch shared by several
@pytest.mark.parametrize("N,M,tau", [(2, 4, 1.0), (2, 4, 0.5), (2, 4, 0.05), (4, 8, 1.0), (4, 8, 0.3), (4, 8, 0.05),
                                     (2, 8, 1.0), (3, 4, 0.8), (8, 16, 0.2), (16, 32, 1.0)])
def test_batch_equals_single_calls(roi, N, M, tau):
    shapes = [(r, c) for r, c in SHAPES if c % M == 0]
    ts = make_set(shapes, 40 + M + int(10 * tau))
    flags = [(k % 3 == 0, k % 2 == 0, k % 4 == 1) for k in range(len(ts))]
    single = run_single(roi, ts, N, M, tau, flags)
    batch = run_batch(roi, ts, N, M, tau, flags)
    for a, b in zip(single, batch):
        assert_same(a, b)


def test_batch_matches_oracle(roi):
    N, M, tau = 2, 4, 1.0
    shapes = [(37, 1000), (5, 96), (64, 3584), (1, 32)]
    ts = make_set(shapes, 90)
    flags = [(True, True, True)] * len(ts)
    res = run_batch(roi, ts, N, M, tau, flags)
    for t, o in zip(ts, res):
        seed, step, tid, lam, roff = t["st"]
        ph, Wb, dWb = t["phi"].cpu().numpy(), _u16(t["W"]), _u16(t["dWm"])
        kw = dict(tensor_id=tid, lam=lam, row_offset=roff)
        f64 = O.mask_fwd(ph, Wb, N, M, tau, seed, step, **kw)
        f32 = O.mask_fwd(ph, Wb, N, M, tau, seed, step, dtype=np.float32, **kw)
        b64 = O.mask_bwd(ph, Wb, dWb, N, M, tau, seed, step, **kw)
        E = t["rows"] * t["cols"]
        outside, _ = C.hard_mismatches(o["hard"].cpu().numpy().view(np.uint32), f64["hard_bits"], f64["keys"], N, M, E)
        assert outside == 0
        tolS = (C.soft_tolerance(f64["soft"], f64["keys"], N, M, tau).ravel()
                + 4.0 * np.abs(f32["soft"].astype(np.float64) - f64["soft"]).ravel())
        assert np.all(np.abs(o["soft"].cpu().numpy().ravel() - f64["soft"].ravel()) <= tolS)
        c = (O.bf16_to_f32(dWb).astype(np.float64) * O.bf16_to_f32(Wb)).ravel()
        assert C.plain_relative(o["dphi"].cpu().numpy(), b64["dlogits"], c, M, tau, lam) <= 1e-5


def test_more_items_than_one_launch_and_empty_items(roi):
    """300 items with empty ones mixed in."""
    import torch
    N, M, tau = 2, 4, 1.0
    shapes = [((k * 7) % 13 + 1, 32 * ((k % 5) + 1)) for k in range(300)]
    ts = make_set(shapes, 7)
    flags = [(False, True, False)] * len(ts)
    empty = {"W": torch.empty(0, 32, dtype=torch.bfloat16, device="cuda"),
             "phi": torch.empty(0, 32, device="cuda"), "dWm": torch.empty(0, 32, dtype=torch.bfloat16, device="cuda"),
             "st": (0, 0, 0, 1.0, 0), "rows": 0, "cols": 32}
    ts = ts[:100] + [empty] + ts[100:] + [empty]
    flags = flags[:100] + [(False, True, False)] + flags[100:] + [(False, True, False)]
    single = run_single(roi, [t for t in ts if t["rows"]], N, M, tau, [f for t, f in zip(ts, flags) if t["rows"]])
    batch = run_batch(roi, ts, N, M, tau, flags)
    batch = [b for t, b in zip(ts, batch) if t["rows"]]
    for a, b in zip(single, batch):
        assert_same(a, b)


def test_batch_launch_counts(roi):
    """Consecutive small tensors with the same tile kernel share one launch: runs of
    at least 8 in the forward, of at least 2 in the plain backward.  A tensor that
    gives every SM at least 12 tiles (2:4: 12288 elements a forward tile, 8192 a
    backward one) keeps a launch of its own and splits the runs around it.  Every
    form gives, bit for bit, what the single calls give."""
    import torch
    N, M, tau = 2, 4, 1.0
    small = [(64, 3584), (16, 512), (37, 1000), (8, 256), (100, 2048), (3, 64), (129, 520), (40, 4096)]
    ts = make_set(small, 3)
    flags = [(False, True, False)] * len(ts)
    run_batch(roi, ts, N, M, tau, flags)
    before = roi.roi_launch_count()
    run_batch(roi, ts, N, M, tau, flags)
    assert roi.roi_launch_count() - before == 2
    before = roi.roi_launch_count()
    run_batch(roi, ts[:3], N, M, tau, flags[:3])
    assert roi.roi_launch_count() - before == 3 + 1
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    big = (12 * sms * 12288 // 4096 + 8, 4096)
    ts = make_set([big] + small + [big, small[0]], 5)
    flags = [(True, True, True)] * len(ts)
    single = run_single(roi, ts, N, M, tau, flags)
    before = roi.roi_launch_count()
    batch = run_batch(roi, ts, N, M, tau, flags)
    # per direction: big, the run of eight small ones, big, one small
    assert roi.roi_launch_count() - before == 2 * 4
    for a, b in zip(single, batch):
        assert_same(a, b)


def test_work_queued_after_a_batch_sees_every_item(roi):
    """Launch chaining keeps stream order: a reduction queued on the same stream right
    after the batched calls (no synchronisation in between) reads every item's
    finished outputs, including those of early items whose successors started
    before they ended."""
    import torch
    N, M, tau = 2, 4, 1.0
    shapes = [(1024, 3584), (64, 512), (8, 256)] * 6 + [(2048, 3584)]
    ts = make_set(shapes, 11)
    flags = [(False, True, False)] * len(ts)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        for rep in range(3):
            res = [outputs(roi, t, *f) for t, f in zip(ts, flags)]
            torch.cuda.current_stream().wait_stream(torch.cuda.default_stream())
            roi.roi_mask_fwd_batch([(t["phi"], t["W"], t["st"], o["Wm"], None, o["hard"])
                                    for t, o in zip(ts, res)], N, M, tau, stream=stream)
            roi.roi_mask_bwd_batch([(t["phi"], t["W"], t["st"], t["dWm"], o["dphi"], None)
                                    for t, o in zip(ts, res)], N, M, tau, stream=stream)
            # queued behind the batch: every output must already be final
            nan_dphi = torch.stack([o["dphi"].isnan().any() for o in res]).any()
            sums = torch.stack([o["Wm"].float().sum() for o in res])
            stream.synchronize()
            assert not bool(nan_dphi)
            again = torch.stack([o["Wm"].float().sum() for o in res])
            assert torch.equal(sums, again)


def test_adamw_batch_equals_single_calls(roi):
    """roi_mask_bwd_adamw_batch: logits, moments, gradients and dW after the step equal
    the single calls' bit for bit (2:4 and 4:8, mixed shapes and noise states; nine
    small tensors, so the batch runs as one multi-tensor launch)."""
    import torch
    for N, M, tau in ((2, 4, 1.0), (4, 8, 0.5), (4, 8, 1.0)):
        shapes = [(r, c) for r, c in SHAPES if c % M == 0]
        ts = make_set(shapes, 70 + M)
        opt = roi.AdamW(1e-3, 0.9, 0.95, 1e-8, 0.05, 4)
        def state():
            out = []
            for k, t in enumerate(ts):
                g = torch.Generator(device="cuda").manual_seed(k)
                out.append({"phi": t["phi"].clone(),
                            "m": 1e-3 * torch.randn(t["phi"].shape, generator=g, device="cuda"),
                            "v": 1e-6 * torch.rand(t["phi"].shape, generator=g, device="cuda"),
                            "dphi": torch.empty_like(t["phi"]),
                            "dW": torch.empty_like(t["W"]) if k % 2 else None})
            return out
        single, batch = state(), state()
        for t, s_ in zip(ts, single):
            roi.roi_mask_bwd_adamw(s_["phi"], t["W"], t["st"], N, M, t["dWm"], tau, s_["m"], s_["v"], opt,
                                   s_["dphi"], s_["dW"])
        roi.roi_mask_bwd_adamw_batch([(b["phi"], t["W"], t["st"], t["dWm"], b["m"], b["v"], b["dphi"], b["dW"])
                                      for t, b in zip(ts, batch)], N, M, tau, opt)
        roi.roi_device_status()
        for a, b in zip(single, batch):
            for k in ("phi", "m", "v", "dphi"):
                assert torch.equal(a[k].view(torch.int32), b[k].view(torch.int32)), k
            if a["dW"] is not None:
                assert torch.equal(a["dW"].view(torch.int16), b["dW"].view(torch.int16))


def test_straight_through_batch_equals_single_calls(roi):
    """roi_mask_{fwd,bwd}_st_batch against the single straight-through calls, bit for
    bit (nine small tensors: one multi-tensor launch per direction)."""
    import torch
    for N, M, tau in ((2, 4, 1.0), (4, 8, 0.5)):
        shapes = [(r, c) for r, c in SHAPES if c % M == 0]
        ts = make_set(shapes, 50 + M)
        res = []
        for k, t in enumerate(ts):
            o = outputs(roi, t, False, True, True)
            roi.roi_mask_fwd_st(t["phi"], t["W"], N, M, tau, t["st"], o["Wm"], None, o["hard"])
            roi.roi_mask_bwd_st(t["phi"], t["W"], t["st"], N, M, t["dWm"], o["hard"], tau, o["dphi"], o["dW"])
            res.append(o)
        bat = [outputs(roi, t, False, True, True) for t in ts]
        roi.roi_mask_fwd_st_batch([(t["phi"], t["W"], t["st"], o["Wm"], None, o["hard"]) for t, o in zip(ts, bat)],
                                  N, M, tau)
        roi.roi_mask_bwd_st_batch([(t["phi"], t["W"], t["st"], t["dWm"], o["hard"], o["dphi"], o["dW"])
                                   for t, o in zip(ts, bat)], N, M, tau)
        roi.roi_device_status()
        for a, b in zip(res, bat):
            assert_same(a, b)


@pytest.mark.parametrize("N,M", [(2, 4), (4, 8)])
def test_batch_mixes_counter_widths(roi, N, M):
    """Items whose noise counters all fit 32 bits (the kernels form them in 32-bit
    arithmetic) followed by items whose flat indices pass 2^34 (64-bit counters), in
    one batch: each equals its single call bit for bit (plain and fused with AdamW,
    tau = 1), and a wide item matches the oracle.  Eight of each: the forward runs
    both widths in one multi-tensor launch, the backwards one launch per width."""
    import torch
    shapes = [(37, 1024), (64, 3584), (29, 1536), (5, 2048)] * 4
    ts = make_set(shapes, 120 + M)
    for k, t in enumerate(ts):
        if k >= 8:  # rows from flat index 2^34 on
            seed, step, tid, lam, _ = t["st"]
            t["st"] = (seed, step, tid, lam, 2 ** 34 // t["cols"] + k)
    flags = [(True, True, True)] * len(ts)
    single = run_single(roi, ts, N, M, 1.0, flags)
    before = roi.roi_launch_count()
    batch = run_batch(roi, ts, N, M, 1.0, flags)
    assert roi.roi_launch_count() - before == 1 + 2
    for a, b in zip(single, batch):
        assert_same(a, b)
    t, o = ts[9], batch[9]
    seed, step, tid, lam, roff = t["st"]
    ph, Wb = t["phi"].cpu().numpy(), WL.bf16_bits(t["W"].cpu())
    ref = O.mask_fwd(ph, Wb, N, M, 1.0, seed, step, tensor_id=tid, lam=lam, row_offset=roff)
    ref32 = O.mask_fwd(ph, Wb, N, M, 1.0, seed, step, tensor_id=tid, lam=lam, row_offset=roff, dtype=np.float32)
    outside, _ = C.hard_mismatches(o["hard"].cpu().numpy().view(np.uint32), ref["hard_bits"], ref["keys"], N, M,
                                   t["rows"] * t["cols"])
    assert outside == 0
    n, _ = C.soft_violations(o["soft"].cpu().numpy(), ref["soft"], ref["keys"], N, M, 1.0,
                             extra=4.0 * np.abs(ref32["soft"].astype(np.float64) - ref["soft"]))
    assert n == 0
    opt = roi.AdamW(1e-3, 0.9, 0.95, 1e-8, 0.05, 4)
    def state():
        return [{"phi": t["phi"].clone(), "m": torch.zeros_like(t["phi"]), "v": torch.full_like(t["phi"], 1e-8),
                 "dphi": torch.empty_like(t["phi"])} for t in ts]
    one, bat = state(), state()
    for t, s_ in zip(ts, one):
        roi.roi_mask_bwd_adamw(s_["phi"], t["W"], t["st"], N, M, t["dWm"], 1.0, s_["m"], s_["v"], opt, s_["dphi"])
    before = roi.roi_launch_count()
    roi.roi_mask_bwd_adamw_batch([(b["phi"], t["W"], t["st"], t["dWm"], b["m"], b["v"], b["dphi"], None)
                                  for t, b in zip(ts, bat)], N, M, 1.0, opt)
    roi.roi_device_status()
    assert roi.roi_launch_count() - before == 2
    for a, b, r in zip(one, bat, single):
        for k in ("phi", "m", "v", "dphi"):
            assert torch.equal(a[k].view(torch.int32), b[k].view(torch.int32)), k
        # the fused step's gradient is the plain backward's (up to the compilers'
        # contraction of the two kernels)
        g, gr = a["dphi"].cpu().numpy(), r["dphi"].cpu().numpy()
        scale = np.abs(gr).reshape(-1, M).max(-1, keepdims=True).repeat(M, -1).reshape(gr.shape)
        assert np.all(np.abs(g - gr) <= 1e-6 * scale + 1e-30)


def _expected_launches(shapes, tile, sms, min_run):
    """Launches of one batched direction: a run of at least min_run consecutive
    tensors with fewer than 12 full tiles per SM each takes one, any other tensor one."""
    small = [r * c // tile < 12 * sms for r, c in shapes]
    n = i = 0
    while i < len(shapes):
        j = i
        while j < len(shapes) and small[j]:
            j += 1
        n += 1
        i = j if j - i >= min_run else i + 1
    return n


@pytest.mark.parametrize("set_name,layers,N,M,tau", [("qwen2.5-0.5b", 4, 2, 4, 0.1), ("qwen2.5-1.5b", 2, 4, 8, 0.5)])
def test_layer_set_batch_equals_single_calls(roi, set_name, layers, N, M, tau):
    """Leading layers of a benchmark layer set at its own N:M and tau, step-keyed noise
    as the benchmark draws it: the batched calls (the 0.5B-shaped set in one forward
    and one backward launch; the 1.5B-shaped forward in one launch, its backward
    sharing each layer's q, k, v, o) give every tensor's Wm, hard bits and logit
    gradients bit for bit as the single calls do."""
    import torch
    dev = torch.device("cuda")
    lset = WL.LAYER_SETS[set_name]
    kind = WL.CONFIGS[set_name].logits
    ts = []
    for layer, p, rows, cols in lset.tensors():
        if layer >= layers:
            break
        W, phi, dWm = WL.make_inputs(rows, cols, kind, WL.tensor_seed(layer, p), device=dev)
        ts.append({"W": W, "phi": phi, "dWm": dWm, "st": (11, 5, 7 * layer + p, 1.0, 0), "rows": rows, "cols": cols})
    flags = [(False, True, False)] * len(ts)
    single = run_single(roi, ts, N, M, tau, flags)
    before = roi.roi_launch_count()
    batch = run_batch(roi, ts, N, M, tau, flags)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    shapes = [(t["rows"], t["cols"]) for t in ts]
    want = (_expected_launches(shapes, 12288 if M == 4 else 8192, sms, 8)
            + _expected_launches(shapes, 8192 if M == 4 else 6144, sms, 2))
    assert roi.roi_launch_count() - before == want
    for a, b in zip(single, batch):
        assert_same(a, b)
