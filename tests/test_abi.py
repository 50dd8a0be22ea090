"""The C ABI: libroi.so loads, exports every function include/roi.h declares, and
validates arguments on the host (these calls return before any CUDA call, so they
run without a GPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "roi.h")


@pytest.fixture(scope="module")
def L():
    from paper_2608_23048_gb300 import _build
    _build.build()
    import paper_2608_23048_gb300 as roi
    return roi.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(roi_[a-z_]+)\s*\(", text)))


def test_header_declares_the_calls():
    names = declared_functions()
    for want in ("roi_mask_fwd", "roi_mask_fwd_ex", "roi_mask_bwd", "roi_hard_mask_export",
                 "roi_status_string", "roi_device_status", "roi_launch_count"):
        assert want in names


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name


def test_binding_names_match_abi():
    import paper_2608_23048_gb300 as roi
    for name in declared_functions():
        assert callable(getattr(roi, name)), name


def _fake(addr):
    return ctypes.c_void_p(addr)


A, B, C, D, E = 0x10000000, 0x20000000, 0x30000000, 0x40000000, 0x50000000


def fwd(L, logits=A, W=B, N=2, M=4, tau=1.0, rows=4, cols=8, Wm=C, soft=None, hard=None, st=None):
    import paper_2608_23048_gb300 as roi
    st = st or roi.NoiseState(0, 0, 0, 1.0, 0)
    return L.roi_mask_fwd_ex(_fake(logits) if logits else None, _fake(W) if W else None, N, M, tau,
                             ctypes.byref(st), rows, cols, _fake(Wm) if Wm else None,
                             _fake(soft) if soft else None, _fake(hard) if hard else None, None)


def test_validation_codes(L):
    import paper_2608_23048_gb300 as roi
    assert fwd(L, logits=0) == 1                    # ROI_ERR_NULL
    assert fwd(L, logits=0, W=0, Wm=0, rows=0) == 0  # empty: pointers may be NULL
    assert fwd(L, Wm=0) == 1
    assert fwd(L, N=0) == 3 and fwd(L, N=4, M=4) == 3 and fwd(L, N=2, M=33, cols=33) == 3   # ROI_ERR_NM
    assert fwd(L, cols=6) == 2 and fwd(L, rows=-1) == 2 and fwd(L, cols=0) == 2            # ROI_ERR_SHAPE
    assert fwd(L, tau=0.0) == 4 and fwd(L, tau=float("nan")) == 4 and fwd(L, tau=float("inf")) == 4
    assert fwd(L, st=roi.NoiseState(0, 0, 0, 0.0, 0)) == 4                                  # lambda
    assert fwd(L, st=roi.NoiseState(0, 0, 0, 1.0, -1)) == 2                                 # row_offset
    assert fwd(L, logits=A + 8) == 5 and fwd(L, hard=D + 4) == 5                            # ROI_ERR_ALIGN
    assert fwd(L, Wm=A + 16) == 6                   # output overlaps logits: ROI_ERR_ALIAS
    assert fwd(L, soft=C + 16) == 6                 # two outputs overlap
    assert fwd(L, rows=0) == 0                      # empty tensor: nothing to do
    st = roi.NoiseState(0, 0, 0, 1.0, 0)
    assert L.roi_mask_bwd(_fake(A), _fake(B), ctypes.byref(st), 2, 4, None, 1.0, 4, 8, _fake(C), None, None) == 1
    assert L.roi_mask_bwd(_fake(A), _fake(B), ctypes.byref(st), 2, 4, _fake(D), 1.0, 4, 8, _fake(D), None, None) == 6
    assert L.roi_hard_mask_export(_fake(A), 2, 4, 4, 8, _fake(C), _fake(B), None, None) == 1
    assert L.roi_hard_mask_export(_fake(A), 2, 4, 4, 8, _fake(C + 4), None, None, None) == 5
    assert L.roi_hard_mask_export(_fake(A), 2, 4, 0, 8, _fake(C), None, None, None) == 0
    # straight-through: as the soft calls; the backward needs the forward's bits when dW is asked for
    assert L.roi_mask_fwd_st(None, _fake(B), 2, 4, 1.0, ctypes.byref(st), 4, 8, _fake(C), None, None, None) == 1
    assert L.roi_mask_fwd_st(_fake(A), _fake(B), 2, 4, 1.0, ctypes.byref(st), 4, 8, _fake(A + 16), None, None,
                             None) == 6
    assert L.roi_mask_bwd_st(_fake(A), _fake(B), ctypes.byref(st), 2, 4, _fake(D), None, 1.0, 4, 8, _fake(C),
                             _fake(E), None) == 1
    assert L.roi_mask_bwd_st(_fake(A), _fake(B), ctypes.byref(st), 2, 4, _fake(D), _fake(E + 4), 1.0, 4, 8,
                             _fake(C), _fake(D + 0x1000), None) == 5
    assert L.roi_mask_bwd_st(_fake(A), _fake(B), ctypes.byref(st), 2, 4, _fake(D), _fake(C), 1.0, 4, 8,
                             _fake(C), _fake(E), None) == 6
    # compressed export: 2:4 only, rows*cols a multiple of 32
    assert L.roi_export_compressed_2of4(_fake(A), _fake(B), 1, 12, _fake(C), _fake(D), None) == 2
    assert L.roi_export_compressed_2of4(_fake(A), _fake(B), 4, 6, _fake(C), _fake(D), None) == 2
    assert L.roi_export_compressed_2of4(None, _fake(B), 4, 8, _fake(C), _fake(D), None) == 1
    assert L.roi_export_compressed_2of4(_fake(A), _fake(B), 4, 8, _fake(C + 2), _fake(D), None) == 5
    assert L.roi_export_compressed_2of4(_fake(A), _fake(B), 4, 8, _fake(A + 16), _fake(D), None) == 6
    assert L.roi_export_compressed_2of4(None, None, 0, 8, None, None, None) == 0
    # fused optimizer: settings checked; logits are in/out and must not overlap m, v or outputs
    opt = roi.AdamW(1e-3, 0.9, 0.95, 1e-8, 0.05, 1)
    bad = roi.AdamW(1e-3, 1.0, 0.95, 1e-8, 0.05, 1)
    zero_t = roi.AdamW(1e-3, 0.9, 0.95, 1e-8, 0.05, 0)
    def bwd_opt(o, m=C, v=D, logits=A, dl=None):
        return L.roi_mask_bwd_adamw(_fake(logits), _fake(B), ctypes.byref(st), 2, 4, _fake(E), 1.0, 4, 8,
                                    _fake(m) if m else None, _fake(v) if v else None,
                                    ctypes.byref(o) if o is not None else None, _fake(dl) if dl else None, None, None)
    assert bwd_opt(None) == 1
    assert bwd_opt(bad) == 9 and bwd_opt(zero_t) == 9
    assert bwd_opt(opt, m=None) == 1
    assert bwd_opt(opt, m=A + 64) == 6               # m overlaps the logits
    assert bwd_opt(opt, dl=D + 16) == 6              # gradient output overlaps v
    assert bwd_opt(opt, v=D + 8) == 5
    assert L.roi_mask_bwd_adamw(None, None, ctypes.byref(st), 2, 4, None, 1.0, 0, 8, None, None,
                                ctypes.byref(opt), None, None, None) == 0
    # masked linear: (2,4), (4,8), (2,8); T <= 256; cols % 8 == 0; Y and workspace are outputs
    def lin(N=2, M=4, T=4, rows=128, cols=64, X=D, logits=A, W=B, Y=C, ws=None, wsb=0, tau=1.0, state=st):
        return L.roi_masked_linear_fwd(_fake(X) if X else None, _fake(logits) if logits else None,
                                       _fake(W) if W else None, N, M, tau, ctypes.byref(state) if state else None,
                                       T, rows, cols, _fake(Y) if Y else None, _fake(ws) if ws else None, wsb, None)
    assert lin(state=None) == 1 and lin(X=0) == 1 and lin(Y=0) == 1
    assert lin(N=1) == 3 and lin(N=3, M=8) == 3 and lin(N=8, M=16, cols=64) == 3
    assert lin(T=257) == 2 and lin(T=-1) == 2 and lin(cols=12) == 2
    assert lin(tau=0.0) == 4
    assert lin(X=D + 8) == 5 and lin(ws=E + 4, wsb=64) == 5
    assert lin(Y=A + 64) == 6                       # Y overlaps the logits
    assert lin(ws=C + 256, wsb=4096) == 6           # workspace overlaps Y
    assert lin(T=0, X=0, logits=0, W=0, Y=0) == 0 and lin(rows=0, X=0, logits=0, W=0, Y=0) == 0
    # the no-workspace variant validates as the workspace call (invalid arguments only: nothing may launch)
    assert L.roi_masked_linear_fwd_noalloc(None, _fake(A), _fake(B), 2, 4, 1.0, ctypes.byref(st), 4, 128, 64,
                                           _fake(C), None) == 1
    assert L.roi_masked_linear_fwd_noalloc(_fake(D), _fake(A), _fake(B), 2, 4, 1.0, ctypes.byref(st), 257, 128, 64,
                                           _fake(C), None) == 2
    assert L.roi_masked_linear_workspace_size(0, 128, 64) == 0 and L.roi_masked_linear_workspace_size(300, 128, 64) == 0
    # batches: every item validated as the single call, plus no output overlapping any other range
    def fitem(logits=A, W=B, Wm=C, soft=None, hard=None, rows=4, cols=8, state=None):
        return roi.FwdItem(logits, W, Wm, soft, hard, rows, cols, state or roi.NoiseState(0, 0, 0, 1.0, 0))
    def fbatch(*its, N=2, M=4, tau=1.0):
        arr = (roi.FwdItem * len(its))(*its)
        return L.roi_mask_fwd_batch(arr, len(its), N, M, tau, None)
    assert L.roi_mask_fwd_batch(None, 2, 2, 4, 1.0, None) == 1
    assert L.roi_mask_fwd_batch(None, -1, 2, 4, 1.0, None) == 2
    assert L.roi_mask_fwd_batch(None, 0, 2, 4, 1.0, None) == 0
    assert fbatch(fitem(), fitem(logits=0x60000000, W=0x61000000, Wm=0)) == 1
    assert fbatch(fitem(), N=4) == 3 and fbatch(fitem(cols=6)) == 2 and fbatch(fitem(), tau=0.0) == 4
    assert fbatch(fitem(state=roi.NoiseState(0, 0, 0, 0.0, 0))) == 4
    assert fbatch(fitem(hard=D + 4)) == 5
    # item 2's output overlaps item 1's logits; item 2's output overlaps item 1's output
    assert fbatch(fitem(), fitem(logits=0x60000000, W=0x61000000, Wm=A + 16)) == 6
    assert fbatch(fitem(), fitem(logits=0x60000000, W=0x61000000, Wm=C + 32)) == 6
    # inputs may be shared between items; empty items only: nothing to do
    assert fbatch(fitem(rows=0, logits=0, W=0, Wm=0), fitem(rows=0, logits=0, W=0, Wm=0)) == 0
    def bitem(logits=A, W=B, dWm=C, dl=D, dW=None, rows=4, cols=8):
        return roi.BwdItem(logits, W, dWm, dl, dW, rows, cols, roi.NoiseState(0, 0, 0, 1.0, 0))
    def bbatch(*its, N=2, M=4):
        arr = (roi.BwdItem * len(its))(*its)
        return L.roi_mask_bwd_batch(arr, len(its), N, M, 1.0, None)
    assert bbatch(bitem(dl=0)) == 1 and bbatch(bitem(dW=E + 2)) == 5
    assert bbatch(bitem(), bitem(logits=0x60000000, W=0x61000000, dWm=0x62000000, dl=B + 16)) == 6
    # AdamW batch: settings first, then every item; logits, m, v are outputs
    def aitem(logits=A, W=B, dWm=C, m=D, v=E, dl=None, rows=4, cols=8):
        return roi.AdamWItem(logits, W, dWm, m, v, dl, None, rows, cols, roi.NoiseState(0, 0, 0, 1.0, 0))
    def abatch(*its, o=opt):
        arr = (roi.AdamWItem * len(its))(*its)
        return L.roi_mask_bwd_adamw_batch(arr, len(its), 2, 4, 1.0, ctypes.byref(o) if o is not None else None, None)
    assert abatch(aitem(), o=None) == 1 and abatch(aitem(), o=bad) == 9
    assert abatch(aitem(m=0)) == 1 and abatch(aitem(v=E + 4)) == 5
    assert abatch(aitem(), aitem(logits=0x60000000, W=0x61000000, dWm=0x62000000, m=0x63000000, v=D + 64)) == 6
    assert abatch(aitem(rows=0, logits=0, W=0, dWm=0, m=0, v=0)) == 0
    # straight-through batches: dW needs the forward's bits
    def sitem(hard=None, dW=E, dl=D, rows=4, cols=8):
        return roi.BwdStItem(A, B, C, hard, dl, dW, rows, cols, roi.NoiseState(0, 0, 0, 1.0, 0))
    sarr = lambda *its: (roi.BwdStItem * len(its))(*its)
    assert L.roi_mask_bwd_st_batch(sarr(sitem()), 1, 2, 4, 1.0, None) == 1
    assert L.roi_mask_bwd_st_batch(sarr(sitem(hard=0x64000004)), 1, 2, 4, 1.0, None) == 5
    assert L.roi_mask_fwd_st_batch(None, 1, 2, 4, 1.0, None) == 1
    for s in range(10):
        assert L.roi_status_string(s)


def test_anneal_schedule_on_the_host(L):
    from oracle import roi_oracle as O
    for t in (0, 1, 700, 1500, 1999):    # the float result of the float64 formula: within 2 float ulps
        for end in (0.05, 0.002):
            want = float(O.anneal(1.0, end, t, 1500))
            assert abs(L.roi_anneal(1.0, end, t, 1500) - want) <= 2 * 2.0 ** -24 * want


def test_short_form_validates_like_ex(L):
    assert L.roi_mask_fwd(None, _fake(B), 2, 4, 1.0, 0, 0, 4, 8, _fake(C), None, None, None) == 1
    assert L.roi_mask_fwd(_fake(A), _fake(B), 2, 4, -1.0, 0, 0, 4, 8, _fake(C), None, None, None) == 4
