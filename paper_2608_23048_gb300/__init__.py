"""RoI mask-learning hot path on GB300: Python binding of libroi.so.

The binding only marshals arguments: every step of the op runs in the CUDA
library declared by include/roi.h.  Function names are the C names.  Tensors
are torch CUDA tensors (bfloat16 tensors are passed by their bit patterns);
calls are asynchronous on the current torch stream unless `stream` is given.
There is no fallback: if libroi.so is missing the import of the binding's
functions fails loudly.
"""
from __future__ import annotations

import ctypes
import os

__all__ = [
    "RoiError", "NoiseState", "lib", "roi_mask_fwd", "roi_mask_fwd_ex", "roi_mask_bwd",
    "roi_hard_mask_export", "roi_device_status", "roi_status_string", "roi_launch_count",
    "library_path", "hard_words", "roi_noise_words", "roi_gumbel_noise",
    "roi_mask_fwd_st", "roi_mask_bwd_st", "roi_export_compressed_2of4", "AdamW", "roi_mask_bwd_adamw",
    "roi_anneal", "roi_set_ring_wait_limit_ns",
]

_PKG = os.path.dirname(os.path.abspath(__file__))
library_path = os.path.join(_PKG, "libroi.so")

ROI_OK = 0
STATUS_NAMES = {0: "ROI_OK", 1: "ROI_ERR_NULL", 2: "ROI_ERR_SHAPE", 3: "ROI_ERR_NM", 4: "ROI_ERR_TAU",
                5: "ROI_ERR_ALIGN", 6: "ROI_ERR_ALIAS", 7: "ROI_ERR_CUDA", 8: "ROI_ERR_TIMEOUT", 9: "ROI_ERR_OPT"}


class RoiError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)} ({roi_status_string(status)})")


class NoiseState(ctypes.Structure):
    """roi_noise_state: seed, step, tensor_id, lambda (sampling temperature), row_offset."""
    _fields_ = [("seed", ctypes.c_uint64), ("step", ctypes.c_uint32), ("tensor_id", ctypes.c_uint32),
                ("lam", ctypes.c_float), ("row_offset", ctypes.c_int64)]


class AdamW(ctypes.Structure):
    """roi_adamw: lr, beta1, beta2, eps, weight_decay, t (1-based step count)."""
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("eps", ctypes.c_float), ("weight_decay", ctypes.c_float), ("t", ctypes.c_uint32)]


class FwdItem(ctypes.Structure):
    """roi_fwd_item: one tensor of roi_mask_fwd_batch."""
    _fields_ = [("logits", ctypes.c_void_p), ("W", ctypes.c_void_p), ("out_Wm", ctypes.c_void_p),
                ("out_soft", ctypes.c_void_p), ("out_hard", ctypes.c_void_p), ("rows", ctypes.c_int64),
                ("cols", ctypes.c_int64), ("st", NoiseState)]


class BwdItem(ctypes.Structure):
    """roi_bwd_item: one tensor of roi_mask_bwd_batch."""
    _fields_ = [("logits", ctypes.c_void_p), ("W", ctypes.c_void_p), ("dWm", ctypes.c_void_p),
                ("out_dlogits", ctypes.c_void_p), ("out_dW", ctypes.c_void_p), ("rows", ctypes.c_int64),
                ("cols", ctypes.c_int64), ("st", NoiseState)]


class AdamWItem(ctypes.Structure):
    """roi_adamw_item: one tensor of roi_mask_bwd_adamw_batch."""
    _fields_ = [("logits", ctypes.c_void_p), ("W", ctypes.c_void_p), ("dWm", ctypes.c_void_p),
                ("m", ctypes.c_void_p), ("v", ctypes.c_void_p), ("out_dlogits", ctypes.c_void_p),
                ("out_dW", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("st", NoiseState)]


class BwdStItem(ctypes.Structure):
    """roi_bwd_st_item: one tensor of roi_mask_bwd_st_batch."""
    _fields_ = [("logits", ctypes.c_void_p), ("W", ctypes.c_void_p), ("dWm", ctypes.c_void_p),
                ("hard", ctypes.c_void_p), ("out_dlogits", ctypes.c_void_p), ("out_dW", ctypes.c_void_p),
                ("rows", ctypes.c_int64), ("cols", ctypes.c_int64), ("st", NoiseState)]


_LIB = None
_P = ctypes.c_void_p


def lib() -> ctypes.CDLL:
    """The loaded libroi.so with argument types declared (loaded once)."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if not os.path.exists(library_path):
        raise ImportError(f"{library_path} is not built; run `python -m paper_2608_23048_gb300._build` "
                          "(or __graft_entry__.build()) first")
    L = ctypes.CDLL(library_path)
    i32, u32, u64, i64, f32 = ctypes.c_int, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int64, ctypes.c_float
    L.roi_mask_fwd.argtypes = [_P, _P, i32, i32, f32, u64, u32, i64, i64, _P, _P, _P, _P]
    L.roi_mask_fwd_ex.argtypes = [_P, _P, i32, i32, f32, ctypes.POINTER(NoiseState), i64, i64, _P, _P, _P, _P]
    L.roi_mask_bwd.argtypes = [_P, _P, ctypes.POINTER(NoiseState), i32, i32, _P, f32, i64, i64, _P, _P, _P]
    L.roi_mask_fwd_st.argtypes = [_P, _P, i32, i32, f32, ctypes.POINTER(NoiseState), i64, i64, _P, _P, _P, _P]
    L.roi_mask_bwd_st.argtypes = [_P, _P, ctypes.POINTER(NoiseState), i32, i32, _P, _P, f32, i64, i64, _P, _P, _P]
    L.roi_export_compressed_2of4.argtypes = [_P, _P, i64, i64, _P, _P, _P]
    L.roi_mask_bwd_adamw.argtypes = [_P, _P, ctypes.POINTER(NoiseState), i32, i32, _P, f32, i64, i64, _P, _P,
                                     ctypes.POINTER(AdamW), _P, _P, _P]
    L.roi_masked_linear_fwd.argtypes = [_P, _P, _P, i32, i32, f32, ctypes.POINTER(NoiseState), i64, i64, i64, _P,
                                        _P, ctypes.c_size_t, _P]
    L.roi_masked_linear_fwd_noalloc.argtypes = [_P, _P, _P, i32, i32, f32, ctypes.POINTER(NoiseState), i64, i64,
                                                i64, _P, _P]
    L.roi_masked_linear_workspace_size.argtypes = [i64, i64, i64]
    L.roi_masked_linear_workspace_size.restype = ctypes.c_size_t
    L.roi_mask_fwd_batch.argtypes = [ctypes.POINTER(FwdItem), i32, i32, i32, f32, _P]
    L.roi_mask_bwd_batch.argtypes = [ctypes.POINTER(BwdItem), i32, i32, i32, f32, _P]
    L.roi_mask_fwd_st_batch.argtypes = [ctypes.POINTER(FwdItem), i32, i32, i32, f32, _P]
    L.roi_mask_bwd_st_batch.argtypes = [ctypes.POINTER(BwdStItem), i32, i32, i32, f32, _P]
    L.roi_mask_bwd_adamw_batch.argtypes = [ctypes.POINTER(AdamWItem), i32, i32, i32, f32, ctypes.POINTER(AdamW), _P]
    L.roi_anneal.argtypes = [f32, f32, u32, u32]
    L.roi_anneal.restype = f32
    L.roi_hard_mask_export.argtypes = [_P, i32, i32, i64, i64, _P, _P, _P, _P]
    L.roi_device_status.argtypes = [_P]
    L.roi_set_ring_wait_limit_ns.argtypes = [u64]
    L.roi_noise_words.argtypes = [ctypes.POINTER(NoiseState), i64, i64, _P, _P]
    L.roi_gumbel_noise.argtypes = [ctypes.POINTER(NoiseState), i64, i64, _P, _P]
    L.roi_status_string.argtypes = [i32]
    L.roi_status_string.restype = ctypes.c_char_p
    L.roi_launch_count.argtypes = []
    L.roi_launch_count.restype = ctypes.c_uint64
    for name in ("roi_mask_fwd", "roi_mask_fwd_ex", "roi_mask_bwd", "roi_hard_mask_export", "roi_device_status",
                 "roi_noise_words", "roi_gumbel_noise", "roi_mask_fwd_st", "roi_mask_bwd_st",
                 "roi_export_compressed_2of4", "roi_mask_bwd_adamw", "roi_masked_linear_fwd",
                 "roi_masked_linear_fwd_noalloc", "roi_mask_fwd_batch", "roi_mask_bwd_batch",
                 "roi_mask_bwd_adamw_batch", "roi_mask_fwd_st_batch", "roi_mask_bwd_st_batch",
                 "roi_set_ring_wait_limit_ns"):
        getattr(L, name).restype = i32
    _LIB = L
    return L


def roi_status_string(status: int) -> str:
    return lib().roi_status_string(int(status)).decode()


def roi_launch_count() -> int:
    return int(lib().roi_launch_count())


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _check_tensor(t, name, dtype, shape=None):
    import torch
    if t is None:
        return
    if t.dtype != dtype:
        raise TypeError(f"{name}: expected {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name}: expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name}: must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: expected shape {tuple(shape)}, got {tuple(t.shape)}")


def hard_words(rows: int, cols: int) -> int:
    """uint32 words of a hard mask over rows * cols elements."""
    return (rows * cols + 31) // 32


def _raise(status, where):
    if status != ROI_OK:
        raise RoiError(status, where)


def roi_mask_fwd_ex(logits, W, N, M, tau, state: NoiseState, out_Wm, out_soft=None, out_hard=None, stream=None):
    """Forward with full noise state; outputs are written in place.  Returns None."""
    import torch
    rows, cols = logits.shape
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(out_Wm, "out_Wm", torch.bfloat16, (rows, cols))
    _check_tensor(out_soft, "out_soft", torch.float32, (rows, cols))
    _check_tensor(out_hard, "out_hard", torch.int32, (hard_words(rows, cols),))
    st = state if isinstance(state, NoiseState) else NoiseState(*state)
    s = lib().roi_mask_fwd_ex(_ptr(logits), _ptr(W), int(N), int(M), float(tau), ctypes.byref(st), rows, cols,
                              _ptr(out_Wm), _ptr(out_soft), _ptr(out_hard), _stream(stream))
    _raise(s, "roi_mask_fwd_ex")


def _addr(t):
    return None if t is None else t.data_ptr()


def make_fwd_items(items):
    """ctypes array of FwdItem from (logits, W, state, out_Wm, out_soft, out_hard) tuples."""
    import torch
    arr = (FwdItem * len(items))()
    for k, (logits, W, state, out_Wm, out_soft, out_hard) in enumerate(items):
        rows, cols = logits.shape
        _check_tensor(logits, "logits", torch.float32)
        _check_tensor(W, "W", torch.bfloat16, (rows, cols))
        _check_tensor(out_Wm, "out_Wm", torch.bfloat16, (rows, cols))
        _check_tensor(out_soft, "out_soft", torch.float32, (rows, cols))
        _check_tensor(out_hard, "out_hard", torch.int32, (hard_words(rows, cols),))
        st = state if isinstance(state, NoiseState) else NoiseState(*state)
        arr[k] = FwdItem(_addr(logits), _addr(W), _addr(out_Wm), _addr(out_soft), _addr(out_hard), rows, cols, st)
    return arr


def make_bwd_items(items):
    """ctypes array of BwdItem from (logits, W, state, dWm, out_dlogits, out_dW) tuples."""
    import torch
    arr = (BwdItem * len(items))()
    for k, (logits, W, state, dWm, out_dlogits, out_dW) in enumerate(items):
        rows, cols = logits.shape
        _check_tensor(logits, "logits", torch.float32)
        _check_tensor(W, "W", torch.bfloat16, (rows, cols))
        _check_tensor(dWm, "dWm", torch.bfloat16, (rows, cols))
        _check_tensor(out_dlogits, "out_dlogits", torch.float32, (rows, cols))
        _check_tensor(out_dW, "out_dW", torch.bfloat16, (rows, cols))
        st = state if isinstance(state, NoiseState) else NoiseState(*state)
        arr[k] = BwdItem(_addr(logits), _addr(W), _addr(dWm), _addr(out_dlogits), _addr(out_dW), rows, cols, st)
    return arr


def make_adamw_items(items):
    """ctypes array of AdamWItem from (logits, W, state, dWm, m, v, out_dlogits, out_dW) tuples."""
    import torch
    arr = (AdamWItem * len(items))()
    for k, (logits, W, state, dWm, m, v, out_dlogits, out_dW) in enumerate(items):
        rows, cols = logits.shape
        _check_tensor(logits, "logits", torch.float32)
        for name, t, dt in (("W", W, torch.bfloat16), ("dWm", dWm, torch.bfloat16), ("m", m, torch.float32),
                            ("v", v, torch.float32), ("out_dlogits", out_dlogits, torch.float32),
                            ("out_dW", out_dW, torch.bfloat16)):
            _check_tensor(t, name, dt, (rows, cols))
        st = state if isinstance(state, NoiseState) else NoiseState(*state)
        arr[k] = AdamWItem(_addr(logits), _addr(W), _addr(dWm), _addr(m), _addr(v), _addr(out_dlogits),
                           _addr(out_dW), rows, cols, st)
    return arr


def roi_mask_bwd_adamw_batch(items, N, M, tau, opt: AdamW, stream=None):
    """Backward fused with the logits' AdamW step for many tensors (AdamWItem array from
    make_adamw_items, or a list of (logits, W, state, dWm, m, v, out_dlogits, out_dW) tuples)."""
    arr = items if isinstance(items, ctypes.Array) else make_adamw_items(items)
    s = lib().roi_mask_bwd_adamw_batch(arr, len(arr), int(N), int(M), float(tau), ctypes.byref(opt), _stream(stream))
    _raise(s, "roi_mask_bwd_adamw_batch")


def make_bwd_st_items(items):
    """ctypes array of BwdStItem from (logits, W, state, dWm, hard, out_dlogits, out_dW) tuples."""
    import torch
    arr = (BwdStItem * len(items))()
    for k, (logits, W, state, dWm, hard, out_dlogits, out_dW) in enumerate(items):
        rows, cols = logits.shape
        _check_tensor(logits, "logits", torch.float32)
        _check_tensor(W, "W", torch.bfloat16, (rows, cols))
        _check_tensor(dWm, "dWm", torch.bfloat16, (rows, cols))
        _check_tensor(hard, "hard", torch.int32, (hard_words(rows, cols),))
        _check_tensor(out_dlogits, "out_dlogits", torch.float32, (rows, cols))
        _check_tensor(out_dW, "out_dW", torch.bfloat16, (rows, cols))
        st = state if isinstance(state, NoiseState) else NoiseState(*state)
        arr[k] = BwdStItem(_addr(logits), _addr(W), _addr(dWm), _addr(hard), _addr(out_dlogits), _addr(out_dW),
                           rows, cols, st)
    return arr


def roi_mask_fwd_st_batch(items, N, M, tau, stream=None):
    """Straight-through forward of many tensors (items as for roi_mask_fwd_batch)."""
    arr = items if isinstance(items, ctypes.Array) else make_fwd_items(items)
    s = lib().roi_mask_fwd_st_batch(arr, len(arr), int(N), int(M), float(tau), _stream(stream))
    _raise(s, "roi_mask_fwd_st_batch")


def roi_mask_bwd_st_batch(items, N, M, tau, stream=None):
    """Straight-through backward of many tensors (BwdStItem array from make_bwd_st_items,
    or a list of (logits, W, state, dWm, hard, out_dlogits, out_dW) tuples)."""
    arr = items if isinstance(items, ctypes.Array) else make_bwd_st_items(items)
    s = lib().roi_mask_bwd_st_batch(arr, len(arr), int(N), int(M), float(tau), _stream(stream))
    _raise(s, "roi_mask_bwd_st_batch")


def roi_mask_fwd_batch(items, N, M, tau, stream=None):
    """Forward of many tensors in one call.  `items`: a FwdItem array from make_fwd_items
    (reusable across calls while its tensors live; update .st.step per step) or a list
    of (logits, W, state, out_Wm, out_soft, out_hard) tuples."""
    arr = items if isinstance(items, ctypes.Array) else make_fwd_items(items)
    s = lib().roi_mask_fwd_batch(arr, len(arr), int(N), int(M), float(tau), _stream(stream))
    _raise(s, "roi_mask_fwd_batch")


def roi_mask_bwd_batch(items, N, M, tau, stream=None):
    """Backward of many tensors in one call (BwdItem array from make_bwd_items, or a list
    of (logits, W, state, dWm, out_dlogits, out_dW) tuples)."""
    arr = items if isinstance(items, ctypes.Array) else make_bwd_items(items)
    s = lib().roi_mask_bwd_batch(arr, len(arr), int(N), int(M), float(tau), _stream(stream))
    _raise(s, "roi_mask_bwd_batch")


def roi_mask_fwd(logits, W, N, M, tau, seed, step, out_Wm, out_soft=None, out_hard=None, stream=None):
    """Forward, short form (lambda = 1, tensor_id = 0, row_offset = 0)."""
    import torch
    rows, cols = logits.shape
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(out_Wm, "out_Wm", torch.bfloat16, (rows, cols))
    _check_tensor(out_soft, "out_soft", torch.float32, (rows, cols))
    _check_tensor(out_hard, "out_hard", torch.int32, (hard_words(rows, cols),))
    s = lib().roi_mask_fwd(_ptr(logits), _ptr(W), int(N), int(M), float(tau), int(seed), int(step), rows, cols,
                           _ptr(out_Wm), _ptr(out_soft), _ptr(out_hard), _stream(stream))
    _raise(s, "roi_mask_fwd")


def roi_mask_bwd(logits, W, state: NoiseState, N, M, dWm, tau, out_dlogits, out_dW=None, stream=None):
    """Backward: logit gradients (overwritten) and optionally dW."""
    import torch
    rows, cols = logits.shape
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(dWm, "dWm", torch.bfloat16, (rows, cols))
    _check_tensor(out_dlogits, "out_dlogits", torch.float32, (rows, cols))
    _check_tensor(out_dW, "out_dW", torch.bfloat16, (rows, cols))
    st = state if isinstance(state, NoiseState) else NoiseState(*state)
    s = lib().roi_mask_bwd(_ptr(logits), _ptr(W), ctypes.byref(st), int(N), int(M), _ptr(dWm), float(tau),
                           rows, cols, _ptr(out_dlogits), _ptr(out_dW), _stream(stream))
    _raise(s, "roi_mask_bwd")


def roi_mask_fwd_st(logits, W, N, M, tau, state: NoiseState, out_Wm, out_soft=None, out_hard=None, stream=None):
    """Straight-through forward: Wm = W where the Gumbel-top-N hard mask is set, +0 elsewhere."""
    import torch
    rows, cols = logits.shape
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(out_Wm, "out_Wm", torch.bfloat16, (rows, cols))
    _check_tensor(out_soft, "out_soft", torch.float32, (rows, cols))
    _check_tensor(out_hard, "out_hard", torch.int32, (hard_words(rows, cols),))
    st = state if isinstance(state, NoiseState) else NoiseState(*state)
    s = lib().roi_mask_fwd_st(_ptr(logits), _ptr(W), int(N), int(M), float(tau), ctypes.byref(st), rows, cols,
                              _ptr(out_Wm), _ptr(out_soft), _ptr(out_hard), _stream(stream))
    _raise(s, "roi_mask_fwd_st")


def roi_mask_bwd_st(logits, W, state: NoiseState, N, M, dWm, hard, tau, out_dlogits, out_dW=None, stream=None):
    """Straight-through backward: logit gradients through the relaxation; dW = dWm where
    the forward's hard mask (`hard`, its out_hard words) is set."""
    import torch
    rows, cols = logits.shape
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(dWm, "dWm", torch.bfloat16, (rows, cols))
    _check_tensor(hard, "hard", torch.int32, (hard_words(rows, cols),))
    _check_tensor(out_dlogits, "out_dlogits", torch.float32, (rows, cols))
    _check_tensor(out_dW, "out_dW", torch.bfloat16, (rows, cols))
    st = state if isinstance(state, NoiseState) else NoiseState(*state)
    s = lib().roi_mask_bwd_st(_ptr(logits), _ptr(W), ctypes.byref(st), int(N), int(M), _ptr(dWm), _ptr(hard),
                              float(tau), rows, cols, _ptr(out_dlogits), _ptr(out_dW), _stream(stream))
    _raise(s, "roi_mask_bwd_st")


def roi_mask_bwd_adamw(logits, W, state: NoiseState, N, M, dWm, tau, m, v, opt: AdamW, out_dlogits=None,
                       out_dW=None, stream=None):
    """Backward fused with one AdamW step: `logits`, `m`, `v` are updated in place."""
    import torch
    rows, cols = logits.shape
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(dWm, "dWm", torch.bfloat16, (rows, cols))
    _check_tensor(m, "m", torch.float32, (rows, cols))
    _check_tensor(v, "v", torch.float32, (rows, cols))
    _check_tensor(out_dlogits, "out_dlogits", torch.float32, (rows, cols))
    _check_tensor(out_dW, "out_dW", torch.bfloat16, (rows, cols))
    st = state if isinstance(state, NoiseState) else NoiseState(*state)
    s = lib().roi_mask_bwd_adamw(_ptr(logits), _ptr(W), ctypes.byref(st), int(N), int(M), _ptr(dWm), float(tau),
                                 rows, cols, _ptr(m), _ptr(v), ctypes.byref(opt), _ptr(out_dlogits), _ptr(out_dW),
                                 _stream(stream))
    _raise(s, "roi_mask_bwd_adamw")


def roi_anneal(init, end, t, T_anneal):
    """Eq. 13: max(end, init * (end / init) ** (t / T_anneal)), evaluated by the library."""
    return float(lib().roi_anneal(float(init), float(end), int(t), int(T_anneal)))


def roi_export_compressed_2of4(logits, W, out_values, out_meta, stream=None):
    """Compressed 2:4 export: kept weights [rows, cols/2] and 4-bit index codes, 8 groups per word."""
    import torch
    rows, cols = logits.shape
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(out_values, "out_values", torch.bfloat16, (rows, cols // 2))
    _check_tensor(out_meta, "out_meta", torch.int32, ((rows * cols) // 32,))
    s = lib().roi_export_compressed_2of4(_ptr(logits), _ptr(W), rows, cols, _ptr(out_values), _ptr(out_meta),
                                         _stream(stream))
    _raise(s, "roi_export_compressed_2of4")


def roi_masked_linear_workspace_size(T, rows, cols) -> int:
    """Bytes of workspace that let roi_masked_linear_fwd split K fully on the current device."""
    return int(lib().roi_masked_linear_workspace_size(int(T), int(rows), int(cols)))


def roi_masked_linear_fwd(X, logits, W, N, M, tau, state: NoiseState, out_Y, workspace=None, stream=None):
    """Y[T, rows] = X[T, cols] @ bf16(W * S)^T with the mask formed inside the GEMM (float32 Y)."""
    import torch
    rows, cols = logits.shape
    T = X.shape[0]
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(X, "X", torch.bfloat16, (T, cols))
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(out_Y, "out_Y", torch.float32, (T, rows))
    ws_bytes = 0
    if workspace is not None:
        _check_tensor(workspace, "workspace", workspace.dtype)
        ws_bytes = workspace.numel() * workspace.element_size()
    st = state if isinstance(state, NoiseState) else NoiseState(*state)
    s = lib().roi_masked_linear_fwd(_ptr(X), _ptr(logits), _ptr(W), int(N), int(M), float(tau), ctypes.byref(st), T,
                                    rows, cols, _ptr(out_Y), _ptr(workspace), ws_bytes, _stream(stream))
    _raise(s, "roi_masked_linear_fwd")


def roi_masked_linear_fwd_noalloc(X, logits, W, N, M, tau, state: NoiseState, out_Y, stream=None):
    """roi_masked_linear_fwd with the library's static split-K scratch (no workspace argument)."""
    import torch
    rows, cols = logits.shape
    T = X.shape[0]
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(X, "X", torch.bfloat16, (T, cols))
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(out_Y, "out_Y", torch.float32, (T, rows))
    st = state if isinstance(state, NoiseState) else NoiseState(*state)
    s = lib().roi_masked_linear_fwd_noalloc(_ptr(X), _ptr(logits), _ptr(W), int(N), int(M), float(tau),
                                            ctypes.byref(st), T, rows, cols, _ptr(out_Y), _stream(stream))
    _raise(s, "roi_masked_linear_fwd_noalloc")


def roi_hard_mask_export(logits, N, M, out_bits, W=None, out_Wpruned=None, stream=None):
    """Deployment mask argtop_N(logits) (+ pruned weights)."""
    import torch
    rows, cols = logits.shape
    _check_tensor(logits, "logits", torch.float32)
    _check_tensor(out_bits, "out_bits", torch.int32, (hard_words(rows, cols),))
    _check_tensor(W, "W", torch.bfloat16, (rows, cols))
    _check_tensor(out_Wpruned, "out_Wpruned", torch.bfloat16, (rows, cols))
    s = lib().roi_hard_mask_export(_ptr(logits), int(N), int(M), rows, cols, _ptr(out_bits), _ptr(W),
                                   _ptr(out_Wpruned), _stream(stream))
    _raise(s, "roi_hard_mask_export")


def roi_noise_words(state: NoiseState, rows, cols, out_words, stream=None):
    """Philox words of every element of a [rows, cols] call (int32 tensor of rows*cols)."""
    import torch
    _check_tensor(out_words, "out_words", torch.int32, (rows * cols,))
    st = state if isinstance(state, NoiseState) else NoiseState(*state)
    _raise(lib().roi_noise_words(ctypes.byref(st), rows, cols, _ptr(out_words), _stream(stream)), "roi_noise_words")


def roi_gumbel_noise(state: NoiseState, rows, cols, out_g, stream=None):
    """Gumbel noise of every element of a [rows, cols] call (float32 tensor of rows*cols)."""
    import torch
    _check_tensor(out_g, "out_g", torch.float32, (rows * cols,))
    st = state if isinstance(state, NoiseState) else NoiseState(*state)
    _raise(lib().roi_gumbel_noise(ctypes.byref(st), rows, cols, _ptr(out_g), _stream(stream)), "roi_gumbel_noise")


def roi_device_status(stream=None):
    """Synchronises the stream; raises RoiError if a kernel timed out or CUDA failed."""
    _raise(lib().roi_device_status(_stream(stream)), "roi_device_status")


ROI_DEFAULT_RING_WAIT_NS = 2_000_000_000


def roi_set_ring_wait_limit_ns(ns: int):
    """Wall-time limit (ns) of the kernels' waits for their staged copies on the
    current device; 0 gives up at once when a stage has not landed (tests)."""
    _raise(lib().roi_set_ring_wait_limit_ns(int(ns)), "roi_set_ring_wait_limit_ns")
