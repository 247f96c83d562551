"""Python binding of libdarb (include/darb.h): argument marshalling only.

Every function has the name of the C call it wraps and forwards torch tensors
as raw device pointers plus the current CUDA stream.  All arithmetic happens in
the library's CUDA kernels; if ``libdarb.so`` is missing or a call fails, a
``DarbError`` is raised -- there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdarb.so")

OK, ERR_INVALID_ARG, ERR_NONFINITE, ERR_OOM, ERR_CUDA, ERR_TIMEOUT, ERR_UNSUPPORTED = range(7)
F32, BF16 = 0, 1
PATH_AUTO, PATH_CUDA_CORES, PATH_TENSOR_CORES = 0, 1, 2
MAX_BLOCK = 256

_lock = threading.Lock()
_lib = None


class DarbError(RuntimeError):
    def __init__(self, status: int, call: str):
        name = status_string(status) if _lib is not None else str(status)
        super().__init__(f"{call} failed: {name}")
        self.status = status


class _Info(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int64), ("cols", ctypes.c_int64), ("nnzb", ctypes.c_int64),
                ("wtype", ctypes.c_int), ("nbins", ctypes.c_int32), ("ngroups", ctypes.c_int32),
                ("value_bytes", ctypes.c_int64), ("offset_bytes", ctypes.c_int64),
                ("meta_bytes", ctypes.c_int64), ("index_bits_min", ctypes.c_int64),
                ("device_bytes", ctypes.c_int64)]


def lib():
    """The loaded libdarb.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise DarbError(ERR_CUDA, f"load {LIB_PATH} (not built; run __graft_entry__.build())")
            L = ctypes.CDLL(LIB_PATH)
            P, I64, I32, S = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p
            sig = {
                "darb_assign_block_sizes": [P, I64, I64, I32, I32, P],
                "darb_assign_from_weights": [P, ctypes.c_int, I64, I64, I64, I64, I32, I32, P, P, S],
                "darb_encode": [P, ctypes.c_int, I64, I64, I64, P, P, S],
                "darb_reencode": [P, P, I64, S],
                "darb_reencode_host": [P, P, I64, P, S],
                "darb_sync_status": [P, S],
                "darb_spmm": [P, P, I64, I64, P, I64, S],
                "darb_spmm_ex": [P, P, I64, I64, P, I64, ctypes.c_int, S],
                "darb_spmm_host": [P, P, I64, I64, P, I64, P, P, S],
                "darb_spmm_path": [P, I64, P, P],
                "darb_lstm_step": [P, I64, I64, I64, P, P, P, P, P, P, S],
                "darb_lstm_step_noalloc": [P, I64, I64, I64, P, P, P, P, P, P, S],
                "darb_gru_step": [P, I64, I64, I64, P, P, P, P, P, S],
                "darb_lstm_sequence": [P, I64, I64, I64, I64, P, P, P, P, P, P, P, S],
                "darb_gru_sequence": [P, I64, I64, I64, I64, P, P, P, P, P, S],
                "darb_rnn_reserve": [P, I64],
                "darb_info": [P, P],
                "darb_export": [P, P, P, P, P],
                "darb_import": [P, P, P, ctypes.c_int, I64, I64, P, S],
                "darb_destroy": [P],
                "darb_set_pdl": [ctypes.c_int],
            }
            for name, args in sig.items():
                fn = getattr(L, name)
                fn.argtypes = args
                fn.restype = ctypes.c_int
            L.darb_status_string.argtypes = [ctypes.c_int]
            L.darb_status_string.restype = ctypes.c_char_p
            _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().darb_status_string(int(status)).decode()


def _check(status: int, call: str):
    if status != OK:
        raise DarbError(status, call)


def _ptr(t) -> int | None:
    if t is None:
        return None
    return int(t.data_ptr())


def _stream(stream) -> int | None:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise DarbError(ERR_INVALID_ARG, f"dtype {t.dtype} (need float32 or bfloat16)")


def _require_cuda_f32(t, name):
    import torch
    if t is None:
        return
    if not t.is_cuda or t.dtype != torch.float32:
        raise DarbError(ERR_INVALID_ARG, f"{name} must be a CUDA float32 tensor")


@dataclass
class Handle:
    """An encoded DARB matrix living on the GPU (owned; free with darb_destroy)."""
    ptr: int
    rows: int
    cols: int
    wtype: int

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        darb_destroy(self)


def darb_assign_block_sizes(row_nnz, cols: int, m_min: int = 1, m_max: int = MAX_BLOCK) -> np.ndarray:
    nnz = np.ascontiguousarray(row_nnz, dtype=np.int64)
    out = np.zeros(nnz.shape[0], dtype=np.int32)
    _check(lib().darb_assign_block_sizes(nnz.ctypes.data, nnz.shape[0], int(cols), int(m_min),
                                         int(m_max), out.ctypes.data), "darb_assign_block_sizes")
    return out


def darb_assign_from_weights(W, keep: int, m_min: int = 1, m_max: int = MAX_BLOCK, stream=None,
                             ldw: int | None = None):
    """(row_nnz, m): each row's count of the `keep` weights of largest magnitude of
    the CUDA tensor W (rows x cols, float32 or bfloat16) and the block sizes they give."""
    code = _dtype_code(W)
    if W.dim() != 2 or not W.is_cuda or W.stride(1) != 1:
        raise DarbError(ERR_INVALID_ARG, "darb_assign_from_weights: W must be a 2-D CUDA tensor with unit column stride")
    rows, cols = W.shape
    ldw = W.stride(0) if ldw is None else ldw
    nnz = np.zeros(rows, dtype=np.int64)
    m = np.zeros(rows, dtype=np.int32)
    _check(lib().darb_assign_from_weights(_ptr(W), code, rows, cols, int(ldw), int(keep), int(m_min), int(m_max),
                                          nnz.ctypes.data, m.ctypes.data, _stream(stream)),
           "darb_assign_from_weights")
    return nnz, m


def darb_encode(W, m, stream=None, ldw: int | None = None) -> Handle:
    """Encode a CUDA tensor W (rows x cols, float32 or bfloat16) with block sizes m."""
    code = _dtype_code(W)
    if W.dim() != 2 or not W.is_cuda or W.stride(1) != 1:
        raise DarbError(ERR_INVALID_ARG, "darb_encode: W must be a 2-D CUDA tensor with unit column stride")
    rows, cols = W.shape
    ldw = W.stride(0) if ldw is None else ldw
    mm = np.ascontiguousarray(m, dtype=np.int32)
    if mm.shape != (rows,):
        raise DarbError(ERR_INVALID_ARG, "darb_encode: m must have one entry per row")
    out = ctypes.c_void_p()
    _check(lib().darb_encode(_ptr(W), code, rows, cols, ldw, mm.ctypes.data, ctypes.byref(out),
                             _stream(stream)), "darb_encode")
    return Handle(out.value, rows, cols, code)


def darb_reencode(h: Handle, W, stream=None):
    _check(lib().darb_reencode(h.ptr, _ptr(W), W.stride(0), _stream(stream)), "darb_reencode")


def darb_reencode_host(h: Handle, W, W_dev, stream=None):
    """darb_reencode from a host W (CPU tensor, rows x cols, row stride ldw) through
    the caller's device buffer W_dev (same shape and row stride)."""
    if W.is_cuda or not W_dev.is_cuda or W.dtype != W_dev.dtype:
        raise DarbError(ERR_INVALID_ARG, "darb_reencode_host: W on the host, W_dev on the device, one dtype")
    if W.shape != W_dev.shape or W.stride() != W_dev.stride() or W.stride(1) != 1:
        raise DarbError(ERR_INVALID_ARG, "darb_reencode_host: W and W_dev of one row-major layout")
    _check(lib().darb_reencode_host(h.ptr, _ptr(W), W.stride(0), _ptr(W_dev), _stream(stream)),
           "darb_reencode_host")


def darb_sync_status(h: Handle, stream=None):
    """Synchronise and raise if the handle's kernels recorded a NaN or a timeout."""
    _check(lib().darb_sync_status(h.ptr, _stream(stream)), "darb_sync_status")


def darb_spmm(h: Handle, X, Y=None, stream=None):
    """Y = W_darb X for X (cols x batch, CUDA float32); returns Y."""
    return darb_spmm_ex(h, X, Y, PATH_AUTO, stream)


def darb_spmm_ex(h: Handle, X, Y=None, path: int = PATH_AUTO, stream=None):
    """darb_spmm with the kernel family chosen (PATH_AUTO, PATH_CUDA_CORES, PATH_TENSOR_CORES)."""
    import torch
    _require_cuda_f32(X, "X")
    if X.dim() == 1:
        X = X.view(-1, 1)
    if X.stride(1) != 1 and X.shape[1] > 1:
        raise DarbError(ERR_INVALID_ARG, "darb_spmm: X must have a contiguous batch dimension")
    batch = X.shape[1]
    if Y is None:
        Y = torch.empty((h.rows, batch), dtype=torch.float32, device=X.device)
    _require_cuda_f32(Y, "Y")
    ldx = X.stride(0) if X.shape[0] > 1 else batch
    ldy = Y.stride(0) if Y.shape[0] > 1 else batch
    if path == PATH_AUTO:
        _check(lib().darb_spmm(h.ptr, _ptr(X), ldx, batch, _ptr(Y), ldy, _stream(stream)), "darb_spmm")
    else:
        _check(lib().darb_spmm_ex(h.ptr, _ptr(X), ldx, batch, _ptr(Y), ldy, int(path), _stream(stream)),
               "darb_spmm_ex")
    return Y


def darb_spmm_host(h: Handle, X, Y, X_dev, Y_dev, stream=None):
    """darb_spmm with X (cols x batch) and Y (rows x batch) host float32 tensors
    (rows strided, columns contiguous) through the caller's dense device buffers
    X_dev (cols x batch) and Y_dev (rows x batch); returns Y."""
    import torch
    for t, n, cuda in ((X, "X", False), (Y, "Y", False), (X_dev, "X_dev", True), (Y_dev, "Y_dev", True)):
        if t.dtype != torch.float32 or t.is_cuda != cuda or t.dim() != 2 or (t.shape[1] > 1 and t.stride(1) != 1):
            raise DarbError(ERR_INVALID_ARG, f"darb_spmm_host: {n} must be a 2-D float32 "
                                             f"{'CUDA' if cuda else 'host'} tensor with contiguous columns")
    batch = X.shape[1]
    if (X_dev.shape != X.shape or Y.shape != (h.rows, batch) or Y_dev.shape != Y.shape or
            not X_dev.is_contiguous() or not Y_dev.is_contiguous()):
        raise DarbError(ERR_INVALID_ARG, "darb_spmm_host: shapes, or device buffers not dense")
    ldx = X.stride(0) if X.shape[0] > 1 else batch
    ldy = Y.stride(0) if Y.shape[0] > 1 else batch
    _check(lib().darb_spmm_host(h.ptr, _ptr(X), ldx, batch, _ptr(Y), ldy, _ptr(X_dev), _ptr(Y_dev),
                                _stream(stream)), "darb_spmm_host")
    return Y


def darb_spmm_path(h: Handle, batch: int) -> tuple[int, int]:
    """(path, kernels): the kernel family darb_spmm takes for this batch and its launches per call."""
    path, kernels = ctypes.c_int(), ctypes.c_int32()
    _check(lib().darb_spmm_path(h.ptr, int(batch), ctypes.byref(path), ctypes.byref(kernels)), "darb_spmm_path")
    return path.value, kernels.value


def darb_lstm_step(h: Handle, I: int, H: int, B: int, x, h_prev, c_prev, bias, h_out, c_out,
                   stream=None):
    for t, n in ((x, "x"), (h_prev, "h_prev"), (c_prev, "c_prev"), (bias, "bias"),
                 (h_out, "h_out"), (c_out, "c_out")):
        _require_cuda_f32(t, n)
    _check(lib().darb_lstm_step(h.ptr, I, H, B, _ptr(x), _ptr(h_prev), _ptr(c_prev), _ptr(bias),
                                _ptr(h_out), _ptr(c_out), _stream(stream)), "darb_lstm_step")


def darb_lstm_step_noalloc(h: Handle, I: int, H: int, B: int, x, h_prev, c_prev, bias, h_out, c_out,
                           stream=None):
    """darb_lstm_step with its scratch in the library's fixed 4 MiB array: no
    allocation at call time (for callers that cannot let a library allocate)."""
    for t, n in ((x, "x"), (h_prev, "h_prev"), (c_prev, "c_prev"), (bias, "bias"),
                 (h_out, "h_out"), (c_out, "c_out")):
        _require_cuda_f32(t, n)
    _check(lib().darb_lstm_step_noalloc(h.ptr, I, H, B, _ptr(x), _ptr(h_prev), _ptr(c_prev),
                                        _ptr(bias), _ptr(h_out), _ptr(c_out), _stream(stream)),
           "darb_lstm_step_noalloc")


def darb_gru_step(h: Handle, I: int, H: int, B: int, x, h_prev, b_ih, b_hh, h_out, stream=None):
    for t, n in ((x, "x"), (h_prev, "h_prev"), (b_ih, "b_ih"), (b_hh, "b_hh"), (h_out, "h_out")):
        _require_cuda_f32(t, n)
    _check(lib().darb_gru_step(h.ptr, I, H, B, _ptr(x), _ptr(h_prev), _ptr(b_ih), _ptr(b_hh),
                               _ptr(h_out), _stream(stream)), "darb_gru_step")


def darb_lstm_sequence(h: Handle, T: int, I: int, H: int, B: int, x_seq, h0, c0, bias, h_seq,
                       c_seq=None, c_last=None, stream=None):
    """T LSTM steps in one persistent launch: x_seq (T, I, B) -> h_seq (T, H, B),
    optionally every c_t (c_seq) and the last c (c_last)."""
    for t, n in ((x_seq, "x_seq"), (h0, "h0"), (c0, "c0"), (bias, "bias"), (h_seq, "h_seq"),
                 (c_seq, "c_seq"), (c_last, "c_last")):
        _require_cuda_f32(t, n)
    _check(lib().darb_lstm_sequence(h.ptr, T, I, H, B, _ptr(x_seq), _ptr(h0), _ptr(c0), _ptr(bias),
                                    _ptr(h_seq), _ptr(c_seq), _ptr(c_last), _stream(stream)),
           "darb_lstm_sequence")


def darb_gru_sequence(h: Handle, T: int, I: int, H: int, B: int, x_seq, h0, b_ih, b_hh, h_seq, stream=None):
    """T GRU steps in one persistent launch: x_seq (T, I, B) -> h_seq (T, H, B)."""
    for t, n in ((x_seq, "x_seq"), (h0, "h0"), (b_ih, "b_ih"), (b_hh, "b_hh"), (h_seq, "h_seq")):
        _require_cuda_f32(t, n)
    _check(lib().darb_gru_sequence(h.ptr, T, I, H, B, _ptr(x_seq), _ptr(h0), _ptr(b_ih), _ptr(b_hh),
                                   _ptr(h_seq), _stream(stream)), "darb_gru_sequence")


def darb_rnn_reserve(h: Handle, max_batch: int):
    _check(lib().darb_rnn_reserve(h.ptr, int(max_batch)), "darb_rnn_reserve")


def darb_info(h: Handle) -> dict:
    info = _Info()
    _check(lib().darb_info(h.ptr, ctypes.byref(info)), "darb_info")
    return {name: getattr(info, name) for name, _ in _Info._fields_}


def darb_export(h: Handle):
    """(val, off, blk_ptr, m) in canonical (row, j) block order; val is float32 or uint16 bf16 bits."""
    info = darb_info(h)
    nnzb = info["nnzb"]
    val = np.zeros(nnzb, dtype=np.uint16 if h.wtype == BF16 else np.float32)
    off = np.zeros(nnzb, dtype=np.uint8)
    bp = np.zeros(h.rows + 1, dtype=np.int64)
    m = np.zeros(h.rows, dtype=np.int32)
    _check(lib().darb_export(h.ptr, val.ctypes.data, off.ctypes.data, bp.ctypes.data, m.ctypes.data),
           "darb_export")
    return val, off, bp, m


def darb_import(val, off, m, wtype: int, rows: int, cols: int, stream=None) -> Handle:
    v = np.ascontiguousarray(val, dtype=np.uint16 if wtype == BF16 else np.float32)
    o = np.ascontiguousarray(off, dtype=np.uint8)
    mm = np.ascontiguousarray(m, dtype=np.int32)
    out = ctypes.c_void_p()
    _check(lib().darb_import(v.ctypes.data, o.ctypes.data, mm.ctypes.data, int(wtype), int(rows),
                             int(cols), ctypes.byref(out), _stream(stream)), "darb_import")
    return Handle(out.value, rows, cols, wtype)


def darb_destroy(h: Handle | None):
    if h is None or h.ptr is None:
        return
    _check(lib().darb_destroy(h.ptr), "darb_destroy")
    h.ptr = None


def darb_set_pdl(enabled: bool):
    """Launch the library's kernels with (default) or without programmatic dependent launch."""
    _check(lib().darb_set_pdl(1 if enabled else 0), "darb_set_pdl")
