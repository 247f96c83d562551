"""Python binding of libdarb_baselines (include/darb_baselines.h) and the host
construction of its inputs.

The comparison of Sec. 4.2 restated on a GPU: the same kept weights as a CSR
matrix (irregular pruning, Sec. 2) and block-pruned matrices of the same
density as BSR, multiplied by cuSPARSE.  Building the CSR and BSR arrays is
host-side numpy work (once per matrix, off any timed path); the products run
in the vendor library.  If ``libdarb_baselines.so`` is missing a ``DarbError``
is raised.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

from . import darb

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libdarb_baselines.so")

_lock = threading.Lock()
_lib = None


def lib():
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise darb.DarbError(darb.ERR_CUDA, f"load {LIB_PATH} (not built; run __graft_entry__.build())")
            L = ctypes.CDLL(LIB_PATH)
            P, I64, S, E = ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_int
            L.darb_baseline_csr_spmm.argtypes = [P, P, P, I64, I64, I64, P, I64, I64, P, I64, E, S]
            L.darb_baseline_bsr_spmm.argtypes = [P, P, P, I64, I64, I64, I64, P, I64, I64, P, I64, E, S]
            L.darb_baseline_csr_spmm.restype = ctypes.c_int
            L.darb_baseline_bsr_spmm.restype = ctypes.c_int
            _lib = L
    return _lib


def csr_from_darb(h: darb.Handle):
    """(row_ptr int32, col_idx int32, vals fp32) of exactly the handle's kept weights."""
    val, off, bp, m = darb.darb_export(h)
    rows = len(m)
    vals = val.astype(np.float32) if val.dtype != np.uint16 else (val.astype(np.uint32) << 16).view(np.float32)
    row_of = np.repeat(np.arange(rows), np.diff(bp))
    j = np.arange(bp[-1]) - bp[row_of]
    cols = j * m[row_of].astype(np.int64) + off.astype(np.int64)
    return bp.astype(np.int32), cols.astype(np.int32), np.ascontiguousarray(vals, dtype=np.float32)


def block_prune(W: np.ndarray, bs: int, nblocks: int):
    """Block pruning of a dense fp32 W (rows, cols multiples of bs): keep the
    `nblocks` bs x bs blocks of largest L1 norm (ties: lowest block index).
    Returns the BSR arrays (brow_ptr, bcol_idx, bvals[nnzb, bs, bs]) and the
    kept-block mask (rows/bs x cols/bs)."""
    R, C = W.shape
    br, bc = R // bs, C // bs
    blocks = W.reshape(br, bs, bc, bs).transpose(0, 2, 1, 3)   # [br, bc, bs, bs]
    norms = np.abs(blocks).sum(axis=(2, 3), dtype=np.float64).ravel()
    nblocks = max(0, min(int(nblocks), norms.size))
    order = np.lexsort((np.arange(norms.size), -norms))[:nblocks]
    mask = np.zeros(norms.size, dtype=bool)
    mask[order] = True
    mask = mask.reshape(br, bc)
    brow_ptr = np.zeros(br + 1, dtype=np.int32)
    brow_ptr[1:] = np.cumsum(mask.sum(axis=1))
    rr, cc = np.nonzero(mask)   # row-major: block rows in order, columns ascending
    return brow_ptr, cc.astype(np.int32), np.ascontiguousarray(blocks[rr, cc], dtype=np.float32), mask


DENSE_ROWS, DENSE_COLS = 0, 1


def _stream(stream):
    return darb._stream(stream)


def _dense(X, Y, rows: int, cols: int, layout: int):
    """(ldx, batch, ldy) of X and Y: DENSE_ROWS takes X (cols, batch) and Y (rows,
    batch); DENSE_COLS takes them stored transposed, X (batch, cols), Y (batch, rows)."""
    darb._require_cuda_f32(X, "X")
    darb._require_cuda_f32(Y, "Y")
    if X.stride(1) != 1 or Y.stride(1) != 1:
        raise darb.DarbError(darb.ERR_INVALID_ARG, "X and Y need unit stride in their last dimension")
    # the stride of a dimension of size 1 is arbitrary: take the row length there
    ld = lambda T: T.stride(0) if T.shape[0] > 1 else T.shape[1]
    if layout == DENSE_ROWS:
        if X.shape[0] != cols or Y.shape != (rows, X.shape[1]):
            raise darb.DarbError(darb.ERR_INVALID_ARG, "shapes: X (cols, batch), Y (rows, batch)")
        return ld(X), X.shape[1], ld(Y)
    if X.shape[1] != cols or Y.shape != (X.shape[0], rows):
        raise darb.DarbError(darb.ERR_INVALID_ARG, "shapes: X (batch, cols), Y (batch, rows)")
    return ld(X), X.shape[0], ld(Y)


def csr_spmm(row_ptr, col_idx, vals, rows: int, cols: int, X, Y, layout: int = DENSE_ROWS, stream=None):
    """Y = A X through cuSPARSE CSR (device tensors, fp32)."""
    for t, n in ((row_ptr, "row_ptr"), (col_idx, "col_idx"), (vals, "vals")):
        if t is None or not t.is_cuda:
            raise darb.DarbError(darb.ERR_INVALID_ARG, f"{n} must be a CUDA tensor")
    ldx, batch, ldy = _dense(X, Y, rows, cols, layout)
    st = lib().darb_baseline_csr_spmm(row_ptr.data_ptr(), col_idx.data_ptr(), vals.data_ptr(), rows, cols,
                                      vals.numel(), X.data_ptr(), ldx, batch, Y.data_ptr(), ldy, layout,
                                      _stream(stream))
    darb._check(st, "darb_baseline_csr_spmm")


def bsr_spmm(brow_ptr, bcol_idx, bvals, rows: int, cols: int, bs: int, X, Y, layout: int = DENSE_ROWS, stream=None):
    """Y = A X through cuSPARSE BSR with bs x bs row-major blocks (device tensors, fp32)."""
    for t, n in ((brow_ptr, "brow_ptr"), (bcol_idx, "bcol_idx"), (bvals, "bvals")):
        if t is None or not t.is_cuda:
            raise darb.DarbError(darb.ERR_INVALID_ARG, f"{n} must be a CUDA tensor")
    ldx, batch, ldy = _dense(X, Y, rows, cols, layout)
    st = lib().darb_baseline_bsr_spmm(brow_ptr.data_ptr(), bcol_idx.data_ptr(), bvals.data_ptr(), rows, cols, bs,
                                      bcol_idx.numel(), X.data_ptr(), ldx, batch, Y.data_ptr(), ldy, layout,
                                      _stream(stream))
    darb._check(st, "darb_baseline_bsr_spmm")
