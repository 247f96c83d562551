"""CPU oracle for DARB -- TEST INFRASTRUCTURE ONLY.

Plain, slow, obviously correct C (``darb_oracle.c``), compiled with gcc and
loaded through ctypes.  Only the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package; the library under
``paper_1911_08020_gb300`` never does, and shares no code with it.

Functions (each follows the passage cited in ``darb_oracle.c``):

* ``assign_block_sizes(row_nnz, cols, m_min, m_max)``  Sec. 3.2 rounding rule
* ``block_pointers(m, cols)``                          ceil(cols/m) blocks per row
* ``encode(W, m, dtype)``                              BMWM, Sec. 3.1 / 3.2
* ``masked_dense(enc, cols)``                          the dense M (.) W
* ``darb_spmm(enc, X)``                                y = W_darb X in fp64
* ``darb_spmm_f32(enc, X)``                            the same sum in fp32, for timing only
* ``lstm_step(enc, I, H, x, h, c, bias)`` / ``gru_step(enc, I, H, x, h, b_ih, b_hh)``
"""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "darb_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, INVALID, NONFINITE = 0, 1, 2


class OracleError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"oracle {what} failed with status {status}")
        self.status = status


def build(force: bool = False) -> str:
    """Compile darb_oracle.c into liboracle.so with gcc (OpenMP when available)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        raise RuntimeError("no C compiler found to build the oracle")
    tmp = _LIB + f".tmp{os.getpid()}"
    base = [cc, "-O2", "-std=c11", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


def load_library(path: str):
    """Load a compiled oracle and declare its C signatures."""
    lib = ctypes.CDLL(path)
    P = ctypes.c_void_p
    I64 = ctypes.c_int64
    I32 = ctypes.c_int32
    lib.oracle_set_threads.argtypes = [ctypes.c_int]
    lib.oracle_set_threads.restype = ctypes.c_int
    lib.oracle_assign_block_sizes.argtypes = [P, I64, I64, I32, I32, P]
    lib.oracle_topk_row_nnz_f32.argtypes = [P, I64, I64, I64, I64, P]
    lib.oracle_topk_row_nnz_bf16.argtypes = [P, I64, I64, I64, I64, P]
    lib.oracle_block_pointers.argtypes = [P, I64, I64, P]
    lib.oracle_encode_f32.argtypes = [P, I64, I64, I64, P, P, P, P]
    lib.oracle_encode_bf16.argtypes = [P, I64, I64, I64, P, P, P, P]
    lib.oracle_masked_dense.argtypes = [P, P, P, P, I64, I64, P]
    lib.oracle_darb_spmm.argtypes = [P, P, P, P, I64, I64, P, I64, I64, P, I64, P]
    lib.oracle_darb_spmm_f32_timed.argtypes = [P, P, P, P, I64, I64, P, I64, I64, P, I64]
    lib.oracle_lstm_step.argtypes = [P, P, P, P, I64, I64, I64, P, P, P, P, P, P, P]
    lib.oracle_gru_step.argtypes = [P, P, P, P, I64, I64, I64, P, P, P, P, P, P]
    for f in ("oracle_assign_block_sizes", "oracle_topk_row_nnz_f32", "oracle_topk_row_nnz_bf16",
              "oracle_block_pointers", "oracle_encode_f32",
              "oracle_encode_bf16", "oracle_masked_dense", "oracle_darb_spmm", "oracle_darb_spmm_f32_timed",
              "oracle_lstm_step", "oracle_gru_step"):
        getattr(lib, f).restype = ctypes.c_int
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            _lib = load_library(_LIB)
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _check(st: int, what: str):
    if st != OK:
        raise OracleError(st, what)


def set_threads(n: int) -> int:
    """Set the OpenMP thread count of the oracle's row loops; returns the count in use."""
    return _load().oracle_set_threads(int(n))


@dataclass
class Encoding:
    """Canonical DARB encoding: blocks in (row, j) order."""
    val: np.ndarray        # float32 or uint16 (bf16 bits), one per block
    off: np.ndarray        # uint8, position of the kept weight inside its block
    blk_ptr: np.ndarray    # int64[rows+1]
    m: np.ndarray          # int32[rows]
    dtype: str             # "f32" or "bf16"
    rows: int
    cols: int

    def values_f64(self) -> np.ndarray:
        if self.dtype == "bf16":
            return (self.val.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        return self.val.astype(np.float64)


def topk_row_nnz(W: np.ndarray, keep: int, dtype: str | None = None) -> np.ndarray:
    """Per-row count of the `keep` weights of largest magnitude (ties at the
    threshold all count): the row densities of Sec. 3.2's first step."""
    if dtype is None:
        dtype = "bf16" if W.dtype == np.uint16 else "f32"
    W = np.ascontiguousarray(W, dtype=np.uint16 if dtype == "bf16" else np.float32)
    rows, cols = W.shape
    out = np.zeros(rows, dtype=np.int64)
    fn = _load().oracle_topk_row_nnz_bf16 if dtype == "bf16" else _load().oracle_topk_row_nnz_f32
    _check(fn(_p(W), rows, cols, cols, int(keep), _p(out)), "topk_row_nnz")
    return out


def assign_block_sizes(row_nnz, cols: int, m_min: int = 1, m_max: int = 256) -> np.ndarray:
    nnz = np.ascontiguousarray(row_nnz, dtype=np.int64)
    out = np.zeros(nnz.shape[0], dtype=np.int32)
    _check(_load().oracle_assign_block_sizes(_p(nnz), nnz.shape[0], cols, m_min, m_max, _p(out)),
           "assign_block_sizes")
    return out


def block_pointers(m, cols: int) -> np.ndarray:
    m = np.ascontiguousarray(m, dtype=np.int32)
    out = np.zeros(m.shape[0] + 1, dtype=np.int64)
    _check(_load().oracle_block_pointers(_p(m), m.shape[0], cols, _p(out)), "block_pointers")
    return out


def encode(W: np.ndarray, m, dtype: str | None = None) -> Encoding:
    """BMWM encode of W (float32, or uint16 bf16 bits when dtype == 'bf16')."""
    if dtype is None:
        dtype = "bf16" if W.dtype == np.uint16 else "f32"
    W = np.ascontiguousarray(W, dtype=np.uint16 if dtype == "bf16" else np.float32)
    rows, cols = W.shape
    m = np.ascontiguousarray(m, dtype=np.int32)
    bp = block_pointers(m, cols)
    nnzb = int(bp[-1])
    val = np.zeros(nnzb, dtype=W.dtype)
    off = np.zeros(nnzb, dtype=np.uint8)
    fn = _load().oracle_encode_bf16 if dtype == "bf16" else _load().oracle_encode_f32
    _check(fn(_p(W), rows, cols, cols, _p(m), _p(val), _p(off), _p(bp)), "encode")
    return Encoding(val, off, bp, m, dtype, rows, cols)


def masked_dense(enc: Encoding) -> np.ndarray:
    out = np.zeros((enc.rows, enc.cols), dtype=np.float64)
    v = enc.values_f64()
    _check(_load().oracle_masked_dense(_p(v), _p(enc.off), _p(enc.blk_ptr), _p(enc.m),
                                       enc.rows, enc.cols, _p(out)), "masked_dense")
    return out


def darb_spmm(enc: Encoding, X: np.ndarray, with_absdot: bool = False):
    """Y = W_darb X in fp64; X is cols x batch (any float dtype, widened exactly)."""
    X = np.ascontiguousarray(X, dtype=np.float64)
    if X.ndim == 1:
        X = X[:, None]
    batch = X.shape[1]
    Y = np.zeros((enc.rows, batch), dtype=np.float64)
    A = np.zeros_like(Y) if with_absdot else None
    v = enc.values_f64()
    _check(_load().oracle_darb_spmm(_p(v), _p(enc.off), _p(enc.blk_ptr), _p(enc.m), enc.rows,
                                    enc.cols, _p(X), batch, batch, _p(Y), batch,
                                    _p(A) if A is not None else None), "darb_spmm")
    return (Y, A) if with_absdot else Y


def darb_spmm_f32(enc: Encoding, X: np.ndarray, values_f32: np.ndarray | None = None):
    """The same product in fp32 (fp32 accumulate, block order): the loop timed
    as the CPU baseline.  Never a reference value: parity is against darb_spmm.
    values_f32 may pass the kept values already widened to float32."""
    X = np.ascontiguousarray(X, dtype=np.float32)
    if X.ndim == 1:
        X = X[:, None]
    batch = X.shape[1]
    Y = np.empty((enc.rows, batch), dtype=np.float32)
    v = values_f32 if values_f32 is not None else enc.values_f64().astype(np.float32)
    _check(_load().oracle_darb_spmm_f32_timed(_p(v), _p(enc.off), _p(enc.blk_ptr), _p(enc.m), enc.rows,
                                              enc.cols, _p(X), batch, batch, _p(Y), batch), "darb_spmm_f32")
    return Y


def lstm_step(enc: Encoding, I: int, H: int, x, h_prev, c_prev, bias=None):
    """One LSTM step in fp64; returns (h, c, gate_abs)."""
    f = lambda a: np.ascontiguousarray(a, dtype=np.float64)
    x, h_prev, c_prev = f(x), f(h_prev), f(c_prev)
    B = h_prev.shape[1]
    b = f(bias) if bias is not None else None
    h = np.zeros((H, B)); c = np.zeros((H, B)); ga = np.zeros((4 * H, B))
    v = enc.values_f64()
    _check(_load().oracle_lstm_step(_p(v), _p(enc.off), _p(enc.blk_ptr), _p(enc.m), I, H, B,
                                    _p(x), _p(h_prev), _p(c_prev),
                                    _p(b) if b is not None else None, _p(h), _p(c), _p(ga)),
           "lstm_step")
    return h, c, ga


def gru_step(enc: Encoding, I: int, H: int, x, h_prev, b_ih=None, b_hh=None):
    """One GRU step in fp64; returns (h, gate_abs[3H, B, 2])."""
    f = lambda a: np.ascontiguousarray(a, dtype=np.float64)
    x, h_prev = f(x), f(h_prev)
    B = h_prev.shape[1]
    bi = f(b_ih) if b_ih is not None else None
    bh = f(b_hh) if b_hh is not None else None
    h = np.zeros((H, B)); ga = np.zeros((3 * H, B, 2))
    v = enc.values_f64()
    _check(_load().oracle_gru_step(_p(v), _p(enc.off), _p(enc.blk_ptr), _p(enc.m), I, H, B,
                                   _p(x), _p(h_prev), _p(bi) if bi is not None else None,
                                   _p(bh) if bh is not None else None, _p(h), _p(ga)),
           "gru_step")
    return h, ga
