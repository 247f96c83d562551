"""The C ABI without a GPU: exported symbols, host-only calls, argument checks.

No test here launches a kernel or dereferences a device pointer; every call
either is host-only or is rejected before any CUDA work.
"""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_1911_08020_gb300 import build as darb_build
from paper_1911_08020_gb300 import darb

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    darb_build.build()
    return darb.lib()


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "darb.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"DARB_API\s+[\w\s\*]+?\b(darb_\w+)\s*\(", src)))


def test_every_declared_symbol_is_exported(L):
    names = _declared_functions()
    assert len(names) >= 13
    for n in names:
        assert hasattr(L, n), n


def test_status_strings(L):
    for code, name in enumerate(["DARB_OK", "DARB_ERR_INVALID_ARG", "DARB_ERR_NONFINITE",
                                 "DARB_ERR_OOM", "DARB_ERR_CUDA", "DARB_ERR_TIMEOUT",
                                 "DARB_ERR_UNSUPPORTED"]):
        assert darb.status_string(code) == name
    assert darb.status_string(99) == "DARB_ERR_UNKNOWN"


def test_assign_block_sizes_matches_oracle(L):
    g = np.random.default_rng(0)
    for trial in range(200):
        rows, cols = int(g.integers(1, 60)), int(g.integers(1, 5000))
        nnz = g.integers(0, cols + 1, size=rows)
        if trial % 7 == 0:
            nnz[:] = nnz[0]
        lo, hi = [(1, 256), (2, 64), (4, 4), (1, 1)][trial % 4]
        np.testing.assert_array_equal(darb.darb_assign_block_sizes(nnz, cols, lo, hi),
                                      oracle.assign_block_sizes(nnz, cols, lo, hi))


def test_assign_block_sizes_worked_example(L):
    # Sec. 3.2: matrix density 7/32; 37.5% -> block size 2, 18.75% -> 8
    np.testing.assert_array_equal(darb.darb_assign_block_sizes([12, 6, 5, 5], 32), [2, 8, 8, 8])


def test_assign_block_sizes_rejects(L):
    out = np.zeros(2, np.int32)
    nnz = np.array([1, 2], np.int64)
    P = lambda a: a.ctypes.data
    assert L.darb_assign_block_sizes(None, 2, 4, 1, 8, P(out)) == darb.ERR_INVALID_ARG
    assert L.darb_assign_block_sizes(P(nnz), 2, 4, 0, 8, P(out)) == darb.ERR_INVALID_ARG
    assert L.darb_assign_block_sizes(P(nnz), 2, 4, 8, 4, P(out)) == darb.ERR_INVALID_ARG
    assert L.darb_assign_block_sizes(P(nnz), 2, 4, 1, 512, P(out)) == darb.ERR_INVALID_ARG
    assert L.darb_assign_block_sizes(P(nnz), 2, 1, 1, 8, P(out)) == darb.ERR_INVALID_ARG  # nnz > cols


def _encode(L, W, wtype, rows, cols, ldw, m):
    out = ctypes.c_void_p(12345)
    st = L.darb_encode(W, wtype, rows, cols, ldw, m, ctypes.byref(out), None)
    return st, out.value


def test_encode_rejects_bad_arguments_before_any_cuda_work(L):
    m = np.full(4, 8, np.int32)
    fake = 4096   # never dereferenced: every call below fails validation first
    mp = m.ctypes.data
    assert _encode(L, None, 0, 4, 32, 32, mp) == (darb.ERR_INVALID_ARG, None)
    assert _encode(L, fake, 7, 4, 32, 32, mp)[0] == darb.ERR_INVALID_ARG       # bad dtype
    assert _encode(L, fake, 0, 0, 32, 32, mp)[0] == darb.ERR_INVALID_ARG       # rows
    assert _encode(L, fake, 0, 4, 32, 16, mp)[0] == darb.ERR_INVALID_ARG       # ldw < cols
    assert _encode(L, fake + 1, 0, 4, 32, 32, mp)[0] == darb.ERR_INVALID_ARG   # misaligned fp32
    assert _encode(L, fake, 0, 4, 32, 32, None)[0] == darb.ERR_INVALID_ARG
    for bad in (0, -3, 257):
        mb = m.copy()
        mb[2] = bad
        assert _encode(L, fake, 1, 4, 32, 32, mb.ctypes.data)[0] == darb.ERR_INVALID_ARG
    assert L.darb_encode(fake, 0, 4, 32, 32, mp, None, None) == darb.ERR_INVALID_ARG


def test_encode_allocation_failure_is_reported(L, monkeypatch):
    monkeypatch.setenv("DARB_FAIL_ALLOC", "1")
    m = np.full(4, 8, np.int32)
    st, h = _encode(L, 4096, 0, 4, 32, 32, m.ctypes.data)
    assert st == darb.ERR_OOM and h is None


def test_assign_from_weights_allocation_failure_is_reported(L, monkeypatch):
    monkeypatch.setenv("DARB_FAIL_ALLOC", "1")
    nnz = np.zeros(4, np.int64)
    m = np.zeros(4, np.int32)
    assert L.darb_assign_from_weights(4096, darb.BF16, 4, 32, 32, 8, 1, 256, nnz.ctypes.data, m.ctypes.data,
                                      None) == darb.ERR_OOM


def test_calls_reject_unknown_handles(L):
    bogus = ctypes.c_void_p(0xDEAD0)
    info = darb._Info()
    assert L.darb_info(bogus, ctypes.byref(info)) == darb.ERR_INVALID_ARG
    assert L.darb_spmm(bogus, 4096, 1, 1, 8192, 1, None) == darb.ERR_INVALID_ARG
    for path in (darb.PATH_AUTO, darb.PATH_CUDA_CORES, darb.PATH_TENSOR_CORES, 3, -1):
        assert L.darb_spmm_ex(bogus, 4096, 1, 1, 8192, 1, path, None) == darb.ERR_INVALID_ARG
    pth, nk = ctypes.c_int(), ctypes.c_int32()
    assert L.darb_spmm_path(bogus, 256, ctypes.byref(pth), ctypes.byref(nk)) == darb.ERR_INVALID_ARG
    assert L.darb_lstm_step(bogus, 1, 1, 1, 4096, 4096, 4096, None, 8192, 8192, None) == darb.ERR_INVALID_ARG
    assert L.darb_gru_step(bogus, 1, 1, 1, 4096, 4096, None, None, 8192, None) == darb.ERR_INVALID_ARG
    assert L.darb_lstm_sequence(bogus, 2, 1, 1, 1, 4096, 4096, 4096, None, 8192, None, None,
                                None) == darb.ERR_INVALID_ARG
    assert L.darb_gru_sequence(bogus, 2, 1, 1, 1, 4096, 4096, None, None, 8192, None) == darb.ERR_INVALID_ARG
    assert L.darb_export(bogus, None, None, None, None) == darb.ERR_INVALID_ARG
    assert L.darb_reencode(bogus, 4096, 8, None) == darb.ERR_INVALID_ARG
    assert L.darb_reencode_host(bogus, 4096, 8, 8192, None) == darb.ERR_INVALID_ARG
    assert L.darb_spmm_host(bogus, 4096, 1, 1, 8192, 1, 12288, 16384, None) == darb.ERR_INVALID_ARG
    assert L.darb_rnn_reserve(bogus, 4) == darb.ERR_INVALID_ARG
    assert L.darb_destroy(bogus) == darb.ERR_INVALID_ARG
    assert L.darb_destroy(None) == darb.OK


def test_assign_from_weights_rejects_bad_arguments_before_any_cuda_work(L):
    nnz = np.zeros(4, np.int64)
    m = np.zeros(4, np.int32)
    call = lambda W, dt, rows, cols, ldw, keep, lo, hi, mo: L.darb_assign_from_weights(
        W, dt, rows, cols, ldw, keep, lo, hi, nnz.ctypes.data, mo, None)
    assert call(None, darb.BF16, 4, 8, 8, 4, 1, 256, m.ctypes.data) == darb.ERR_INVALID_ARG      # no W
    assert call(4096, darb.BF16, 4, 8, 8, 4, 1, 256, None) == darb.ERR_INVALID_ARG               # no m_out
    assert call(4096, 7, 4, 8, 8, 4, 1, 256, m.ctypes.data) == darb.ERR_INVALID_ARG              # dtype
    assert call(4096, darb.BF16, 0, 8, 8, 4, 1, 256, m.ctypes.data) == darb.ERR_INVALID_ARG      # rows
    assert call(4096, darb.BF16, 4, 8, 7, 4, 1, 256, m.ctypes.data) == darb.ERR_INVALID_ARG      # ldw < cols
    assert call(4096, darb.BF16, 4, 8, 8, 0, 1, 256, m.ctypes.data) == darb.ERR_INVALID_ARG      # keep < 1
    assert call(4096, darb.BF16, 4, 8, 8, 33, 1, 256, m.ctypes.data) == darb.ERR_INVALID_ARG     # keep > rows*cols
    assert call(4096, darb.BF16, 4, 8, 8, 4, 0, 256, m.ctypes.data) == darb.ERR_INVALID_ARG      # m_min
    assert call(4096, darb.BF16, 4, 8, 8, 4, 8, 4, m.ctypes.data) == darb.ERR_INVALID_ARG        # m_max < m_min
    assert call(4097, darb.F32, 4, 8, 8, 4, 1, 256, m.ctypes.data) == darb.ERR_INVALID_ARG       # misaligned
    assert call(4096, darb.BF16, 1 << 17, 1 << 16, 1 << 16, 4, 1, 256, m.ctypes.data) == darb.ERR_UNSUPPORTED


def test_import_rejects_bad_arguments(L):
    out = ctypes.c_void_p()
    v = np.zeros(8, np.float32)
    o = np.zeros(8, np.uint8)
    m = np.full(2, 8, np.int32)
    assert L.darb_import(None, o.ctypes.data, m.ctypes.data, 0, 2, 32, ctypes.byref(out), None) == darb.ERR_INVALID_ARG
    assert L.darb_import(v.ctypes.data, o.ctypes.data, m.ctypes.data, 0, 2, 32, None, None) == darb.ERR_INVALID_ARG
    o[3] = 8   # offset outside its block of 8
    assert L.darb_import(v.ctypes.data, o.ctypes.data, m.ctypes.data, 0, 2, 32, ctypes.byref(out), None) == darb.ERR_INVALID_ARG
    assert out.value is None


def test_binding_fails_loudly_without_the_library(monkeypatch, tmp_path):
    monkeypatch.setattr(darb, "_lib", None)
    monkeypatch.setattr(darb, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(darb.DarbError):
        darb.lib()
