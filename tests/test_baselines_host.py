"""The cuSPARSE comparison library without a GPU: exported symbols, argument
checks before any CUDA work, and the host-side block pruning that feeds it."""
import os
import re

import numpy as np
import pytest

from paper_1911_08020_gb300 import baselines, darb
from paper_1911_08020_gb300 import build as darb_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def BL():
    darb_build.build()
    return baselines.lib()


def test_every_declared_symbol_is_exported(BL):
    src = open(os.path.join(ROOT, "include", "darb_baselines.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = sorted(set(re.findall(r"DARB_API\s+[\w\s\*]+?\b(darb_\w+)\s*\(", src)))
    assert names == ["darb_baseline_bsr_spmm", "darb_baseline_csr_spmm"]
    for n in names:
        assert hasattr(BL, n), n


def test_baselines_are_not_in_libdarb():
    darb_build.build()
    assert not hasattr(darb.lib(), "darb_baseline_csr_spmm")


def test_calls_reject_bad_arguments_before_any_cuda_work(BL):
    f = 4096   # never dereferenced: every call below fails validation first
    csr = BL.darb_baseline_csr_spmm
    assert csr(None, f, f, 8, 8, 4, f, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG       # no row_ptr
    assert csr(f, None, f, 8, 8, 4, f, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG       # nnz > 0, no columns
    assert csr(f, f, f, 0, 8, 4, f, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG          # rows
    assert csr(f, f, f, 8, 8, -1, f, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG         # nnz
    assert csr(f, f, f, 8, 8, 4, f, 1, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG          # ldx < batch
    assert csr(f, f, f, 8, 8, 4, None, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG       # no X
    assert csr(f, f, f, 8, 8, 1 << 31, f, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG    # nnz beyond int32
    bsr = BL.darb_baseline_bsr_spmm
    assert bsr(f, f, f, 8, 8, 1, 4, f, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG       # bs = 1
    assert bsr(f, f, f, 8, 8, 64, 4, f, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG      # bs > 32
    assert bsr(f, f, f, 10, 8, 4, 4, f, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG      # rows % bs
    assert bsr(f, f, f, 8, 8, 4, 4, f, 2, 0, f, 2, 0, None) == darb.ERR_INVALID_ARG       # batch
    assert bsr(None, f, f, 8, 8, 4, 4, f, 2, 2, f, 2, 0, None) == darb.ERR_INVALID_ARG    # no brow_ptr
    assert csr(f, f, f, 8, 8, 4, f, 2, 2, f, 2, 7, None) == darb.ERR_INVALID_ARG         # unknown layout
    assert csr(f, f, f, 8, 6, 4, f, 5, 2, f, 8, 1, None) == darb.ERR_INVALID_ARG         # column-major: ldx < cols
    assert csr(f, f, f, 8, 6, 4, f, 6, 2, f, 7, 1, None) == darb.ERR_INVALID_ARG         # column-major: ldy < rows


def _block_prune_brute(W, bs, k):
    R, C = W.shape
    scored = []
    for i in range(R // bs):
        for j in range(C // bs):
            scored.append((-float(np.abs(W[i * bs:(i + 1) * bs, j * bs:(j + 1) * bs]).astype(np.float64).sum()),
                           i * (C // bs) + j, i, j))
    scored.sort()
    keep = sorted((i, j) for _, _, i, j in scored[:k])
    return keep


@pytest.mark.parametrize("bs", [2, 4, 8])
def test_block_prune_keeps_the_largest_blocks(bs):
    g = np.random.default_rng(bs)
    for trial in range(20):
        R, C = bs * int(g.integers(1, 6)), bs * int(g.integers(1, 7))
        W = g.standard_normal((R, C)).astype(np.float32)
        if trial % 4 == 0:   # ties: equal-norm blocks, lowest block index wins
            W = np.round(W)
        nb = (R // bs) * (C // bs)
        k = int(g.integers(0, nb + 1))
        brow_ptr, bcol, bvals, mask = baselines.block_prune(W, bs, k)
        keep = _block_prune_brute(W, bs, k)
        assert sorted(zip(*np.nonzero(mask))) == keep
        assert brow_ptr[-1] == k and len(bcol) == k
        # the BSR arrays reproduce the pruned matrix
        dense = np.zeros_like(W)
        for i in range(R // bs):
            for p in range(brow_ptr[i], brow_ptr[i + 1]):
                j = bcol[p]
                dense[i * bs:(i + 1) * bs, j * bs:(j + 1) * bs] = bvals[p]
        expect = np.where(np.kron(mask, np.ones((bs, bs), dtype=bool)), W, 0)
        np.testing.assert_array_equal(dense, expect)
