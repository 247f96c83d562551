"""Block sizes from the weights on the GPU (darb_assign_from_weights) against the oracle.

The row counts of the top-K magnitude mask are integers: they must equal the
oracle's exactly, and so must the block sizes the rounding rule makes of them.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from paper_1911_08020_gb300 import darb, synth
from tests.gpu_helpers import assert_encoding_equal, dev, weight_tensor
from tests.oracle_pins import _golden_lines, _kv

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1911_08020_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _stored(w, dtype):
    return synth.f32_to_bf16_bits(w) if dtype == "bf16" else w.astype(np.float32)


def _gpu(stored, dtype, keep, m_min=1, m_max=256, pad=0):
    rows, cols = stored.shape
    if pad:
        big = np.zeros((rows, cols + pad), stored.dtype)
        big[:, :cols] = stored
        W = weight_tensor(big, dtype)[:, :cols]
    else:
        W = weight_tensor(stored, dtype)
    return darb.darb_assign_from_weights(W, keep, m_min, m_max)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_counts_and_block_sizes_match_oracle(dtype):
    g = np.random.default_rng(60)
    for rows, cols, pad in ((1, 1, 0), (3, 7, 0), (37, 91, 3), (100, 257, 0), (257, 1030, 5), (64, 4096, 0)):
        w = (0.05 * g.standard_normal((rows, cols)) * np.exp(0.5 * g.standard_normal((rows, 1)))).astype(np.float32)
        stored = _stored(w, dtype)
        n = rows * cols
        for keep in sorted(k for k in {1, 2, max(1, n // 25), max(1, n // 3), max(1, n - 1), n} if k <= n):
            nnz, m = _gpu(stored, dtype, keep, pad=pad)
            ref = oracle.topk_row_nnz(stored, keep, dtype)
            assert np.array_equal(nnz, ref), (rows, cols, keep)
            assert np.array_equal(m, oracle.assign_block_sizes(ref, cols)), (rows, cols, keep)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_ties_zeros_and_infinities(dtype):
    g = np.random.default_rng(61)
    rows, cols = 50, 300
    w = (np.round(g.standard_normal((rows, cols)) * 2) / 4).astype(np.float32)   # few distinct magnitudes
    w[g.random((rows, cols)) < 0.1] = 0.0
    w[g.random((rows, cols)) < 0.05] = -0.0
    w[3, 17] = np.inf
    w[9, 2] = -np.inf
    stored = _stored(w, dtype)
    for keep in (1, 2, 3, 50, 1000, 7000, rows * cols):
        nnz, m = _gpu(stored, dtype, keep, m_min=2, m_max=64)
        ref = oracle.topk_row_nnz(stored, keep, dtype)
        assert np.array_equal(nnz, ref), keep
        assert np.array_equal(m, oracle.assign_block_sizes(ref, cols, 2, 64)), keep


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_nan_is_reported(dtype):
    w = np.ones((8, 40), np.float32)
    w[5, 31] = np.nan
    with pytest.raises(darb.DarbError) as e:
        _gpu(_stored(w, dtype), dtype, 10)
    assert e.value.status == darb.ERR_NONFINITE


def test_worked_example_of_the_paper():
    lines = _golden_lines("topk_worked_example.txt")
    head = _kv(lines[0])
    rows, cols, keep = int(head["rows"]), int(head["cols"]), int(head["keep"])
    cases = [_kv(ln) for ln in lines[1:]]
    g = np.random.default_rng(62)
    W = (g.uniform(0.01, 0.5, (rows, cols)) * g.choice([-1, 1], (rows, cols))).astype(np.float32)
    for c in cases:
        r, k = int(c["row"]), int(c["kept"])
        W[r, :k] = (1.0 + np.arange(k) / 64.0 + r / 8.0) * g.choice([-1, 1], k)
    nnz, m = _gpu(W, "f32", keep)
    assert list(nnz) == [int(c["kept"]) for c in cases]
    assert list(m) == [int(c["block_size"]) for c in cases]


def test_full_size_top4_percent_then_encode():
    """The FC6 shape with block sizes from a 4% top-K mask (the row scales make
    dense rows), then the encoding of W with them, all on the GPU."""
    wl = synth.WORKLOADS["fc6_fc7"]
    _, stored, _ = synth.matrix(wl, 0)
    rows, cols = stored.shape
    keep = rows * cols // 25
    W = weight_tensor(stored, "bf16")
    nnz, m = darb.darb_assign_from_weights(W, keep, 1, 256)
    ref = oracle.topk_row_nnz(stored, keep, "bf16")
    assert np.array_equal(nnz, ref)
    m_ref = oracle.assign_block_sizes(ref, cols)
    assert np.array_equal(m, m_ref)
    assert len(np.unique(m)) > 1   # density-adaptive: the rows differ
    h = darb.darb_encode(W, m)
    try:
        assert_encoding_equal(h, oracle.encode(stored, m_ref, "bf16"))
    finally:
        darb.darb_destroy(h)
