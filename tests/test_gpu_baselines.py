"""cuSPARSE comparison products (include/darb_baselines.h) on the GPU: the CSR
of a DARB handle's kept weights and block-pruned BSR matrices against fp64
references, and the CSR against darb_spmm on full-size FC6."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from paper_1911_08020_gb300 import baselines, darb, synth
from tests.gpu_helpers import TOL, assert_product_close, dev, encode_both, t

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1911_08020_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _run(fn, X: np.ndarray, rows: int, layout: int) -> np.ndarray:
    """Call fn(Xd, Yd, layout) with X (cols x batch) in the given dense layout; Y as rows x batch."""
    B = X.shape[1]
    if layout == baselines.DENSE_ROWS:
        Y = torch.empty((rows, B), device=dev())
        fn(t(X), Y, layout)
        return Y.cpu().numpy()
    Y = torch.empty((B, rows), device=dev())
    fn(t(np.ascontiguousarray(X.T)), Y, layout)
    return Y.cpu().numpy().T


LAYOUTS = [0, 1]


@pytest.mark.parametrize("layout", LAYOUTS)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_csr_of_darb_weights_matches_the_oracle(dtype, layout):
    g = np.random.default_rng(50)
    for rows, cols, B in ((5, 7, 1), (64, 300, 3), (200, 1000, 16), (96, 513, 40)):
        w = (0.1 * g.standard_normal((rows, cols))).astype(np.float32)
        stored = synth.f32_to_bf16_bits(w) if dtype == "bf16" else w
        m = g.choice(np.asarray((1, 3, 8, 16, 32), np.int32), size=rows)
        h, ref = encode_both(stored, m, dtype)
        try:
            rp, ci, vv = baselines.csr_from_darb(h)
            X = synth.activations(cols, B, seed=rows)
            Y = _run(lambda Xd, Yd, lay: baselines.csr_spmm(t(rp), t(ci), t(vv), rows, cols, Xd, Yd, lay), X, rows,
                     layout)
            yref, absdot = oracle.darb_spmm(ref, X, with_absdot=True)
            # the same kept weights in another format: the fp32 product bound holds
            assert_product_close(Y, yref, absdot, TOL["f32"])
        finally:
            darb.darb_destroy(h)


@pytest.mark.parametrize("layout", LAYOUTS)
@pytest.mark.parametrize("bs", [4, 8])
def test_bsr_block_pruned_matches_dense_reference(bs, layout):
    g = np.random.default_rng(51 + bs)
    for rows, cols, B, keep in ((bs, bs, 1, 1), (8 * bs, 12 * bs, 5, 20), (32 * bs, 40 * bs, 64, 200)):
        W = (0.1 * g.standard_normal((rows, cols))).astype(np.float32)
        brow_ptr, bcol, bvals, mask = baselines.block_prune(W, bs, keep)
        X = synth.activations(cols, B, seed=rows + bs)
        Y = _run(lambda Xd, Yd, lay: baselines.bsr_spmm(t(brow_ptr), t(bcol), t(bvals.reshape(-1)), rows, cols, bs,
                                                        Xd, Yd, lay), X, rows, layout)
        Wm = np.where(np.kron(mask, np.ones((bs, bs), dtype=bool)), W, 0).astype(np.float64)
        yref = Wm @ X.astype(np.float64)
        absdot = np.abs(Wm) @ np.abs(X.astype(np.float64))
        assert_product_close(Y, yref, absdot, TOL["f32"])


def test_csr_of_fc6_matches_the_oracle():
    """Full-size FC6: the CSR of the kept weights against the oracle, next to darb_spmm."""
    wl = synth.WORKLOADS["fc6_fc7"]
    _, stored, m = synth.matrix(wl, 0)
    h, ref = encode_both(stored, m, wl.dtype)
    try:
        rows, cols = ref.rows, ref.cols
        rp, ci, vv = baselines.csr_from_darb(h)
        info = darb.darb_info(h)
        assert len(vv) == info["nnzb"] and rp[-1] == info["nnzb"]
        X = synth.activations(cols, 16, seed=9)
        Yc = torch.empty((rows, 16), device=dev())
        baselines.csr_spmm(t(rp), t(ci), t(vv), rows, cols, t(X), Yc)
        Yd = darb.darb_spmm(h, t(X))
        yref, absdot = oracle.darb_spmm(ref, X, with_absdot=True)
        assert_product_close(Yc.cpu().numpy(), yref, absdot, TOL["f32"])
        assert_product_close(Yd.cpu().numpy(), yref, absdot, TOL[wl.dtype])
    finally:
        darb.darb_destroy(h)
