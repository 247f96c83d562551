"""The tensor-core product (densified tiles, tcgen05 kind::f16) against the oracle.

darb_spmm sends bf16 weights with more than 32 batch columns to the tensor cores;
darb_spmm_ex picks the path explicitly, so both kernel families are checked on
the same inputs.  Activations enter the tensor cores as two bf16 parts
(x = hi + lo, |x - hi - lo| <= 2^-16 |x|), so the error of that path is about
2^-16 * sum |val * x| plus fp32 accumulation: TC_TOL checks it far inside the
bf16 tolerance every product must meet, tight enough that dropping the low
part (an error near 2^-9) fails.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from paper_1911_08020_gb300 import darb, synth
from tests.gpu_helpers import TOL, assert_product_close, dev, encode_both, t

pytestmark = pytest.mark.gpu

TC_TOL = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1911_08020_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _case(g, rows, cols, mset):
    w = (0.05 * g.standard_normal((rows, cols)) * np.exp(0.5 * g.standard_normal((rows, 1)))).astype(np.float32)
    m = g.choice(np.asarray(mset, np.int32), size=rows)
    return synth.f32_to_bf16_bits(w), m


def _both_paths(h, ref, X):
    Xd = t(X)
    out = {}
    for path in (darb.PATH_TENSOR_CORES, darb.PATH_CUDA_CORES):
        out[path] = darb.darb_spmm_ex(h, Xd, path=path).cpu().numpy()
    Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
    return out, Yr, A


@pytest.mark.parametrize("rows,cols,mset", [
    (1, 1, (1,)),
    (37, 91, (1, 2, 3, 8)),
    (100, 257, (10, 15, 20, 30)),
    (257, 1030, (1, 2, 3, 8, 10, 16, 17, 32, 64, 200)),
    (300, 700, (16, 32, 64)),
    (513, 2000, (255, 256, 7)),
    (64, 20, (4, 16)),            # fewer than one 32-column stage
])
def test_tensor_path_matches_oracle(rows, cols, mset):
    g = np.random.default_rng(rows * 7 + cols)
    stored, m = _case(g, rows, cols, mset)
    h, ref = encode_both(stored, m, "bf16")
    try:
        for B in (4, 16, 20, 32, 64, 100, 128, 200, 256, 300, 520):
            X = synth.activations(cols, B, seed=B + cols)
            out, Yr, A = _both_paths(h, ref, X)
            assert_product_close(out[darb.PATH_TENSOR_CORES], Yr, A, TC_TOL)
            assert_product_close(out[darb.PATH_CUDA_CORES], Yr, A, TOL["bf16"])
    finally:
        darb.darb_destroy(h)


@pytest.mark.parametrize("name,index", [("fc6_fc7", 0), ("fc6_fc7", 1), ("gru_1024", 0), ("lstm_lm_1500", 0)])
def test_tensor_path_full_size(name, index):
    wl = synth.WORKLOADS[name]
    _, stored, m = synth.matrix(wl, index)
    h, ref = encode_both(stored, m, wl.dtype)
    try:
        for B in (16, 20, 64, 256):
            X = synth.activations(wl.shapes[index][1], B, seed=wl.seed + 70 + B)
            Y = darb.darb_spmm_ex(h, t(X), path=darb.PATH_TENSOR_CORES).cpu().numpy()
            Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
            assert_product_close(Y, Yr, A, TC_TOL)
    finally:
        darb.darb_destroy(h)


def test_tensor_path_is_deterministic_and_graph_capturable():
    g = np.random.default_rng(5)
    stored, m = _case(g, 1000, 3000, (16, 32, 64))
    h, ref = encode_both(stored, m, "bf16")
    try:
        X = t(synth.activations(3000, 256, seed=9))
        Y1 = darb.darb_spmm(h, X).clone()
        Y2 = darb.darb_spmm(h, X).clone()
        assert torch.equal(Y1, Y2)
        Y = torch.empty_like(Y1)
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            darb.darb_spmm(h, X, Y)
        torch.cuda.current_stream().wait_stream(s)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            darb.darb_spmm(h, X, Y)
        Y.zero_()
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(Y, Y1)
        Yr, A = oracle.darb_spmm(ref, X.cpu().numpy(), with_absdot=True)
        assert_product_close(Y.cpu().numpy(), Yr, A, TC_TOL)
        darb.darb_sync_status(h)   # raises unless the kernels reported nothing
    finally:
        darb.darb_destroy(h)


def test_tensor_path_strides_and_untouched_columns():
    g = np.random.default_rng(6)
    rows, cols = 200, 500
    stored, m = _case(g, rows, cols, (8, 32))
    h, ref = encode_both(stored, m, "bf16")
    try:
        for B, pad in ((16, 4), (40, 8), (64, 0), (96, 12), (33, 2), (130, 3)):
            Xbig = synth.activations(cols, B + pad, seed=B)
            Xd = t(Xbig)[:, :B]                          # ldx = B + pad, any alignment
            Yd = torch.full((rows, B + 6), 7.0, device=dev())   # ldy = B + 6
            darb.darb_spmm_ex(h, Xd, Yd[:, :B], path=darb.PATH_TENSOR_CORES)
            Yr, A = oracle.darb_spmm(ref, Xbig[:, :B], with_absdot=True)
            Yh = Yd.cpu().numpy()
            assert_product_close(Yh[:, :B], Yr, A, TC_TOL)
            assert np.all(Yh[:, B:] == 7.0), "wrote outside Y's columns"
    finally:
        darb.darb_destroy(h)


def test_path_query_reports_the_gather_for_every_batch():
    g = np.random.default_rng(8)
    w = (0.1 * g.standard_normal((64, 256))).astype(np.float32)
    m = np.full(64, 16, np.int32)
    h32, _ = encode_both(w, m, "f32")
    h16, _ = encode_both(synth.f32_to_bf16_bits(w), m, "bf16")
    try:
        assert darb.darb_spmm_path(h32, 512) == (darb.PATH_CUDA_CORES, 1)
        # darb_spmm never picks the tensor cores on its own: they are opt-in
        for B in (1, 32, 33, 64, 256, 4096):
            assert darb.darb_spmm_path(h16, B) == (darb.PATH_CUDA_CORES, 1)
        with pytest.raises(darb.DarbError):
            darb.darb_spmm_path(h16, 0)
    finally:
        darb.darb_destroy(h32)
        darb.darb_destroy(h16)


def test_tensor_path_refuses_what_it_cannot_take():
    g = np.random.default_rng(7)
    w = (0.1 * g.standard_normal((64, 128))).astype(np.float32)
    m = np.full(64, 8, np.int32)
    h32, ref32 = encode_both(w, m, "f32")
    stored, _ = _case(g, 64, 128, (8,))
    h16, ref16 = encode_both(stored, m, "bf16")
    try:
        X = t(synth.activations(128, 64, seed=1))
        with pytest.raises(darb.DarbError) as e:
            darb.darb_spmm_ex(h32, X, path=darb.PATH_TENSOR_CORES)
        assert e.value.status == darb.ERR_UNSUPPORTED
        # the automatic choice falls back to the CUDA cores for fp32 weights
        Y = darb.darb_spmm(h32, t(synth.activations(128, 200, seed=2))).cpu().numpy()
        Yr, A = oracle.darb_spmm(ref32, synth.activations(128, 200, seed=2), with_absdot=True)
        assert_product_close(Y, Yr, A, TOL["f32"])
        with pytest.raises(darb.DarbError) as e:
            darb.darb_spmm_ex(h16, X, path=7)
        assert e.value.status == darb.ERR_INVALID_ARG
    finally:
        darb.darb_destroy(h32)
        darb.darb_destroy(h16)
