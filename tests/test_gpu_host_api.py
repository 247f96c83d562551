"""The host-buffer entry points against the CPU oracle (needs a GB300).

darb_reencode_host and darb_spmm_host take W, X and Y in host memory and copy
them through caller-owned device buffers: encodings must match the oracle bit
for bit and products stay inside the gpu_helpers tolerance, for pinned and
pageable host memory, with host rows wider than the data.  The padding past
each row holds NaN: it is never read (a NaN weight would be reported by
darb_sync_status, a NaN activation would reach Y), and the padding of Y is
never written.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from paper_1911_08020_gb300 import darb, synth
from tests.gpu_helpers import TOL, assert_encoding_equal, assert_product_close, dev, encode_both, weight_tensor

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1911_08020_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _weights(g, rows, cols, dtype):
    w = (0.05 * g.standard_normal((rows, cols))).astype(np.float32)
    return synth.f32_to_bf16_bits(w) if dtype == "bf16" else w


def _host(a, pinned):
    x = torch.from_numpy(np.ascontiguousarray(a))
    return x.pin_memory() if pinned else x


@pytest.mark.parametrize("pinned", [True, False])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_reencode_from_host_matches_oracle(dtype, pinned):
    g = np.random.default_rng(60)
    rows, cols, pad = 70, 300, 5
    m = g.choice(np.asarray((1, 3, 8, 16, 33, 100), np.int32), size=rows)
    h = darb.darb_encode(weight_tensor(_weights(g, rows, cols, dtype), dtype), m)
    try:
        for trial in range(2):
            w = _weights(g, rows, cols, dtype)
            nan = np.uint16(0x7FC0) if dtype == "bf16" else np.float32(np.nan)
            wide = np.full((rows, cols + pad), nan, dtype=w.dtype)
            wide[:, :cols] = w
            host = _host(wide.view(np.int16) if dtype == "bf16" else wide, pinned)
            if dtype == "bf16":
                host = host.view(torch.bfloat16)
            W = host[:, :cols]
            W_dev = torch.empty_strided((rows, cols), (cols + pad, 1), dtype=W.dtype, device=dev())
            s = torch.cuda.Stream()
            darb.darb_reencode_host(h, W, W_dev, stream=s)
            darb.darb_sync_status(h, stream=s)   # the NaN padding was never read
            assert_encoding_equal(h, oracle.encode(w, m, dtype))
    finally:
        darb.darb_destroy(h)


@pytest.mark.parametrize("pinned", [True, False])
def test_spmm_from_host_matches_oracle(pinned):
    g = np.random.default_rng(61)
    rows, cols = 257, 1030
    for dtype in ("f32", "bf16"):
        m = g.choice(np.asarray((2, 8, 16, 17, 64), np.int32), size=rows)
        h, ref = encode_both(_weights(g, rows, cols, dtype), m, dtype)
        try:
            for B, padx, pady in ((1, 0, 0), (5, 3, 0), (17, 0, 2), (64, 1, 1), (130, 0, 0)):
                X = synth.activations(cols, B, seed=B)
                xw = np.full((cols, B + padx), np.nan, np.float32)
                xw[:, :B] = X
                Xh = _host(xw, pinned)[:, :B]
                Yfull = _host(np.full((rows, B + pady), 7.0, np.float32), pinned)
                Yh = Yfull[:, :B]
                X_dev = torch.empty((cols, B), device=dev())
                Y_dev = torch.empty((rows, B), device=dev())
                s = torch.cuda.Stream()
                darb.darb_spmm_host(h, Xh, Yh, X_dev, Y_dev, stream=s)
                s.synchronize()
                Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
                assert_product_close(Yh.numpy(), Yr, A, TOL[dtype])
                assert np.all(Yfull.numpy()[:, B:] == 7.0), "wrote outside Y's columns"
        finally:
            darb.darb_destroy(h)


def test_host_calls_reject_bad_buffers():
    g = np.random.default_rng(62)
    rows, cols = 40, 96
    m = np.full(rows, 8, np.int32)
    h, _ = encode_both(_weights(g, rows, cols, "f32"), m, "f32")
    try:
        L = darb.lib()
        X = torch.zeros((cols, 4)).pin_memory()
        Y = torch.zeros((rows, 4)).pin_memory()
        buf = torch.empty((cols + rows) * 4, device=dev())
        s = torch.cuda.current_stream().cuda_stream
        P = lambda t: t.data_ptr()
        # null device buffers, device buffers that overlap
        assert L.darb_spmm_host(h.ptr, P(X), 4, 4, P(Y), 4, None, P(buf), s) == darb.ERR_INVALID_ARG
        assert L.darb_spmm_host(h.ptr, P(X), 4, 4, P(Y), 4, P(buf), P(buf) + 64, s) == darb.ERR_INVALID_ARG
        assert L.darb_spmm_host(h.ptr, P(X), 3, 4, P(Y), 4, P(buf), P(buf) + cols * 16, s) == darb.ERR_INVALID_ARG
        W = torch.zeros((rows, cols)).pin_memory()
        assert L.darb_reencode_host(h.ptr, P(W), cols, None, s) == darb.ERR_INVALID_ARG
        assert L.darb_reencode_host(h.ptr, P(W), cols - 1, P(buf), s) == darb.ERR_INVALID_ARG
        darb.darb_sync_status(h)
    finally:
        darb.darb_destroy(h)
