"""CUDA path against the CPU oracle, element by element (needs a GB300).

Encodings must match bit for bit; products and RNN steps must stay inside the
tolerances derived in gpu_helpers.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from paper_1911_08020_gb300 import darb, synth
from tests.gpu_helpers import (TOL, assert_encoding_equal, assert_product_close, dev, encode_both,
                               gru_bound, lstm_bounds, t, weight_tensor)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1911_08020_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _random_case(g, rows, cols, dtype, mset=None):
    w = (0.05 * g.standard_normal((rows, cols)) * np.exp(0.5 * g.standard_normal((rows, 1)))).astype(np.float32)
    if mset is None:
        m = g.integers(1, 257, size=rows).astype(np.int32)
    else:
        m = g.choice(np.asarray(mset, np.int32), size=rows)
    stored = synth.f32_to_bf16_bits(w) if dtype == "bf16" else w
    return stored, m


# --------------------------------------------------------------------------- encode
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_encode_small_ragged_shapes(dtype):
    g = np.random.default_rng(10)
    shapes = [(1, 1), (1, 7), (3, 33), (33, 17), (31, 100), (64, 129), (70, 300), (5, 1000),
              (40, 12289), (2, 20000)]
    for rows, cols in shapes:
        for mset in (None, (1, 2, 3), (10, 15, 20, 30), (16, 32, 64), (255, 256), (5, 8, 13, 200)):
            stored, m = _random_case(g, rows, cols, dtype, mset)
            h, ref = encode_both(stored, m, dtype)
            try:
                assert_encoding_equal(h, ref)
            finally:
                darb.darb_destroy(h)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_encode_ties_zeros_and_infinities(dtype):
    g = np.random.default_rng(11)
    rows, cols = 67, 301
    for mode in range(4):
        if mode == 0:
            w = np.round(g.standard_normal((rows, cols)) * 2).astype(np.float32)       # many ties
        elif mode == 1:
            w = np.where(g.random((rows, cols)) < 0.5, 0.0, -0.0).astype(np.float32)  # all +-0
        elif mode == 2:
            w = np.where(g.random((rows, cols)) < 0.5, 1.0, -1.0).astype(np.float32)  # all tied
        else:
            w = g.standard_normal((rows, cols)).astype(np.float32)
            w[g.random((rows, cols)) < 0.05] = np.inf
            w[g.random((rows, cols)) < 0.05] = -np.inf
        m = g.integers(1, 70, size=rows).astype(np.int32)
        stored = synth.f32_to_bf16_bits(w) if dtype == "bf16" else w
        h, ref = encode_both(stored, m, dtype)
        try:
            assert_encoding_equal(h, ref)
        finally:
            darb.darb_destroy(h)


@pytest.mark.parametrize("name", list(synth.WORKLOADS))
def test_encode_workloads_full_size(name):
    wl = synth.WORKLOADS[name]
    for i in range(len(wl.shapes)):
        _, stored, m = synth.matrix(wl, i)
        h, ref = encode_both(stored, m, wl.dtype)
        try:
            assert_encoding_equal(h, ref)
            info = darb.darb_info(h)
            assert info["nnzb"] == int(ref.blk_ptr[-1])
            ratio = info["rows"] * info["cols"] / info["nnzb"]
            want = synth.expected_ratio(wl.choices, wl.probs)
            assert abs(ratio / want - 1) < 0.1, (ratio, want)
        finally:
            darb.darb_destroy(h)


def test_encode_strided_and_misaligned_rows():
    g = np.random.default_rng(12)
    rows, cols = 50, 203
    for dtype in ("f32", "bf16"):
        big, m = _random_case(g, rows, cols + 13, dtype, (4, 7, 16, 64))
        Wt = weight_tensor(big, dtype)
        for c0 in (0, 1, 3):
            sub = Wt[:, c0:c0 + cols]
            h = darb.darb_encode(sub, m)
            ref = oracle.encode(np.ascontiguousarray(big[:, c0:c0 + cols]), m, dtype)
            try:
                assert_encoding_equal(h, ref)
            finally:
                darb.darb_destroy(h)


@pytest.mark.parametrize("mset", [(8,), (128, 256), (8, 16, 32, 64, 128, 256)])
def test_encode_bf16_power_of_two_block_sizes(mset):
    """bf16 weights whose block sizes are all powers of two from 8 to 256, in
    rows padded to a multiple of 8 elements: the encoder's row path (tiles of
    2048 columns, one 16-byte unit per lane; several lanes per block above
    m = 64).  Every row length, so that a row's last block and last 8-element
    unit may be partial; Gaussian, tied, signed-zero and infinite weights; the
    padding past each row holds NaNs, which must never be read."""
    g = np.random.default_rng(14)
    for rows, cols in ((1, 8), (3, 17), (33, 100), (64, 1000), (40, 2049), (7, 4296), (5, 12289)):
        ldw = (cols + 7) // 8 * 8 + 8
        for mode in range(4):
            if mode == 1:
                w = np.round(g.standard_normal((rows, cols)) * 2).astype(np.float32)       # many ties
            elif mode == 2:
                w = np.where(g.random((rows, cols)) < 0.5, 0.0, -0.0).astype(np.float32)  # all +-0
            else:
                w = g.standard_normal((rows, cols)).astype(np.float32)
                if mode == 3:
                    w[g.random((rows, cols)) < 0.05] = np.inf
                    w[g.random((rows, cols)) < 0.05] = -np.inf
            m = g.choice(np.asarray(mset, np.int32), size=rows)
            stored = synth.f32_to_bf16_bits(w)
            big = np.full((rows, ldw), 0x7FC1, np.uint16)   # NaN past each row's end
            big[:, :cols] = stored
            Wt = weight_tensor(big, "bf16")[:, :cols]
            h = darb.darb_encode(Wt, m)
            try:
                assert_encoding_equal(h, oracle.encode(stored, m, "bf16"))
            finally:
                darb.darb_destroy(h)


def test_encode_nan_is_reported():
    w = np.ones((40, 64), np.float32)
    w[37, 61] = np.nan
    with pytest.raises(darb.DarbError) as e:
        darb.darb_encode(t(w), np.full(40, 8, np.int32))
    assert e.value.status == darb.ERR_NONFINITE
    wb = torch.from_numpy(w).to(dev()).to(torch.bfloat16)
    with pytest.raises(darb.DarbError) as e:
        darb.darb_encode(wb, np.full(40, 8, np.int32))
    assert e.value.status == darb.ERR_NONFINITE


def test_reencode_and_status():
    g = np.random.default_rng(13)
    w1, m = _random_case(g, 90, 400, "f32", (8, 16, 32))
    w2, _ = _random_case(g, 90, 400, "f32", (8,))
    h = darb.darb_encode(t(w1), m)
    try:
        darb.darb_reencode(h, t(w2))
        darb.darb_sync_status(h)
        assert_encoding_equal(h, oracle.encode(w2, m))
        w3 = w2.copy()
        w3[5, 5] = np.nan
        darb.darb_reencode(h, t(w3))
        with pytest.raises(darb.DarbError) as e:
            darb.darb_sync_status(h)
        assert e.value.status == darb.ERR_NONFINITE
        darb.darb_sync_status(h)   # flag cleared
    finally:
        darb.darb_destroy(h)


def test_import_export_roundtrip():
    g = np.random.default_rng(14)
    for dtype in ("f32", "bf16"):
        stored, m = _random_case(g, 77, 345, dtype, (1, 3, 16, 17, 100))
        ref = oracle.encode(stored, m, dtype)
        h = darb.darb_import(ref.val, ref.off, m, darb.BF16 if dtype == "bf16" else darb.F32, 77, 345)
        try:
            assert_encoding_equal(h, ref)
            X = synth.activations(345, 5, seed=1)
            Y = darb.darb_spmm(h, t(X)).cpu().numpy()
            Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
            assert_product_close(Y, Yr, A, TOL[dtype])
        finally:
            darb.darb_destroy(h)


# --------------------------------------------------------------------------- product
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_spmm_batches_and_ragged(dtype):
    g = np.random.default_rng(20)
    for rows, cols in ((1, 1), (37, 91), (100, 257), (257, 1030)):
        stored, m = _random_case(g, rows, cols, dtype, (1, 2, 3, 8, 10, 16, 17, 32, 64, 200))
        h, ref = encode_both(stored, m, dtype)
        try:
            for B in (1, 2, 3, 4, 5, 8, 9, 16, 17, 31, 33, 64, 100, 129, 256):
                X = synth.activations(cols, B, seed=B)
                Y = darb.darb_spmm(h, t(X)).cpu().numpy()
                Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
                assert_product_close(Y, Yr, A, TOL[dtype])
        finally:
            darb.darb_destroy(h)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_spmm_wide_column_slices(dtype):
    """Wide matrices at batches above 16, where the columns are split over a
    cluster: block sizes whose least common multiple divides the slice (no
    block crosses a slice; the last slice runs past the matrix at 7000 and
    9000 columns), one that divides it exactly (7000 columns, m in {10, 20,
    40}), and sizes whose slices need the rows past their end (m up to 200)."""
    g = np.random.default_rng(25)
    for rows, cols, mset in ((300, 7000, (16, 32, 64)), (300, 7000, (10, 20, 40)), (260, 9000, (16, 64, 256)),
                             (200, 6000, (3, 7, 16, 200)), (130, 12000, (8, 32))):
        stored, m = _random_case(g, rows, cols, dtype, mset)
        h, ref = encode_both(stored, m, dtype)
        try:
            for B in (17, 40, 64):
                X = synth.activations(cols, B, seed=B + cols)
                Y = darb.darb_spmm(h, t(X)).cpu().numpy()
                Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
                assert_product_close(Y, Yr, A, TOL[dtype])
        finally:
            darb.darb_destroy(h)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_spmm_too_wide_for_resident_slices(dtype):
    """Matrices whose activation slice does not fit shared memory even split 8
    ways (tens of thousands of columns) take the staged-rounds kernel at every
    batch; products still match the oracle, ragged tiles included."""
    g = np.random.default_rng(26)
    for rows, cols, mset in ((100, 20000, (16, 64)), (70, 30000, (5, 32, 256))):
        stored, m = _random_case(g, rows, cols, dtype, mset)
        h, ref = encode_both(stored, m, dtype)
        try:
            for B in (17, 40, 100):
                X = synth.activations(cols, B, seed=B + 7)
                Y = darb.darb_spmm(h, t(X)).cpu().numpy()
                Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
                assert_product_close(Y, Yr, A, TOL[dtype])
        finally:
            darb.darb_destroy(h)


def test_spmm_leading_dimensions_and_alignment():
    g = np.random.default_rng(21)
    rows, cols = 130, 300
    stored, m = _random_case(g, rows, cols, "f32", (4, 16, 48))
    h, ref = encode_both(stored, m, "f32")
    try:
        for B, pad, shift in ((1, 3, 0), (6, 2, 1), (20, 5, 1), (64, 4, 0), (64, 4, 1), (130, 7, 3)):
            Xbig = synth.activations(cols, B + pad + shift, seed=B)
            Xd = t(Xbig)[:, shift:shift + B]           # ldx = B + pad + shift, maybe unaligned
            Yd = torch.full((rows, B + 5), 7.0, device=dev())
            darb.darb_spmm(h, Xd, Yd[:, :B])
            Yr, A = oracle.darb_spmm(ref, Xbig[:, shift:shift + B], with_absdot=True)
            Yh = Yd.cpu().numpy()
            assert_product_close(Yh[:, :B], Yr, A, TOL["f32"])
            assert np.all(Yh[:, B:] == 7.0), "wrote outside Y's columns"
    finally:
        darb.darb_destroy(h)


def test_spmm_unselected_infinities_do_not_leak():
    g = np.random.default_rng(22)
    rows, cols = 100, 512
    stored, m = _random_case(g, rows, cols, "f32", (8, 32, 100))
    h, ref = encode_both(stored, m, "f32")
    try:
        used = np.zeros(cols, bool)
        for r in range(rows):
            p0, p1 = ref.blk_ptr[r], ref.blk_ptr[r + 1]
            used[np.arange(p1 - p0) * m[r] + ref.off[p0:p1]] = True
        for B in (1, 4, 16, 64):
            X = synth.activations(cols, B, seed=3)
            X[~used, :] = np.inf
            Y = darb.darb_spmm(h, t(X)).cpu().numpy()
            Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
            assert np.isfinite(Y).all()
            assert_product_close(Y, Yr, A, TOL["f32"])
    finally:
        darb.darb_destroy(h)


@pytest.mark.parametrize("B", [64, 256])
def test_spmm_fc6_bf16_unselected_nonfinite_stay_out(B):
    """FC6 (4096 x 9216 bf16) through darb_spmm at the bench's wide batches:
    +Inf and NaN in activation rows that no kept weight selects must not reach
    Y (Fig. 6(b): each block contributes only the activation it selects), and
    every output matches the oracle element by element.  Every 7th column of
    W is zeroed so that BMWM never keeps a weight there (a block's maximum
    magnitude is never 0 for these Gaussian weights)."""
    wl = synth.WORKLOADS["fc6_fc7"]
    _, stored, m = synth.matrix(wl, 0)
    stored = stored.copy()
    stored[:, 3::7] = 0
    h, ref = encode_both(stored, m, wl.dtype)
    try:
        cols = wl.shapes[0][1]
        used = np.zeros(cols, bool)
        nb = ref.blk_ptr[1:] - ref.blk_ptr[:-1]
        rows_of_block = np.repeat(np.arange(len(m)), nb)
        j = np.arange(ref.blk_ptr[-1]) - ref.blk_ptr[rows_of_block]
        used[j * m[rows_of_block] + ref.off] = True
        assert (~used).sum() >= cols // 7, "the case needs unselected activation rows"
        X = synth.activations(cols, B, seed=wl.seed + 70 + B)
        unused = np.flatnonzero(~used)
        X[unused[0::2], :] = np.inf
        X[unused[1::2], :] = np.nan
        assert darb.darb_spmm_path(h, B) == (darb.PATH_CUDA_CORES, 1)
        Y = darb.darb_spmm(h, t(X)).cpu().numpy()
        Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
        assert np.isfinite(Yr).all() and np.isfinite(Y).all()
        assert_product_close(Y, Yr, A, TOL[wl.dtype])
    finally:
        darb.darb_destroy(h)


@pytest.mark.parametrize("name", list(synth.WORKLOADS))
def test_spmm_workloads_full_size(name):
    wl = synth.WORKLOADS[name]
    batches = sorted(set(wl.batches) | {1})
    for i in range(len(wl.shapes)):
        _, stored, m = synth.matrix(wl, i)
        h, ref = encode_both(stored, m, wl.dtype)
        try:
            for B in batches:
                X = synth.activations(wl.shapes[i][1], B, seed=wl.seed + 50 + B)
                Y = darb.darb_spmm(h, t(X)).cpu().numpy()
                Yr, A = oracle.darb_spmm(ref, X, with_absdot=True)
                assert_product_close(Y, Yr, A, TOL[wl.dtype])
        finally:
            darb.darb_destroy(h)


def test_spmm_in_cuda_graph():
    g = np.random.default_rng(23)
    stored, m = _random_case(g, 300, 700, "bf16", (16, 32, 64))
    h, ref = encode_both(stored, m, "bf16")
    try:
        for B in (1, 16, 64):
            X = t(synth.activations(700, B, seed=B))
            Y = torch.empty((300, B), device=dev())
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
            Yr, A = oracle.darb_spmm(ref, X.cpu().numpy(), with_absdot=True)
            assert_product_close(Y.cpu().numpy(), Yr, A, TOL["bf16"])
    finally:
        darb.darb_destroy(h)


# --------------------------------------------------------------------------- RNN steps
def _lstm_case(g, I, H, dtype, mset):
    w = (0.3 * g.standard_normal((4 * H, I + H))).astype(np.float32)
    stored = synth.f32_to_bf16_bits(w) if dtype == "bf16" else w
    m = g.choice(np.asarray(mset, np.int32), size=4 * H)
    return stored, m


def _run_lstm(h, ref, I, H, B, x, hp, cp, bias, tol):
    ho = torch.empty((H, B), device=dev())
    co = torch.empty((H, B), device=dev())
    darb.darb_lstm_step(h, I, H, B, t(x) if I else None, t(hp), t(cp),
                        t(bias) if bias is not None else None, ho, co)
    hg, cg = ho.cpu().numpy().astype(np.float64), co.cpu().numpy().astype(np.float64)
    hr, cr, ga = oracle.lstm_step(ref, I, H, x, hp, cp, bias)
    bc, bh = lstm_bounds(ga, cp, tol)
    assert np.all(np.abs(cg - cr) <= bc), float(np.max(np.abs(cg - cr) - bc))
    assert np.all(np.abs(hg - hr) <= bh), float(np.max(np.abs(hg - hr) - bh))
    return ho.cpu().numpy(), co.cpu().numpy()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_lstm_step_small(dtype):
    g = np.random.default_rng(30)
    for I, H, B in ((0, 5, 1), (3, 4, 2), (7, 33, 3), (20, 40, 8), (64, 100, 9), (10, 70, 33)):
        stored, m = _lstm_case(g, I, H, dtype, (1, 2, 3, 4, 8, 17))
        h, ref = encode_both(stored, m, dtype)
        try:
            x = synth.activations(I, B, seed=I)
            hp, cp = synth.state(H, B, seed=H), synth.state(H, B, seed=H + 1, scale=1.0)
            for bias in (None, synth.bias(4 * H, seed=I)):
                _run_lstm(h, ref, I, H, B, x, hp, cp, bias, TOL[dtype])
        finally:
            darb.darb_destroy(h)


def _run_gru(h, ref, I, H, B, x, hp, bi, bh, tol):
    ho = torch.empty((H, B), device=dev())
    darb.darb_gru_step(h, I, H, B, t(x) if I else None, t(hp), t(bi) if bi is not None else None,
                       t(bh) if bh is not None else None, ho)
    hg = ho.cpu().numpy().astype(np.float64)
    hr, ga = oracle.gru_step(ref, I, H, x, hp, bi, bh)
    bound = gru_bound(ga, hp, hr, tol)
    assert np.all(np.abs(hg - hr) <= bound), float(np.max(np.abs(hg - hr) - bound))
    return ho.cpu().numpy()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_gru_step_small(dtype):
    g = np.random.default_rng(31)
    for I, H, B in ((0, 5, 1), (3, 4, 2), (7, 33, 3), (20, 40, 8), (64, 100, 9), (10, 70, 33)):
        w = (0.3 * g.standard_normal((3 * H, I + H))).astype(np.float32)
        stored = synth.f32_to_bf16_bits(w) if dtype == "bf16" else w
        m = g.choice(np.asarray((1, 2, 5, 8, 16), np.int32), size=3 * H)
        h, ref = encode_both(stored, m, dtype)
        try:
            x = synth.activations(I, B, seed=I)
            hp = synth.state(H, B, seed=H)
            _run_gru(h, ref, I, H, B, x, hp, None, None, TOL[dtype])
            _run_gru(h, ref, I, H, B, x, hp, synth.bias(3 * H, seed=1), synth.bias(3 * H, seed=2), TOL[dtype])
        finally:
            darb.darb_destroy(h)


@pytest.mark.parametrize("name,batch", [("lstm_1024", 1), ("lstm_1024", 32), ("lstm_lm_1500", 20)])
def test_lstm_workload_steps(name, batch):
    """A few full-size steps, each checked against the oracle fed the GPU's own state."""
    wl = synth.WORKLOADS[name]
    I, H = wl.input_size, wl.hidden
    _, stored, m = synth.matrix(wl, 0)
    h, ref = encode_both(stored, m, wl.dtype)
    try:
        xs = synth.rnn_inputs(wl, batch, 3)
        hp = np.zeros((H, batch), np.float32)
        cp = np.zeros((H, batch), np.float32)
        bias = synth.bias(4 * H, seed=wl.seed)
        for step in range(3):
            hp, cp = _run_lstm(h, ref, I, H, batch, xs[step], hp, cp, bias, TOL[wl.dtype])
    finally:
        darb.darb_destroy(h)


def test_gru_workload_steps():
    wl = synth.WORKLOADS["gru_1024"]
    I, H, B = wl.input_size, wl.hidden, wl.batches[0]
    _, stored, m = synth.matrix(wl, 0)
    h, ref = encode_both(stored, m, wl.dtype)
    try:
        xs = synth.rnn_inputs(wl, B, 3)
        hp = np.zeros((H, B), np.float32)
        bi, bh = synth.bias(3 * H, seed=1), synth.bias(3 * H, seed=2)
        for step in range(3):
            hp = _run_gru(h, ref, I, H, B, xs[step], hp, bi, bh, TOL[wl.dtype])
    finally:
        darb.darb_destroy(h)


def test_step_argument_checks():
    g = np.random.default_rng(32)
    stored, m = _lstm_case(g, 4, 6, "f32", (2, 4))
    h = darb.darb_encode(t(stored), m)
    try:
        z = torch.zeros((6, 2), device=dev())
        o1, o2 = torch.empty_like(z), torch.empty_like(z)
        x = torch.zeros((4, 2), device=dev())
        with pytest.raises(darb.DarbError):
            darb.darb_lstm_step(h, 5, 6, 2, x, z, z, None, o1, o2)      # I + H != cols
        with pytest.raises(darb.DarbError):
            darb.darb_lstm_step(h, 4, 6, 2, x, z, z, None, z, o2)       # output aliases input
        with pytest.raises(darb.DarbError):
            darb.darb_gru_step(h, 4, 6, 2, x, z, None, None, o1)       # 4H rows is not a GRU
    finally:
        darb.darb_destroy(h)
