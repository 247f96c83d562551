"""Checks that pin the CPU oracle to facts outside itself.

Each check raises AssertionError on failure.  They take the oracle module as
an argument so that the mutation test can run them against deliberately
broken builds of the oracle and confirm that every planted mistake is caught.

What each check leans on:

* golden fixtures under tests/golden/ (numbers printed in the paper, cited there);
* closed forms (sum_k ceil(1500 / 2^k) = 1478, ceil block counts);
* numpy's argmax (first maximum) on every block, for BMWM;
* a dense masked matrix times X with numpy's matmul, for the product
  (exact on integer-valued inputs);
* torch.nn.LSTMCell / GRUCell in float64, for the cell equations;
* hand-evaluated closed forms for an all-zero gate matrix.
"""
from __future__ import annotations

import math
import os
from fractions import Fraction

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _golden_lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]


def _kv(line):
    return dict(tok.split("=", 1) for tok in line.split())


# --------------------------------------------------------------------------- top-K row densities
def check_topk_worked_example(orc):
    """Sec. 3.2 example through the mask: K = 28 of 4 x 32 weights, kept 12/6/5/5 -> m = 2/8/8/8."""
    lines = _golden_lines("topk_worked_example.txt")
    head = _kv(lines[0])
    rows, cols, keep = int(head["rows"]), int(head["cols"]), int(head["keep"])
    cases = [_kv(ln) for ln in lines[1:]]
    g = np.random.default_rng(40)
    for dtype in ("f32", "bf16"):
        # row i: its first kept[i] columns hold large weights (magnitudes 1..2, distinct,
        # random signs), the rest small ones (magnitude below 0.5)
        W = (g.uniform(0.01, 0.5, (rows, cols)) * g.choice([-1, 1], (rows, cols))).astype(np.float32)
        for c in cases:
            r, k = int(c["row"]), int(c["kept"])
            W[r, :k] = (1.0 + np.arange(k) / 64.0 + r / 8.0) * g.choice([-1, 1], k)
        stored = W
        if dtype == "bf16":
            stored = (W.view(np.uint32) >> 16).astype(np.uint16)   # magnitudes chosen exact in bf16 above 1
        nnz = orc.topk_row_nnz(stored, keep, dtype)
        assert list(nnz) == [int(c["kept"]) for c in cases], (dtype, nnz)
        m = orc.assign_block_sizes(nnz, cols)
        assert list(m) == [int(c["block_size"]) for c in cases], (dtype, m)


def _threshold_by_enumeration(mag, keep):
    """The K-th largest magnitude as the unique candidate t with
    #(|w| > t) < keep <= #(|w| >= t) (every distinct magnitude is tried)."""
    for t in np.unique(mag):
        if np.count_nonzero(mag > t) < keep <= np.count_nonzero(mag >= t):
            return t
    raise AssertionError("no threshold")


def check_topk_random(orc):
    """Brute force on small matrices: counts of |w| >= t with t found by enumeration;
    with distinct magnitudes the counts add up to exactly K; K = all keeps every weight."""
    g = np.random.default_rng(41)
    for rows, cols in ((3, 4), (5, 7), (8, 33)):
        n = rows * cols
        # distinct magnitudes: a permutation of 1..n, random signs
        W = (g.permutation(n).reshape(rows, cols) + 1).astype(np.float32) * g.choice([-1, 1], (rows, cols))
        for keep in (1, 2, n // 3, n - 1, n):
            nnz = orc.topk_row_nnz(W, keep, "f32")
            t = _threshold_by_enumeration(np.abs(W), keep)
            assert list(nnz) == list(np.count_nonzero(np.abs(W) >= t, axis=1)), (rows, cols, keep)
            assert int(nnz.sum()) == keep
        assert list(orc.topk_row_nnz(W, n, "f32")) == [cols] * rows
        # K = 1 keeps only the largest magnitude's row
        one = orc.topk_row_nnz(W, 1, "f32")
        assert int(one.sum()) == 1 and one[np.unravel_index(np.argmax(np.abs(W)), W.shape)[0]] == 1


def check_topk_ties(orc):
    """Ties at the K-th magnitude all count; +0 and -0 tie; infinities are largest; NaN is refused."""
    W = np.array([[2.0, -2.0, 1.0, 0.0], [-0.0, 2.0, -1.0, 3.0]], np.float32)
    assert list(orc.topk_row_nnz(W, 1, "f32")) == [0, 1]          # 3
    assert list(orc.topk_row_nnz(W, 2, "f32")) == [2, 2]          # 3, then three 2s tie
    assert list(orc.topk_row_nnz(W, 5, "f32")) == [3, 3]          # the two 1s tie
    assert list(orc.topk_row_nnz(W, 7, "f32")) == [4, 4]          # +0 and -0 tie
    W2 = W.copy()
    W2[0, 2] = -np.inf
    assert list(orc.topk_row_nnz(W2, 1, "f32")) == [1, 0]
    W2[1, 1] = np.nan
    try:
        orc.topk_row_nnz(W2, 1, "f32")
    except orc.OracleError as e:
        assert e.status == 2
    else:
        raise AssertionError("NaN accepted")


# --------------------------------------------------------------------------- assignment
def check_assign_worked_example(orc):
    """Sec. 3.2 example: D = 7/32; 37.5% -> m = 2, 18.75% -> m = 8."""
    lines = _golden_lines("assign_worked_example.txt")
    num = int(_kv(lines[0])["matrix_density_num"])
    den = int(_kv(lines[1])["matrix_density_den"])
    cases = [_kv(ln) for ln in lines[2:]]
    cols = 32
    # rows whose densities are the example's, padded with rows at 5/32 so that
    # the matrix density is exactly num/den.
    nnz = [int(Fraction(c["row_density_pct"]) / 100 * cols) for c in cases]
    rows = 4
    nnz += [5] * (rows - len(nnz))
    assert Fraction(sum(nnz), rows * cols) == Fraction(num, den)
    m = orc.assign_block_sizes(nnz, cols)
    for i, c in enumerate(cases):
        assert m[i] == int(c["block_size"]), (i, m[i], c)


def _reference_block_size(nnz, total, rows, cols, m_min, m_max):
    """The rounding rule through log2 of the inverse density (independent form).

    Densities are powers of two 2^-e.  Rounding a density d UP to one means the
    largest e with 2^e <= 1/d, i.e. floor(log2(cols/nnz)); rounding DOWN means
    ceil(log2(cols/nnz)).  Both are taken with int.bit_length on exact integers.
    """
    if nnz == 0:
        m = m_max
    elif Fraction(nnz, cols) >= Fraction(total, rows * cols):
        m = 2 ** ((cols // nnz).bit_length() - 1)
    else:
        m = 2 ** ((-(-cols // nnz) - 1).bit_length())
    return min(max(m, m_min), m_max)


def check_assign_random(orc, seed=0):
    g = np.random.default_rng(seed)
    for trial in range(40):
        rows = int(g.integers(1, 40))
        cols = int(g.integers(1, 300))
        nnz = g.integers(0, cols + 1, size=rows)
        if trial % 5 == 0:
            nnz[:] = nnz[0]          # every row exactly at the matrix density
        m_min, m_max = (1, 256) if trial % 3 else (2, 32)
        got = orc.assign_block_sizes(nnz, cols, m_min, m_max)
        total = int(nnz.sum())
        for r in range(rows):
            want = _reference_block_size(int(nnz[r]), total, rows, cols, m_min, m_max)
            assert got[r] == want, (trial, r, int(nnz[r]), total, rows, cols, got[r], want)


# --------------------------------------------------------------------------- block counts
def check_block_counts(orc):
    for ln in _golden_lines("block_counts.txt"):
        kv = _kv(ln)
        cols, m = int(kv["cols"]), int(kv["block_size"])
        bp = orc.block_pointers([m], cols)
        if "blocks" in kv:
            assert bp[1] == int(kv["blocks"]), (kv, bp)
        if "density_pct" in kv:
            assert Fraction(int(bp[1]), cols) == Fraction(kv["density_pct"]) / 100
    lines = _golden_lines("decoding_1478.txt")
    width = int(lines[0].split("=")[1])
    sizes = [int(s) for s in lines[1].split("=")[1].split(",")]
    want = int(lines[2].split("=")[1])
    bp = orc.block_pointers(sizes, width)
    assert bp[-1] == want, (bp[-1], want)
    assert sum(width // s for s in sizes) != want    # flooring would give 1474


def check_pruning_ratio_identity(orc):
    """ratio = rows*cols / sum(blocks); the paper's printed triples agree to rounding."""
    for ln in _golden_lines("pruning_ratios.txt"):
        params, ratio, kept = (float(t) for t in ln.split())
        assert abs(params / ratio - kept) <= 0.006, ln
    g = np.random.default_rng(1)
    for _ in range(10):
        rows, cols = int(g.integers(1, 20)), int(g.integers(1, 200))
        m = g.integers(1, 70, size=rows).astype(np.int32)
        W = g.standard_normal((rows, cols)).astype(np.float32)
        enc = orc.encode(W, m)
        assert int(enc.blk_ptr[-1]) == sum(-(-cols // int(x)) for x in m)
        for r in range(rows):
            if cols % m[r] == 0:
                assert Fraction(int(enc.blk_ptr[r + 1] - enc.blk_ptr[r]), cols) == Fraction(1, int(m[r]))


# --------------------------------------------------------------------------- BMWM encode
def _numpy_bmwm(Wf, m):
    """Per-block first-argmax of |W| with numpy (np.argmax returns the first max)."""
    rows, cols = Wf.shape
    offs, picks = [], []
    for r in range(rows):
        for lo in range(0, cols, int(m[r])):
            blk = np.abs(Wf[r, lo:lo + int(m[r])].astype(np.float64))
            o = int(np.argmax(blk))
            offs.append(o)
            picks.append((r, lo + o))
    return np.array(offs, dtype=np.uint8), picks


def check_encode_random(orc, seed=2):
    g = np.random.default_rng(seed)
    for trial in range(60):
        rows, cols = int(g.integers(1, 12)), int(g.integers(1, 80))
        m = g.integers(1, min(cols, 40) + 3, size=rows).astype(np.int32)
        W = g.standard_normal((rows, cols)).astype(np.float32)
        if trial % 4 == 1:
            W = np.round(W * 2).astype(np.float32)            # many exact ties and zeros
        if trial % 4 == 2:
            W[g.random(W.shape) < 0.3] = -0.0
        if trial % 4 == 3:
            W = np.where(g.random(W.shape) < 0.5, 1.0, -1.0).astype(np.float32)
        enc = orc.encode(W, m)
        offs, picks = _numpy_bmwm(W, m)
        np.testing.assert_array_equal(enc.off, offs)
        want = np.array([W[r, c] for r, c in picks], dtype=np.float32)
        np.testing.assert_array_equal(enc.val.view(np.uint32), want.view(np.uint32))


def check_encode_bf16(orc, seed=3):
    from paper_1911_08020_gb300 import synth
    g = np.random.default_rng(seed)
    for trial in range(20):
        rows, cols = int(g.integers(1, 10)), int(g.integers(1, 70))
        m = g.integers(1, 33, size=rows).astype(np.int32)
        W = g.standard_normal((rows, cols)).astype(np.float32)
        bits = synth.f32_to_bf16_bits(W)
        enc = orc.encode(bits, m, "bf16")
        offs, picks = _numpy_bmwm(synth.bf16_bits_to_f32(bits), m)
        np.testing.assert_array_equal(enc.off, offs)
        np.testing.assert_array_equal(enc.val, np.array([bits[r, c] for r, c in picks], np.uint16))


def check_encode_special_values(orc):
    inf = np.float32(np.inf)
    W = np.array([[0.0, -0.0, 0.0, -0.0,   -0.0, 0.0, 0.0, 0.0,   2.0, -2.0, 2.0, 1.0,
                   1.0, -inf, inf, 3.0,    5.0, 5.0, -5.0, 5.0,   0.0, 0.0, 0.0, 7.5]],
                 dtype=np.float32)
    enc = orc.encode(W, [4])
    assert list(enc.off) == [0, 0, 0, 1, 0, 3]
    assert enc.val.view(np.uint32)[1] == np.float32(-0.0).view(np.uint32)
    assert list(enc.val[[2, 3, 4, 5]]) == [2.0, -inf, 5.0, 7.5]
    # one block spanning the row (m >= cols) and a short tail block
    enc = orc.encode(np.array([[1, 9, -9, 3, 4]], np.float32), [8])
    assert list(enc.off) == [1] and enc.val[0] == 9
    enc = orc.encode(np.array([[1, 2, 3, 4, 5, -6, 0]], np.float32), [3])
    assert list(enc.off) == [2, 2, 0] and list(enc.val) == [3, -6, 0]
    # m = 1 keeps every weight
    W = np.arange(-3, 4, dtype=np.float32)[None, :]
    enc = orc.encode(W, [1])
    np.testing.assert_array_equal(enc.val, W[0])
    assert not enc.off.any()


def check_encode_nan(orc):
    W = np.ones((2, 8), np.float32)
    W[1, 5] = np.nan
    try:
        orc.encode(W, [4, 4])
    except orc.OracleError as e:
        assert e.status == orc.NONFINITE
    else:
        raise AssertionError("NaN weight was accepted")


# --------------------------------------------------------------------------- product
def _numpy_masked(enc):
    """Dense M (.) W built from (row, j, off) with numpy indexing."""
    Wd = np.zeros((enc.rows, enc.cols))
    v = enc.values_f64()
    for r in range(enc.rows):
        js = np.arange(enc.blk_ptr[r + 1] - enc.blk_ptr[r])
        cols = js * int(enc.m[r]) + enc.off[enc.blk_ptr[r]:enc.blk_ptr[r + 1]]
        Wd[r, cols] = v[enc.blk_ptr[r]:enc.blk_ptr[r + 1]]
    return Wd


def check_product_exhaustive(orc, seed=4):
    """Every m in 1..cols on tiny integer matrices: exact equality with numpy."""
    g = np.random.default_rng(seed)
    for cols in range(1, 25):
        for mm in range(1, cols + 1):
            rows = int(g.integers(1, 9))
            m = np.full(rows, mm, np.int32)
            m[g.random(rows) < 0.4] = int(g.integers(1, cols + 1))
            W = g.integers(-8, 9, size=(rows, cols)).astype(np.float32)
            X = g.integers(-5, 6, size=(cols, 3)).astype(np.float32)
            enc = orc.encode(W, m)
            Wd = _numpy_masked(enc)
            np.testing.assert_array_equal(orc.masked_dense(enc), Wd)
            # each block keeps exactly one entry of W and it is the block's max |w|
            for r in range(rows):
                for lo in range(0, cols, int(m[r])):
                    seg = Wd[r, lo:lo + int(m[r])]
                    assert np.count_nonzero(seg) <= 1
                    assert np.abs(seg).max() == np.abs(W[r, lo:lo + int(m[r])]).max()
            Y = orc.darb_spmm(enc, X)
            np.testing.assert_array_equal(Y, Wd @ X.astype(np.float64))


def check_product_random(orc, seed=5):
    g = np.random.default_rng(seed)
    for _ in range(10):
        rows, cols, B = int(g.integers(1, 60)), int(g.integers(1, 300)), int(g.integers(1, 7))
        m = g.integers(1, 65, size=rows).astype(np.int32)
        W = g.standard_normal((rows, cols)).astype(np.float32)
        X = g.standard_normal((cols, B)).astype(np.float32)
        enc = orc.encode(W, m)
        Y, A = orc.darb_spmm(enc, X, with_absdot=True)
        Wd = _numpy_masked(enc)
        np.testing.assert_allclose(Y, Wd @ X.astype(np.float64), rtol=0, atol=1e-12)
        np.testing.assert_allclose(A, np.abs(Wd) @ np.abs(X.astype(np.float64)), rtol=1e-14, atol=0)


def check_product_f32_timed(orc, seed=11):
    """The single-precision loop timed as the CPU baseline: exact on small
    integer inputs (every partial sum is an exactly representable integer),
    and within fp32 summation error of numpy's masked dense product in
    float64 on Gaussian inputs (|err| <= n * 2^-24 * sum |w x|)."""
    g = np.random.default_rng(seed)
    for _ in range(10):
        rows, cols, B = int(g.integers(1, 60)), int(g.integers(1, 300)), int(g.integers(1, 7))
        m = g.integers(1, 65, size=rows).astype(np.int32)
        Wi = g.integers(-8, 9, size=(rows, cols)).astype(np.float32)
        Xi = g.integers(-5, 6, size=(cols, B)).astype(np.float32)
        enc = orc.encode(Wi, m)
        np.testing.assert_array_equal(orc.darb_spmm_f32(enc, Xi), _numpy_masked(enc) @ Xi.astype(np.float64))
        W = g.standard_normal((rows, cols)).astype(np.float32)
        X = g.standard_normal((cols, B)).astype(np.float32)
        enc = orc.encode(W, m)
        Wd = _numpy_masked(enc)
        exact = Wd @ X.astype(np.float64)
        bound = (np.abs(Wd) @ np.abs(X.astype(np.float64))) * (cols + 1) * 2.0 ** -24
        assert np.all(np.abs(orc.darb_spmm_f32(enc, X) - exact) <= bound)


# --------------------------------------------------------------------------- RNN cells
def _enc_rnn(orc, rows, cols, seed):
    g = np.random.default_rng(seed)
    m = g.integers(1, 9, size=rows).astype(np.int32)
    W = (0.5 * g.standard_normal((rows, cols))).astype(np.float32)
    return orc.encode(W, m), g


def check_lstm_vs_torch(orc, seed=6):
    import torch
    for I, H, B in ((5, 4, 3), (0, 3, 2), (7, 6, 1)):
        enc, g = _enc_rnn(orc, 4 * H, I + H, seed + I)
        x = g.standard_normal((I, B)); h = g.standard_normal((H, B)); c = g.standard_normal((H, B))
        bias = g.standard_normal(4 * H)
        ho, co, _ = orc.lstm_step(enc, I, H, x, h, c, bias)
        Wd = torch.from_numpy(_numpy_masked(enc))
        cell = torch.nn.LSTMCell(I, H, bias=True).double()
        with torch.no_grad():
            cell.weight_ih.copy_(Wd[:, :I]); cell.weight_hh.copy_(Wd[:, I:])
            cell.bias_ih.copy_(torch.from_numpy(bias)); cell.bias_hh.zero_()
            ht, ct = cell(torch.from_numpy(x.T.copy()), (torch.from_numpy(h.T.copy()),
                                                         torch.from_numpy(c.T.copy())))
        np.testing.assert_allclose(ho, ht.numpy().T, rtol=0, atol=1e-12)
        np.testing.assert_allclose(co, ct.numpy().T, rtol=0, atol=1e-12)


def check_gru_vs_torch(orc, seed=7):
    import torch
    for I, H, B in ((5, 4, 3), (0, 3, 2), (6, 6, 1)):
        enc, g = _enc_rnn(orc, 3 * H, I + H, seed + I)
        x = g.standard_normal((I, B)); h = g.standard_normal((H, B))
        bi, bh = g.standard_normal(3 * H), g.standard_normal(3 * H)
        ho, _ = orc.gru_step(enc, I, H, x, h, bi, bh)
        Wd = torch.from_numpy(_numpy_masked(enc))
        cell = torch.nn.GRUCell(I, H, bias=True).double()
        with torch.no_grad():
            cell.weight_ih.copy_(Wd[:, :I]); cell.weight_hh.copy_(Wd[:, I:])
            cell.bias_ih.copy_(torch.from_numpy(bi)); cell.bias_hh.copy_(torch.from_numpy(bh))
            ht = cell(torch.from_numpy(x.T.copy()), torch.from_numpy(h.T.copy()))
        np.testing.assert_allclose(ho, ht.numpy().T, rtol=0, atol=1e-12)


def _sig(v):
    return 1.0 / (1.0 + math.exp(-v))


def check_rnn_zero_weights(orc):
    """W = 0: every gate equals its bias; closed forms evaluated by hand."""
    I, H = 2, 3
    z = np.zeros((4 * H, I + H), np.float32)
    enc = orc.encode(z, np.full(4 * H, 2, np.int32))
    c0 = np.array([[0.3], [-1.2], [2.0]])
    b = np.array([0.1, -0.2, 0.3, 1.0, 2.0, -1.0, -0.5, 0.25, 0.0, 0.7, -0.7, 1.5])
    ho, co, _ = orc.lstm_step(enc, I, H, np.ones((I, 1)), np.full((H, 1), 9.0), c0, b)
    for j in range(H):
        c = _sig(b[H + j]) * c0[j, 0] + _sig(b[j]) * math.tanh(b[2 * H + j])
        assert abs(co[j, 0] - c) < 1e-15 and abs(ho[j, 0] - _sig(b[3 * H + j]) * math.tanh(c)) < 1e-15
    enc = orc.encode(np.zeros((3 * H, I + H), np.float32), np.full(3 * H, 3, np.int32))
    bi, bh = b[:3 * H], np.linspace(-1, 1, 3 * H)
    h0 = np.array([[0.5], [-0.25], [1.0]])
    ho, _ = orc.gru_step(enc, I, H, np.ones((I, 1)), h0, bi, bh)
    for j in range(H):
        r = _sig(bi[j] + bh[j]); zz = _sig(bi[H + j] + bh[H + j])
        n = math.tanh(bi[2 * H + j] + r * bh[2 * H + j])
        assert abs(ho[j, 0] - ((1 - zz) * n + zz * h0[j, 0])) < 1e-15


def check_gru_split_columns(orc):
    """One kept weight per row (m >= cols): a GRU n-gate whose weight sits on the
    h side is scaled by r, one on the x side is not."""
    I, H = 2, 1
    W = np.zeros((3, 3), np.float32)
    W[0, 0] = 0.5     # r row: x side
    W[1, 2] = -0.4    # z row: h side
    W[2, 2] = 0.8     # n row: h side
    enc = orc.encode(W, np.full(3, 4, np.int32))
    x = np.array([[1.5], [0.0]]); h = np.array([[0.6]])
    ho, _ = orc.gru_step(enc, I, H, x, h)
    w04, w08 = float(np.float32(-0.4)), float(np.float32(0.8))   # the stored fp32 weights
    r = _sig(0.5 * 1.5); zz = _sig(w04 * 0.6)
    n = math.tanh(r * (w08 * 0.6))
    assert abs(ho[0, 0] - ((1 - zz) * n + zz * 0.6)) < 1e-15
    W[2, 2] = 0.0
    W[2, 0] = 0.8     # n row: x side
    enc = orc.encode(W, np.full(3, 4, np.int32))
    ho, _ = orc.gru_step(enc, I, H, x, h)
    n = math.tanh(w08 * 1.5)
    assert abs(ho[0, 0] - ((1 - zz) * n + zz * 0.6)) < 1e-15


ALL_CHECKS = [
    check_topk_worked_example, check_topk_random, check_topk_ties,
    check_assign_worked_example, check_assign_random, check_block_counts,
    check_pruning_ratio_identity, check_encode_random, check_encode_bf16,
    check_encode_special_values, check_encode_nan, check_product_exhaustive,
    check_product_random, check_product_f32_timed, check_lstm_vs_torch, check_gru_vs_torch, check_rnn_zero_weights,
    check_gru_split_columns,
]
