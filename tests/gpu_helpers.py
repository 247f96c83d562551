"""Shared helpers of the GPU parity tests: tensors, oracle comparisons, tolerances.

Tolerances (the bar every product is held to, from the arithmetic):

* a product output y against the fp64 oracle ref:  |y - ref| <= tol * S, where
  S = sum_j |val_j * x_j| over the kept weights of that output (for S = 0, y
  must be 0).  tol = 1e-5 for fp32 weights and 2e-3 for bf16 weights; both
  kernels compute fp32 products of exactly widened weights and fp32 inputs and
  add them in fp32, whose rounding error is far inside either bound;
* RNN cells: the gate pre-activation errors (tol * S per gate, S including
  |bias|) pushed through the cell with |sigmoid'| <= 1/4, |tanh'| <= 1 and
  |sigmoid|, |tanh| <= 1, plus 2e-6 for the fp32 expf / tanhf calls.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_1911_08020_gb300 import darb, synth

TOL = {"f32": 1e-5, "bf16": 2e-3}
TRANSCENDENTAL_SLACK = 2e-6


def dev():
    return torch.device("cuda:0")


def t(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev())


def weight_tensor(w_stored, dtype):
    """Device tensor holding exactly the stored weights (fp32, or bf16 bits)."""
    if dtype == "bf16":
        return t(w_stored.view(np.int16)).view(torch.bfloat16)
    return t(w_stored)


def encode_both(w_stored, m, dtype):
    h = darb.darb_encode(weight_tensor(w_stored, dtype), m)
    ref = oracle.encode(w_stored, m, dtype)
    return h, ref


def assert_encoding_equal(h, ref):
    val, off, bp, m = darb.darb_export(h)
    np.testing.assert_array_equal(bp, ref.blk_ptr)
    np.testing.assert_array_equal(m, ref.m)
    np.testing.assert_array_equal(off, ref.off)
    view = np.uint16 if ref.dtype == "bf16" else np.uint32
    np.testing.assert_array_equal(val.view(view), ref.val.view(view))


def assert_product_close(Y, ref_Y, absdot, tol):
    Y = np.asarray(Y, dtype=np.float64)
    err = np.abs(Y - ref_Y)
    zero = absdot == 0
    assert np.all(Y[zero] == 0), "output with no contributing terms is not zero"
    bound = tol * absdot
    bad = err > bound
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{bad.sum()} outputs out of tolerance, first at {tuple(i)}: "
                             f"got {Y[tuple(i)]!r}, want {ref_Y[tuple(i)]!r}, bound {bound[tuple(i)]!r}")
    rel = np.where(zero, 0.0, err / np.where(zero, 1.0, absdot))
    return float(rel.max(initial=0.0))


def lstm_bounds(ga, c_prev, tol):
    """Per-(unit, b) error bounds for c and h from gate scales ga (4H x B)."""
    H = ga.shape[0] // 4
    Si, Sf, Sg, So = ga[:H], ga[H:2 * H], ga[2 * H:3 * H], ga[3 * H:]
    bc = tol * (Si / 4 + Sf * np.abs(c_prev) / 4 + Sg) + TRANSCENDENTAL_SLACK
    bh = tol * So / 4 + bc + TRANSCENDENTAL_SLACK
    return bc, bh


def gru_bound(ga, h_prev, h_ref, tol):
    """Per-(unit, b) error bound for h from gate scales ga (3H x B x 2: x part, h part)."""
    H = ga.shape[0] // 3
    Sa, Sb = ga[..., 0], ga[..., 1]
    dr = tol * (Sa[:H] + Sb[:H]) / 4
    dz = tol * (Sa[H:2 * H] + Sb[H:2 * H]) / 4
    # |bh_n| <= Sb_n ; |n - h_prev| <= 1 + |h_prev|
    dn = tol * (Sa[2 * H:] + Sb[2 * H:]) + dr * Sb[2 * H:]
    return dz * (1 + np.abs(h_prev)) + dn + 2 * TRANSCENDENTAL_SLACK
