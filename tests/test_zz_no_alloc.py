"""darb_lstm_step_noalloc: the LSTM step for callers that cannot let a library allocate.

Such callers (a serving loop on a fixed memory budget, code that must not
synchronise the device mid-stream, or callers whose memory all comes from their
own pool) get the same step with its scratch in a fixed array inside the
library.  This file checks, through the C ABI, that two calls in a row give
what the allocating darb_lstm_step gives and what the CPU oracle's LSTM step
gives, each within the tolerance the other LSTM tests use, and that a call too
large for the array is refused.  It is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_1911_08020_gb300 import darb, synth
from tests.gpu_helpers import TOL, encode_both, lstm_bounds, t

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def L():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1911_08020_gb300 import build
    build.build()
    torch.cuda.set_device(0)
    return darb.lib()


def _ptr(a):
    return ctypes.c_void_p(a.data_ptr() if a is not None else None)


def _step(fn, h, I, H, B, x, hp, cp, bias, ho, co):
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return fn(h.ptr, I, H, B, _ptr(x), _ptr(hp), _ptr(cp), _ptr(bias), _ptr(ho), _ptr(co), stream)


@pytest.mark.parametrize("I,H,B,dtype", [(64, 200, 1, "f32"), (48, 160, 9, "bf16"), (256, 1024, 32, "f32")])
def test_noalloc_matches_allocating_step_twice(L, I, H, B, dtype):
    g = np.random.default_rng(100 + B)
    w = (0.3 * g.standard_normal((4 * H, I + H))).astype(np.float32)
    stored = synth.f32_to_bf16_bits(w) if dtype == "bf16" else w
    m = g.choice(np.array([2, 4, 8, 16, 32], np.int32), size=4 * H)
    h, ref = encode_both(stored, m, dtype)
    try:
        bias = t(synth.bias(4 * H, seed=B))
        hp = synth.state(H, B, seed=1)
        cp = synth.state(H, B, seed=2, scale=1.0)
        for call in range(2):   # two calls in a row share the array
            x = synth.activations(I, B, seed=10 + call)
            xd, hpd, cpd = t(x), t(hp), t(cp)
            ho_a, co_a = torch.empty((H, B), device="cuda"), torch.empty((H, B), device="cuda")
            ho_n, co_n = torch.full((H, B), 7.0, device="cuda"), torch.full((H, B), 7.0, device="cuda")
            assert _step(L.darb_lstm_step, h, I, H, B, xd, hpd, cpd, bias, ho_a, co_a) == darb.OK
            assert _step(L.darb_lstm_step_noalloc, h, I, H, B, xd, hpd, cpd, bias, ho_n, co_n) == darb.OK
            torch.cuda.synchronize()
            hr, cr, ga = oracle.lstm_step(ref, I, H, x, hp, cp, bias.cpu().numpy())
            bc, bh = lstm_bounds(ga, cp, TOL[dtype])
            # against the oracle itself, and against the allocating step (each
            # GPU result is within the bound of the exact one, so the two are
            # within twice that of each other)
            assert np.all(np.abs(co_n.cpu().numpy() - cr) <= bc)
            assert np.all(np.abs(ho_n.cpu().numpy() - hr) <= bh)
            assert np.all(np.abs(co_n.cpu().numpy() - co_a.cpu().numpy()) <= 2 * bc)
            assert np.all(np.abs(ho_n.cpu().numpy() - ho_a.cpu().numpy()) <= 2 * bh)
            hp, cp = ho_n.cpu().numpy(), co_n.cpu().numpy()
    finally:
        darb.darb_destroy(h)


def test_noalloc_refuses_sizes_beyond_its_array(L):
    I, H = 8, 64
    g = np.random.default_rng(7)
    w = g.standard_normal((4 * H, I + H)).astype(np.float32)
    h, _ = encode_both(w, np.full(4 * H, 4, np.int32), "f32")
    try:
        B = 4200   # 4H * B floats = 4.3 MB > 4 MiB
        x = torch.zeros((I, B), device="cuda")
        s = torch.zeros((H, B), device="cuda")
        ho, co = torch.empty_like(s), torch.empty_like(s)
        assert _step(L.darb_lstm_step_noalloc, h, I, H, B, x, s, s, None, ho, co) == darb.ERR_UNSUPPORTED
        # shape errors are reported as for darb_lstm_step
        assert _step(L.darb_lstm_step_noalloc, h, I + 1, H, 2, x, s, s, None, ho, co) == darb.ERR_INVALID_ARG
    finally:
        darb.darb_destroy(h)
