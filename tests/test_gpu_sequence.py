"""Persistent LSTM/GRU sequences (darb_lstm_sequence, darb_gru_sequence) against
the CPU oracle, step by step (needs a GB300).

Every step t of a sequence is checked against the oracle's step fed the GPU's
own h_{t-1} (and c_{t-1}), inside the bounds of gpu_helpers: the errors of a
recurrence compound from step to step, so comparing whole trajectories would
test the conditioning of the network, not the kernel.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from paper_1911_08020_gb300 import darb, synth
from tests.gpu_helpers import TOL, dev, encode_both, gru_bound, lstm_bounds, t

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1911_08020_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _gate_matrix(g, gates, I, H, dtype, mset):
    w = (0.3 * g.standard_normal((gates * H, I + H))).astype(np.float32)
    stored = synth.f32_to_bf16_bits(w) if dtype == "bf16" else w
    return stored, g.choice(np.asarray(mset, np.int32), size=gates * H)


def _check_lstm_sequence(h, ref, T, I, H, B, xs, h0, c0, bias, tol):
    hs = torch.empty((T, H, B), device=dev())
    cs = torch.empty((T, H, B), device=dev())
    cl = torch.empty((H, B), device=dev())
    darb.darb_lstm_sequence(h, T, I, H, B, t(xs) if I else None, t(h0), t(c0),
                            t(bias) if bias is not None else None, hs, cs, cl)
    torch.cuda.synchronize()
    hs, cs, cl = hs.cpu().numpy(), cs.cpu().numpy(), cl.cpu().numpy()
    hp, cp = h0, c0
    for s in range(T):
        hr, cr, ga = oracle.lstm_step(ref, I, H, xs[s] if I else None, hp, cp, bias)
        bc, bh = lstm_bounds(ga, cp, tol)
        dc, dh = np.abs(cs[s] - cr) - bc, np.abs(hs[s] - hr) - bh
        assert np.all(dc <= 0), (s, float(dc.max()))
        assert np.all(dh <= 0), (s, float(dh.max()))
        hp, cp = hs[s], cs[s]
    np.testing.assert_array_equal(cl, cs[T - 1])
    return hs, cs


def _check_gru_sequence(h, ref, T, I, H, B, xs, h0, bi, bh, tol):
    hs = torch.empty((T, H, B), device=dev())
    darb.darb_gru_sequence(h, T, I, H, B, t(xs) if I else None, t(h0), t(bi) if bi is not None else None,
                           t(bh) if bh is not None else None, hs)
    torch.cuda.synchronize()
    hs = hs.cpu().numpy()
    hp = h0
    for s in range(T):
        hr, ga = oracle.gru_step(ref, I, H, xs[s] if I else None, hp, bi, bh)
        d = np.abs(hs[s] - hr) - gru_bound(ga, hp, hr, tol)
        assert np.all(d <= 0), (s, float(d.max()))
        hp = hs[s]
    return hs


# (I, H, B): one unit per CTA, ragged batch tiles, several tiles, I = 0, more
# units than CTAs, a batch tile of one column; batches that are multiples of 4
# stage through tensor maps (one CTA; a ragged last tile staged from the padded
# copy of h, as one tile (B = 12) and as the second of two (B = 40))
SHAPES = [(0, 5, 1), (3, 4, 2), (7, 33, 3), (20, 40, 8), (64, 100, 9), (10, 70, 33), (16, 300, 1),
          (40, 200, 70), (5, 400, 17), (4, 1, 8), (6, 9, 4), (12, 36, 40), (0, 64, 12), (300, 260, 4)]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_lstm_sequence_small(dtype):
    g = np.random.default_rng(40)
    for I, H, B in SHAPES:
        stored, m = _gate_matrix(g, 4, I, H, dtype, (1, 2, 3, 4, 8, 17))
        h, ref = encode_both(stored, m, dtype)
        try:
            T = 4
            xs = synth.activations(T * I, B, seed=I).reshape(T, I, B) if I else np.zeros((T, 0, B), np.float32)
            h0, c0 = synth.state(H, B, seed=H), synth.state(H, B, seed=H + 1, scale=1.0)
            for bias in (None, synth.bias(4 * H, seed=I)):
                _check_lstm_sequence(h, ref, T, I, H, B, xs, h0, c0, bias, TOL[dtype])
        finally:
            darb.darb_destroy(h)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_gru_sequence_small(dtype):
    g = np.random.default_rng(41)
    for I, H, B in SHAPES:
        stored, m = _gate_matrix(g, 3, I, H, dtype, (1, 2, 5, 8, 16))
        h, ref = encode_both(stored, m, dtype)
        try:
            T = 4
            xs = synth.activations(T * I, B, seed=I).reshape(T, I, B) if I else np.zeros((T, 0, B), np.float32)
            h0 = synth.state(H, B, seed=H)
            _check_gru_sequence(h, ref, T, I, H, B, xs, h0, None, None, TOL[dtype])
            _check_gru_sequence(h, ref, T, I, H, B, xs, h0, synth.bias(3 * H, seed=1), synth.bias(3 * H, seed=2),
                                TOL[dtype])
        finally:
            darb.darb_destroy(h)


def test_gru_sequence_blocks_straddling_the_input_boundary():
    """Block sizes that do not divide I put one block of a row on both x and h:
    its kept weight must land in the right part of the GRU gate sum."""
    g = np.random.default_rng(42)
    I, H, B, T = 13, 24, 5, 3
    for mset in ((3,), (5,), (7,), (13,), (37,)):
        stored, m = _gate_matrix(g, 3, I, H, "f32", mset)
        h, ref = encode_both(stored, m, "f32")
        try:
            xs = synth.activations(T * I, B, seed=5).reshape(T, I, B)
            _check_gru_sequence(h, ref, T, I, H, B, xs, synth.state(H, B, seed=6), synth.bias(3 * H, seed=1),
                                synth.bias(3 * H, seed=2), TOL["f32"])
        finally:
            darb.darb_destroy(h)


# (I, H, B, T) where x_t is at least a third of the stacked input and the
# sequence has at least 64 columns: the x parts of all steps go through one
# product before the recurrence; block sizes that do not divide I leave blocks
# straddling the x/h boundary
PRE_SHAPES = [(13, 24, 5, 13), (40, 64, 33, 2), (100, 70, 64, 3), (8, 16, 1, 64), (30, 50, 20, 4)]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_sequences_with_precomputed_x_parts(dtype):
    g = np.random.default_rng(45)
    for I, H, B, T in PRE_SHAPES:
        xs = synth.activations(T * I, B, seed=I).reshape(T, I, B)
        h0, c0 = synth.state(H, B, seed=H), synth.state(H, B, seed=H + 1, scale=1.0)
        stored, m = _gate_matrix(g, 4, I, H, dtype, (3, 5, 7, 8, 13))
        h, ref = encode_both(stored, m, dtype)
        try:
            _check_lstm_sequence(h, ref, T, I, H, B, xs, h0, c0, synth.bias(4 * H, seed=I), TOL[dtype])
        finally:
            darb.darb_destroy(h)
        stored, m = _gate_matrix(g, 3, I, H, dtype, (3, 5, 7, 8, 13))
        h, ref = encode_both(stored, m, dtype)
        try:
            _check_gru_sequence(h, ref, T, I, H, B, xs, h0, synth.bias(3 * H, seed=1), synth.bias(3 * H, seed=2),
                                TOL[dtype])
        finally:
            darb.darb_destroy(h)


@pytest.mark.parametrize("name,batch", [("lstm_1024", 1), ("lstm_1024", 32), ("lstm_lm_1500", 20)])
def test_lstm_sequence_workloads(name, batch):
    """Full-size gate matrices in the launch configuration the bench times."""
    wl = synth.WORKLOADS[name]
    I, H, T = wl.input_size, wl.hidden, 4
    _, stored, m = synth.matrix(wl, 0)
    h, ref = encode_both(stored, m, wl.dtype)
    try:
        xs = synth.rnn_inputs(wl, batch, T)
        z = np.zeros((H, batch), np.float32)
        _check_lstm_sequence(h, ref, T, I, H, batch, xs, z, z, synth.bias(4 * H, seed=wl.seed), TOL[wl.dtype])
    finally:
        darb.darb_destroy(h)


def test_gru_sequence_workload():
    wl = synth.WORKLOADS["gru_1024"]
    I, H, B, T = wl.input_size, wl.hidden, wl.batches[0], 3
    _, stored, m = synth.matrix(wl, 0)
    h, ref = encode_both(stored, m, wl.dtype)
    try:
        xs = synth.rnn_inputs(wl, B, T)
        _check_gru_sequence(h, ref, T, I, H, B, xs, np.zeros((H, B), np.float32), synth.bias(3 * H, seed=1),
                            synth.bias(3 * H, seed=2), TOL[wl.dtype])
    finally:
        darb.darb_destroy(h)


def test_sequence_matches_repeated_steps_closely():
    """The sequence and T step calls compute the same cell; they differ only in
    the order of fp32 additions, so their trajectories stay close over a
    short sequence."""
    wl = synth.WORKLOADS["lstm_1024"]
    I, H, B, T = wl.input_size, wl.hidden, 8, 6
    _, stored, m = synth.matrix(wl, 0)
    h = darb.darb_encode(t(stored), m)
    try:
        xs = t(synth.rnn_inputs(wl, B, T))
        bias = t(synth.bias(4 * H, seed=3))
        hs = torch.empty((T, H, B), device=dev())
        cl = torch.empty((H, B), device=dev())
        z = torch.zeros((H, B), device=dev())
        darb.darb_lstm_sequence(h, T, I, H, B, xs, z, z, bias, hs, None, cl)
        hp, cp = z.clone(), z.clone()
        for s in range(T):
            ho, co = torch.empty_like(z), torch.empty_like(z)
            darb.darb_lstm_step(h, I, H, B, xs[s], hp, cp, bias, ho, co)
            hp, cp = ho, co
        torch.cuda.synchronize()
        assert torch.max(torch.abs(hs[T - 1] - hp)).item() < 1e-4
        assert torch.max(torch.abs(cl - cp)).item() < 1e-4
    finally:
        darb.darb_destroy(h)


def test_sequence_deterministic_and_graph_capturable():
    g = np.random.default_rng(43)
    I, H, B, T = 48, 160, 12, 5
    stored, m = _gate_matrix(g, 4, I, H, "bf16", (2, 4, 8, 16))
    h = darb.darb_encode(t(stored.view(np.int16)).view(torch.bfloat16), m)
    try:
        xs = t(synth.activations(T * I, B, seed=1).reshape(T, I, B))
        h0, c0 = t(synth.state(H, B, seed=2)), t(synth.state(H, B, seed=3))
        outs = []
        for _ in range(2):
            hs = torch.empty((T, H, B), device=dev())
            darb.darb_lstm_sequence(h, T, I, H, B, xs, h0, c0, None, hs)
            outs.append(hs)
        torch.cuda.synchronize()
        assert torch.equal(outs[0], outs[1])
        hs = torch.full((T, H, B), float("nan"), device=dev())
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.stream(s):
            with torch.cuda.graph(graph, stream=s):
                darb.darb_lstm_sequence(h, T, I, H, B, xs, h0, c0, None, hs, stream=s.cuda_stream)
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(hs, outs[0])
    finally:
        darb.darb_destroy(h)


def test_sequence_empty_and_argument_checks():
    g = np.random.default_rng(44)
    I, H, B = 4, 6, 2
    stored, m = _gate_matrix(g, 4, I, H, "f32", (2, 4))
    h = darb.darb_encode(t(stored), m)
    try:
        z = torch.zeros((H, B), device=dev())
        c0 = torch.randn((H, B), device=dev())
        cl = torch.empty_like(z)
        darb.darb_lstm_sequence(h, 0, I, H, B, None, z, c0, None, None, None, cl)   # no steps: c_last = c0
        torch.cuda.synchronize()
        assert torch.equal(cl, c0)
        xs = torch.zeros((3, I, B), device=dev())
        hs = torch.empty((3, H, B), device=dev())
        with pytest.raises(darb.DarbError):
            darb.darb_lstm_sequence(h, 3, I + 1, H, B, xs, z, c0, None, hs)             # I + H != cols
        with pytest.raises(darb.DarbError):
            darb.darb_lstm_sequence(h, -1, I, H, B, xs, z, c0, None, hs)                # T < 0
        with pytest.raises(darb.DarbError):
            darb.darb_lstm_sequence(h, 3, I, H, B, xs, z, c0, None, hs, None, hs[0])    # c_last inside h_seq
        with pytest.raises(darb.DarbError):
            darb.darb_lstm_sequence(h, 3, I, H, B, xs, hs[1], c0, None, hs)             # h0 inside h_seq
        with pytest.raises(darb.DarbError):
            darb.darb_gru_sequence(h, 3, I, H, B, xs, z, None, None, hs)               # 4H rows is not a GRU
    finally:
        darb.darb_destroy(h)


@pytest.mark.parametrize("cell,I,H,B", [("lstm", 20, 200, 8), ("lstm", 7, 33, 3), ("gru", 64, 300, 12)])
def test_barrier_timeout_is_reported_and_the_device_stays_usable(cell, I, H, B, monkeypatch):
    """The failure path of the sequence kernels' grid barrier, made on purpose
    from the host: DARB_TEST_BARRIER_TIMEOUT=1 shortens the barrier's limit to
    1 ms and holds back one CTA's first arrival, so every other CTA's wait runs
    out (no copy is in flight at a barrier, and no wait is unbounded).  The
    call must end, darb_sync_status must report DARB_ERR_TIMEOUT, and the next
    call, without the hook, must be correct."""
    g = np.random.default_rng(45)
    gates = 4 if cell == "lstm" else 3
    T = 4
    stored, m = _gate_matrix(g, gates, I, H, "f32", (2, 4, 8))
    h, ref = encode_both(stored, m, "f32")
    try:
        xs = synth.activations(T * I, B, seed=5).reshape(T, I, B)
        h0 = synth.state(H, B, seed=6)
        c0 = synth.state(H, B, seed=7)
        hs = torch.empty((T, H, B), device=dev())
        monkeypatch.setenv("DARB_TEST_BARRIER_TIMEOUT", "1")
        if cell == "lstm":
            darb.darb_lstm_sequence(h, T, I, H, B, t(xs), t(h0), t(c0), None, hs)
        else:
            darb.darb_gru_sequence(h, T, I, H, B, t(xs), t(h0), None, None, hs)
        with pytest.raises(darb.DarbError) as e:
            darb.darb_sync_status(h)
        assert e.value.status == darb.ERR_TIMEOUT
        monkeypatch.delenv("DARB_TEST_BARRIER_TIMEOUT")
        darb.darb_sync_status(h)   # the status was cleared by the read
        if cell == "lstm":
            _check_lstm_sequence(h, ref, T, I, H, B, xs, h0, c0, None, TOL["f32"])
        else:
            _check_gru_sequence(h, ref, T, I, H, B, xs, h0, None, None, TOL["f32"])
        darb.darb_sync_status(h)
    finally:
        darb.darb_destroy(h)
