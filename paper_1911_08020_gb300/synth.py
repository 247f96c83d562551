"""Seeded synthetic inputs shaped like the paper's RNN and FC workloads.

This module only draws numbers: weights, per-row block sizes, activations and
RNN state.  It holds none of DARB's arithmetic (no block-size rounding, no
block-max selection, no product), so both the CUDA path and the CPU oracle can
take their inputs from it without sharing any of the method's code.

Recipe (the shapes come from the models of Sec. 4.1 and the FC6/FC7 layers of
AlexNet in Sec. 3.1):

* weights  W[r, c] = 0.05 * z[r, c] * s[r],  z ~ N(0, 1),  s[r] = exp(0.5 * z'[r])
  (a per-row lognormal(0, 0.5) scale, so that some rows are much denser in
  salient weights than others, like the row-density spread of Figs. 3-4);
  bf16 workloads round the fp32 draw to nearest-even bf16;
* block sizes  m[r]  drawn per row from a small categorical distribution whose
  weights put the expected pruning ratio 1 / E[1/m] near the ratios the paper
  reports for the model class (13x-25x);
* activations  X ~ N(0, 1) in fp32; RNN initial state h = c = 0.

Every array comes from its own numpy PCG64 stream keyed by (seed, stream id,
sub-id), so a workload is reproducible bit for bit on any machine.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Sequence

import numpy as np

_STREAM_ROW_SCALE = 1
_STREAM_WEIGHTS = 2
_STREAM_BLOCK_SIZES = 3
_STREAM_ACTIVATIONS = 4
_STREAM_STATE = 5
_STREAM_BIAS = 6


def rng(seed: int, stream: int, sub: int = 0) -> np.random.Generator:
    """Independent, reproducible generator for (seed, stream, sub)."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, stream, sub])))


def weights(rows: int, cols: int, seed: int, sub: int = 0) -> np.ndarray:
    """fp32 rows x cols, row-major: 0.05 * N(0,1) * lognormal(0, 0.5) row scale."""
    z_row = rng(seed, _STREAM_ROW_SCALE, sub).standard_normal(rows)
    scale = np.exp(0.5 * z_row)
    z = rng(seed, _STREAM_WEIGHTS, sub).standard_normal((rows, cols))
    return (0.05 * z * scale[:, None]).astype(np.float32)


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round fp32 to nearest-even bf16; returns the uint16 bit patterns."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp32."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def block_sizes(rows: int, choices: Sequence[int], probs: Sequence[float], seed: int,
                sub: int = 0) -> np.ndarray:
    """int32[rows] drawn i.i.d. from `choices` with probabilities `probs`."""
    g = rng(seed, _STREAM_BLOCK_SIZES, sub)
    return g.choice(np.asarray(choices, dtype=np.int32), size=rows, p=np.asarray(probs))


def activations(rows: int, cols: int, seed: int, sub: int = 0) -> np.ndarray:
    """fp32 rows x cols of N(0, 1) (X is cols_of_W x batch, batch contiguous)."""
    return rng(seed, _STREAM_ACTIVATIONS, sub).standard_normal((rows, cols)).astype(np.float32)


def state(rows: int, cols: int, seed: int, sub: int = 0, scale: float = 0.5) -> np.ndarray:
    """fp32 RNN state-like values, N(0, scale^2) (used by single-step tests)."""
    g = rng(seed, _STREAM_STATE, sub)
    return (scale * g.standard_normal((rows, cols))).astype(np.float32)


def bias(n: int, seed: int, sub: int = 0, scale: float = 0.1) -> np.ndarray:
    """fp32 bias vector, N(0, scale^2)."""
    return (scale * rng(seed, _STREAM_BIAS, sub).standard_normal(n)).astype(np.float32)


def expected_ratio(choices: Sequence[int], probs: Sequence[float]) -> float:
    """1 / E[1/m] for a block-size distribution (what rows*cols / sum(blocks) tends to)."""
    return 1.0 / float(sum(p / m for m, p in zip(choices, probs)))


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: the matrices, their block-size law and the batch/steps."""
    name: str
    kind: str                       # "gemv", "lstm", "gru", "fc"
    dtype: str                      # "f32" or "bf16" (the weight storage type)
    shapes: tuple                   # ((rows, cols), ...) one entry per matrix
    choices: tuple
    probs: tuple
    seed: int
    batches: tuple = (1,)
    steps: int = 1
    input_size: int = 0             # RNN: I
    hidden: int = 0                 # RNN: H
    real_features: int = 0          # RNN: features before zero padding (0 = none)
    layers: int = 1
    notes: str = ""
    extra: dict = field(default_factory=dict)


WORKLOADS = {
    "gemv_1024": Workload(
        name="gemv_1024", kind="gemv", dtype="f32", shapes=((1024, 1024),),
        choices=(8, 16, 32, 64), probs=(0.1, 0.2, 0.3, 0.4), seed=0, batches=(1,),
        notes="single fp32 matrix, DARB encode plus GEMV at batch 1"),
    "lstm_1024": Workload(
        name="lstm_1024", kind="lstm", dtype="f32", shapes=((4096, 1280),),
        choices=(4, 8, 16, 32), probs=(0.1, 0.1, 0.4, 0.4), seed=1, batches=(1, 32),
        steps=100, input_size=256, hidden=1024, real_features=153,
        notes="LSTM hidden 1024, input 256 zero-padded from 153 features"),
    "lstm_lm_1500": Workload(
        name="lstm_lm_1500", kind="lstm", dtype="bf16", shapes=((6000, 3000), (6000, 3000)),
        choices=(10, 15, 20, 30), probs=(0.25, 0.25, 0.25, 0.25), seed=2, batches=(20,),
        steps=35, input_size=1500, hidden=1500, layers=2,
        notes="two-layer LSTM language-model shape (Sec. 4.1, PTB model)"),
    "gru_1024": Workload(
        name="gru_1024", kind="gru", dtype="bf16", shapes=((3072, 2048),),
        choices=(8, 16, 32, 64), probs=(0.2, 0.15, 0.3, 0.35), seed=3, batches=(64,),
        steps=200, input_size=1024, hidden=1024,
        notes="GRU hidden 1024, input 1024 (Sec. 4.1, TIMIT GRU)"),
    "fc6_fc7": Workload(
        name="fc6_fc7", kind="fc", dtype="bf16", shapes=((4096, 9216), (4096, 4096)),
        choices=(16, 32, 64), probs=(0.4, 0.3, 0.3), seed=4, batches=(1, 16, 64, 256),
        notes="AlexNet FC6 4096x9216 and FC7 4096x4096 (Sec. 4.1, Table 6)"),
}


def matrix(wl: Workload, index: int = 0):
    """(W_f32, W_stored, m) for matrix `index` of a workload.

    W_stored is fp32 for "f32" workloads and uint16 bf16 bits for "bf16" ones;
    W_f32 is the exact fp32 value of what is stored.
    """
    rows, cols = wl.shapes[index]
    w = weights(rows, cols, wl.seed, sub=index)
    m = block_sizes(rows, wl.choices, wl.probs, wl.seed, sub=index)
    if wl.dtype == "bf16":
        bits = f32_to_bf16_bits(w)
        return bf16_bits_to_f32(bits), bits, m
    return w, w, m


def rnn_inputs(wl: Workload, batch: int, steps: int, layer: int = 0):
    """x_t for every step, I x batch each, with feature rows >= real_features zeroed."""
    xs = activations(steps * wl.input_size, batch, wl.seed, sub=100 + 10 * layer + batch)
    xs = xs.reshape(steps, wl.input_size, batch)
    if wl.real_features:
        xs[:, wl.real_features:, :] = 0.0
    return xs
