"""The seeded input generators: reproducible, shaped and distributed as stated."""
import numpy as np
import torch

from paper_1911_08020_gb300 import synth


def test_expected_ratios_match_workload_targets():
    # 1 / E[1/m] for each workload's block-size law (the "~Nx" pruning ratios)
    want = {"gemv_1024": 24.6, "lstm_1024": 13.3, "lstm_lm_1500": 16.0, "gru_1024": 20.3,
            "fc6_fc7": 25.6}
    for name, r in want.items():
        wl = synth.WORKLOADS[name]
        assert abs(synth.expected_ratio(wl.choices, wl.probs) - r) < 0.05, name


def test_reproducible_and_distinct_streams():
    a = synth.weights(64, 48, seed=3)
    b = synth.weights(64, 48, seed=3)
    c = synth.weights(64, 48, seed=3, sub=1)
    assert a.dtype == np.float32 and a.shape == (64, 48)
    np.testing.assert_array_equal(a, b)
    assert not np.array_equal(a, c)
    m = synth.block_sizes(5000, (8, 16, 32, 64), (0.1, 0.2, 0.3, 0.4), seed=0)
    freq = np.array([(m == v).mean() for v in (8, 16, 32, 64)])
    assert np.all(np.abs(freq - np.array([0.1, 0.2, 0.3, 0.4])) < 0.03)


def test_weight_row_scale_is_lognormal():
    w = synth.weights(4000, 256, seed=11).astype(np.float64)
    row_sd = w.std(axis=1)
    log_scale = np.log(row_sd / 0.05)
    assert abs(log_scale.mean()) < 0.05 and abs(log_scale.std() - 0.5) < 0.05


def test_bf16_rounding_matches_torch():
    g = np.random.default_rng(0)
    a = (g.standard_normal(100000) * np.exp(g.uniform(-30, 30, 100000))).astype(np.float32)
    a[:4] = [0.0, -0.0, np.inf, -np.inf]
    bits = synth.f32_to_bf16_bits(a)
    ref = torch.from_numpy(a).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(bits, ref)
    back = synth.bf16_bits_to_f32(bits)
    np.testing.assert_array_equal(back, torch.from_numpy(a).to(torch.bfloat16).float().numpy())


def test_rnn_inputs_zero_padding():
    wl = synth.WORKLOADS["lstm_1024"]
    xs = synth.rnn_inputs(wl, batch=2, steps=3)
    assert xs.shape == (3, 256, 2)
    assert not xs[:, 153:, :].any() and xs[:, :153, :].any()
