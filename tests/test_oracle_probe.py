"""Pins of the oracle's copy-intent probe (Eq. 3) and its two-layer extension.

The oracle sums in double in index order.  The pins use library routines with their own bf16
decoding (torch's bfloat16 -> float64 conversion) and their own reductions (torch.dot, torch.matmul
in float64), plus closed forms.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth


def _torch_bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits, np.uint16).view(np.int16)).view(torch.bfloat16)


def test_bf16_decode_matches_torch():
    bits = np.array([0x0000, 0x8000, 0x3F80, 0xBF80, 0x4049, 0x0001, 0x7F7F, 0xFF7F, 0x3C00],
                    np.uint16)
    ref = _torch_bf16(bits).double().numpy()
    got = np.array([oracle.bf16_to_double(int(v)) for v in bits])
    assert np.array_equal(got, ref)
    assert oracle.bf16_to_double(0x3F80) == 1.0 and oracle.bf16_to_double(0xC000) == -2.0


@pytest.mark.parametrize("d", [1, 8, 4096, 5120])
def test_linear_probe_matches_torch_float64(d):
    rng = np.random.default_rng(d)
    h = synth.bf16_bits_from_f32(rng.standard_normal(d).astype(np.float32))
    w = synth.bf16_bits_from_f32((rng.standard_normal(d) / math.sqrt(d)).astype(np.float32))
    ref = torch.dot(_torch_bf16(w).double(), _torch_bf16(h).double()).item()
    assert abs(oracle.probe_linear(h, w) - ref) <= 1e-12 * max(1.0, abs(ref))


def test_linear_probe_closed_forms():
    d = 64
    one = np.full(d, 0x3F80, np.uint16)       # 1.0
    half = np.full(d, 0x3F00, np.uint16)      # 0.5
    assert oracle.probe_linear(one, half) == 32.0
    neg = np.full(d, 0xBF80, np.uint16)       # -1.0
    assert oracle.probe_linear(one, neg) == -64.0
    # no bias term: the zero vector scores exactly 0 (Eq. 3 has no bias)
    assert oracle.probe_linear(np.zeros(d, np.uint16), half) == 0.0
    # one non-zero coordinate selects that product
    e = np.zeros(d, np.uint16)
    e[17] = 0x4040                             # 3.0
    w = np.zeros(d, np.uint16)
    w[17] = 0xC000                             # -2.0
    assert oracle.probe_linear(e, w) == -6.0


def test_mlp_probe_matches_torch_float64():
    rng = np.random.default_rng(3)
    d, H1 = 320, 48
    h = synth.bf16_bits_from_f32(rng.standard_normal(d).astype(np.float32))
    W1 = synth.bf16_bits_from_f32((rng.standard_normal((H1, d)) / math.sqrt(d)).astype(np.float32))
    w2 = synth.bf16_bits_from_f32((rng.standard_normal(H1) / math.sqrt(H1)).astype(np.float32))
    b1 = rng.standard_normal(H1).astype(np.float32) * 0.1
    b2 = np.float32(0.25)
    th, tW1, tw2 = (_torch_bf16(a).double() for a in (h, W1, w2))
    ref = (torch.relu(tW1 @ th + torch.from_numpy(b1).double()) @ tw2 + float(b2)).item()
    got = oracle.probe_mlp(h, W1, w2, b1=b1, b2=float(b2))
    assert abs(got - ref) <= 1e-12 * max(1.0, abs(ref))
    # without biases
    ref0 = (torch.relu(tW1 @ th) @ tw2).item()
    assert abs(oracle.probe_mlp(h, W1, w2) - ref0) <= 1e-12 * max(1.0, abs(ref0))


def test_mlp_reduces_to_linear_with_one_positive_unit():
    """With one hidden unit, w2 = 1 and a positive pre-activation, the two-layer probe is the linear
    probe of its weight row (a special case that reduces to Eq. 3)."""
    d = 256
    rng = np.random.default_rng(11)
    h = synth.bf16_bits_from_f32(np.abs(rng.standard_normal(d)).astype(np.float32))
    w = synth.bf16_bits_from_f32(np.abs(rng.standard_normal(d) / 16).astype(np.float32))
    lin = oracle.probe_linear(h, w)
    assert lin > 0
    mlp = oracle.probe_mlp(h, w.reshape(1, d), np.array([0x3F80], np.uint16))
    assert mlp == lin
    # ReLU clips a negative pre-activation to exactly 0 (plus b2)
    wneg = w ^ np.uint16(0x8000)
    assert oracle.probe_mlp(h, wneg.reshape(1, d), np.array([0x3F80], np.uint16), b2=0.5) == 0.5


def test_logit_space_decision_is_sigmoid_decision():
    """Eq. 4 compares sigma(z) with tau; sigma is monotone, so z >= logit(tau) is the same test.
    Checked with math.exp on values well away from the threshold."""
    for tau in (0.1, 0.4, 0.5, 0.9):
        lt = math.log(tau / (1 - tau))
        for z in np.linspace(-8, 8, 401):
            if abs(z - lt) < 1e-9:
                continue
            assert (1 / (1 + math.exp(-z)) >= tau) == (z >= lt)
    assert synth.get_workload("uniform_8k").logit_tau == 0.0


def test_planted_probe_signs():
    """The planted workload builds w_j = s |g_j| sign(h_j), so the logit has sign s."""
    for name, sign in (("planted_copy", 1), ("planted_nocopy", -1)):
        wl = synth.get_workload(name)
        z = oracle.probe_linear(wl.hidden(0)[0], wl.probe_weights())
        assert np.sign(z) == sign and abs(z) > 1.0
