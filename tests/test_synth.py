"""Checks of the seeded input generators and the host harness (no controller arithmetic here)."""
import numpy as np

import synth
from synth.rng import splitmix64, splitmix64_int, harness_key


def test_splitmix64_published_sequence():
    # SplitMix64 seeded with 0 (Vigna's reference generator): the state advances by the golden gamma
    # and each output is the finaliser of the state; the first three outputs are:
    g = 0x9E3779B97F4A7C15
    expect = [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    assert [splitmix64_int((i * g) % (1 << 64)) for i in range(3)] == expect
    got = splitmix64(np.array([(i * g) % (1 << 64) for i in range(3)], np.uint64))
    assert [int(v) for v in got] == expect


def test_harness_key_is_a_chain():
    a = harness_key(7, 3, 11, np.arange(5, dtype=np.uint64))
    k = splitmix64_int(7)
    k = splitmix64_int(k ^ 3)
    k = splitmix64_int(k ^ 11)
    assert [int(v) for v in a] == [splitmix64_int(k ^ s) for s in range(5)]


def test_bf16_rounding():
    f = np.array([1.0, -2.0, 1.00390625, 1.005859375, 3.0e38, 0.0], np.float32)
    bits = synth.bf16_bits_from_f32(f)
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: round to even (1.0); 1 + 3*2^-9 rounds up
    assert bits.tolist() == [0x3F80, 0xC000, 0x3F80, 0x3F81, 0x7F62, 0x0000]
    assert np.array_equal(synth.f32_from_bf16_bits(bits[:2]), np.array([1.0, -2.0], np.float32))


def test_workload_shapes_and_determinism():
    for name, wl in synth.WORKLOADS.items():
        assert wl.cap % 4 == 0 and wl.cap >= wl.L0 + wl.steps * (wl.k + 1)
        small = wl.scaled(B=min(wl.B, 2), L0=min(wl.L0, 4096), steps=2)
        a = small.context_row(1 if small.B > 1 else 0)
        b = small.context_row(1 if small.B > 1 else 0)
        assert np.array_equal(a, b) and a.min() >= 0 and a.max() < wl.V
    wl = synth.get_workload("uniform_8k")
    assert wl.probe_weights().shape == (wl.d,)
    assert wl.hidden(3).shape == (wl.B, wl.d)
    mlp = synth.get_workload("code_16k")
    assert mlp.probe_weights().shape == (mlp.probe_hidden * mlp.d + mlp.probe_hidden,)


def test_planted_spans_are_verbatim_earlier_copies():
    wl = synth.get_workload("uniform_8k").scaled(B=1)
    x = wl.context_row(0)
    # with uniform ids over 128K, an 8-gram repeat only arises from a planted copy; about 10 % of
    # positions end such a repeat
    seen = {}
    ends = 0
    for e in range(7, x.shape[0]):
        g = tuple(x[e - 7: e + 1].tolist())
        if g in seen:
            ends += 1
        seen.setdefault(g, e)
    assert 0.05 * x.shape[0] < ends < 0.12 * x.shape[0]


def test_future_stream():
    """The target's continuation keeps the row's token law and plants copies of earlier spans with
    about 10 % edits."""
    wl = synth.get_workload("uniform_8k").scaled(B=1, steps=600, future_coverage=0.5)
    g = wl.future_row(0)
    assert g.shape == (wl.cap - wl.L0,) and g.min() >= 0 and g.max() < wl.V
    assert np.array_equal(g, wl.future_row(0))
    x = np.concatenate([wl.context_row(0), g])
    # fraction of future positions that end an 8-gram seen earlier (uniform ids: only copies do)
    seen = set()
    ends = 0
    for e in range(7, x.shape[0]):
        gram = tuple(x[e - 7: e + 1].tolist())
        if e >= wl.L0 and gram in seen:
            ends += 1
        seen.add(gram)
    frac = ends / g.shape[0]
    assert 0.15 < frac < 0.5          # 50 % coverage, 8-grams broken by 10 % edits: ~0.5 * 0.9^8


def test_harness_law():
    wl = synth.get_workload("uniform_8k").scaled(B=64, steps=16)
    params = wl.harness_params()
    B, k = wl.B, wl.k
    rng = np.random.default_rng(0)
    draft = rng.integers(0, wl.V, (B, k)).astype(np.int32)
    mode = np.array([1, 0, 2] * 21 + [1], np.int32)
    dlen = np.where(mode == 1, rng.integers(0, k + 1, B), 0).astype(np.int32)
    lens = (wl.L0 + rng.integers(0, 100, B)).astype(np.int32)
    assert wl.cap - wl.L0 >= 100 + k + 1
    future = rng.integers(0, wl.V, (B, wl.cap - wl.L0)).astype(np.int32)
    vd, vl, t = synth.harness_targets(params, 0, lens, mode, draft, dlen, future)
    # the target reads the future stream at the row's current length
    for b in range(B):
        assert t[b].tolist() == future[b, lens[b] - wl.L0: lens[b] - wl.L0 + k + 1].tolist()
    copy = mode == 1
    assert np.array_equal(vl[copy], dlen[copy]) and np.all(vl[~copy] == params["gamma"])
    for b in np.nonzero(copy)[0]:
        assert vd[b, : vl[b]].tolist() == draft[b, : vl[b]].tolist()
        assert np.all(vd[b, vl[b]:] == 0)
    g = params["gamma"]
    agree = (vd[~copy, :g] == t[~copy, :g])
    assert 0.65 < agree.mean() < 0.85          # p_neural = 0.75
    assert np.all(vd[~copy, g:] == 0)
    # positions past the stream read as 0
    lens2 = np.full(B, wl.cap - 3, np.int32)
    _, _, t2 = synth.harness_targets(params, 1, lens2, mode, draft, dlen, future)
    assert np.all(t2[:, 3:] == 0) and np.array_equal(t2[:, :3], future[:, -3:])
