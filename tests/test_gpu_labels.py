"""Copy-mode labels (§3.2) on the GPU vs the oracle, through the C ABI.

Labels are integers: bit-exact.  Small rows (several structures, lengths, n) compare every position
with oracle.copy_labels; the full-size contexts of the zipf_32k workload compare sampled positions
with the oracle's single-window test (a position is labelled iff one of the n windows covering it
repeats) and check the runs-of-n invariant everywhere.
"""
import itertools

import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu


def _labels(ctx: np.ndarray, lens: np.ndarray, n: int) -> np.ndarray:
    import torch
    from paper_2609_20186_gb300 import binding as bd
    c = torch.from_numpy(np.ascontiguousarray(ctx, np.int32)).cuda()
    ln = torch.from_numpy(np.ascontiguousarray(lens, np.int32)).cuda()
    out = torch.full(c.shape, 7, dtype=torch.uint8, device="cuda")
    bd.switchsd_copy_labels(c, ln, out, n=n)
    return out.cpu().numpy()


def _rows(seed, B, cap):
    rng = np.random.default_rng(seed)
    ctx = np.zeros((B, cap), np.int32)
    lens = np.zeros(B, np.int32)
    for b in range(B):
        L = int(rng.integers(0, cap + 1))
        kind = b % 4
        if kind == 0:                      # small alphabet: many short repeats
            x = rng.integers(0, 3, L)
        elif kind == 1:                    # large alphabet with planted copies of earlier spans
            x = rng.integers(0, 100000, L)
            for _ in range(4):
                if L > 40:
                    ln = int(rng.integers(5, 30))
                    src = int(rng.integers(0, L - ln))
                    dst = int(rng.integers(src, L - ln + 1))
                    x[dst:dst + ln] = x[src:src + ln].copy()
        elif kind == 2:                    # a periodic run
            x = np.tile(rng.integers(0, 5, int(rng.integers(1, 7))), L // 1 + 1)[:L]
        else:                              # Zipf-like ids
            x = np.minimum(rng.zipf(1.3, L), 50000)
        ctx[b, :L] = x
        ctx[b, L:] = rng.integers(0, 3, cap - L)  # garbage past the length must not matter
        lens[b] = L
    return ctx, lens


@pytest.mark.parametrize("n", [5, 1, 3, 8, 32])
def test_small_rows_every_position(n):
    ctx, lens = _rows(10 + n, 24, 700)
    got = _labels(ctx, lens, n)
    for b in range(ctx.shape[0]):
        L = int(lens[b])
        ref = oracle.copy_labels(ctx[b, :L], n)
        assert np.array_equal(got[b, :L], ref), (b, L, n)
        assert not got[b, L:].any()


def test_bad_and_short_lengths():
    ctx, lens = _rows(3, 6, 64)
    lens[:] = [0, 3, 64, -1, 65, 5]
    got = _labels(ctx, lens, 5)
    assert not got[[0, 1, 3, 4]].any()                  # empty, shorter than n, out of range
    assert np.array_equal(got[2], oracle.copy_labels(ctx[2], 5))
    assert np.array_equal(got[5, :5], oracle.copy_labels(ctx[5, :5], 5))


def test_full_size_sampled_positions():
    wl = synth.WORKLOADS["zipf_32k"]
    ctx, lens = wl.contexts()
    got = _labels(ctx, lens, 5)
    rng = np.random.default_rng(0)
    for b in (0, 9, 33, 63):
        L = int(lens[b])
        x = ctx[b, :L]
        y = got[b, :L]
        runs = [len(list(g)) for k, g in itertools.groupby(y.tolist()) if k == 1]
        assert all(r >= 5 for r in runs)
        assert not got[b, L:].any()
        for j in rng.integers(0, L, 60):
            j = int(j)
            ref = any(oracle.window_repeats(x, 5, s) for s in range(max(0, j - 4), j + 1))
            assert bool(y[j]) == ref, (b, j)
        assert 0.02 < y.mean() < 0.98                   # the workload has both kinds of positions


@pytest.mark.parametrize("n", [1, 5])
def test_long_runs_and_short_periods(n):
    """Rows where thousands of windows are equal (one run, period 2, a 2-token alphabet: every insert
    lands on a few table slots) beside ordinary rows in one batch; every position against the oracle."""
    rng = np.random.default_rng(77 + n)
    B, cap = 6, 12000
    ctx = np.zeros((B, cap), np.int32)
    ctx[0] = 7                                          # one run: every window equal
    ctx[1] = np.tile([3, 9], cap // 2)                  # period 2
    ctx[2] = rng.integers(0, 2, cap)                    # two-letter alphabet: few distinct windows
    ctx[3] = rng.integers(0, 100000, cap)               # distinct windows
    ctx[4, :6000] = 5                                   # half a run, then distinct tokens
    ctx[4, 6000:] = rng.integers(0, 100000, cap - 6000)
    ctx[5] = np.minimum(rng.zipf(1.3, cap), 50000)      # Zipf ids
    lens = np.array([cap, cap - 1, cap, cap, cap - 3, 9001], np.int32)
    got = _labels(ctx, lens, n)
    for b in range(B):
        L = int(lens[b])
        assert np.array_equal(got[b, :L], oracle.copy_labels(ctx[b, :L], n)), b
        assert not got[b, L:].any()
