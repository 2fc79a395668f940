"""Pins of the oracle's copy-mode labels (§3.2: a position is a copy-mode instance when it belongs to a
verbatim sequence of at least n_train tokens that appears earlier in the context).

The pins do not re-run the oracle's loops: an independent brute force that, for every position,
enumerates every verbatim sequence of length >= n containing it (any length, not only n) and every
earlier start; hand-built contexts; and the invariant that labelled positions come in runs of at least n.
"""
import itertools

import numpy as np
import pytest

import oracle


def _brute(x, n):
    L = len(x)
    y = [0] * L
    for j in range(L):
        for s in range(0, j + 1):
            for t in range(max(j, s + n - 1), L):           # sequence x[s..t] of length >= n holding j
                seq = x[s:t + 1]
                if any(x[s2:s2 + len(seq)] == seq for s2 in range(0, s)):
                    y[j] = 1
                    break
            if y[j]:
                break
    return y


@pytest.mark.parametrize("n", [1, 2, 3])
def test_brute_force_small_alphabet(n):
    for L in range(0, 9):
        for x in itertools.product(range(3), repeat=L):
            assert oracle.copy_labels(np.array(x, np.int32), n).tolist() == _brute(list(x), n), (x, n)


def test_brute_force_random():
    rng = np.random.default_rng(2)
    for _ in range(300):
        L = int(rng.integers(0, 40))
        x = rng.integers(0, 3, L).astype(np.int32)
        n = int(rng.integers(1, 6))
        assert oracle.copy_labels(x, n).tolist() == _brute(x.tolist(), n)


def test_hand_cases():
    # the second occurrence of a 5-gram is labelled, the first and the separator are not
    assert oracle.copy_labels([1, 2, 3, 4, 5, 9, 1, 2, 3, 4, 5], 5).tolist() == [0] * 6 + [1] * 5
    # a periodic run matches itself one token later
    assert oracle.copy_labels([7] * 7, 5).tolist() == [0] + [1] * 6
    # four tokens repeated are too short for n = 5
    assert oracle.copy_labels([1, 2, 3, 4, 8, 1, 2, 3, 4], 5).sum() == 0
    # shorter than n: nothing
    assert oracle.copy_labels([1, 1, 1], 5).sum() == 0
    # window starting at s: the earlier occurrence must start strictly before s
    assert not oracle.window_repeats([1, 2, 3, 4, 5], 5, 0)
    assert oracle.window_repeats([3, 3, 3, 3, 3, 3], 5, 1)
    assert not oracle.window_repeats([3, 3, 3, 3, 3, 3], 5, 2)   # does not fit


def test_labels_come_in_runs_of_n():
    rng = np.random.default_rng(4)
    for _ in range(200):
        x = rng.integers(0, 4, int(rng.integers(5, 80))).astype(np.int32)
        y = oracle.copy_labels(x, 5)
        runs = [len(list(g)) for k, g in itertools.groupby(y.tolist()) if k == 1]
        assert all(r >= 5 for r in runs)
        for j in np.flatnonzero(y):     # every labelled position is covered by a repeating window
            assert any(oracle.window_repeats(x, 5, s) for s in range(max(0, j - 4), j + 1))
