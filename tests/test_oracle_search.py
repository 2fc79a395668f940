"""Pins of the oracle's longest-suffix n-gram search (§3.3, kappa-gram gate and recency ranking).

The oracle scans n from n_max down and e from L-2 down.  The brute force below is an independent
formulation: it lists every (n, e) pair whose n-gram ends at e and equals the context's last n
tokens, sorts by (longest n, most recent e) and takes the first.  It is run over every context on a
three-letter alphabet up to length 9 and over random short contexts.
"""
import itertools

import numpy as np
import pytest

import oracle


def brute_force(x, n_min, n_max):
    L = len(x)
    hits = []
    for n in range(n_min, n_max + 1):
        if n > L:
            continue
        suffix = tuple(x[L - n:])
        for e in range(0, L - 1):          # a prior occurrence ends before the last token
            s = e - n + 1
            if s < 0:
                continue
            if tuple(x[s: e + 1]) == suffix:
                hits.append((n, e))
    if not hits:
        return 0, -1
    hits.sort(key=lambda t: (-t[0], -t[1]))
    return hits[0]


@pytest.mark.parametrize("n_min,n_max", [(1, 1), (1, 3), (2, 4), (3, 8), (2, 2)])
def test_exhaustive_ternary(n_min, n_max):
    count = 0
    for L in range(0, 10):
        for x in itertools.product(range(3), repeat=L):
            got = oracle.longest_suffix_match(np.array(x, np.int32), n_min, n_max, L=L) \
                if L > 0 else oracle.longest_suffix_match(np.zeros(1, np.int32), n_min, n_max, L=0)
            assert got == brute_force(list(x), n_min, n_max), (x, n_min, n_max, got)
            count += 1
    assert count == sum(3 ** L for L in range(10))


def test_random_small_alphabet():
    rng = np.random.default_rng(7)
    for trial in range(3000):
        L = int(rng.integers(1, 65))
        a = int(rng.integers(2, 6))
        x = rng.integers(0, a, L).astype(np.int32)
        n_min = int(rng.integers(1, 5))
        n_max = int(rng.integers(n_min, 13))
        assert oracle.longest_suffix_match(x, n_min, n_max) == brute_force(x.tolist(), n_min, n_max)


def test_hand_cases():
    # periodic run: the suffix "7 7 7 7" overlaps itself; the longest prior occurrence is the
    # 4-gram ending at e = 3 (x[0..3]), with n capped by e + 1
    assert oracle.longest_suffix_match(np.array([7, 7, 7, 7, 7], np.int32), 1, 8) == (4, 3)
    # unique last token: no repetition at all (Fig. 1 case i)
    assert oracle.longest_suffix_match(np.array([1, 2, 3, 4], np.int32), 1, 4) == (0, -1)
    # recency: "1 2" occurs ending at 1 and at 4; the later one wins
    x = np.array([1, 2, 9, 1, 2, 8, 1, 2], np.int32)
    assert oracle.longest_suffix_match(x, 2, 2) == (2, 4)
    # length beats recency: "5 1 2" ends at 2; "1 2" alone ends at 5 more recently
    x = np.array([5, 1, 2, 0, 1, 2, 7, 5, 1, 2], np.int32)
    assert oracle.longest_suffix_match(x, 2, 3) == (3, 2)
    # n capped at n_max even when a longer match exists; most recent among the n_max matches
    x = np.array([4, 5, 6, 7, 0, 4, 5, 6, 7], np.int32)
    assert oracle.longest_suffix_match(x, 1, 2) == (2, 3)
    # a match at the earliest possible position (e = n - 1)
    x = np.array([3, 4, 9, 9, 9, 3, 4], np.int32)
    assert oracle.longest_suffix_match(x, 2, 4) == (2, 1)
    # too short for n_min: L < n_min + 1 -> no match
    assert oracle.longest_suffix_match(np.array([2, 2], np.int32), 2, 4) == (0, -1)
    assert oracle.longest_suffix_match(np.array([2, 2, 2], np.int32), 2, 4) == (2, 1)
    # the last token itself (e = L-1) is never a prior occurrence
    assert oracle.longest_suffix_match(np.array([6], np.int32), 1, 1) == (0, -1)


def test_planted_construction():
    """The planted workload fixes the answer by construction: the context ends with a verbatim copy of
    the 64 tokens starting at 300, so n* = n_max and e* = 363 (§3.3 recency: the copy's source is the
    only earlier occurrence)."""
    import synth
    for name in ("planted_copy", "planted_nocopy"):
        wl = synth.get_workload(name)
        x = wl.context_row(0)
        assert oracle.longest_suffix_match(x, wl.n_min, wl.n_max) == (8, 363)
        assert brute_force(x.tolist(), wl.n_min, wl.n_max) == (8, 363)
    wl = synth.get_workload("planted_norep")
    x = wl.context_row(0)
    assert oracle.longest_suffix_match(x, wl.n_min, wl.n_max) == (0, -1)
