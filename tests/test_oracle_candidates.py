"""Pins of the oracle's W copy candidates and their verification (§3.3, App. D).

No pin re-runs the oracle's loops: an independent brute force by slicing, the relation to the single
longest-then-most-recent search (with kappa = n*, the first candidate is e*), invariants of the
candidate list, and hand cases for choosing the longest validated candidate.
"""
import itertools

import numpy as np
import pytest

import oracle


def _brute(x, n_min, n_max, kappa, W, D, copy_ok=True):
    L = len(x)
    ms = {}
    for e in range(L - 1):
        m = max([n for n in range(1, n_max + 1) if n <= e + 1 and x[e - n + 1:e + 1] == x[L - n:]] + [0])
        ms[e] = m
    has = any(m >= n_min for m in ms.values())
    ends = sorted([e for e, m in ms.items() if m >= kappa], reverse=True)[:W]
    if not has:
        return 0, [], []
    if not ends or not copy_ok:
        return 2, [], []
    return 1, [x[e + 1:e + 1 + min(D, L - 1 - e)] for e in ends], ends


@pytest.mark.parametrize("n_min,n_max,kappa,W,D", [(1, 3, 1, 3, 2), (2, 4, 3, 2, 4), (2, 3, 2, 5, 1)])
def test_brute_force_ternary(n_min, n_max, kappa, W, D):
    for L in range(1, 9):
        for x in itertools.product(range(3), repeat=L):
            x = list(x)
            for z, ok in ((1.0, True), (-1.0, False)):
                mode, cands, ends = oracle.candidates(np.array(x, np.int32), n_min=n_min, n_max=n_max,
                                                      kappa=kappa, z=z, logit_tau=0.0, W=W, D=D)
                assert (mode, cands, ends) == _brute(x, n_min, n_max, kappa, W, D, ok), (x, z)


def test_brute_force_random():
    rng = np.random.default_rng(5)
    for _ in range(400):
        L = int(rng.integers(2, 60))
        x = rng.integers(0, 4, L).astype(np.int32)
        n_min = int(rng.integers(1, 4))
        n_max = int(rng.integers(n_min, 7))
        kappa = int(rng.integers(n_min, n_max + 2))
        W, D = int(rng.integers(1, 11)), int(rng.integers(1, 21))
        got = oracle.candidates(x, n_min=n_min, n_max=n_max, kappa=kappa, z=0.5, logit_tau=0.0, W=W, D=D)
        assert got == _brute(x.tolist(), n_min, n_max, kappa, W, D)


def test_first_candidate_is_the_longest_match_end():
    rng = np.random.default_rng(6)
    checked = 0
    for _ in range(500):
        x = rng.integers(0, 3, int(rng.integers(3, 50))).astype(np.int32)
        n_star, e_star = oracle.longest_suffix_match(x, 2, 6)
        if n_star == 0:
            continue
        mode, cands, ends = oracle.candidates(x, n_min=2, n_max=6, kappa=n_star, z=1.0, logit_tau=0.0, W=4, D=8)
        assert mode == 1 and ends[0] == e_star
        checked += 1
    assert checked > 100


def test_invariants():
    rng = np.random.default_rng(7)
    for _ in range(300):
        x = rng.integers(0, 3, int(rng.integers(3, 80))).astype(np.int32)
        L = len(x)
        mode, cands, ends = oracle.candidates(x, n_min=2, n_max=5, kappa=3, z=1.0, logit_tau=0.0, W=10, D=20)
        assert ends == sorted(ends, reverse=True) and len(set(ends)) == len(ends)
        for c, e in zip(cands, ends):
            assert e <= L - 2 and list(x[e - 2:e + 1]) == list(x[L - 3:])      # the kappa-gram recurs at e
            assert c == list(x[e + 1:e + 1 + min(20, L - 1 - e)])


def test_verify_candidates_hand_cases():
    row = np.zeros(32, np.int32)
    row[:3] = [1, 2, 3]
    # candidate 1 validates 3 tokens, candidate 0 only 1: candidate 1 is kept, its bonus appended
    got = oracle.verify_candidates_row(row, 3, 32, [[4, 5, 6], [4, 7, 8, 9]],
                                       [[4, 0, 0, 0, 0], [4, 7, 8, 1, 0]])
    assert got == (7, 3, 1, 0) and row[:7].tolist() == [1, 2, 3, 4, 7, 8, 1]
    # a tie keeps the most recent candidate (the lowest index)
    row = np.zeros(32, np.int32)
    got = oracle.verify_candidates_row(row, 1, 32, [[4, 5], [4, 6]], [[4, 9, 0], [4, 8, 0]])
    assert got == (3, 1, 0, 0) and row[1:3].tolist() == [4, 9]
    # no candidate: the target's next token only
    row = np.zeros(8, np.int32)
    assert oracle.verify_candidates_row(row, 1, 8, [], [[5]]) == (2, 0, 0, 0) and row[1] == 5
    # capacity: untouched
    row = np.zeros(6, np.int32)
    row[:4] = [1, 2, 3, 4]
    assert oracle.verify_candidates_row(row, 4, 6, [[5, 6]], [[5, 6, 7]]) == (4, -1, 0, 1)
    assert row.tolist() == [1, 2, 3, 4, 0, 0]


def test_one_candidate_is_greedy_verification():
    rng = np.random.default_rng(8)
    for _ in range(300):
        L, k = int(rng.integers(1, 20)), int(rng.integers(0, 9))
        cap = L + k + 1 + int(rng.integers(-2, 3))
        prefix = rng.integers(0, 5, L).astype(np.int32)
        draft = rng.integers(0, 3, k).astype(np.int32)
        target = rng.integers(0, 3, k + 1).astype(np.int32)
        r1 = np.zeros(max(cap, L), np.int32)
        r1[:L] = prefix
        r2 = r1.copy()
        g = oracle.verify_row(r1, L, cap, draft, target)
        c = oracle.verify_candidates_row(r2, L, cap, [draft.tolist()], [target.tolist()])
        assert (c[0], c[1], c[3]) == g and np.array_equal(r1, r2)
