"""Pins of the oracle's verification at temperature T > 0 (App. A; speculative sampling).

Nothing here re-runs the oracle's own formula: the pins are hand cases at the acceptance boundary,
the reduction to greedy verification as T -> 0 (the target's probabilities become one-hot), the closed
form of the expected accepted length of a copy draft, and the defining property of speculative
sampling -- the first emitted token is distributed as the target -- checked by simulation with the
residual draw done here.
"""
import numpy as np
import pytest

import oracle


def _row(prefix, cap):
    r = np.zeros(cap, np.int32)
    r[: len(prefix)] = prefix
    return r


def test_boundary_hand_cases():
    # u * q < p accepts; equality rejects; p = 0 never accepts; u = 0 accepts any p > 0
    r = _row([1, 2, 3], 16)
    assert oracle.verify_sampled_row(r, 3, 16, [4, 5, 6], [0.6, 0.4, 0.9], [0.5, 0.5, 0.5], [7, 8, 9, 10]) \
        == (5, 1, 0)
    assert r[:5].tolist() == [1, 2, 3, 4, 8]             # draft[0], then the resample at the rejection
    r = _row([1], 8)
    assert oracle.verify_sampled_row(r, 1, 8, [4], [0.5], [0.5], [7, 9]) == (2, 0, 0)   # tie rejects
    assert r[:2].tolist() == [1, 7]
    r = _row([1], 8)
    assert oracle.verify_sampled_row(r, 1, 8, [4, 5], [0.0, 1.0], [0.0, 0.0], [7, 8, 9])[1] == 0
    r = _row([1], 8)
    assert oracle.verify_sampled_row(r, 1, 8, [4, 5], [1e-30, 1e-30], [0.0, 0.0], [7, 8, 9]) == (4, 2, 0)
    assert r[:4].tolist() == [1, 4, 5, 9]                # all accepted: the bonus draw is appended
    # a neural draft: q scales the threshold (accept iff u < p / q)
    r = _row([1], 8)
    assert oracle.verify_sampled_row(r, 1, 8, [4, 5], [0.3, 0.3], [0.5, 0.7], [7, 8, 9], q=[0.5, 0.5])[1] == 1
    # q = None is q = 1
    for u in (0.1, 0.49, 0.5, 0.51, 0.9):
        r1, r2 = _row([1], 8), _row([1], 8)
        a = oracle.verify_sampled_row(r1, 1, 8, [4], [0.5], [u], [7, 8])
        b = oracle.verify_sampled_row(r2, 1, 8, [4], [0.5], [u], [7, 8], q=[1.0])
        assert a == b and np.array_equal(r1, r2)


def test_binary32_product():
    # The product u*q is rounded to binary32 before the compare: pick u, q whose exact product lies
    # just below p while the binary32 product equals p (so the draft is rejected).
    u = np.float32(0.1)
    q = np.float32(0.3)
    exact = float(u) * float(q)
    p32 = np.float32(u * q)                       # binary32 rounding of the product
    assert float(p32) != exact
    r = _row([1], 8)
    acc = oracle.verify_sampled_row(r, 1, 8, [4], [float(p32)], [float(u)], [7, 8], q=[float(q)])[1]
    assert acc == 0                               # product == p in binary32: not strictly below
    nxt = float(np.nextafter(p32, np.float32(1)))
    r = _row([1], 8)
    assert oracle.verify_sampled_row(r, 1, 8, [4], [nxt], [float(u)], [7, 8], q=[float(q)])[1] == 1


def test_capacity_leaves_row_untouched():
    r = _row([1, 2, 3, 4], 6)
    before = r.copy()
    assert oracle.verify_sampled_row(r, 4, 6, [5, 6, 7], [1, 1, 1], [0, 0, 0], [8, 9, 10, 11]) == (4, -1, 1)
    assert np.array_equal(r, before)


def test_temperature_zero_is_greedy():
    """With one-hot target probabilities (T -> 0) and the target's argmax as the resample, the
    sampled verification is the greedy one for every draw of u."""
    rng = np.random.default_rng(7)
    for _ in range(400):
        L = int(rng.integers(1, 20))
        k = int(rng.integers(0, 9))
        cap = L + k + 1 + int(rng.integers(0, 3))
        prefix = rng.integers(0, 5, L).astype(np.int32)
        draft = rng.integers(0, 3, k).astype(np.int32)
        target = rng.integers(0, 3, k + 1).astype(np.int32)
        p = (draft == target[:k]).astype(np.float32)
        u = rng.random(k).astype(np.float32)
        r1, r2 = _row(prefix, cap), _row(prefix, cap)
        g = oracle.verify_row(r1, L, cap, draft, target)
        s = oracle.verify_sampled_row(r2, L, cap, draft, p, u, target)
        assert g == s and np.array_equal(r1, r2)


def test_expected_accepted_length_closed_form():
    """A copy draft (q = 1) of n tokens each with target probability p: P(a >= j) = p^j, so
    E[a] = sum_{j=1..n} p^j."""
    rng = np.random.default_rng(11)
    n, N = 8, 20000
    for p in (0.3, 0.7, 0.95):
        acc = np.empty(N)
        for t in range(N):
            r = np.zeros(n + 2, np.int32)
            acc[t] = oracle.verify_sampled_row(r, 1, n + 2, np.arange(n), np.full(n, p),
                                               rng.random(n).astype(np.float32), np.zeros(n + 1))[1]
        mean = sum(p ** j for j in range(1, n + 1))
        var = sum((2 * j - 1) * p ** j for j in range(1, n + 1)) - mean ** 2
        assert abs(acc.mean() - mean) <= 5 * np.sqrt(var / N), (p, acc.mean(), mean)


@pytest.mark.parametrize("seed", [0, 1])
def test_first_token_follows_target(seed):
    """The defining property of speculative sampling: draft x ~ Q, accept with the oracle's rule,
    else emit a draw from max(0, P - Q) renormalised -- the emitted token is distributed as P."""
    rng = np.random.default_rng(seed)
    V, N = 5, 40000
    P = rng.dirichlet(np.ones(V)).astype(np.float32)
    Q = rng.dirichlet(np.ones(V)).astype(np.float32)
    res = np.maximum(P.astype(np.float64) - Q, 0)
    res /= res.sum()
    counts = np.zeros(V)
    for _ in range(N):
        x = int(rng.choice(V, p=Q / Q.sum()))
        r_tok = int(rng.choice(V, p=res))
        row = np.zeros(4, np.int32)
        _, a, _ = oracle.verify_sampled_row(row, 1, 4, [x], [P[x]], [np.float32(rng.random())], [r_tok, 0],
                                            q=[Q[x]])
        counts[row[1]] += 1
    emp = counts / N
    tol = 5 * np.sqrt(P * (1 - P) / N) + 1e-3
    assert np.all(np.abs(emp - P) <= tol), (emp, P)
