"""Pins of the oracle's switch (Fig. 1, Eq. 4) and greedy verification (§3.3, temperature 0).

Hand-built cases, one per switch case, the PLD and never-copy special cases (tau = 0 and tau = 1,
i.e. logit(tau) = -inf / +inf), clipping of the continuation, and the invariants of verification:
accepted <= draft length, the context grows by accepted + 1, and the appended tokens are exactly the
target's greedy tokens (the exactness property of speculative decoding).
"""
import numpy as np
import pytest

import oracle
import synth

NO_REP, COPY, REP_NO_COPY = 0, 1, 2
INF = float("inf")


def test_three_cases():
    x = np.array([10, 11, 12, 13, 14, 99, 11, 12, 13], np.int32)   # suffix "11 12 13" ends at e=3
    hit, (n, e) = True, oracle.longest_suffix_match(x, 2, 4)
    assert (n, e) == (3, 3)
    # (ii) repetition with copy intent -> copy the continuation after e: x[4..]
    mode, draft = oracle.switch(hit, n, e, 0.7, 0.0, 2, 3, x)
    assert mode == COPY and draft == [14, 99, 11]
    # (iii) repetition without copy intent -> neural draft (empty copy draft)
    mode, draft = oracle.switch(hit, n, e, -0.7, 0.0, 2, 3, x)
    assert mode == REP_NO_COPY and draft == []
    # (i) no repetition -> neural draft whatever the probe says
    mode, draft = oracle.switch(False, 0, -1, 5.0, 0.0, 2, 3, x)
    assert mode == NO_REP and draft == []


def test_kappa_gate():
    """§3.3: copy needs the kappa-gram ending at the current token to occur earlier; a shorter match
    counts as repetition without copy intent."""
    x = np.array([1, 2, 3, 4, 2, 3], np.int32)
    n, e = oracle.longest_suffix_match(x, 2, 8)
    assert (n, e) == (2, 2)
    assert oracle.switch(True, n, e, 3.0, 0.0, 3, 4, x)[0] == REP_NO_COPY
    assert oracle.switch(True, n, e, 3.0, 0.0, 2, 4, x) == (COPY, [4, 2, 3])


def test_threshold_edges():
    x = np.array([5, 6, 7, 5, 6], np.int32)
    n, e = oracle.longest_suffix_match(x, 2, 2)
    assert (n, e) == (2, 1)
    # exact tie z == logit(tau) copies (Eq. 4 uses >=)
    assert oracle.switch(True, n, e, 0.0, 0.0, 2, 8, x)[0] == COPY
    assert oracle.switch(True, n, e, -1e-30, 0.0, 2, 8, x)[0] == REP_NO_COPY
    # tau -> 0 (logit -inf): copy whenever a match exists (prompt-lookup decoding)
    assert oracle.switch(True, n, e, -1e30, -INF, 2, 8, x)[0] == COPY
    # tau -> 1 (logit +inf): never copy
    assert oracle.switch(True, n, e, 1e30, INF, 2, 8, x)[0] == REP_NO_COPY
    # the decision is taken in binary32: a logit that rounds up to the threshold copies
    assert oracle.switch(True, n, e, 0.5 - 1e-12, 0.5, 2, 8, x)[0] == COPY


def test_continuation_clipped_at_context_end():
    x = np.array([8, 9, 1, 2, 8, 9], np.int32)      # "8 9" ends at e=1 and the end
    n, e = oracle.longest_suffix_match(x, 2, 2)
    assert (n, e) == (2, 1)
    mode, draft = oracle.switch(True, n, e, 1.0, 0.0, 2, 16, x)
    assert mode == COPY and draft == [1, 2, 8, 9]    # L-1-e = 4 < k
    # periodic run: continuation of the overlapped occurrence is only the last token
    x = np.array([4, 4, 4, 4], np.int32)
    n, e = oracle.longest_suffix_match(x, 1, 8)
    assert (n, e) == (3, 2)
    assert oracle.switch(True, n, e, 1.0, 0.0, 1, 8, x) == (COPY, [4])


def _row(tokens, cap):
    r = np.zeros(cap, np.int32)
    r[: len(tokens)] = tokens
    return r


def test_verify_full_zero_partial():
    cap = 16
    ctx = [1, 2, 3]
    # full accept: all 4 draft tokens agree, bonus token 77 appended -> +5
    row = _row(ctx, cap)
    L, a, st = oracle.verify_row(row, 3, cap, [4, 5, 6, 7], [4, 5, 6, 7, 77])
    assert (L, a, st) == (8, 4, 0) and row[:8].tolist() == [1, 2, 3, 4, 5, 6, 7, 77]
    # zero accept: the first token disagrees; the target's own token is appended -> +1
    row = _row(ctx, cap)
    L, a, st = oracle.verify_row(row, 3, cap, [4, 5], [9, 5, 6])
    assert (L, a, st) == (4, 0, 0) and row[:4].tolist() == [1, 2, 3, 9]
    # partial: agree on 2 then disagree
    row = _row(ctx, cap)
    L, a, st = oracle.verify_row(row, 3, cap, [4, 5, 6], [4, 5, 0, 1])
    assert (L, a, st) == (6, 2, 0) and row[:6].tolist() == [1, 2, 3, 4, 5, 0]
    # empty draft: plain autoregressive step appends target[0]
    row = _row(ctx, cap)
    L, a, st = oracle.verify_row(row, 3, cap, [], [42])
    assert (L, a, st) == (4, 0, 0) and row[3] == 42


def test_verify_capacity_leaves_row_untouched():
    cap = 6
    row = _row([1, 2, 3, 4], cap)
    before = row.copy()
    L, a, st = oracle.verify_row(row, 4, cap, [5, 6, 7], [5, 6, 7, 8])   # would need 4 slots
    assert (L, a, st) == (4, -1, oracle.ROW_CAPACITY)
    assert np.array_equal(row, before)
    L, a, st = oracle.verify_row(row, 4, cap, [5, 9], [5, 6, 7])          # needs 2 slots: fits
    assert (L, a, st) == (6, 1, 0) and row.tolist() == [1, 2, 3, 4, 5, 6]


def test_greedy_exactness_invariant():
    """Whatever the drafts, the appended stream equals the target's greedy tokens: every appended
    token is target[j] for the j it lands on, and accepted <= draft length."""
    rng = np.random.default_rng(5)
    cap = 4096
    row = _row([0], cap)
    L = 1
    for _ in range(300):
        k = int(rng.integers(0, 9))
        draft = rng.integers(0, 3, k).astype(np.int32)
        target = rng.integers(0, 3, k + 1).astype(np.int32)
        L0 = L
        L, a, st = oracle.verify_row(row, L, cap, draft, target)
        assert st == 0 and 0 <= a <= k and L == L0 + a + 1
        assert row[L0: L].tolist() == target[: a + 1].tolist()


def test_batched_step_and_verify_match_single_row_calls():
    wl = synth.get_workload("uniform_8k").scaled(B=4, L0=600, steps=3)
    ctx, lens = wl.contexts()
    h = wl.hidden(0)
    w = wl.probe_weights()
    out = oracle.step(ctx, lens, h, w, k=wl.k, n_min=wl.n_min, n_max=wl.n_max,
                      logit_tau=wl.logit_tau)
    for b in range(wl.B):
        n, e = oracle.longest_suffix_match(ctx[b], wl.n_min, wl.n_max, L=int(lens[b]))
        assert (out["match_n"][b], out["match_end"][b]) == (n, e)
        z = oracle.probe_linear(h[b], w)
        assert out["score"][b] == z
        mode, draft = oracle.switch(n > 0, n, e, z, wl.logit_tau, wl.n_min, wl.k, ctx[b],
                                    L=int(lens[b]))
        assert out["mode"][b] == mode and out["draft"][b, : out["len"][b]].tolist() == draft
