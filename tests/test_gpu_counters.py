"""The per-mode controller tallies (switchsd_params.counters) against the oracle's trace.

The paper reports, per benchmark, the share of iterations that copy and the mean accepted length of each
drafter (§4, Table 1).  With counters the fused calls tally, for every row, the mode its step chose and,
for the draft its verification checked, the previous step's mode (copy or neural) and the accepted
length.  The oracle's lockstep trace gives the same tallies directly: every step's mode, and for the
verification inside launch t the mode and accepted length of step t - 1 (the last draft is verified by
switchsd_verify, which does not count).  They must be equal.
"""
import numpy as np
import pytest

import synth
from tests import lockstep

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS


def _expected(o_trace, rows):
    c = np.zeros(7, np.int64)
    for t, o in enumerate(o_trace):
        for b in rows:
            c[int(o["mode"][b])] += 1
            if t + 1 < len(o_trace) and o["accept"][b] >= 0:   # verified inside launch t + 1
                slot = 3 if o["mode"][b] == 1 else 5
                c[slot] += 1
                c[slot + 1] += int(o["accept"][b])
    return c


@pytest.mark.parametrize("name,use_index", [("zipf", False), ("code", False), ("mixed", False),
                                            ("zipf", True)])
def test_counters_match_oracle(name, use_index):
    wl = {"zipf": W["zipf_32k"].scaled(name="zipf_ctr", B=12, L0=6000, steps=20),
          "code": W["code_16k"].scaled(name="code_ctr", B=24, L0=4000, steps=12),
          "mixed": W["mixed_128k"].scaled(name="mixed_ctr", B=4, L0=20003, steps=10)}[name]
    rows = range(wl.B)
    o_trace, _, _ = lockstep.oracle_trace(wl, rows, wl.steps)
    extras = {}
    g_trace, _, _ = lockstep.gpu_trace(wl, wl.steps, fused=True, use_index=use_index, extras=extras)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, rows)
    assert not flips          # a flipped row would diverge; these seeds have none
    exp = _expected(o_trace, rows)
    assert np.array_equal(extras["counters"], exp), (extras["counters"], exp)
    assert exp[1] > 0 and exp[3] > 0 and exp[5] > 0           # both drafters were exercised
