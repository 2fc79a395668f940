"""The rescan kernel's hash instance against the oracle, through the C ABI.

The library takes the instance that hashes every old end before the grid-dependency wait (one byte an
end; the scan after the wait then compares bytes and tests only the ends whose byte matches) when a
launch's grid has at least one CTA per SM and the extra shared memory keeps the resident CTAs per SM.
The small lockstep cases of the other files run grids below the SM count, so the cases here force grids
above it (rows x CTAs per row >= the SM count) on short rows: filter depths 3, 2 and 1 (n_min 3, 2, 1),
greedy, sampled and W-candidate verification, fused and separate, the linear and the two-layer probe.
The same rows with fewer CTAs than SMs (the other instance) are held to the oracle beside them.
"""
import numpy as np
import pytest

import synth
from tests import lockstep
from tests.test_gpu_candidates import compare as cand_compare, gpu_loop as cand_gpu_loop, \
    oracle_loop as cand_oracle_loop

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS

# (workload, CTAs per row): rows x CTAs >= 152 SMs takes the hash instance
HASHED = {
    "zipf_f3": (W["zipf_32k"].scaled(name="zipf_f3", B=48, L0=5001, steps=12), 4),
    "mixed_f2": (W["mixed_128k"].scaled(name="mixed_f2", B=40, L0=6003, steps=10), 4),
    "uniform_f1": (W["uniform_8k"].scaled(name="uniform_f1", B=48, L0=3001, steps=12, n_min=1), 4),
    "code_mlp": (W["code_16k"].scaled(name="code_mlp", B=160, L0=2001, steps=6), 1),
}


def _sms():
    import torch
    return torch.cuda.get_device_properties(0).multi_processor_count


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("name", list(HASHED))
def test_hash_instance_lockstep(name, fused):
    wl, split = HASHED[name]
    assert wl.B * split >= _sms()  # the grid that selects the hash instance
    rows = range(wl.B)
    o_trace, o_ctx, _ = lockstep.oracle_trace(wl, rows, wl.steps)
    g_trace, g_ctx, _ = lockstep.gpu_trace(wl, wl.steps, split=split, fused=fused)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert stats["checked"] > 0 and len(flips) <= 1
    if name != "code_mlp":
        # the same rows on a grid below the SM count (the instance without the hash bytes)
        g2, g2_ctx, _ = lockstep.gpu_trace(wl, wl.steps, split=1, fused=fused)
        assert wl.B * 1 < _sms()
        lockstep.compare(wl, o_trace, g2, rows, o_ctx, g2_ctx)


@pytest.mark.parametrize("name", ["zipf_f3", "mixed_f2"])
def test_hash_instance_sampled(name):
    wl, split = HASHED[name]
    rows = range(wl.B)
    o_trace, o_ctx, _ = lockstep.oracle_trace(wl, rows, wl.steps, sampled=True)
    g_trace, g_ctx, _ = lockstep.gpu_trace(wl, wl.steps, sampled=True, split=split, fused=True)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert stats["checked"] > 0 and len(flips) <= 1


@pytest.mark.parametrize("Wc,D", [(10, 20), (3, 8)])
@pytest.mark.parametrize("name", ["zipf_f3", "uniform_f1"])
def test_hash_instance_candidates(name, Wc, D):
    wl, split = HASHED[name]
    wl = wl.scaled(k=max(wl.k, D))  # row capacity for appends of up to D + 1 tokens a step
    rows = range(wl.B)
    o_trace, o_ctx = cand_oracle_loop(wl, rows, wl.steps, Wc, D)
    g_trace, g_ctx = cand_gpu_loop(wl, wl.steps, Wc, D, split=split, fused=True)
    checked, _ = cand_compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert checked > 0
