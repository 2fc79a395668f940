"""Verification at temperature T > 0 (App. A): the CUDA path vs the oracle, through the C ABI.

The loop is step -> sampled stand-in -> switchsd_verify_sampled (or the fused
switchsd_verify_sampled_step) on both sides from the same seeded inputs; accepted lengths, appended contexts and everything the step produces must match the oracle
bit for bit (the acceptance test is taken in binary32 on both sides), the probe logit within 1e-3.
"""
import numpy as np
import pytest

import oracle
import synth
from tests import lockstep

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS

SMALL = {
    "uniform_small": W["uniform_8k"].scaled(name="uniform_small", B=8, L0=3000, steps=20),
    "zipf_small": W["zipf_32k"].scaled(name="zipf_small", B=8, L0=9001, steps=24),
    "code_small": W["code_16k"].scaled(name="code_small", B=12, L0=5000, steps=16),
    "mixed_small": W["mixed_128k"].scaled(name="mixed_small", B=4, L0=20003, steps=12),
}


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("name", list(SMALL))
def test_sampled_lockstep(name, fused):
    wl = SMALL[name]
    rows = range(wl.B)
    o_trace, o_ctx, _ = lockstep.oracle_trace(wl, rows, wl.steps, sampled=True)
    g_trace, g_ctx, _ = lockstep.gpu_trace(wl, wl.steps, sampled=True, fused=fused)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert stats["checked"] > 0
    # the sampled rule accepted something and rejected something over the run
    acc = np.concatenate([t["accept"] for t in o_trace])
    assert acc.max() > 0 and (acc == 0).any()


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("name", ["zipf_small", "code_small", "mixed_small"])
def test_sampled_index_lockstep(name, fused):
    """The incremental index with the sampled rule: verification and inserts in the index kernel."""
    wl = SMALL[name]
    rows = range(wl.B)
    o_trace, o_ctx, _ = lockstep.oracle_trace(wl, rows, wl.steps, sampled=True)
    g_trace, g_ctx, _ = lockstep.gpu_trace(wl, wl.steps, sampled=True, fused=fused, use_index=True)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert stats["checked"] > 0


def test_device_sampled_harness_matches_host():
    import torch
    from paper_2609_20186_gb300 import binding as bd

    wl = W["zipf_32k"].scaled(B=64, steps=8)
    rng = np.random.default_rng(3)
    B, k = wl.B, wl.k
    lens = (wl.L0 + rng.integers(-3, 50, B)).astype(np.int32)
    lens[5] = wl.cap - 2
    mode = rng.integers(0, 3, B).astype(np.int32)
    future = rng.integers(0, 50, (B, wl.cap - wl.L0)).astype(np.int32)
    draft = np.zeros((B, k), np.int32)
    for b in range(B):  # copy drafts that agree with the stream for a while, then not
        pos = lens[b] - wl.L0 + np.arange(k)
        ok = (pos >= 0) & (pos < future.shape[1])
        g = np.where(ok, future[b, np.clip(pos, 0, future.shape[1] - 1)], 0)
        cut = rng.integers(0, k + 1)
        draft[b] = np.where(np.arange(k) < cut, g, rng.integers(0, 50, k))
    dlen = np.where(mode == 1, rng.integers(1, k + 1, B), 0).astype(np.int32)
    hp = wl.harness_params()
    for step in (0, 5):
        vd, vl, p, q, u, rs = synth.harness_sampled(hp, step, lens, mode, draft, dlen, future)
        dev = {n: torch.from_numpy(a).cuda() for n, a in
               (("lens", lens), ("mode", mode), ("draft", draft), ("dlen", dlen), ("future", future))}
        i32 = dict(dtype=torch.int32, device="cuda")
        f32 = dict(dtype=torch.float32, device="cuda")
        g = dict(vd=torch.zeros(B, k, **i32), vl=torch.zeros(B, **i32), p=torch.zeros(B, k, **f32),
                 q=torch.zeros(B, k, **f32), u=torch.zeros(B, k, **f32), rs=torch.zeros(B, k + 1, **i32))
        bd.switchsd_harness_sampled(dev["lens"], dev["mode"], dev["draft"], dev["dlen"], dev["future"],
                                    g["vd"], g["vl"], g["p"], g["q"], g["u"], g["rs"], step=step,
                                    **{x: hp[x] for x in ("seed", "V", "L0", "gamma", "thr_neural",
                                                          "p_hit", "p_miss", "q_neural")})
        for name, ref in (("vd", vd), ("vl", vl), ("p", p), ("q", q), ("u", u), ("rs", rs)):
            got = g[name].cpu().numpy()
            assert np.array_equal(got, ref), name   # floats too: both sides build them exactly


def test_temperature_zero_matches_greedy_kernel():
    """One-hot target probabilities and the argmax as the resample: switchsd_verify_sampled and
    switchsd_verify leave identical contexts, lengths and accepted counts, equal to the oracle's."""
    import torch
    from paper_2609_20186_gb300 import binding as bd

    rng = np.random.default_rng(5)
    B, k, cap = 200, 16, 96
    L0 = rng.integers(1, 60, B).astype(np.int32)
    L0[0], L0[1] = cap - k - 1, cap - 3          # the first fits exactly, the second overflows
    ctx = rng.integers(0, 4, (B, cap)).astype(np.int32)
    draft = rng.integers(0, 3, (B, k)).astype(np.int32)
    target = rng.integers(0, 3, (B, k + 1)).astype(np.int32)
    dlen = rng.integers(0, k + 1, B).astype(np.int32)
    draft[1], dlen[1] = target[1, :k], k          # accepts all k tokens: does not fit
    p = (draft == target[:, :k]).astype(np.float32)
    u = rng.random((B, k)).astype(np.float32)
    results = []
    for sampled in (False, True):
        c = torch.from_numpy(ctx.copy()).cuda()
        ln = torch.from_numpy(L0.copy()).cuda()
        acc = torch.zeros(B, dtype=torch.int32, device="cuda")
        st = torch.zeros(B, dtype=torch.int32, device="cuda")
        d = torch.from_numpy(draft).cuda()
        t = torch.from_numpy(target).cuda()
        dl = torch.from_numpy(dlen).cuda()
        if sampled:
            bd.switchsd_verify_sampled(d, torch.from_numpy(p).cuda(), torch.from_numpy(u).cuda(), t, acc,
                                       draft_len=dl, ctx_tokens=c, ctx_lens=ln, status=st)
        else:
            bd.switchsd_verify(d, t, acc, draft_len=dl, ctx_tokens=c, ctx_lens=ln, status=st)
        results.append((c.cpu().numpy(), ln.cpu().numpy(), acc.cpu().numpy(), st.cpu().numpy()))
    for x, y in zip(*results):
        assert np.array_equal(x, y)
    octx, olens = ctx.copy(), L0.copy()
    oacc, ost = oracle.verify_sampled(octx, olens, draft, dlen, p, u, target)
    assert np.array_equal(results[1][0], octx) and np.array_equal(results[1][1], olens)
    assert np.array_equal(results[1][2], oacc) and np.array_equal(results[1][3], ost)
    assert (ost == 1).any()


def test_full_size_sampled_rows():
    """zipf_32k in the benchmark's shape: every row runs on the GPU at T > 0; the oracle replays a sample
    of rows over every step (rows are independent, so a replayed row is exact)."""
    wl = W["zipf_32k"].scaled(steps=16)
    g_trace, g_ctx, _ = lockstep.gpu_trace(wl, wl.steps, sampled=True, fused=True)
    rows = [0, 17, 40, 63]
    o_trace, o_ctx, _ = lockstep.oracle_trace(wl, rows, wl.steps, sampled=True)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert stats["checked"] > 0
