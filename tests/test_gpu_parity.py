"""GPU path vs the CPU oracle, through the C ABI (libswitchsd.so via the ctypes binding).

Bar: bit-exact on match length / end position, modes, draft tokens, accepted lengths and contexts;
probe logits within 1e-3 absolute; no switch flip outside 1e-3 of the threshold (lockstep.compare).

Small cases compare every row at every step and span several staged tiles with ragged tails; the
full-size workloads run every row on the GPU in the launch configuration the benchmark uses, and the
oracle replays every row of every step (its calls split over the host cores), 64 of the 256 rows for the
two-layer-probe workload.
"""
import numpy as np
import pytest

import synth
from tests import lockstep

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS

SMALL = {
    "uniform_small": W["uniform_8k"].scaled(name="uniform_small", B=8, L0=3000, steps=20),
    "zipf_small": W["zipf_32k"].scaled(name="zipf_small", B=8, L0=9001, steps=24),
    "code_small": W["code_16k"].scaled(name="code_small", B=12, L0=5000, steps=16),
    "mixed_small": W["mixed_128k"].scaled(name="mixed_small", B=4, L0=20003, steps=12),
    "zipf_kappa5": W["zipf_32k"].scaled(name="zipf_kappa5", B=8, L0=6000, steps=16, kappa=5),
}


def _run_small(wl, split=0, fused=False):
    rows = range(wl.B)
    o_trace, o_ctx, _ = lockstep.oracle_trace(wl, rows, wl.steps)
    g_trace, g_ctx, _ = lockstep.gpu_trace(wl, wl.steps, split=split, fused=fused)
    return lockstep.compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("name", list(SMALL))
def test_small_lockstep(name, fused):
    flips, stats = _run_small(SMALL[name], fused=fused)
    assert stats["checked"] > 0
    assert len(flips) <= 1


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("split", [1, 2, 4, 8, 16])
def test_split_invariance(split, fused):
    wl = SMALL["zipf_small"].scaled(steps=8)
    _run_small(wl, split=split, fused=fused)


def test_multi_tile_ring():
    """Rows long enough for several kTileMax tiles per CTA (two-stage ring), fused and separate."""
    wl = W["mixed_128k"].scaled(name="mixed_ring", B=2, L0=70001, steps=6)
    for fused in (False, True):
        _run_small(wl, split=2, fused=fused)


def test_fused_copy_heavy():
    """The code workload copies often: fused appends land in the staged tiles of the last CTA."""
    wl = W["code_16k"].scaled(name="code_fused", B=16, L0=3001, steps=24, probe_kind=0, d=4096)
    flips, stats = _run_small(wl, split=4, fused=True)
    assert stats["copy"] > 0


@pytest.mark.parametrize("variant", ["copy", "nocopy", "norep"])
def test_planted(variant):
    wl = W[f"planted_{variant}"]
    exp = wl.expected_planted()
    o_trace, o_ctx, _ = lockstep.oracle_trace(wl, [0], 1)
    g_trace, g_ctx, g_lens = lockstep.gpu_trace(wl, 1)
    lockstep.compare(wl, o_trace, g_trace, [0], o_ctx, g_ctx)
    g = g_trace[0]
    assert g["mode"][0] == exp["mode"]
    assert g["match_n"][0] == exp["match_n"] and g["match_end"][0] == exp["match_end"]
    assert g["draft"][0, : g["len"][0]].tolist() == exp["draft"]
    if "accept" in exp:
        assert g["accept"][0] == exp["accept"] and g_lens[0] == wl.L0 + exp["accept"] + 1


FULL_ROWS = {"uniform_8k": 64, "zipf_32k": 64, "code_16k": 64, "mixed_128k": 16}


@pytest.mark.parametrize("name", list(FULL_ROWS))
def test_full_size_every_row(name):
    """Full-size workload in the benchmark's launch configuration (fused verify + step), every step:
    every row (the first 64 of the code workload's 256) against the oracle."""
    wl = W[name]
    n = FULL_ROWS[name]
    g_trace, g_ctx, _ = lockstep.gpu_trace(wl, wl.steps, fused=True)
    o_trace, o_ctx, _ = lockstep.oracle_trace_rows(wl, n, wl.steps)
    rows = range(n)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert stats["checked"] >= (n - len(flips)) * wl.steps
    assert len(flips) <= 2
    # every row of the batch stayed healthy on the GPU
    for t in g_trace:
        assert np.all(t["status"] == 0) and np.all(t["vstatus"] == 0)
        assert np.all(t["len"] <= wl.k)


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("name", ["mixed_small", "zipf_small", "code_small", "zipf_kappa5"])
def test_index_lockstep(name, fused):
    """The incremental n-gram index against the oracle's rescan, in lockstep (build, inserts on every
    verification, lookups), with the two-layer probe for the code workload."""
    wl = SMALL[name]
    rows = range(wl.B)
    o_trace, o_ctx, _ = lockstep.oracle_trace(wl, rows, wl.steps)
    g_trace, g_ctx, _ = lockstep.gpu_trace(wl, wl.steps, fused=fused, use_index=True)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert stats["checked"] > 0 and len(flips) <= 1


def test_index_rewind_and_replay():
    """Lowering ctx_lens and appending the same tokens again leaves the index consistent: the replayed
    steps reproduce the first pass exactly (the insertions of known positions are no-ops)."""
    import torch
    from paper_2609_20186_gb300 import Session, bf16_tensor

    wl = SMALL["mixed_small"].scaled(steps=10)
    ctx, lens = wl.contexts()
    sess = Session(ctx, lens, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max,
                   logit_tau=wl.logit_tau, future=wl.future(), harness=wl.harness_params(), d=wl.d,
                   use_index=True)
    hid = [bf16_tensor(wl.hidden(t), sess.device) for t in range(wl.steps)]
    sess.step(hid[0])
    sess.harness(0)
    for t in range(1, 4):
        sess.verify_step(hid[t])
        sess.harness(t)
    state = [(x, x.clone()) for x in (sess.lens, sess.vdraft, sess.vlen, sess.target, sess.mode,
                                      sess.draft, sess.len)]

    def run():
        outs = []
        for t in range(4, wl.steps):
            sess.verify_step(hid[t])
            outs.append({n: getattr(sess, n).clone() for n in ("mode", "len", "draft", "match_n",
                                                               "match_end", "accept", "lens")})
            sess.harness(t)
        return outs

    first = run()
    for dst, src in state:
        dst.copy_(src)
    second = run()
    for a, b in zip(first, second):
        for n in a:
            assert torch.equal(a[n], b[n]), n


@pytest.mark.parametrize("name", ["mixed_128k", "zipf_32k"])
def test_index_equals_rescan_full_size(name):
    """Every row at every step of the full workload: the index path and the rescan path (both on the
    GPU, fused launches) produce identical matches, modes, drafts and contexts."""
    wl = W[name]
    a, a_ctx, _ = lockstep.gpu_trace(wl, wl.steps, fused=True)
    b, b_ctx, _ = lockstep.gpu_trace(wl, wl.steps, fused=True, use_index=True)
    for t, (x, y) in enumerate(zip(a, b)):
        for key in ("match_n", "match_end", "mode", "len", "accept", "lens_after", "status"):
            assert np.array_equal(x[key], y[key]), (name, t, key)
        for r in range(wl.B):
            n = int(x["len"][r])
            assert np.array_equal(x["draft"][r, :n], y["draft"][r, :n]), (name, t, r)
        assert np.allclose(x["score"], y["score"], atol=1e-3)
    assert np.array_equal(a_ctx, b_ctx)


def test_threshold_extremes():
    """tau -> 0 (logit -inf) copies on every kappa-match (prompt-lookup decoding); tau -> 1 never
    copies."""
    base = SMALL["zipf_small"].scaled(steps=6)
    for tau, expect_copy in ((0.0, True), (1.0, False)):
        wl = base.scaled(tau=tau)
        _, _ = _run_small(wl)
        g_trace, _, _ = lockstep.gpu_trace(wl, wl.steps)
        for t in g_trace:
            hit = t["match_n"] >= wl.kappa_eff
            if expect_copy:
                assert np.array_equal(t["mode"] == 1, hit)
            else:
                assert not np.any(t["mode"] == 1)


def test_edge_lengths_and_status():
    """Rows of length 1, 2, n_min, n_min + 1, a full row and out-of-range lengths in one batch."""
    import torch
    from paper_2609_20186_gb300 import Session, bf16_tensor
    import oracle

    wl = W["uniform_8k"].scaled(B=10, L0=256, steps=1)
    ctx, _ = wl.contexts()
    ctx[:, :] = np.random.default_rng(0).integers(0, 3, ctx.shape)   # dense small-alphabet repeats
    cap = wl.cap
    lens = np.array([1, 2, 3, 4, 9, cap - 4, cap, 0, cap + 1, -7], np.int32)
    sess = Session(ctx, lens, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max,
                   logit_tau=wl.logit_tau, future=wl.future(), harness=wl.harness_params())
    h = wl.hidden(0)
    sess.step(bf16_tensor(h, sess.device))
    g = sess.step_outputs()
    for b in range(7):
        o = oracle.step(ctx, lens, h, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max,
                        logit_tau=wl.logit_tau, rows=(b, b + 1))
        assert g["status"][b] == 0
        assert (g["match_n"][b], g["match_end"][b]) == (o["match_n"][b], o["match_end"][b]), b
        assert g["mode"][b] == o["mode"][b] and g["len"][b] == o["len"][b]
        assert np.array_equal(g["draft"][b, : g["len"][b]], o["draft"][b, : o["len"][b]])
    for b in range(7, 10):
        assert g["status"][b] == 2 and g["mode"][b] == 0 and g["len"][b] == 0
    # verification: the full row (L = cap) cannot take even the bonus token
    sess.vdraft.zero_()
    sess.target.zero_()
    sess.vlen.zero_()
    sess.vlen[5] = 3
    sess.target[5, :4] = torch.tensor([0, 0, 0, 9], dtype=torch.int32, device=sess.device)
    before = sess.ctx.clone()
    sess.verify()
    acc = sess.accept.cpu().numpy()
    st = sess.vstatus.cpu().numpy()
    ln = sess.lens.cpu().numpy()
    assert st[6] == 1 and acc[6] == -1 and ln[6] == cap
    assert torch.equal(sess.ctx[6], before[6])
    # row 5: L = cap - 4, accepts 3 zeros, appends 9 -> exactly full
    assert st[5] == 0 and acc[5] == 3 and ln[5] == cap
    assert sess.ctx[5, cap - 4:].tolist() == [0, 0, 0, 9]
    # rows 0..4: empty drafts append target[0] = 0
    assert np.all(acc[:5] == 0) and np.all(ln[:5] == lens[:5] + 1)
    for b in range(7, 10):
        assert st[b] == 2 and acc[b] == -1


def test_device_harness_matches_host():
    import torch
    from paper_2609_20186_gb300 import binding as bd

    wl = W["zipf_32k"].scaled(B=64, steps=8)
    rng = np.random.default_rng(1)
    B, k = wl.B, wl.k
    lens = (wl.L0 + rng.integers(-3, 50, B)).astype(np.int32)
    lens[5] = wl.cap - 2                       # future positions past the stream read as 0
    mode = rng.integers(0, 3, B).astype(np.int32)
    draft = rng.integers(0, wl.V, (B, k)).astype(np.int32)
    dlen = np.where(mode == 1, rng.integers(1, k + 1, B), 0).astype(np.int32)
    future = rng.integers(0, wl.V, (B, wl.cap - wl.L0)).astype(np.int32)
    hp = wl.harness_params()
    for step in (0, 5):
        vd, vl, tg = synth.harness_targets(hp, step, lens, mode, draft, dlen, future)
        dev = {n: torch.from_numpy(a).cuda() for n, a in
               (("lens", lens), ("mode", mode), ("draft", draft), ("dlen", dlen), ("future", future))}
        gvd = torch.zeros(B, k, dtype=torch.int32, device="cuda")
        gvl = torch.zeros(B, dtype=torch.int32, device="cuda")
        gtg = torch.zeros(B, k + 1, dtype=torch.int32, device="cuda")
        bd.switchsd_harness_target(dev["lens"], dev["mode"], dev["draft"], dev["dlen"], dev["future"],
                                   gvd, gvl, gtg, step=step, **{x: hp[x] for x in
                                                                ("seed", "V", "L0", "gamma",
                                                                 "thr_neural")})
        assert np.array_equal(gvd.cpu().numpy(), vd)
        assert np.array_equal(gvl.cpu().numpy(), vl)
        assert np.array_equal(gtg.cpu().numpy(), tg)


@pytest.mark.parametrize("B,d,H1,bias", [(256, 5120, 256, False), (130, 4096, 100, True),
                                         (7, 1000, 64, True), (1, 64, 1, False),
                                         (300, 8192, 1024, True), (129, 5120, 200, True)])
def test_two_layer_probe_tensor_cores(B, d, H1, bias):
    """The tcgen05 two-layer probe vs the oracle (double), through switchsd_step: ragged B (M tiles),
    H1 (N tiles) and d (K chunks), with and without biases."""
    import math
    import torch
    import oracle
    from paper_2609_20186_gb300 import binding as bd, bf16_tensor

    rng = np.random.default_rng(B * 7 + d + H1)
    h = synth.bf16_bits_from_f32(rng.standard_normal((B, d)).astype(np.float32))
    W1 = synth.bf16_bits_from_f32((rng.standard_normal((H1, d)) / math.sqrt(d)).astype(np.float32))
    w2 = synth.bf16_bits_from_f32((rng.standard_normal(H1) / math.sqrt(H1)).astype(np.float32))
    b1 = (rng.standard_normal(H1) * 0.2).astype(np.float32) if bias else None
    b2 = 0.125 if bias else 0.0
    cap = 64
    ctx = torch.zeros(B, cap, dtype=torch.int32, device="cuda")
    lens = torch.full((B,), 10, dtype=torch.int32, device="cuda")
    out = dict(draft=torch.zeros(B, 8, dtype=torch.int32, device="cuda"),
               len=torch.zeros(B, dtype=torch.int32, device="cuda"),
               mode=torch.zeros(B, dtype=torch.int32, device="cuda"),
               score=torch.zeros(B, dtype=torch.float32, device="cuda"))
    pw = np.concatenate([W1.reshape(-1), w2])
    bd.switchsd_step(ctx, lens, bf16_tensor(h, "cuda"), bf16_tensor(pw, "cuda"), out["draft"],
                     out["len"], out["mode"], out["score"], k=8, n_min=2, n_max=4,
                     probe_kind=bd.PROBE_MLP, probe_hidden=H1,
                     b1=torch.from_numpy(b1).cuda() if bias else None, b2=b2)
    got = out["score"].cpu().numpy()
    for b in range(B):
        ref = oracle.probe_mlp(h[b], W1, w2, b1=b1, b2=b2)
        assert abs(got[b] - ref) <= 1e-3, (b, got[b], ref)
