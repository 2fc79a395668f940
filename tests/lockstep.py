"""Lockstep drivers used by the parity tests.

The oracle side and the GPU side each run the full decoding loop on their own state, from the same
seeded inputs (synth): step -> harness (target stand-in) -> verify.  Nothing computed by one side is
fed to the other; the tests compare the two traces step by step.

Near-threshold rule: if the modes differ and the oracle's logit is within 1e-3 of logit(tau), the row is a
permitted flip -- the two probes round differently at the threshold, so both sides have taken a valid
decision; their contexts diverge from then on, and the row is compared no further.  Any other difference
fails.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

import oracle
import synth

SCORE_TOL = 1e-3


def oracle_trace(wl: synth.Workload, rows, steps: int, ctx=None, lens=None, sampled: bool = False):
    """Runs the oracle loop on the given rows; returns a list (per step) of dicts of per-row arrays
    plus the final ctx / lens.  sampled: verification at T > 0 with the sampled stand-in."""
    if ctx is None:
        ctx, lens = wl.contexts()
    ctx = ctx.copy()
    lens = lens.copy()
    future = wl.future()
    pw = wl.probe_weights()
    hp = wl.harness_params()
    rows = list(rows)
    trace = []
    for t in range(steps):
        h = wl.hidden(t)
        out = None
        for b in rows:
            o = oracle.step(ctx, lens, h, pw, k=wl.k, n_min=wl.n_min, n_max=wl.n_max,
                            kappa=wl.kappa, logit_tau=wl.logit_tau, probe_kind=wl.probe_kind,
                            probe_hidden=wl.probe_hidden, rows=(b, b + 1))
            if out is None:
                out = o
            else:
                for key in out:
                    out[key][b] = o[key][b]
        if sampled:
            vd, vl, pp, qq, uu, rs = synth.harness_sampled(hp, t, lens, out["mode"], out["draft"],
                                                           out["len"], future, rows=rows)
        else:
            vd, vl, tg = synth.harness_targets(hp, t, lens, out["mode"], out["draft"], out["len"],
                                               future, rows=rows)
        acc = np.zeros(wl.B, np.int32)
        st = np.zeros(wl.B, np.int32)
        for b in rows:
            if sampled:
                a, s = oracle.verify_sampled(ctx, lens, vd, vl, pp, uu, rs, q=qq, rows=(b, b + 1))
            else:
                a, s = oracle.verify(ctx, lens, vd, vl, tg, rows=(b, b + 1))
            acc[b], st[b] = a[b], s[b]
        out["accept"] = acc
        out["vstatus"] = st
        out["lens_after"] = lens.copy()
        trace.append(out)
    return trace, ctx, lens


def oracle_trace_rows(wl: synth.Workload, n_rows: int, steps: int, threads: int | None = None):
    """oracle_trace on rows 0 .. n_rows-1 with every oracle call split into contiguous row ranges run on
    host threads (rows are independent and the oracle's C calls release the interpreter lock): the same
    trace, in a fraction of the time.  The host target stand-in runs once per step on all the rows."""
    ctx, lens = wl.contexts()
    future = wl.future()
    pw = wl.probe_weights()
    hp = wl.harness_params()
    R = min(n_rows, wl.B)
    try:
        cores = len(os.sched_getaffinity(0))
    except AttributeError:
        cores = os.cpu_count() or 1
    nt = max(1, min(threads or cores, R))
    chunks = [(R * i // nt, R * (i + 1) // nt) for i in range(nt)]
    rows = range(R)
    trace = []
    with ThreadPoolExecutor(nt) as pool:
        for t in range(steps):
            h = wl.hidden(t)
            parts = list(pool.map(lambda c: oracle.step(
                ctx, lens, h, pw, k=wl.k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                logit_tau=wl.logit_tau, probe_kind=wl.probe_kind, probe_hidden=wl.probe_hidden,
                rows=c), chunks))
            out = parts[0]
            for (b0, b1), part in zip(chunks[1:], parts[1:]):
                for key in out:
                    out[key][b0:b1] = part[key][b0:b1]
            vd, vl, tg = synth.harness_targets(hp, t, lens, out["mode"], out["draft"], out["len"], future,
                                               rows=rows)
            acc = np.zeros(wl.B, np.int32)
            st = np.zeros(wl.B, np.int32)
            for (b0, b1), (a, s) in zip(chunks, pool.map(
                    lambda c: oracle.verify(ctx, lens, vd, vl, tg, rows=c), chunks)):
                acc[b0:b1], st[b0:b1] = a[b0:b1], s[b0:b1]
            out["accept"] = acc
            out["vstatus"] = st
            out["lens_after"] = lens.copy()
            trace.append(out)
    return trace, ctx, lens


def gpu_trace(wl: synth.Workload, steps: int, split: int = 0, ctx=None, lens=None, device="cuda",
              fused: bool = False, use_index: bool = False, sampled: bool = False, extras: dict | None = None):
    """Runs the GPU loop on all rows; returns the per-step host copies of every output.

    fused=False: switchsd_step, target stand-in, switchsd_verify per iteration.
    fused=True:  switchsd_verify_step (verification of iteration t-1, then step t) and the target
                 stand-in per iteration; the last draft is verified by switchsd_verify.
    sampled=True: the sampled stand-in and switchsd_verify_sampled / switchsd_verify_sampled_step (T > 0).
    extras: if given, the run keeps the per-mode counters (switchsd_params.counters) and stores them
    there under "counters" (host int64 array)."""
    import torch
    from paper_2609_20186_gb300 import Session, bf16_tensor

    if ctx is None:
        ctx, lens = wl.contexts()
    sess = Session(ctx, lens, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max,
                   kappa=wl.kappa, logit_tau=wl.logit_tau, probe_kind=wl.probe_kind,
                   probe_hidden=wl.probe_hidden, future=wl.future(), harness=wl.harness_params(),
                   split=split, d=wl.d, use_index=use_index, device=device, counters=extras is not None)
    trace = []
    for t in range(steps):
        hidden = bf16_tensor(wl.hidden(t), sess.device)
        if fused and t > 0:
            if sampled:
                sess.verify_sampled_step(hidden)
            else:
                sess.verify_step(hidden)
            prev = trace[-1]
            st = sess.status.cpu().numpy()
            prev["accept"] = sess.accept.cpu().numpy()
            prev["vstatus"] = np.where((st == 1) | (st == 2), st, 0)
            prev["lens_after"] = sess.lens.cpu().numpy()
        else:
            sess.step(hidden)
        out = sess.step_outputs()
        if sampled:
            sess.harness_sampled(t)
        else:
            sess.harness(t)
        if not fused or t == steps - 1:
            if sampled:
                sess.verify_sampled()
            else:
                sess.verify()
            out["accept"] = sess.accept.cpu().numpy()
            out["vstatus"] = sess.vstatus.cpu().numpy()
            out["lens_after"] = sess.lens.cpu().numpy()
        trace.append(out)
    torch.cuda.synchronize()
    if extras is not None:
        extras["counters"] = sess.counters.cpu().numpy()
    return trace, sess.ctx.cpu().numpy(), sess.lens.cpu().numpy()


def compare(wl: synth.Workload, o_trace, g_trace, rows, o_ctx=None, g_ctx=None):
    """Asserts parity on the given rows; returns (flips, stats)."""
    kappa = wl.kappa_eff
    active = set(rows)
    flips = []
    stats = {"copy": 0, "rep_no_copy": 0, "no_rep": 0, "checked": 0}
    for t, (o, g) in enumerate(zip(o_trace, g_trace)):
        for b in sorted(active):
            where = f"{wl.name} step {t} row {b}"
            assert g["status"][b] == 0, where
            # integer outputs of the search: bit-exact
            assert g["match_n"][b] == o["match_n"][b], (where, g["match_n"][b], o["match_n"][b])
            assert g["match_end"][b] == o["match_end"][b], (where, g["match_end"][b],
                                                            o["match_end"][b])
            # probe logit within tolerance
            assert abs(float(g["score"][b]) - float(o["score"][b])) <= SCORE_TOL, \
                (where, g["score"][b], o["score"][b])
            if g["mode"][b] != o["mode"][b]:
                near = abs(float(o["score"][b]) - wl.logit_tau) <= SCORE_TOL
                both_match = o["match_n"][b] >= kappa
                assert near and both_match, (where, "switch flip outside the threshold band",
                                             g["mode"][b], o["mode"][b], o["score"][b])
                flips.append((t, b))
                active.discard(b)
                continue
            m = int(o["mode"][b])
            stats[("no_rep", "copy", "rep_no_copy")[m]] += 1
            assert g["len"][b] == o["len"][b], where
            ln = int(o["len"][b])
            assert np.array_equal(g["draft"][b, :ln], o["draft"][b, :ln]), where
            assert g["accept"][b] == o["accept"][b], (where, g["accept"][b], o["accept"][b])
            assert g["vstatus"][b] == o["vstatus"][b], where
            assert g["lens_after"][b] == o["lens_after"][b], where
            stats["checked"] += 1
    if o_ctx is not None and g_ctx is not None:
        for b in active:
            L = int(o_trace[-1]["lens_after"][b])
            assert np.array_equal(o_ctx[b, :L], g_ctx[b, :L]), f"{wl.name} final context row {b}"
    return flips, stats
