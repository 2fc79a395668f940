"""W recency-ranked copy candidates (§3.3, App. D) on the GPU vs the oracle, through the C ABI.

Both sides run step -> candidate stand-in -> candidate verification from the same seeded inputs.  The
candidates, their lengths and count, the mode, the match, the kept candidate, the accepted length and
the contexts must match bit for bit; the probe logit within 1e-3; a mode may differ only within 1e-3
of the threshold (the row is then compared no further, as in lockstep.compare).
"""
import ctypes

import numpy as np
import pytest

import oracle
import synth
from tests import lockstep

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS
SMALL = {
    "uniform_small": W["uniform_8k"].scaled(name="uniform_small", B=8, L0=3000, steps=16),
    "zipf_small": W["zipf_32k"].scaled(name="zipf_small", B=8, L0=9001, steps=16),
    "code_small": W["code_16k"].scaled(name="code_small", B=12, L0=5000, steps=12),
    "mixed_small": W["mixed_128k"].scaled(name="mixed_small", B=4, L0=20003, steps=10),
    "zipf_kappa5": W["zipf_32k"].scaled(name="zipf_kappa5", B=8, L0=6000, steps=12, kappa=5),
}


def oracle_loop(wl, rows, steps, Wc, D):
    ctx, lens = wl.contexts()
    future, pw, hp = wl.future(), wl.probe_weights(), wl.harness_params()
    rows = list(rows)
    trace = []
    for t in range(steps):
        h = wl.hidden(t)
        out = None
        for b in rows:
            o = oracle.step_candidates(ctx, lens, h, pw, W=Wc, D=D, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                                       logit_tau=wl.logit_tau, probe_kind=wl.probe_kind,
                                       probe_hidden=wl.probe_hidden, rows=(b, b + 1))
            if out is None:
                out = o
            else:
                for key in out:
                    out[key][b] = o[key][b]
        vc, vl, vn, tg = synth.harness_candidates(hp, t, lens, out["mode"], out["cand"], out["cand_len"],
                                                  out["ncand"], future, rows=rows)
        acc = np.zeros(wl.B, np.int32)
        ch = np.zeros(wl.B, np.int32)
        for b in rows:
            a, c, _ = oracle.verify_candidates(ctx, lens, vc, vl, vn, tg, rows=(b, b + 1))
            acc[b], ch[b] = a[b], c[b]
        out.update(accept=acc, choice=ch, lens_after=lens.copy())
        trace.append(out)
    return trace, ctx


def gpu_loop(wl, steps, Wc, D, split=0, fused=False, use_index=False):
    """fused: switchsd_verify_candidates_step verifies iteration t-1's candidates and searches step t's in
    one launch; the last iteration's candidates are verified by switchsd_verify_candidates.  use_index:
    the incremental n-gram index (built from the initial contexts) searches, verifies and inserts."""
    import torch
    from paper_2609_20186_gb300 import binding as bd, bf16_tensor
    lib = bd.load()
    ctx, lens = wl.contexts()
    B, cap = ctx.shape
    dev = torch.device("cuda")
    i32 = dict(dtype=torch.int32, device=dev)
    c = torch.from_numpy(ctx).to(dev)
    ln = torch.from_numpy(lens).to(dev)
    fut = torch.from_numpy(np.ascontiguousarray(wl.future(), np.int32)).to(dev)
    pw = bf16_tensor(wl.probe_weights().reshape(-1), dev)
    cand, clen = torch.zeros(B, Wc, D, **i32), torch.zeros(B, Wc, **i32)
    ncand, mode = torch.zeros(B, **i32), torch.zeros(B, **i32)
    score = torch.zeros(B, dtype=torch.float32, device=dev)
    mn, me, st = torch.zeros(B, **i32), torch.zeros(B, **i32), torch.zeros(B, **i32)
    vc, vl, vn = torch.zeros(B, Wc, D, **i32), torch.zeros(B, Wc, **i32), torch.zeros(B, **i32)
    tg = torch.zeros(B, Wc, D + 1, **i32)
    acc, ch, vst = torch.zeros(B, **i32), torch.zeros(B, **i32), torch.zeros(B, **i32)
    p = bd.switchsd_params()
    p.B, p.cap, p.d, p.k = B, cap, wl.d, wl.k
    p.n_min, p.n_max, p.kappa, p.logit_tau = wl.n_min, wl.n_max, wl.kappa, wl.logit_tau
    p.probe_kind, p.probe_hidden, p.split = wl.probe_kind, wl.probe_hidden, split
    ws = torch.empty(max(256, bd.switchsd_workspace_bytes(B, wl.probe_kind, wl.probe_hidden, wl.d)),
                     dtype=torch.uint8, device=dev)
    p.workspace, p.workspace_bytes = ws.data_ptr(), ws.numel()
    p.out_match_n, p.out_match_end, p.status = mn.data_ptr(), me.data_ptr(), st.data_ptr()
    p.stream = torch.cuda.current_stream().cuda_stream
    idx = None
    if use_index:
        idx = bd.NgramIndex(B, cap, wl.n_min, wl.n_max)
        idx.build(c, ln)
        p.index = idx.handle
    h = wl.harness_params()
    hp = bd.switchsd_harness_params()
    hp.B, hp.k, hp.V, hp.L0, hp.n_future = B, wl.k, h["V"], h["L0"], fut.shape[1]
    hp.gamma, hp.seed, hp.thr_neural = h["gamma"], h["seed"], h["thr_neural"]
    hp.stream = p.stream
    vp = bd.switchsd_candidates_verify_params()
    vp.B, vp.cap, vp.W, vp.D = B, cap, Wc, D
    vp.cand_len, vp.ncand, vp.ctx_tokens, vp.ctx_lens = vl.data_ptr(), vn.data_ptr(), c.data_ptr(), ln.data_ptr()
    vp.status, vp.stream = vst.data_ptr(), p.stream
    vp.index = idx.handle if idx is not None else None
    trace = []
    for t in range(steps):
        hid = bf16_tensor(wl.hidden(t), dev)
        if fused and t > 0:
            assert lib.switchsd_verify_candidates_step(
                vc.data_ptr(), tg.data_ptr(), vl.data_ptr(), vn.data_ptr(), acc.data_ptr(), ch.data_ptr(),
                c.data_ptr(), ln.data_ptr(), hid.data_ptr(), pw.data_ptr(), ctypes.byref(p), Wc, D, cand.data_ptr(),
                clen.data_ptr(), ncand.data_ptr(), mode.data_ptr(), score.data_ptr()) == 0
            s_ = st.cpu().numpy()
            trace[-1].update(accept=acc.cpu().numpy(), choice=ch.cpu().numpy(), lens_after=ln.cpu().numpy(),
                             vstatus=np.where((s_ == 1) | (s_ == 2), s_, 0))
        else:
            assert lib.switchsd_step_candidates(c.data_ptr(), ln.data_ptr(), hid.data_ptr(), pw.data_ptr(),
                                                ctypes.byref(p), Wc, D, cand.data_ptr(), clen.data_ptr(),
                                                ncand.data_ptr(), mode.data_ptr(), score.data_ptr()) == 0
        out = {"cand": cand.cpu().numpy(), "cand_len": clen.cpu().numpy(), "ncand": ncand.cpu().numpy(),
               "mode": mode.cpu().numpy(), "score": score.cpu().numpy(), "match_n": mn.cpu().numpy(),
               "match_end": me.cpu().numpy(), "status": st.cpu().numpy()}
        hp.step = t
        assert lib.switchsd_harness_candidates(ln.data_ptr(), mode.data_ptr(), cand.data_ptr(), clen.data_ptr(),
                                               ncand.data_ptr(), fut.data_ptr(), Wc, D, vc.data_ptr(), vl.data_ptr(),
                                               vn.data_ptr(), tg.data_ptr(), ctypes.byref(hp)) == 0
        if not fused or t == steps - 1:
            assert lib.switchsd_verify_candidates(vc.data_ptr(), tg.data_ptr(), acc.data_ptr(), ch.data_ptr(),
                                                  ctypes.byref(vp)) == 0
            out.update(accept=acc.cpu().numpy(), choice=ch.cpu().numpy(), lens_after=ln.cpu().numpy(),
                       vstatus=vst.cpu().numpy())
        trace.append(out)
    torch.cuda.synchronize()
    if idx is not None:
        idx.close()
    return trace, c.cpu().numpy()


def compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx):
    active = set(rows)
    checked = copies = 0
    for t, (o, g) in enumerate(zip(o_trace, g_trace)):
        for b in sorted(active):
            where = f"{wl.name} step {t} row {b}"
            assert g["status"][b] == 0 and g["vstatus"][b] == 0, where
            assert g["match_n"][b] == o["match_n"][b] and g["match_end"][b] == o["match_end"][b], where
            assert abs(float(g["score"][b]) - float(o["score"][b])) <= lockstep.SCORE_TOL, where
            if g["mode"][b] != o["mode"][b]:
                assert abs(float(o["score"][b]) - wl.logit_tau) <= lockstep.SCORE_TOL, (where, "flip")
                active.discard(b)
                continue
            n = int(o["ncand"][b])
            assert g["ncand"][b] == n, (where, g["ncand"][b], n)
            for w in range(n):
                ln = int(o["cand_len"][b, w])
                assert g["cand_len"][b, w] == ln, where
                assert np.array_equal(g["cand"][b, w, :ln], o["cand"][b, w, :ln]), (where, w)
            assert g["accept"][b] == o["accept"][b] and g["choice"][b] == o["choice"][b], where
            assert g["lens_after"][b] == o["lens_after"][b], where
            checked += 1
            copies += n > 0
    for b in active:
        L = int(o_trace[-1]["lens_after"][b])
        assert np.array_equal(o_ctx[b, :L], g_ctx[b, :L]), f"{wl.name} context row {b}"
    return checked, copies


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("Wc,D", [(10, 20), (3, 8), (16, 64), (1, 4)])
@pytest.mark.parametrize("name", list(SMALL))
def test_candidates_lockstep(name, Wc, D, fused):
    wl = SMALL[name]
    rows = range(wl.B)
    o_trace, o_ctx = oracle_loop(wl, rows, wl.steps, Wc, D)
    g_trace, g_ctx = gpu_loop(wl, wl.steps, Wc, D, fused=fused)
    checked, copies = compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert checked > 0


KAPPA_LOW = {
    "zipf_kappa2": W["zipf_32k"].scaled(name="zipf_kappa2", B=4, L0=20003, steps=8, kappa=2),
    "code_kappa1": W["code_16k"].scaled(name="code_kappa1", B=4, L0=20003, steps=6, kappa=1),
}


@pytest.mark.parametrize("split", [0, 1], ids=["rescan_kernel", "step_kernel"])
@pytest.mark.parametrize("name", list(KAPPA_LOW))
def test_candidates_kappa_below_n_min(name, split):
    """kappa below n_min on the scan path: a candidate needs only kappa tokens of common suffix, fewer
    than a match that decides the mode, so the scan's filter must not test more than kappa tokens.  The
    library's split takes the rescan kernel; one CTA over 20K-token rows takes the step kernel."""
    wl = KAPPA_LOW[name]
    rows = range(wl.B)
    o_trace, o_ctx = oracle_loop(wl, rows, wl.steps, 10, 20)
    g_trace, g_ctx = gpu_loop(wl, wl.steps, 10, 20, split=split, fused=True)
    checked, copies = compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert checked > 0 and copies > 0


@pytest.mark.parametrize("split", [1, 2, 4, 8, 16])
def test_candidates_split_invariance(split):
    wl = SMALL["zipf_small"]
    rows = range(wl.B)
    o_trace, o_ctx = oracle_loop(wl, rows, 8, 10, 20)
    g_trace, g_ctx = gpu_loop(wl, 8, 10, 20, split=split)
    compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)


def test_candidates_multi_stage_ring():
    """One CTA per row over 70,001 tokens: the scan runs a ring of staged tiles and the candidate bitmap
    spans every stage."""
    wl = W["mixed_128k"].scaled(name="mixed_ring", B=2, L0=70001, steps=4)
    rows = range(wl.B)
    o_trace, o_ctx = oracle_loop(wl, rows, wl.steps, 10, 20)
    g_trace, g_ctx = gpu_loop(wl, wl.steps, 10, 20, split=1)
    compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)


def test_candidates_full_size_sampled_rows():
    wl = W["zipf_32k"].scaled(steps=8)
    g_trace, g_ctx = gpu_loop(wl, wl.steps, 10, 20, fused=True)
    rows = [0, 21, 42, 63]
    o_trace, o_ctx = oracle_loop(wl, rows, wl.steps, 10, 20)
    checked, copies = compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert checked > 0


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("Wc,D", [(10, 20), (16, 64), (1, 4)])
@pytest.mark.parametrize("name", list(SMALL))
def test_candidates_index_lockstep(name, Wc, D, fused):
    """The index's candidate mode: the kappa-gram chain lists the ends, the index kernel verifies the
    candidates and inserts the appended positions; everything as the rescan's lockstep."""
    wl = SMALL[name]
    rows = range(wl.B)
    o_trace, o_ctx = oracle_loop(wl, rows, wl.steps, Wc, D)
    g_trace, g_ctx = gpu_loop(wl, wl.steps, Wc, D, fused=fused, use_index=True)
    checked, copies = compare(wl, o_trace, g_trace, rows, o_ctx, g_ctx)
    assert checked > 0


def test_candidates_index_kappa_below_n_min_is_rejected():
    import ctypes
    import torch
    from paper_2609_20186_gb300 import binding as bd
    lib = bd.load()
    wl = SMALL["mixed_small"]  # n_min = 2
    B, cap = 2, 64
    idx = bd.NgramIndex(B, cap, 3, 8)
    z = torch.zeros(B, cap, dtype=torch.int32, device="cuda")
    ln = torch.full((B,), 10, dtype=torch.int32, device="cuda")
    idx.build(z, ln)
    p = bd.switchsd_params()
    p.B, p.cap, p.d, p.k, p.n_min, p.n_max, p.kappa = B, cap, 8, 4, 3, 8, 2
    p.index = idx.handle
    p.stream = torch.cuda.current_stream().cuda_stream
    h = torch.zeros(B, 8, dtype=torch.bfloat16, device="cuda")
    o = torch.zeros(B, 4, 4, dtype=torch.int32, device="cuda")
    v = torch.zeros(B, 4, dtype=torch.int32, device="cuda")
    f = torch.zeros(B, dtype=torch.float32, device="cuda")
    assert lib.switchsd_step_candidates(z.data_ptr(), ln.data_ptr(), h.data_ptr(), h.data_ptr(), ctypes.byref(p),
                                        4, 4, o.data_ptr(), v.data_ptr(), v.data_ptr(), v.data_ptr(),
                                        f.data_ptr()) == bd.ERR_SHAPE
    idx.close()
