"""The fused verification reading the probe's state from the target's [B, k+1, d] output (params
.hidden_rows = k + 1): row a_b of each row, row 0 when nothing was appended.  The code workload runs the
two-layer probe (its rows gathered by a separate kernel before the tensor-core probe kernel), with a
batch of 130 rows spanning two 128-row tiles of that kernel.

The oracle side gathers the same row on the host from its own accepted lengths and runs the oracle step
on the gathered [B, d] states; everything must match as in the other lockstep tests (a wrong row changes
the logit).
"""
import numpy as np
import pytest

import oracle
import synth
from tests import lockstep

pytestmark = pytest.mark.gpu
W = synth.WORKLOADS


def _hidden_all(wl, t):
    """Seeded bf16 bits [B, k+1, d]: a different state for every verification position."""
    rng = np.random.default_rng(7_000_003 * wl.seed + t)
    return synth.bf16_bits_from_f32(rng.standard_normal((wl.B, wl.k + 1, wl.d)).astype(np.float32))


def _oracle(wl, steps, sampled):
    ctx, lens = wl.contexts()
    future, pw, hp = wl.future(), wl.probe_weights(), wl.harness_params()
    acc_prev = np.full(wl.B, -1, np.int32)
    trace = []
    for t in range(steps):
        ha = _hidden_all(wl, t)
        pos = np.where(acc_prev > 0, acc_prev, 0) if t > 0 else np.zeros(wl.B, np.int64)
        h = np.ascontiguousarray(ha[np.arange(wl.B), pos])
        out = oracle.step(ctx, lens, h, pw, k=wl.k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                          logit_tau=wl.logit_tau, probe_kind=wl.probe_kind, probe_hidden=wl.probe_hidden)
        if sampled:
            vd, vl, pp, qq, uu, rs = synth.harness_sampled(hp, t, lens, out["mode"], out["draft"], out["len"],
                                                           future)
            acc, st = oracle.verify_sampled(ctx, lens, vd, vl, pp, uu, rs, q=qq)
        else:
            vd, vl, tg = synth.harness_targets(hp, t, lens, out["mode"], out["draft"], out["len"], future)
            acc, st = oracle.verify(ctx, lens, vd, vl, tg)
        out.update(accept=acc, vstatus=st, lens_after=lens.copy())
        acc_prev = acc.copy()
        trace.append(out)
    return trace, ctx


def _gpu(wl, steps, sampled, use_index=False):
    import torch
    from paper_2609_20186_gb300 import Session, bf16_tensor
    ctx, lens = wl.contexts()
    sess = Session(ctx, lens, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                   logit_tau=wl.logit_tau, probe_kind=wl.probe_kind, probe_hidden=wl.probe_hidden,
                   future=wl.future(), harness=wl.harness_params(), d=wl.d, hidden_rows=wl.k + 1,
                   use_index=use_index)
    trace = []
    for t in range(steps):
        ha = bf16_tensor(_hidden_all(wl, t), sess.device)
        if t == 0:
            sess.step(ha[:, 0].contiguous())
        else:
            (sess.verify_sampled_step if sampled else sess.verify_step)(ha)
            s_ = sess.status.cpu().numpy()
            trace[-1].update(accept=sess.accept.cpu().numpy(), lens_after=sess.lens.cpu().numpy(),
                             vstatus=np.where((s_ == 1) | (s_ == 2), s_, 0))
        out = sess.step_outputs()
        (sess.harness_sampled if sampled else sess.harness)(t)
        if t == steps - 1:
            (sess.verify_sampled if sampled else sess.verify)()
            out.update(accept=sess.accept.cpu().numpy(), vstatus=sess.vstatus.cpu().numpy(),
                       lens_after=sess.lens.cpu().numpy())
        trace.append(out)
    torch.cuda.synchronize()
    return trace, sess.ctx.cpu().numpy()


@pytest.mark.parametrize("sampled", [False, True], ids=["greedy", "sampled"])
@pytest.mark.parametrize("name,B,L0,steps", [("uniform_8k", 8, 3000, 16), ("zipf_32k", 8, 9001, 16),
                                             ("mixed_128k", 4, 20003, 10), ("code_16k", 8, 5000, 12),
                                             ("code_16k", 130, 3001, 6)])
def test_gather_lockstep(name, B, L0, steps, sampled):
    wl = W[name].scaled(name=f"{name}_gather", B=B, L0=L0, steps=steps)
    o_trace, o_ctx = _oracle(wl, steps, sampled)
    g_trace, g_ctx = _gpu(wl, steps, sampled)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, range(wl.B), o_ctx, g_ctx)
    assert stats["checked"] > 0
    # the accepted lengths vary, so rows other than 0 were read
    assert any((t["accept"] > 0).any() for t in o_trace)


@pytest.mark.parametrize("sampled", [False, True], ids=["greedy", "sampled"])
@pytest.mark.parametrize("name,B,L0,steps", [("zipf_32k", 8, 9001, 12), ("code_16k", 8, 5000, 10)])
def test_gather_index_lockstep(name, B, L0, steps, sampled):
    """The same with the incremental index: its kernel verifies, inserts and probes row a_b."""
    wl = W[name].scaled(name=f"{name}_gather_index", B=B, L0=L0, steps=steps)
    o_trace, o_ctx = _oracle(wl, steps, sampled)
    g_trace, g_ctx = _gpu(wl, steps, sampled, use_index=True)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, range(wl.B), o_ctx, g_ctx)
    assert stats["checked"] > 0
