"""params.prefetch: the context and probe copies start before the preceding kernel finishes.

The serving order is verify_step(t) -> target -> verify_step(t+1), launched back to back with no host
synchronisation, so each call's context copies overlap the target stand-in's kernel while the rows
were written by the call before it (the hidden states are uploaded once, before the chain).  With and without prefetch the whole run must give identical
outputs (the same kernels in the same order, so bit-identical, the probe logits included) and
identical contexts; the no-prefetch path is itself held to the oracle by test_gpu_parity.py.
"""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS
KEYS = ("draft", "len", "mode", "score", "match_n", "match_end", "status", "accept")


def _chain(wl, prefetch: int, steps: int, record_every: int, len_bound: int = 0, use_index: bool = False):
    import torch
    from paper_2609_20186_gb300 import Session, bf16_tensor

    ctx, lens = wl.contexts()
    sess = Session(ctx, lens, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max,
                   kappa=wl.kappa, logit_tau=wl.logit_tau, probe_kind=wl.probe_kind,
                   probe_hidden=wl.probe_hidden, future=wl.future(), harness=wl.harness_params(),
                   d=wl.d, prefetch=prefetch, len_bound=len_bound, use_index=use_index)
    hidden = bf16_tensor(np.stack([wl.hidden(t) for t in range(steps)]), sess.device)
    torch.cuda.synchronize()
    rec = {}
    for t in range(steps):
        if t == 0:
            sess.step(hidden[0])
        else:
            sess.verify_step(hidden[t])
        if t % record_every == 0:  # recorded on the device; the other steps chain kernel to kernel
            rec[t] = {key: getattr(sess, key).clone() for key in KEYS}
        sess.harness(t)
    sess.verify()
    torch.cuda.synchronize()
    out = {t: {key: v.cpu().numpy() for key, v in r.items()} for t, r in rec.items()}
    return out, sess.ctx.cpu().numpy(), sess.lens.cpu().numpy()


@pytest.mark.parametrize("name,steps", [("zipf_32k", 40), ("code_16k", 24), ("mixed_128k", 24),
                                        ("uniform_8k", 40)])
def test_prefetch_matches_back_to_back(name, steps):
    wl = W[name].scaled(steps=steps)
    from paper_2609_20186_gb300 import binding as bd
    a, a_ctx, a_lens = _chain(wl, 0, steps, record_every=3)
    b, b_ctx, b_lens = _chain(wl, bd.PREFETCH_CONTEXT | bd.PREFETCH_PROBE, steps, record_every=3)
    assert np.array_equal(a_lens, b_lens)
    assert (a_lens > wl.L0).all()  # every row grew: the chain really appended
    assert np.array_equal(a_ctx, b_ctx)
    for t in a:
        for key in KEYS:
            if key == "draft":
                for r in range(wl.B):
                    n = int(a[t]["len"][r])
                    assert np.array_equal(a[t]["draft"][r, :n], b[t]["draft"][r, :n]), (t, r)
            else:
                assert np.array_equal(a[t][key], b[t][key]), (name, t, key)


@pytest.mark.parametrize("name,steps", [("zipf_32k", 40), ("mixed_128k", 24), ("code_16k", 16)])
def test_prefetch_matches_back_to_back_index(name, steps):
    """The same with the incremental index: its kernel reads the row's length and tail and computes the
    linear probe before the wait."""
    wl = W[name].scaled(steps=steps)
    from paper_2609_20186_gb300 import binding as bd
    a, a_ctx, a_lens = _chain(wl, 0, steps, record_every=3, use_index=True)
    b, b_ctx, b_lens = _chain(wl, bd.PREFETCH_CONTEXT | bd.PREFETCH_PROBE, steps, record_every=3, use_index=True)
    assert np.array_equal(a_lens, b_lens) and (a_lens > wl.L0).all()
    assert np.array_equal(a_ctx, b_ctx)
    for t in a:
        for key in KEYS:
            if key != "draft":
                assert np.array_equal(a[t][key], b[t][key]), (name, t, key)


@pytest.mark.parametrize("name,steps", [("zipf_32k", 40), ("uniform_8k", 40), ("mixed_128k", 24),
                                        ("code_16k", 16)])
def test_length_bound_matches(name, steps):
    """params.len_bound = cap splits every row's ends on cap (copies before the length read): the run
    must be bit-identical to the plain one, rows far from full (uniform_8k) included."""
    from paper_2609_20186_gb300 import binding as bd
    wl = W[name].scaled(steps=steps)
    cap = wl.contexts()[0].shape[1]
    a, a_ctx, a_lens = _chain(wl, 0, steps, record_every=4)
    b, b_ctx, b_lens = _chain(wl, bd.PREFETCH_CONTEXT | bd.PREFETCH_PROBE, steps, record_every=4, len_bound=cap)
    assert np.array_equal(a_lens, b_lens) and np.array_equal(a_ctx, b_ctx)
    for t in a:
        for key in KEYS:
            if key != "draft":
                assert np.array_equal(a[t][key], b[t][key]), (name, t, key)


def test_length_above_bound_is_bad_length():
    import torch
    from paper_2609_20186_gb300 import Session, bf16_tensor
    wl = W["uniform_8k"].scaled(B=6, L0=2000, steps=2)
    ctx, lens = wl.contexts()
    lens[:] = [1990, 2000, 2001, 2005, 1, 1500]
    sess = Session(ctx, lens, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                   logit_tau=wl.logit_tau, d=wl.d, len_bound=2000)
    sess.step(bf16_tensor(wl.hidden(0), sess.device))
    torch.cuda.synchronize()
    st = sess.status.cpu().numpy()
    assert st.tolist() == [0, 0, 2, 2, 0, 0]
    ref = Session(ctx, lens, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                  logit_tau=wl.logit_tau, d=wl.d)
    ref.step(bf16_tensor(wl.hidden(0), ref.device))
    torch.cuda.synchronize()
    for r in (0, 1, 4, 5):                         # rows within the bound: the plain step's results
        assert sess.mode.cpu()[r] == ref.mode.cpu()[r] and sess.match_end.cpu()[r] == ref.match_end.cpu()[r]
