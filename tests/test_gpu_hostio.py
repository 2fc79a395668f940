"""The host-staged entry points and the read ceiling on the GPU, through the C ABI.

switchsd_step_host / switchsd_verify_step_host, and switchsd_plan replays of them, must give exactly
what the device-buffer calls give (same contexts, outputs and accepted lengths, step after step) with
the hidden states taken from host memory and the results delivered to host memory; the plan replays
(the benchmark's e2e path) are also held to the oracle directly.  switchsd_harness_read must fold exactly the words it
is documented to read (checked against numpy)."""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu


def _session(wl, prefetch, use_index=False):
    from paper_2609_20186_gb300 import Session, binding
    ctx, lens = wl.contexts()
    return Session(ctx, lens, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                   logit_tau=wl.logit_tau, probe_kind=wl.probe_kind, probe_hidden=wl.probe_hidden,
                   future=wl.future(), harness=wl.harness_params(), d=wl.d, use_index=use_index,
                   prefetch=(binding.PREFETCH_CONTEXT | binding.PREFETCH_PROBE) if prefetch else 0)


@pytest.mark.parametrize("name", ["zipf_32k", "code_16k"])
@pytest.mark.parametrize("prefetch", [False, True])
def test_host_staged_matches_device_calls(name, prefetch):
    import torch
    from paper_2609_20186_gb300 import bf16_tensor
    wl = synth.WORKLOADS[name].scaled(B=8, L0=6001, steps=10)
    a, b = _session(wl, prefetch), _session(wl, prefetch)
    B, d, k = wl.B, wl.d, wl.k
    dev_h = torch.empty(B, d, dtype=torch.bfloat16, device="cuda")
    host_h = torch.empty(B, d, dtype=torch.int16).pin_memory()
    host_out = torch.empty(B * (k + 3), dtype=torch.int32).pin_memory()
    for t in range(wl.steps):
        hid = wl.hidden(t)
        host_h.copy_(torch.from_numpy(hid.view(np.int16)))
        if t == 0:
            a.step(bf16_tensor(hid, "cuda"), debug=False)
            got = b.step_host(host_h, dev_h, host_out)
        else:
            a.harness(t - 1)
            b.harness(t - 1)
            a.verify_step(bf16_tensor(hid, "cuda"), debug=False)
            got = b.verify_step_host(host_h, dev_h, host_out)
        torch.cuda.synchronize()
        want = a.results.cpu().numpy()
        assert np.array_equal(host_out.numpy(), want), (name, t)
        assert np.array_equal(got["draft"].numpy(), want[3 * B:].reshape(B, k))
        assert np.array_equal(a.lens.cpu().numpy(), b.lens.cpu().numpy()), (name, t)
        assert np.array_equal(a.score.cpu().numpy(), b.score.cpu().numpy()), (name, t)
    assert np.array_equal(a.ctx.cpu().numpy(), b.ctx.cpu().numpy())


def test_host_staged_without_sync_then_stream_sync():
    import torch
    wl = synth.WORKLOADS["uniform_8k"].scaled(B=4, L0=3000, steps=3)
    s = _session(wl, False)
    B, d, k = wl.B, wl.d, wl.k
    dev_h = torch.empty(B, d, dtype=torch.bfloat16, device="cuda")
    host_h = torch.from_numpy(wl.hidden(0).view(np.int16)).pin_memory()
    host_out = torch.full((B * (k + 3),), -7, dtype=torch.int32).pin_memory()
    s.step_host(host_h, dev_h, host_out, synchronize=False)
    torch.cuda.current_stream().synchronize()
    assert np.array_equal(host_out.numpy(), s.results.cpu().numpy())


@pytest.mark.parametrize("prefetch", [0, 1])
@pytest.mark.parametrize("split", [1, 3, 8, 32])
def test_read_ceiling_folds_what_it_reads(split, prefetch):
    import torch
    from paper_2609_20186_gb300 import binding as bd
    lib = bd.load()
    rng = np.random.default_rng(5)
    B, cap, d = 5, 4100, 136
    ctx = rng.integers(-2**31, 2**31 - 1, size=(B, cap), dtype=np.int64).astype(np.int32)
    lens = np.array([0, 1, 4099, 4100, 1234], np.int32)
    hid = rng.integers(0, 2**16, size=(B, d), dtype=np.int64).astype(np.uint16)
    c, ln = torch.from_numpy(ctx).cuda(), torch.from_numpy(lens).cuda()
    h = torch.from_numpy(hid.view(np.int16)).cuda()
    out = torch.full((B * split,), 0x5A5A, dtype=torch.int32, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    assert lib.switchsd_harness_read(c.data_ptr(), ln.data_ptr(), B, cap, h.data_ptr(), d, split, prefetch,
                                     out.data_ptr(), s) == 0
    got = out.cpu().numpy().view(np.uint32).reshape(B, split)
    for b in range(B):
        words = 4 * ((int(lens[b]) + 3) // 4)   # whole 16-byte words covering the first L tokens
        want = np.bitwise_xor.reduce(ctx[b, :words].view(np.uint32)) if words else np.uint32(0)
        want ^= np.bitwise_xor.reduce(hid[b].view(np.uint32))
        assert np.bitwise_xor.reduce(got[b]) == want, b


@pytest.mark.parametrize("use_index", [False, True], ids=["rescan", "index"])
@pytest.mark.parametrize("name", ["zipf_32k", "code_16k"])
@pytest.mark.parametrize("prefetch", [False, True])
def test_plan_replays_match_device_calls(name, prefetch, use_index):
    """Replays alternate between two host hidden buffers and two host result buffers, so the recorded
    copies are retargeted on every replay.  With the index, the recorded graph holds the index kernel."""
    import torch
    from paper_2609_20186_gb300 import bf16_tensor
    wl = synth.WORKLOADS[name].scaled(B=8, L0=6001, steps=12)
    a, b = _session(wl, prefetch, use_index), _session(wl, prefetch, use_index)
    B, d, k = wl.B, wl.d, wl.k
    dev_h = torch.empty(B, d, dtype=torch.bfloat16, device="cuda")
    host_h = [torch.empty(B, d, dtype=torch.int16).pin_memory() for _ in range(2)]
    host_out = [torch.empty(B * (k + 3), dtype=torch.int32).pin_memory() for _ in range(2)]
    first = b.host_plan(host_h[0], dev_h, host_out[0], verify=False)
    plan = b.host_plan(host_h[1], dev_h, host_out[1], verify=True)
    for t in range(wl.steps):
        hid = wl.hidden(t)
        hh, ho = host_h[t % 2], host_out[(t // 2) % 2]
        hh.copy_(torch.from_numpy(hid.view(np.int16)))
        if t == 0:
            a.step(bf16_tensor(hid, "cuda"), debug=False)
            first.run(hh, ho)
            got = first.results()
        else:
            a.harness(t - 1)
            b.harness(t - 1)
            a.verify_step(bf16_tensor(hid, "cuda"), debug=False)
            plan.run(hh, ho)
            got = plan.results()
        torch.cuda.synchronize()
        want = a.results.cpu().numpy()
        assert np.array_equal(ho.numpy(), want), (name, t)
        assert np.array_equal(got["mode"].numpy(), want[:B])
        assert np.array_equal(a.lens.cpu().numpy(), b.lens.cpu().numpy()), (name, t)
        assert np.array_equal(a.score.cpu().numpy(), b.score.cpu().numpy()), (name, t)
    assert np.array_equal(a.ctx.cpu().numpy(), b.ctx.cpu().numpy())
    first.close()
    plan.close()
    plan.close()  # idempotent


@pytest.mark.parametrize("pinned", [False, True])
def test_host_staged_pageable_and_pinned(pinned):
    """Pageable host buffers take the copy engine, pinned ones the copy kernels: same results."""
    import torch
    from paper_2609_20186_gb300 import bf16_tensor
    wl = synth.WORKLOADS["zipf_32k"].scaled(B=4, L0=5003, steps=5)
    a, b = _session(wl, True), _session(wl, True)
    B, d, k = wl.B, wl.d, wl.k
    dev_h = torch.empty(B, d, dtype=torch.bfloat16, device="cuda")
    host_h = torch.empty(B, d, dtype=torch.int16)
    host_out = torch.empty(B * (k + 3), dtype=torch.int32)
    if pinned:
        host_h, host_out = host_h.pin_memory(), host_out.pin_memory()
    for t in range(wl.steps):
        hid = wl.hidden(t)
        host_h.copy_(torch.from_numpy(hid.view(np.int16)))
        if t == 0:
            a.step(bf16_tensor(hid, "cuda"), debug=False)
            b.step_host(host_h, dev_h, host_out)
        else:
            a.harness(t - 1)
            b.harness(t - 1)
            a.verify_step(bf16_tensor(hid, "cuda"), debug=False)
            b.verify_step_host(host_h, dev_h, host_out)
        torch.cuda.synchronize()
        assert np.array_equal(host_out.numpy(), a.results.cpu().numpy()), t
    assert np.array_equal(a.ctx.cpu().numpy(), b.ctx.cpu().numpy())


@pytest.mark.parametrize("use_index", [False, True], ids=["rescan", "index"])
def test_sampled_host_staged_and_plan_match_device_calls(use_index):
    """The sampled fused step from host buffers: switchsd_verify_sampled_step_host on one session, a
    plan of it on another, the device call on a third; all three agree step after step."""
    import torch
    from paper_2609_20186_gb300 import bf16_tensor
    wl = synth.WORKLOADS["zipf_32k"].scaled(B=8, L0=6001, steps=10)
    a, b, c = (_session(wl, True, use_index) for _ in range(3))
    B, d, k = wl.B, wl.d, wl.k
    dev_b = torch.empty(B, d, dtype=torch.bfloat16, device="cuda")
    dev_c = torch.empty(B, d, dtype=torch.bfloat16, device="cuda")
    host_h = [torch.empty(B, d, dtype=torch.int16).pin_memory() for _ in range(2)]
    out_b = torch.empty(B * (k + 3), dtype=torch.int32).pin_memory()
    out_c = torch.empty(B * (k + 3), dtype=torch.int32).pin_memory()
    plan = c.host_plan(host_h[1], dev_c, out_c, verify=False, sampled=True)
    for t in range(wl.steps):
        hid = wl.hidden(t)
        hh = host_h[t % 2]
        hh.copy_(torch.from_numpy(hid.view(np.int16)))
        if t == 0:
            for s_, dh, ho in ((a, None, None), (b, dev_b, out_b), (c, dev_c, out_c)):
                if dh is None:
                    s_.step(bf16_tensor(hid, "cuda"), debug=False)
                else:
                    s_.step_host(hh, dh, ho)
        else:
            for s_ in (a, b, c):
                s_.harness_sampled(t - 1)
            a.verify_sampled_step(bf16_tensor(hid, "cuda"), debug=False)
            b.verify_sampled_step_host(hh, dev_b, out_b)
            plan.run(hh, out_c)
        torch.cuda.synchronize()
        want = a.results.cpu().numpy()
        assert np.array_equal(out_b.numpy(), want), t
        assert np.array_equal(out_c.numpy(), want), t
    assert np.array_equal(a.ctx.cpu().numpy(), b.ctx.cpu().numpy())
    assert np.array_equal(a.ctx.cpu().numpy(), c.ctx.cpu().numpy())
    plan.close()


@pytest.mark.parametrize("name", ["zipf_32k", "code_16k"])
def test_plan_replays_match_the_oracle(name):
    """The e2e path itself -- switchsd_plan replays of switchsd_verify_step_host, the hidden states taken
    from pinned host memory and the results read back into it, prefetch on -- against the oracle step by
    step (lockstep.compare: bit-exact integers, logits within 1e-3)."""
    import torch
    from tests import lockstep
    wl = synth.WORKLOADS[name].scaled(B=8, L0=6001, steps=10)
    s = _session(wl, True)
    B, d, k = wl.B, wl.d, wl.k
    dev_h = torch.empty(B, d, dtype=torch.bfloat16, device="cuda")
    host_h = torch.empty(B, d, dtype=torch.int16).pin_memory()
    host_out = torch.empty(B * (k + 3), dtype=torch.int32).pin_memory()
    first = s.host_plan(host_h, dev_h, host_out, verify=False, debug=True)
    plan = s.host_plan(host_h, dev_h, host_out, verify=True, debug=True)
    g_trace = []
    for t in range(wl.steps):
        host_h.copy_(torch.from_numpy(wl.hidden(t).view(np.int16)))
        if t == 0:
            first.run(host_h, host_out)
        else:
            s.harness(t - 1)
            plan.run(host_h, host_out)
        torch.cuda.synchronize()
        res = host_out.numpy().copy()                   # mode [B], len [B], accept [B], draft [B, k]
        out = s.step_outputs()
        assert np.array_equal(res[:B], out["mode"]) and np.array_equal(res[B:2 * B], out["len"])
        if t > 0:                                       # this replay verified the previous step's draft
            st = out["status"]
            g_trace[-1]["accept"] = res[2 * B:3 * B]
            g_trace[-1]["vstatus"] = np.where((st == 1) | (st == 2), st, 0)
            g_trace[-1]["lens_after"] = s.lens.cpu().numpy()
        out["draft"] = res[3 * B:].reshape(B, k)
        g_trace.append(out)
    s.harness(wl.steps - 1)
    s.verify()
    torch.cuda.synchronize()
    g_trace[-1]["accept"] = s.accept.cpu().numpy()
    g_trace[-1]["vstatus"] = s.vstatus.cpu().numpy()
    g_trace[-1]["lens_after"] = s.lens.cpu().numpy()
    rows = range(B)
    o_trace, o_ctx, _ = lockstep.oracle_trace(wl, rows, wl.steps)
    flips, stats = lockstep.compare(wl, o_trace, g_trace, rows, o_ctx, s.ctx.cpu().numpy())
    assert stats["checked"] > 0 and len(flips) <= 1
    first.close()
    plan.close()
