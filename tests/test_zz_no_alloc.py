"""switchsd_step_static_workspace: switchsd_step for callers that cannot allocate device memory.

Some callers cannot give the library device memory at call time (an inference server that hands all
of the GPU's memory to its own pool at start-up, or a host program without a CUDA allocator).  This
entry point keeps the two-layer probe's scratch in an array compiled into the library.  Here it is
called through the C ABI and compared with switchsd_step given a caller workspace, on two calls in a
row (the second reuses the array the first one left behind), with the two-layer probe and with the
linear one (which needs no scratch).  Around the calls the device's free memory and the caching
allocator's count must not move: the entry point allocates nothing.  The file runs last so that a
failure here leaves every other test already run; it also passes on its own in a fresh process.
"""
import ctypes
import math

import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu

SCORE_TOL = 1e-3


def _problem(seed, B, d, H1, cap, k, mlp):
    rng = np.random.default_rng(seed)
    ctx = rng.integers(0, 5, (B, cap)).astype(np.int32)           # dense repeats: modes vary
    lens = rng.integers(cap // 2, cap, B).astype(np.int32)
    h = synth.bf16_bits_from_f32(rng.standard_normal((B, d)).astype(np.float32))
    if not mlp:
        w = synth.bf16_bits_from_f32((rng.standard_normal(d) / math.sqrt(d)).astype(np.float32))
        return ctx, lens, h, w, None
    W1 = synth.bf16_bits_from_f32((rng.standard_normal((H1, d)) / math.sqrt(d)).astype(np.float32))
    w2 = synth.bf16_bits_from_f32((rng.standard_normal(H1) / math.sqrt(H1)).astype(np.float32))
    b1 = (rng.standard_normal(H1) * 0.1).astype(np.float32)
    return ctx, lens, h, np.concatenate([W1.reshape(-1), w2]), b1


class _Call:
    """Device buffers and parameters of one call, made before any call so that the calls themselves
    run with no allocation by the test either."""

    def __init__(self, prob, B, d, H1, k, mlp, workspace=None):
        import torch
        from paper_2609_20186_gb300 import binding as bd, bf16_tensor

        ctx, lens, h, pw, b1 = prob
        dev = "cuda"
        self.t = [torch.from_numpy(ctx).to(dev), torch.from_numpy(lens).to(dev), bf16_tensor(h, dev),
                  bf16_tensor(pw, dev)]
        self.b1 = torch.from_numpy(b1).to(dev) if b1 is not None else None
        self.out = {"draft": torch.zeros(B, k, dtype=torch.int32, device=dev),
                    "len": torch.zeros(B, dtype=torch.int32, device=dev),
                    "mode": torch.zeros(B, dtype=torch.int32, device=dev),
                    "score": torch.zeros(B, dtype=torch.float32, device=dev),
                    "match_n": torch.zeros(B, dtype=torch.int32, device=dev),
                    "match_end": torch.zeros(B, dtype=torch.int32, device=dev)}
        p = bd.switchsd_params()
        p.B, p.cap, p.d, p.k, p.n_min, p.n_max, p.kappa, p.logit_tau = B, ctx.shape[1], d, k, 2, 6, 0, 0.0
        if mlp:
            p.probe_kind, p.probe_hidden, p.b1, p.b2 = bd.PROBE_MLP, H1, self.b1.data_ptr(), 0.25
        else:
            p.probe_kind, p.probe_hidden, p.b1, p.b2 = bd.PROBE_LINEAR, 0, None, 0.0
        p.split = 0
        if workspace is not None:
            p.workspace, p.workspace_bytes = workspace.data_ptr(), workspace.numel()
        p.out_match_n, p.out_match_end = self.out["match_n"].data_ptr(), self.out["match_end"].data_ptr()
        p.stream = torch.cuda.current_stream().cuda_stream
        self.p = p

    def __call__(self, lib, entry):
        from paper_2609_20186_gb300 import binding as bd

        o = self.out
        code = getattr(lib, entry)(self.t[0].data_ptr(), self.t[1].data_ptr(), self.t[2].data_ptr(),
                                   self.t[3].data_ptr(), ctypes.byref(self.p), o["draft"].data_ptr(),
                                   o["len"].data_ptr(), o["mode"].data_ptr(), o["score"].data_ptr())
        assert code == bd.OK, (entry, code, bd.strerror(code))

    def result(self):
        return {n: t.cpu().numpy() for n, t in self.out.items()}


def _compare(got, ref, B, seed):
    assert np.max(np.abs(got["score"] - ref["score"])) <= SCORE_TOL
    for name in ("mode", "len", "match_n", "match_end"):
        assert np.array_equal(got[name], ref[name]), (seed, name)
    for b in range(B):
        n = int(ref["len"][b])
        assert np.array_equal(got["draft"][b, :n], ref["draft"][b, :n]), (seed, b)
    assert len(set(ref["mode"].tolist())) >= 2        # the comparison exercised the switch


@pytest.mark.parametrize("mlp", [True, False], ids=["two_layer", "linear"])
def test_static_workspace_matches_caller_workspace(mlp):
    import torch
    from paper_2609_20186_gb300 import binding as bd

    lib = bd.load()
    B, d, H1, cap, k = 300, 4096, 200, 640, 8
    ws = torch.empty(max(256, bd.switchsd_workspace_bytes(B, bd.PROBE_MLP if mlp else bd.PROBE_LINEAR, H1, d)),
                     dtype=torch.uint8, device="cuda")
    seeds = (11, 12)                                       # two calls in a row on the shared static array
    refs = [_Call(_problem(s, B, d, H1, cap, k, mlp), B, d, H1, k, mlp, workspace=ws) for s in seeds]
    gots = [_Call(_problem(s, B, d, H1, cap, k, mlp), B, d, H1, k, mlp) for s in seeds]
    for r in refs:
        r(lib, "switchsd_step")
    torch.cuda.synchronize()
    gots[0](lib, "switchsd_step_static_workspace")         # first call: the per-device set-up
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    alloc0 = torch.cuda.memory_allocated()
    for g in gots:                                         # the first problem again, then the second
        g(lib, "switchsd_step_static_workspace")
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0 and torch.cuda.memory_allocated() == alloc0    # nothing was allocated
    for s, r, g in zip(seeds, refs, gots):
        _compare(g.result(), r.result(), B, s)


def test_static_workspace_rejects_requests_beyond_its_size():
    from paper_2609_20186_gb300 import binding as bd

    lib = bd.load()
    p = bd.switchsd_params()
    p.B, p.cap, p.d, p.k, p.n_min, p.n_max = 16385, 64, 4096, 8, 2, 6
    p.probe_kind, p.probe_hidden = bd.PROBE_MLP, 256       # 16 x 16,385 rows x 256 units > 4 Mi floats
    fake = 0x10000
    code = lib.switchsd_step_static_workspace(fake, fake, fake, fake, ctypes.byref(p), fake, fake, fake,
                                              fake)
    assert code == bd.ERR_SHAPE
