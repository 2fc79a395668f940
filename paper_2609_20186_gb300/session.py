"""Device-resident state of one batch of sequences and the controller loop around it.

A ``Session`` owns the context buffer, lengths and every output buffer on one CUDA device, and runs
one decoding iteration as three library calls on one stream:

    switchsd_step            (controller: search, probe, switch, copy draft)
    switchsd_harness_target  (stand-in for the neural drafter and the target forward)
    switchsd_verify          (controller: greedy verification and append)

For inputs that arrive in host memory and decisions read back on the host, ``step_host`` and
``verify_step_host`` make the host-to-device copy, the step and one device-to-host copy of every
per-row result in a single library call (switchsd_step_host / switchsd_verify_step_host).

Inputs arrive as numpy arrays (token ids int32, bf16 values as uint16 bit patterns) and are copied to
the device once.  The buffers are checked once at construction; each call then passes the cached
argument list straight to the C function, so the per-call host cost is one foreign call.  Nothing
here computes any part of the controller.
"""
from __future__ import annotations

import ctypes

import numpy as np
import torch

from . import binding as bd


def bf16_tensor(bits: np.ndarray, device) -> torch.Tensor:
    """uint16 bf16 bit patterns (numpy) -> torch.bfloat16 tensor on ``device``."""
    b = np.ascontiguousarray(bits, np.uint16).view(np.int16)
    return torch.from_numpy(b).view(torch.bfloat16).to(device)


class Session:
    def __init__(self, ctx: np.ndarray, lens: np.ndarray, probe_w_bits: np.ndarray, *, k: int,
                 n_min: int, n_max: int, kappa: int = 0, logit_tau: float = 0.0,
                 probe_kind: int = bd.PROBE_LINEAR, probe_hidden: int = 0, future=None,
                 harness: dict | None = None, split: int = 0, d: int | None = None,
                 use_index: bool = False, device="cuda", stream: torch.cuda.Stream | None = None,
                 prefetch: int = 0, hidden_rows: int = 0, len_bound: int = 0, counters: bool = False):
        self.lib = bd.load()
        self.hidden_rows = int(hidden_rows)
        self.device = torch.device(device)
        if self.device.type == "cuda" and self.device.index is None:
            self.device = torch.device("cuda", torch.cuda.current_device())
        self.B, self.cap = ctx.shape
        self.k = k
        dev = self.device
        self.ctx = torch.from_numpy(np.ascontiguousarray(ctx, np.int32)).to(dev)
        self.lens = torch.from_numpy(np.ascontiguousarray(lens, np.int32)).to(dev)
        self.probe_w = bf16_tensor(probe_w_bits.reshape(-1), dev)
        B = self.B
        i32 = dict(dtype=torch.int32, device=dev)
        # The per-step results a caller reads back live in one buffer, so one copy brings them to the
        # host (outputs_to): mode [B], draft length [B], accepted length [B], draft [B, k].
        self.results = torch.zeros(B * (k + 3), **i32)
        self.mode = self.results[0:B]
        self.len = self.results[B:2 * B]
        self.accept = self.results[2 * B:3 * B]
        self.draft = self.results[3 * B:].view(B, k)
        self.score = torch.zeros(B, dtype=torch.float32, device=dev)
        self.match_n = torch.zeros(B, **i32)
        self.match_end = torch.zeros(B, **i32)
        self.status = torch.zeros(B, **i32)
        self.vdraft = torch.zeros(B, k, **i32)
        self.vlen = torch.zeros(B, **i32)
        self.target = torch.zeros(B, k + 1, **i32)
        self.vstatus = torch.zeros(B, **i32)
        # per-mode tallies (switchsd_params.counters; uint64 on the device, int64 here), when asked for
        self.counters = torch.zeros(bd.COUNTERS, dtype=torch.int64, device=dev) if counters else None
        fut = future if future is not None else np.zeros((B, 0), np.int32)
        self.future = torch.from_numpy(np.ascontiguousarray(fut, np.int32)).to(dev)
        self.stream = stream
        sp = (stream or torch.cuda.current_stream(dev)).cuda_stream
        if d is None:
            d = probe_w_bits.size if probe_kind == bd.PROBE_LINEAR else None
        self.d = d

        # workspace of the two-layer probe (none for the linear probe)
        probe = bd.switchsd_params()
        probe.B, probe.d, probe.probe_kind, probe.probe_hidden = B, d or 0, probe_kind, probe_hidden
        probe.hidden_rows = int(hidden_rows)  # k + 1 with the two-layer probe: room for the gathered rows
        ws_bytes = int(self.lib.switchsd_workspace_bytes(ctypes.byref(probe)))
        self.workspace = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=dev)

        # incremental n-gram index (optional): built once from the initial contexts, then kept current
        # by the verification calls
        self.index = None
        if use_index:
            self.index = bd.NgramIndex(B, self.cap, n_min, n_max)
            self.index.build(self.ctx, self.lens, stream=stream)

        # switchsd_step: two cached parameter blocks (with and without the debug outputs)
        def params(debug: bool):
            p = bd.switchsd_params()
            p.B, p.cap, p.d, p.k = B, self.cap, d or 0, k
            p.n_min, p.n_max, p.kappa, p.logit_tau = n_min, n_max, kappa, logit_tau
            p.probe_kind, p.probe_hidden, p.b1, p.b2, p.split = probe_kind, probe_hidden, None, 0.0, split
            p.workspace, p.workspace_bytes = self.workspace.data_ptr(), self.workspace.numel()
            p.index = self.index.handle if self.index is not None else None
            p.out_match_n = self.match_n.data_ptr() if debug else None
            p.out_match_end = self.match_end.data_ptr() if debug else None
            p.status = self.status.data_ptr() if debug else None
            p.stream = sp
            p.prefetch = int(prefetch)
            p.hidden_rows = int(hidden_rows)  # k + 1: verify_step reads row a_b of a [B, k+1, d] hidden
            p.len_bound = int(len_bound)      # > 0: split on this bound, copies before the length read
            p.counters = self.counters.data_ptr() if self.counters is not None else None
            return p
        self._p_dbg, self._p_fast = params(True), params(False)
        self._step_head = (self.ctx.data_ptr(), self.lens.data_ptr())
        self._step_tail = (self.probe_w.data_ptr(),)
        self._step_outs = (self.draft.data_ptr(), self.len.data_ptr(), self.mode.data_ptr(),
                           self.score.data_ptr())

        def vparams(debug: bool):
            vp = bd.switchsd_verify_params()
            vp.B, vp.cap, vp.k = B, self.cap, k
            vp.draft_len = self.vlen.data_ptr()
            vp.ctx_tokens = self.ctx.data_ptr()
            vp.ctx_lens = self.lens.data_ptr()
            vp.status = self.vstatus.data_ptr() if debug else None
            vp.index = self.index.handle if self.index is not None else None
            vp.stream = sp
            return vp
        self._vp_dbg, self._vp_fast = vparams(True), vparams(False)
        self._verify_args = (self.vdraft.data_ptr(), self.target.data_ptr(), self.accept.data_ptr())
        self._vs_head = (self.vdraft.data_ptr(), self.target.data_ptr(), self.vlen.data_ptr(),
                         self.accept.data_ptr())

        self._hp = None
        if harness is not None:
            hp = bd.switchsd_harness_params()
            hp.B, hp.k, hp.V, hp.L0 = B, k, harness["V"], harness["L0"]
            hp.n_future = self.future.shape[1]
            hp.gamma, hp.step = harness["gamma"], 0
            hp.seed, hp.thr_neural = harness["seed"], harness["thr_neural"]
            hp.p_hit = harness.get("p_hit", 0.9)
            hp.p_miss = harness.get("p_miss", 0.05)
            hp.q_neural = harness.get("q_neural", 0.8)
            hp.stream = sp
            self._hp = hp
            self._harness_args = (self.lens.data_ptr(), self.mode.data_ptr(), self.draft.data_ptr(),
                                  self.len.data_ptr(),
                                  self.future.data_ptr() if self.future.numel() else None,
                                  self.vdraft.data_ptr(), self.vlen.data_ptr(),
                                  self.target.data_ptr())
        # sampled verification (T > 0): target / drafter probabilities and uniforms of the last draft;
        # self.target then holds the residual and bonus draws
        f32 = dict(dtype=torch.float32, device=dev)
        self.vp = torch.zeros(B, k, **f32)
        self.vq = torch.ones(B, k, **f32)
        self.vu = torch.zeros(B, k, **f32)
        self._io = bd.switchsd_host_io()  # host_io of the host-staged calls, refilled per call

    # --- the three calls ---------------------------------------------------------------------
    def _check_hidden(self, hidden: torch.Tensor, rows: int = 1) -> None:
        """hidden: bf16 [B, d], or [B, rows, d] when rows > 1 (the fused verification's gather)."""
        shape_ok = hidden.shape[0] == self.B and (
            (rows <= 1 and hidden.dim() == 2) or (rows > 1 and hidden.dim() == 3 and hidden.shape[1] == rows))
        if (hidden.dtype != torch.bfloat16 or hidden.device != self.device
                or not hidden.is_contiguous() or not shape_ok
                or (self.d is not None and hidden.shape[-1] != self.d)):
            raise ValueError("hidden must be a contiguous bf16 [B, d] (or [B, k+1, d]) tensor on the session device")
        if self.d is None:
            self._p_dbg.d = self._p_fast.d = hidden.shape[1]
            self.d = hidden.shape[1]

    def step(self, hidden: torch.Tensor, debug: bool = True) -> None:
        """switchsd_step (no verification): hidden is [B, d] whatever hidden_rows is."""
        self._check_hidden(hidden)
        p = self._p_dbg if debug else self._p_fast
        rows, p.hidden_rows = p.hidden_rows, 0
        code = self.lib.switchsd_step(*self._step_head, hidden.data_ptr(), *self._step_tail,
                                      ctypes.byref(p), *self._step_outs)
        p.hidden_rows = rows
        if code != bd.OK:
            raise RuntimeError(f"switchsd_step failed: {code} ({bd.strerror(code)})")

    def verify_step(self, hidden: torch.Tensor, debug: bool = True) -> None:
        """Verification of the last harness draft (vdraft / target / vlen) and the next step, fused.
        With hidden_rows = k + 1, hidden is the target's [B, k+1, d] output and row a_b is probed."""
        self._check_hidden(hidden, self.hidden_rows)
        p = self._p_dbg if debug else self._p_fast
        code = self.lib.switchsd_verify_step(*self._vs_head, self.ctx.data_ptr(), self.lens.data_ptr(),
                                             hidden.data_ptr(), *self._step_tail, ctypes.byref(p),
                                             *self._step_outs)
        if code != bd.OK:
            raise RuntimeError(f"switchsd_verify_step failed: {code} ({bd.strerror(code)})")

    def harness(self, t: int) -> None:
        self._hp.step = t
        code = self.lib.switchsd_harness_target(*self._harness_args, ctypes.byref(self._hp))
        if code != bd.OK:
            raise RuntimeError(f"switchsd_harness_target failed: {code} ({bd.strerror(code)})")

    def verify(self, debug: bool = True) -> None:
        code = self.lib.switchsd_verify(*self._verify_args,
                                        ctypes.byref(self._vp_dbg if debug else self._vp_fast))
        if code != bd.OK:
            raise RuntimeError(f"switchsd_verify failed: {code} ({bd.strerror(code)})")

    def verify_sampled_step(self, hidden: torch.Tensor, debug: bool = True) -> None:
        """Sampled verification (T > 0) of the last sampled-harness draft and the next step, fused."""
        self._check_hidden(hidden, self.hidden_rows)
        p = self._p_dbg if debug else self._p_fast
        code = self.lib.switchsd_verify_sampled_step(
            self.vdraft.data_ptr(), self.vp.data_ptr(), self.vq.data_ptr(), self.vu.data_ptr(),
            self.target.data_ptr(), self.vlen.data_ptr(), self.accept.data_ptr(), self.ctx.data_ptr(),
            self.lens.data_ptr(), hidden.data_ptr(), *self._step_tail, ctypes.byref(p), *self._step_outs)
        if code != bd.OK:
            raise RuntimeError(f"switchsd_verify_sampled_step failed: {code} ({bd.strerror(code)})")

    def harness_sampled(self, t: int) -> None:
        """The target stand-in at T > 0: vdraft / vlen, vp / vq / vu and the resample tokens in target."""
        self._hp.step = t
        a = self._harness_args
        code = self.lib.switchsd_harness_sampled(*a[:7], self.vp.data_ptr(), self.vq.data_ptr(),
                                                 self.vu.data_ptr(), a[7], ctypes.byref(self._hp))
        if code != bd.OK:
            raise RuntimeError(f"switchsd_harness_sampled failed: {code} ({bd.strerror(code)})")

    def verify_sampled(self, debug: bool = True) -> None:
        """switchsd_verify_sampled of the last harness draft (no index)."""
        vp = self._vp_dbg if debug else self._vp_fast
        code = self.lib.switchsd_verify_sampled(self.vdraft.data_ptr(), self.vp.data_ptr(), self.vq.data_ptr(),
                                                self.vu.data_ptr(), self.target.data_ptr(), self.accept.data_ptr(),
                                                ctypes.byref(vp))
        if code != bd.OK:
            raise RuntimeError(f"switchsd_verify_sampled failed: {code} ({bd.strerror(code)})")

    def iterate(self, hidden: torch.Tensor, t: int, debug: bool = True) -> None:
        self.step(hidden, debug)
        self.harness(t)
        self.verify(debug)

    def outputs_to(self, host: torch.Tensor) -> dict:
        """One asynchronous device-to-host copy of mode, draft length, accepted length and draft into
        `host` (pinned int32 [B * (k + 3)]); returns views of it.  Synchronise the stream before use."""
        host.copy_(self.results, non_blocking=True)
        return self._host_views(host)

    # --- host-staged calls (inputs and results in host memory) ------------------------------------
    def _host_io(self, hidden_host: torch.Tensor, hidden: torch.Tensor, results_host: torch.Tensor,
                 synchronize: bool):
        if (hidden_host.device.type != "cpu" or not hidden_host.is_contiguous()
                or hidden_host.numel() * hidden_host.element_size() != hidden.numel() * hidden.element_size()):
            raise ValueError("hidden_host must be a contiguous host tensor with the bytes of hidden")
        if (results_host.device.type != "cpu" or results_host.dtype != torch.int32
                or not results_host.is_contiguous() or results_host.numel() != self.results.numel()):
            raise ValueError("results_host must be a contiguous host int32 tensor of B * (k + 3) entries")
        io = self._io
        io.in_host, io.in_dev = hidden_host.data_ptr(), hidden.data_ptr()
        io.in_bytes = hidden.numel() * hidden.element_size()
        io.out_dev, io.out_host = self.results.data_ptr(), results_host.data_ptr()
        io.out_bytes = self.results.numel() * 4
        io.synchronize = int(bool(synchronize))
        return io

    def _host_views(self, host: torch.Tensor) -> dict:
        B, k = self.B, self.k
        return {"mode": host[0:B], "len": host[B:2 * B], "accept": host[2 * B:3 * B],
                "draft": host[3 * B:].view(B, k)}

    def step_host(self, hidden_host: torch.Tensor, hidden: torch.Tensor, results_host: torch.Tensor,
                  debug: bool = False, synchronize: bool = True) -> dict:
        """switchsd_step_host: the bytes of hidden_host (host, pinned) are copied into `hidden` (the
        device [B, d] buffer the step reads), the step runs, and mode / draft length / accepted length /
        draft come back into results_host (host int32 [B * (k + 3)], pinned) in one copy -- one library
        call.  With synchronize the call returns when results_host is filled.  Returns its views."""
        self._check_hidden(hidden)
        io = self._host_io(hidden_host, hidden, results_host, synchronize)
        p = self._p_dbg if debug else self._p_fast
        rows, p.hidden_rows = p.hidden_rows, 0
        code = self.lib.switchsd_step_host(ctypes.byref(io), *self._step_head, hidden.data_ptr(), *self._step_tail,
                                           ctypes.byref(p), *self._step_outs)
        p.hidden_rows = rows
        if code != bd.OK:
            raise RuntimeError(f"switchsd_step_host failed: {code} ({bd.strerror(code)})")
        return self._host_views(results_host)

    def verify_step_host(self, hidden_host: torch.Tensor, hidden: torch.Tensor, results_host: torch.Tensor,
                         debug: bool = False, synchronize: bool = True) -> dict:
        """switchsd_verify_step_host: verify_step between the copies of step_host, in one library call."""
        self._check_hidden(hidden, self.hidden_rows)
        io = self._host_io(hidden_host, hidden, results_host, synchronize)
        p = self._p_dbg if debug else self._p_fast
        code = self.lib.switchsd_verify_step_host(ctypes.byref(io), *self._vs_head, self.ctx.data_ptr(),
                                                  self.lens.data_ptr(), hidden.data_ptr(), *self._step_tail,
                                                  ctypes.byref(p), *self._step_outs)
        if code != bd.OK:
            raise RuntimeError(f"switchsd_verify_step_host failed: {code} ({bd.strerror(code)})")
        return self._host_views(results_host)

    def host_plan(self, hidden_host: torch.Tensor, hidden: torch.Tensor, results_host: torch.Tensor,
                  verify: bool = True, debug: bool = False, sampled: bool = False) -> "HostPlan":
        """switchsd_plan_create: what verify_step_host (verify=True), verify_sampled_step_host
        (sampled=True: the sampled verification of vdraft with vp / vq / vu and the resample tokens in
        target) or step_host does with these buffers, recorded once as a CUDA graph; HostPlan.run
        replays it with this step's host buffers."""
        self._check_hidden(hidden, self.hidden_rows if (verify or sampled) else 1)
        io = bd.switchsd_host_io.from_buffer_copy(self._host_io(hidden_host, hidden, results_host, False))
        p = bd.switchsd_params.from_buffer_copy(self._p_dbg if debug else self._p_fast)
        if not (verify or sampled):
            p.hidden_rows = 0
        a = bd.switchsd_step_args()
        if verify or sampled:
            a.draft, a.target_argmax, a.draft_len, a.out_accept = self._vs_head
        if sampled:
            a.p_draft, a.q_draft, a.u = self.vp.data_ptr(), self.vq.data_ptr(), self.vu.data_ptr()
        a.ctx_tokens, a.ctx_lens = self._step_head
        a.hidden, a.probe_w = hidden.data_ptr(), self.probe_w.data_ptr()
        a.params = ctypes.pointer(p)
        a.out_draft, a.out_len, a.out_mode, a.out_score = self._step_outs
        h = ctypes.c_void_p()
        code = self.lib.switchsd_plan_create(ctypes.byref(a), ctypes.byref(io), ctypes.byref(h))
        if code != bd.OK:
            raise RuntimeError(f"switchsd_plan_create failed: {code} ({bd.strerror(code)})")
        return HostPlan(self, h, io.in_bytes, (hidden_host, hidden, results_host))

    def verify_sampled_step_host(self, hidden_host: torch.Tensor, hidden: torch.Tensor,
                                 results_host: torch.Tensor, debug: bool = False, synchronize: bool = True) -> dict:
        """switchsd_verify_sampled_step_host: verify_sampled_step between the copies of step_host."""
        self._check_hidden(hidden, self.hidden_rows)
        io = self._host_io(hidden_host, hidden, results_host, synchronize)
        p = self._p_dbg if debug else self._p_fast
        code = self.lib.switchsd_verify_sampled_step_host(
            ctypes.byref(io), self.vdraft.data_ptr(), self.vp.data_ptr(), self.vq.data_ptr(), self.vu.data_ptr(),
            self.target.data_ptr(), self.vlen.data_ptr(), self.accept.data_ptr(), self.ctx.data_ptr(),
            self.lens.data_ptr(), hidden.data_ptr(), *self._step_tail, ctypes.byref(p), *self._step_outs)
        if code != bd.OK:
            raise RuntimeError(f"switchsd_verify_sampled_step_host failed: {code} ({bd.strerror(code)})")
        return self._host_views(results_host)

    # --- host views ------------------------------------------------------------------------------
    def step_outputs(self) -> dict:
        return {"draft": self.draft.cpu().numpy(), "len": self.len.cpu().numpy(),
                "mode": self.mode.cpu().numpy(), "score": self.score.cpu().numpy(),
                "match_n": self.match_n.cpu().numpy(), "match_end": self.match_end.cpu().numpy(),
                "status": self.status.cpu().numpy()}


class HostPlan:
    """A recorded host-staged step (switchsd_plan) of a Session.  run() replays it: H2D of this step's
    hidden states from host memory, the step, one D2H of the results, and (by default) a host wait."""

    def __init__(self, session: Session, handle: ctypes.c_void_p, in_bytes: int, keep):
        self.session, self.handle, self.in_bytes = session, handle, in_bytes
        self._keep = keep  # the buffers recorded at creation stay alive with the plan

    def run(self, hidden_host: torch.Tensor | None = None, results_host: torch.Tensor | None = None,
            synchronize: bool = True) -> None:
        """hidden_host: host tensor with the hidden states' bytes (pinned; None: the last one);
        results_host: pinned host int32 [B * (k + 3)] (None: the last one).  After a synchronised run
        (or a stream synchronisation) ``results()`` holds this replay's results."""
        if self.handle is None:
            raise RuntimeError("the plan was closed")
        hp = rp = None
        if hidden_host is not None:
            if hidden_host.device.type != "cpu" or hidden_host.numel() * hidden_host.element_size() != self.in_bytes:
                raise ValueError("hidden_host must be a host tensor with the bytes of the recorded hidden states")
            hp = hidden_host.data_ptr()
        if results_host is not None:
            if results_host.device.type != "cpu" or results_host.numel() != self.session.results.numel():
                raise ValueError("results_host must be a host int32 tensor of B * (k + 3) entries")
            rp = results_host.data_ptr()
            self._keep = self._keep[:2] + (results_host,)
        code = self.session.lib.switchsd_plan_run(self.handle, hp, rp, int(bool(synchronize)))
        if code != bd.OK:
            raise RuntimeError(f"switchsd_plan_run failed: {code} ({bd.strerror(code)})")

    def results(self) -> dict:
        """Views (mode, len, accept, draft) of the host buffer the last replay wrote."""
        return self.session._host_views(self._keep[2])

    def close(self) -> None:
        if self.handle is not None:
            self.session.lib.switchsd_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
