"""Device-resident state of one batch of sequences and the controller loop around it.

A ``Session`` owns the context buffer, lengths and every output buffer on one CUDA device, and runs
one decoding iteration as three library calls on one stream:

    switchsd_step            (controller: search, probe, switch, copy draft)
    switchsd_harness_target  (stand-in for the neural drafter and the target forward)
    switchsd_verify          (controller: greedy verification and append)

Inputs arrive as numpy arrays (token ids int32, bf16 values as uint16 bit patterns) and are copied to
the device once; nothing here computes any part of the controller.
"""
from __future__ import annotations

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
                 probe_kind: int = bd.PROBE_LINEAR, probe_hidden: int = 0, labels=None,
                 harness: dict | None = None, split: int = 0, device="cuda", stream=None):
        self.device = torch.device(device)
        self.B, self.cap = ctx.shape
        self.k = k
        self.cfg = dict(k=k, n_min=n_min, n_max=n_max, kappa=kappa, logit_tau=logit_tau,
                        probe_kind=probe_kind, probe_hidden=probe_hidden, split=split)
        dev = self.device
        self.ctx = torch.from_numpy(np.ascontiguousarray(ctx, np.int32)).to(dev)
        self.lens = torch.from_numpy(np.ascontiguousarray(lens, np.int32)).to(dev)
        self.probe_w = bf16_tensor(probe_w_bits.reshape(-1), dev)
        B = self.B
        i32 = dict(dtype=torch.int32, device=dev)
        self.draft = torch.zeros(B, k, **i32)
        self.len = torch.zeros(B, **i32)
        self.mode = torch.zeros(B, **i32)
        self.score = torch.zeros(B, dtype=torch.float32, device=dev)
        self.match_n = torch.zeros(B, **i32)
        self.match_end = torch.zeros(B, **i32)
        self.status = torch.zeros(B, **i32)
        self.vdraft = torch.zeros(B, k, **i32)
        self.vlen = torch.zeros(B, **i32)
        self.target = torch.zeros(B, k + 1, **i32)
        self.accept = torch.zeros(B, **i32)
        self.vstatus = torch.zeros(B, **i32)
        lab = labels if labels is not None else np.zeros((B, 0), np.uint8)
        self.labels = torch.from_numpy(np.ascontiguousarray(lab, np.uint8)).to(dev)
        self.harness_cfg = harness
        self.stream = stream

    # --- the three calls ---------------------------------------------------------------------
    def step(self, hidden: torch.Tensor, debug: bool = True) -> None:
        bd.switchsd_step(self.ctx, self.lens, hidden, self.probe_w, self.draft, self.len, self.mode,
                         self.score, out_match_n=self.match_n if debug else None,
                         out_match_end=self.match_end if debug else None,
                         status=self.status if debug else None, stream=self.stream, **self.cfg)

    def harness(self, t: int) -> None:
        h = self.harness_cfg
        bd.switchsd_harness_target(self.lens, self.mode, self.draft, self.len, self.labels,
                                   self.vdraft, self.vlen, self.target, seed=h["seed"], V=h["V"],
                                   L0=h["L0"], agree_cap=h["agree_cap"], thr_in=h["thr_in"],
                                   thr_out=h["thr_out"], step=t, stream=self.stream)

    def verify(self, debug: bool = True) -> None:
        bd.switchsd_verify(self.vdraft, self.target, self.accept, draft_len=self.vlen,
                           ctx_tokens=self.ctx, ctx_lens=self.lens,
                           status=self.vstatus if debug else None, stream=self.stream)

    def iterate(self, hidden: torch.Tensor, t: int, debug: bool = True) -> None:
        self.step(hidden, debug)
        self.harness(t)
        self.verify(debug)

    # --- host views ------------------------------------------------------------------------------
    def step_outputs(self) -> dict:
        return {"draft": self.draft.cpu().numpy(), "len": self.len.cpu().numpy(),
                "mode": self.mode.cpu().numpy(), "score": self.score.cpu().numpy(),
                "match_n": self.match_n.cpu().numpy(), "match_end": self.match_end.cpu().numpy(),
                "status": self.status.cpu().numpy()}
