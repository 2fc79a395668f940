"""ctypes binding of libswitchsd.so: the C ABI of include/switchsd.h and include/switchsd_harness.h.

Argument marshalling only: every function takes torch CUDA tensors, checks dtype / device / layout,
and passes raw device pointers and the current CUDA stream to the library.  All computation runs in
the library's kernels.  If the library is missing the first call raises; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

MODE_NO_REP, MODE_COPY, MODE_REP_NO_COPY = 0, 1, 2
PROBE_LINEAR, PROBE_MLP = 0, 1
OK, ERR_ARG, ERR_SHAPE, ERR_CUDA = 0, -1, -2, -3
ROW_OK, ROW_CAPACITY, ROW_BAD_LEN, ROW_TIMEOUT = 0, 1, 2, 3
NMAX, KMAX = 32, 64
ABI_VERSION = 8  # SWITCHSD_ABI_VERSION this binding marshals for
PREFETCH_CONTEXT, PREFETCH_PROBE = 1, 2  # switchsd_params.prefetch bits

_c_i32p = ctypes.c_void_p


class switchsd_params(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("cap", ctypes.c_int32), ("d", ctypes.c_int32), ("k", ctypes.c_int32),
        ("n_min", ctypes.c_int32), ("n_max", ctypes.c_int32), ("kappa", ctypes.c_int32),
        ("logit_tau", ctypes.c_float),
        ("probe_kind", ctypes.c_int32), ("probe_hidden", ctypes.c_int32),
        ("b1", ctypes.c_void_p), ("b2", ctypes.c_float),
        ("split", ctypes.c_int32),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t),
        ("index", ctypes.c_void_p),
        ("out_match_n", ctypes.c_void_p), ("out_match_end", ctypes.c_void_p),
        ("status", ctypes.c_void_p),
        ("stream", ctypes.c_void_p),
        ("prefetch", ctypes.c_int32),
        ("hidden_rows", ctypes.c_int32),
        ("len_bound", ctypes.c_int32),
        ("counters", ctypes.c_void_p),
    ]


# slots of switchsd_params.counters (include/switchsd.h)
CTR_STEPS, CTR_COPY_DRAFTS, CTR_COPY_ACCEPTED, CTR_NEURAL_DRAFTS, CTR_NEURAL_ACCEPTED, COUNTERS = 0, 3, 4, 5, 6, 7


class switchsd_verify_params(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("cap", ctypes.c_int32), ("k", ctypes.c_int32),
        ("draft_len", ctypes.c_void_p), ("ctx_tokens", ctypes.c_void_p),
        ("ctx_lens", ctypes.c_void_p), ("status", ctypes.c_void_p), ("index", ctypes.c_void_p),
        ("stream", ctypes.c_void_p),
    ]


class switchsd_candidates_verify_params(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("cap", ctypes.c_int32), ("W", ctypes.c_int32), ("D", ctypes.c_int32),
        ("cand_len", ctypes.c_void_p), ("ncand", ctypes.c_void_p), ("ctx_tokens", ctypes.c_void_p),
        ("ctx_lens", ctypes.c_void_p), ("status", ctypes.c_void_p), ("stream", ctypes.c_void_p),
        ("index", ctypes.c_void_p),
    ]


class switchsd_host_io(ctypes.Structure):
    _fields_ = [
        ("in_host", ctypes.c_void_p), ("in_dev", ctypes.c_void_p), ("in_bytes", ctypes.c_size_t),
        ("out_dev", ctypes.c_void_p), ("out_host", ctypes.c_void_p), ("out_bytes", ctypes.c_size_t),
        ("synchronize", ctypes.c_int32),
    ]


class switchsd_step_args(ctypes.Structure):
    _fields_ = [
        ("draft", ctypes.c_void_p), ("target_argmax", ctypes.c_void_p), ("draft_len", ctypes.c_void_p),
        ("out_accept", ctypes.c_void_p), ("ctx_tokens", ctypes.c_void_p), ("ctx_lens", ctypes.c_void_p),
        ("hidden", ctypes.c_void_p), ("probe_w", ctypes.c_void_p),
        ("params", ctypes.POINTER(switchsd_params)),
        ("out_draft", ctypes.c_void_p), ("out_len", ctypes.c_void_p), ("out_mode", ctypes.c_void_p),
        ("out_score", ctypes.c_void_p),
        ("p_draft", ctypes.c_void_p), ("q_draft", ctypes.c_void_p), ("u", ctypes.c_void_p),
    ]


class switchsd_harness_params(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("k", ctypes.c_int32), ("V", ctypes.c_int32), ("L0", ctypes.c_int32),
        ("n_future", ctypes.c_int32), ("gamma", ctypes.c_int32), ("step", ctypes.c_int32),
        ("seed", ctypes.c_uint64), ("thr_neural", ctypes.c_uint64),
        ("stream", ctypes.c_void_p),
        ("p_hit", ctypes.c_float), ("p_miss", ctypes.c_float), ("q_neural", ctypes.c_float),
    ]


_lock = threading.Lock()
_lib = None

# Every symbol the headers declare, with its ctypes signature.
_SIGNATURES = {
    "switchsd_step": (ctypes.c_int, [ctypes.c_void_p] * 4 + [ctypes.POINTER(switchsd_params)]
                      + [ctypes.c_void_p] * 4),
    "switchsd_verify": (ctypes.c_int, [ctypes.c_void_p] * 3
                        + [ctypes.POINTER(switchsd_verify_params)]),
    "switchsd_verify_sampled": (ctypes.c_int, [ctypes.c_void_p] * 6
                                + [ctypes.POINTER(switchsd_verify_params)]),
    "switchsd_verify_step": (ctypes.c_int, [ctypes.c_void_p] * 8 + [ctypes.POINTER(switchsd_params)]
                             + [ctypes.c_void_p] * 4),
    "switchsd_verify_sampled_step": (ctypes.c_int, [ctypes.c_void_p] * 11 + [ctypes.POINTER(switchsd_params)]
                                     + [ctypes.c_void_p] * 4),
    "switchsd_step_host": (ctypes.c_int, [ctypes.POINTER(switchsd_host_io)] + [ctypes.c_void_p] * 4
                           + [ctypes.POINTER(switchsd_params)] + [ctypes.c_void_p] * 4),
    "switchsd_verify_step_host": (ctypes.c_int, [ctypes.POINTER(switchsd_host_io)] + [ctypes.c_void_p] * 8
                                  + [ctypes.POINTER(switchsd_params)] + [ctypes.c_void_p] * 4),
    "switchsd_verify_sampled_step_host": (ctypes.c_int, [ctypes.POINTER(switchsd_host_io)] + [ctypes.c_void_p] * 11
                                          + [ctypes.POINTER(switchsd_params)] + [ctypes.c_void_p] * 4),
    "switchsd_harness_read": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32,
                                             ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                             ctypes.c_void_p, ctypes.c_void_p]),
    "switchsd_plan_create": (ctypes.c_int, [ctypes.POINTER(switchsd_step_args), ctypes.POINTER(switchsd_host_io),
                                            ctypes.POINTER(ctypes.c_void_p)]),
    "switchsd_plan_run": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32]),
    "switchsd_plan_destroy": (None, [ctypes.c_void_p]),
    "switchsd_step_static_workspace": (ctypes.c_int, [ctypes.c_void_p] * 4
                                       + [ctypes.POINTER(switchsd_params)] + [ctypes.c_void_p] * 4),
    "switchsd_index_create": (ctypes.c_int, [ctypes.POINTER(switchsd_params),
                                             ctypes.POINTER(ctypes.c_void_p)]),
    "switchsd_index_build": (ctypes.c_int, [ctypes.c_void_p] * 4),
    "switchsd_index_bytes": (ctypes.c_size_t, [ctypes.c_void_p]),
    "switchsd_index_destroy": (None, [ctypes.c_void_p]),
    "switchsd_strerror": (ctypes.c_char_p, [ctypes.c_int]),
    "switchsd_workspace_bytes": (ctypes.c_size_t, [ctypes.POINTER(switchsd_params)]),
    "switchsd_abi_version": (ctypes.c_int, []),
    "switchsd_step_candidates": (ctypes.c_int, [ctypes.c_void_p] * 4 + [ctypes.POINTER(switchsd_params),
                                                                        ctypes.c_int32, ctypes.c_int32]
                                 + [ctypes.c_void_p] * 5),
    "switchsd_verify_candidates": (ctypes.c_int, [ctypes.c_void_p] * 4
                                   + [ctypes.POINTER(switchsd_candidates_verify_params)]),
    "switchsd_verify_candidates_step": (ctypes.c_int, [ctypes.c_void_p] * 10 + [ctypes.POINTER(switchsd_params),
                                                                             ctypes.c_int32, ctypes.c_int32]
                                        + [ctypes.c_void_p] * 5),
    "switchsd_harness_candidates": (ctypes.c_int, [ctypes.c_void_p] * 6 + [ctypes.c_int32, ctypes.c_int32]
                                    + [ctypes.c_void_p] * 4 + [ctypes.POINTER(switchsd_harness_params)]),
    "switchsd_labels_workspace_bytes": (ctypes.c_size_t, [ctypes.c_int32, ctypes.c_int32]),
    "switchsd_copy_labels": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32,
                                            ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t,
                                            ctypes.c_void_p]),
    "switchsd_harness_target": (ctypes.c_int, [ctypes.c_void_p] * 8
                                + [ctypes.POINTER(switchsd_harness_params)]),
    "switchsd_harness_sampled": (ctypes.c_int, [ctypes.c_void_p] * 11
                                 + [ctypes.POINTER(switchsd_harness_params)]),
}


def library_path() -> str:
    return _build.LIB


def load(path: str | None = None):
    """Loads (once) and returns the ctypes handle.  Raises if the library was not built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or _build.LIB
        if not os.path.exists(p):
            raise RuntimeError(f"{p} is missing: build it with __graft_entry__.build() "
                               "(python -m paper_2609_20186_gb300.build); there is no fallback")
        lib = ctypes.CDLL(p)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        if lib.switchsd_abi_version() != ABI_VERSION:
            raise RuntimeError(f"{p} has ABI {lib.switchsd_abi_version()}, the binding wants {ABI_VERSION}: rebuild it")
        _lib = lib
        return lib


def strerror(code: int) -> str:
    return load().switchsd_strerror(code).decode()


def abi_version() -> int:
    return load().switchsd_abi_version()


def _check(code: int, what: str):
    if code != OK:
        raise RuntimeError(f"{what} failed: {code} ({strerror(code)})")


def _dev(t: torch.Tensor | None, dtype, name: str, shape=None):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return t.data_ptr()


def _stream_ptr(stream) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _bf16(t: torch.Tensor, name: str, shape=None):
    return _dev(t, torch.bfloat16, name, shape)


def switchsd_step(ctx_tokens, ctx_lens, hidden, probe_w, out_draft, out_len, out_mode, out_score, *,
                  k: int, n_min: int, n_max: int, kappa: int = 0, logit_tau: float = 0.0,
                  probe_kind: int = PROBE_LINEAR, probe_hidden: int = 0, b1=None, b2: float = 0.0,
                  split: int = 0, out_match_n=None, out_match_end=None, status=None,
                  workspace=None, stream=None, prefetch: int = 0) -> None:
    """switchsd_step of include/switchsd.h on torch tensors (see the header for semantics).

    ctx_tokens int32 [B, cap]; ctx_lens int32 [B]; hidden bf16 [B, d]; probe_w bf16 (w[d] or
    W1[H1, d] + w2[H1] flattened); outputs int32 [B, k], int32 [B], int32 [B], float32 [B].
    """
    B, cap = ctx_tokens.shape
    d = hidden.shape[1]
    p = switchsd_params()
    p.B, p.cap, p.d, p.k = B, cap, d, k
    p.n_min, p.n_max, p.kappa = n_min, n_max, kappa
    p.logit_tau = logit_tau
    p.probe_kind, p.probe_hidden = probe_kind, probe_hidden
    p.b1 = _dev(b1, torch.float32, "b1", (probe_hidden,)) if b1 is not None else None
    p.b2 = b2
    p.split = split
    p.out_match_n = _dev(out_match_n, torch.int32, "out_match_n", (B,))
    p.out_match_end = _dev(out_match_end, torch.int32, "out_match_end", (B,))
    p.status = _dev(status, torch.int32, "status", (B,))
    p.stream = _stream_ptr(stream)
    p.prefetch = int(prefetch)  # PREFETCH_* bits (see the header for the caller's guarantee)
    nw = d if probe_kind == PROBE_LINEAR else probe_hidden * d + probe_hidden
    ws = _attach_workspace(p, workspace, ctx_tokens.device)  # noqa: F841 (kept alive for the call)
    code = load().switchsd_step(
        _dev(ctx_tokens, torch.int32, "ctx_tokens"), _dev(ctx_lens, torch.int32, "ctx_lens", (B,)),
        _bf16(hidden, "hidden", (B, d)), _bf16(probe_w, "probe_w", (nw,)), ctypes.byref(p),
        _dev(out_draft, torch.int32, "out_draft", (B, k)), _dev(out_len, torch.int32, "out_len", (B,)),
        _dev(out_mode, torch.int32, "out_mode", (B,)), _dev(out_score, torch.float32, "out_score", (B,)))
    _check(code, "switchsd_step")


def switchsd_workspace_bytes(B: int, probe_kind: int = PROBE_LINEAR, probe_hidden: int = 0, d: int = 0,
                             hidden_rows: int = 0) -> int:
    """switchsd_workspace_bytes of include/switchsd.h for a batch of B rows of hidden size d."""
    p = switchsd_params()
    p.B, p.d, p.probe_kind, p.probe_hidden, p.hidden_rows = B, d, probe_kind, probe_hidden, hidden_rows
    return int(load().switchsd_workspace_bytes(ctypes.byref(p)))


class NgramIndex:
    """switchsd_index_* of include/switchsd.h: the incremental n-gram index of B rows (device memory
    owned by the library, freed by close() or when the object is collected)."""

    def __init__(self, B: int, cap: int, n_min: int, n_max: int):
        p = switchsd_params()
        p.B, p.cap, p.n_min, p.n_max = B, cap, n_min, n_max
        h = ctypes.c_void_p()
        _check(load().switchsd_index_create(ctypes.byref(p), ctypes.byref(h)), "switchsd_index_create")
        self.handle = h.value
        self.B, self.cap, self.n_min, self.n_max = B, cap, n_min, n_max

    def build(self, ctx_tokens: torch.Tensor, ctx_lens: torch.Tensor, stream=None) -> None:
        _check(load().switchsd_index_build(self.handle, _dev(ctx_tokens, torch.int32, "ctx_tokens",
                                                             (self.B, self.cap)),
                                           _dev(ctx_lens, torch.int32, "ctx_lens", (self.B,)),
                                           _stream_ptr(stream)), "switchsd_index_build")

    @property
    def nbytes(self) -> int:
        return int(load().switchsd_index_bytes(self.handle))

    def close(self) -> None:
        if self.handle:
            load().switchsd_index_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _attach_workspace(p: switchsd_params, workspace, device) -> torch.Tensor | None:
    """Points p at `workspace` (a CUDA uint8 tensor), allocating one from torch when the probe needs it
    and none was given.  Returns the tensor so the caller keeps it alive for the call."""
    need = int(load().switchsd_workspace_bytes(ctypes.byref(p)))
    if need == 0 and workspace is None:
        return None
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=device)
    if not workspace.is_cuda or workspace.numel() * workspace.element_size() < need:
        raise ValueError(f"workspace must be a CUDA tensor of at least {need} bytes")
    p.workspace = workspace.data_ptr()
    p.workspace_bytes = workspace.numel() * workspace.element_size()
    return workspace


def switchsd_verify_step(draft, target_argmax, draft_len, out_accept, ctx_tokens, ctx_lens, hidden,
                         probe_w, out_draft, out_len, out_mode, out_score, *, k: int, n_min: int,
                         n_max: int, kappa: int = 0, logit_tau: float = 0.0,
                         probe_kind: int = PROBE_LINEAR, probe_hidden: int = 0, b1=None,
                         b2: float = 0.0, split: int = 0, out_match_n=None, out_match_end=None,
                         status=None, workspace=None, stream=None, prefetch: int = 0) -> None:
    """switchsd_verify_step of include/switchsd.h: verification of the previous draft, then the next
    step, in one launch."""
    B, cap = ctx_tokens.shape
    d = hidden.shape[1]
    p = switchsd_params()
    p.B, p.cap, p.d, p.k = B, cap, d, k
    p.n_min, p.n_max, p.kappa = n_min, n_max, kappa
    p.logit_tau = logit_tau
    p.probe_kind, p.probe_hidden = probe_kind, probe_hidden
    p.b1 = _dev(b1, torch.float32, "b1", (probe_hidden,)) if b1 is not None else None
    p.b2 = b2
    p.split = split
    p.out_match_n = _dev(out_match_n, torch.int32, "out_match_n", (B,))
    p.out_match_end = _dev(out_match_end, torch.int32, "out_match_end", (B,))
    p.status = _dev(status, torch.int32, "status", (B,))
    p.stream = _stream_ptr(stream)
    p.prefetch = int(prefetch)  # PREFETCH_* bits (see the header for the caller's guarantee)
    nw = d if probe_kind == PROBE_LINEAR else probe_hidden * d + probe_hidden
    ws = _attach_workspace(p, workspace, ctx_tokens.device)  # noqa: F841 (kept alive for the call)
    code = load().switchsd_verify_step(
        _dev(draft, torch.int32, "draft", (B, k)),
        _dev(target_argmax, torch.int32, "target_argmax", (B, k + 1)),
        _dev(draft_len, torch.int32, "draft_len", (B,)), _dev(out_accept, torch.int32, "out_accept", (B,)),
        _dev(ctx_tokens, torch.int32, "ctx_tokens"), _dev(ctx_lens, torch.int32, "ctx_lens", (B,)),
        _bf16(hidden, "hidden", (B, d)), _bf16(probe_w, "probe_w", (nw,)), ctypes.byref(p),
        _dev(out_draft, torch.int32, "out_draft", (B, k)), _dev(out_len, torch.int32, "out_len", (B,)),
        _dev(out_mode, torch.int32, "out_mode", (B,)), _dev(out_score, torch.float32, "out_score", (B,)))
    _check(code, "switchsd_verify_step")


def switchsd_verify(draft, target_argmax, out_accept, *, draft_len, ctx_tokens, ctx_lens,
                    status=None, stream=None) -> None:
    """switchsd_verify of include/switchsd.h on torch tensors."""
    B, cap = ctx_tokens.shape
    k = draft.shape[1]
    vp = switchsd_verify_params()
    vp.B, vp.cap, vp.k = B, cap, k
    vp.draft_len = _dev(draft_len, torch.int32, "draft_len", (B,))
    vp.ctx_tokens = _dev(ctx_tokens, torch.int32, "ctx_tokens")
    vp.ctx_lens = _dev(ctx_lens, torch.int32, "ctx_lens", (B,))
    vp.status = _dev(status, torch.int32, "status", (B,))
    vp.stream = _stream_ptr(stream)
    code = load().switchsd_verify(_dev(draft, torch.int32, "draft", (B, k)),
                                  _dev(target_argmax, torch.int32, "target_argmax", (B, k + 1)),
                                  _dev(out_accept, torch.int32, "out_accept", (B,)), ctypes.byref(vp))
    _check(code, "switchsd_verify")


def switchsd_verify_sampled(draft, p_draft, u, resample, out_accept, *, draft_len, ctx_tokens, ctx_lens,
                            q_draft=None, status=None, stream=None) -> None:
    """switchsd_verify_sampled of include/switchsd.h on torch tensors: draft int32 [B, k], p_draft /
    q_draft (None: copy drafts) / u float32 [B, k], resample int32 [B, k + 1]."""
    B, cap = ctx_tokens.shape
    k = draft.shape[1]
    vp = switchsd_verify_params()
    vp.B, vp.cap, vp.k = B, cap, k
    vp.draft_len = _dev(draft_len, torch.int32, "draft_len", (B,))
    vp.ctx_tokens = _dev(ctx_tokens, torch.int32, "ctx_tokens")
    vp.ctx_lens = _dev(ctx_lens, torch.int32, "ctx_lens", (B,))
    vp.status = _dev(status, torch.int32, "status", (B,))
    vp.stream = _stream_ptr(stream)
    code = load().switchsd_verify_sampled(
        _dev(draft, torch.int32, "draft", (B, k)), _dev(p_draft, torch.float32, "p_draft", (B, k)),
        _dev(q_draft, torch.float32, "q_draft", (B, k)), _dev(u, torch.float32, "u", (B, k)),
        _dev(resample, torch.int32, "resample", (B, k + 1)), _dev(out_accept, torch.int32, "out_accept", (B,)),
        ctypes.byref(vp))
    _check(code, "switchsd_verify_sampled")


def switchsd_harness_target(ctx_lens, mode, draft, draft_len, future, vdraft, vlen, target, *,
                            seed: int, V: int, L0: int, gamma: int, thr_neural: int, step: int,
                            stream=None) -> None:
    """switchsd_harness_target of include/switchsd_harness.h (the target-model stand-in)."""
    B, k = draft.shape
    hp = switchsd_harness_params()
    hp.B, hp.k, hp.V, hp.L0 = B, k, V, L0
    hp.n_future = future.shape[1]
    hp.gamma, hp.step = gamma, step
    hp.seed, hp.thr_neural = seed, thr_neural
    hp.stream = _stream_ptr(stream)
    code = load().switchsd_harness_target(
        _dev(ctx_lens, torch.int32, "ctx_lens", (B,)), _dev(mode, torch.int32, "mode", (B,)),
        _dev(draft, torch.int32, "draft", (B, k)), _dev(draft_len, torch.int32, "draft_len", (B,)),
        _dev(future, torch.int32, "future"), _dev(vdraft, torch.int32, "vdraft", (B, k)),
        _dev(vlen, torch.int32, "vlen", (B,)), _dev(target, torch.int32, "target", (B, k + 1)),
        ctypes.byref(hp))
    _check(code, "switchsd_harness_target")


def switchsd_harness_sampled(ctx_lens, mode, draft, draft_len, future, vdraft, vlen, p, q, u, resample, *,
                             seed: int, V: int, L0: int, gamma: int, thr_neural: int, step: int,
                             p_hit: float, p_miss: float, q_neural: float, stream=None) -> None:
    """switchsd_harness_sampled of include/switchsd_harness.h (the stand-in at T > 0)."""
    B, k = draft.shape
    hp = switchsd_harness_params()
    hp.B, hp.k, hp.V, hp.L0 = B, k, V, L0
    hp.n_future = future.shape[1]
    hp.gamma, hp.step = gamma, step
    hp.seed, hp.thr_neural = seed, thr_neural
    hp.p_hit, hp.p_miss, hp.q_neural = p_hit, p_miss, q_neural
    hp.stream = _stream_ptr(stream)
    code = load().switchsd_harness_sampled(
        _dev(ctx_lens, torch.int32, "ctx_lens", (B,)), _dev(mode, torch.int32, "mode", (B,)),
        _dev(draft, torch.int32, "draft", (B, k)), _dev(draft_len, torch.int32, "draft_len", (B,)),
        _dev(future, torch.int32, "future"), _dev(vdraft, torch.int32, "vdraft", (B, k)),
        _dev(vlen, torch.int32, "vlen", (B,)), _dev(p, torch.float32, "p", (B, k)),
        _dev(q, torch.float32, "q", (B, k)), _dev(u, torch.float32, "u", (B, k)),
        _dev(resample, torch.int32, "resample", (B, k + 1)), ctypes.byref(hp))
    _check(code, "switchsd_harness_sampled")


def switchsd_copy_labels(ctx_tokens, ctx_lens, out_labels, *, n: int = 5, workspace=None, stream=None) -> None:
    """switchsd_copy_labels of include/switchsd.h (§3.2 copy-mode labels): ctx_tokens int32 [B, cap],
    ctx_lens int32 [B], out_labels uint8 [B, cap].  Allocates the workspace from torch when none is given."""
    B, cap = ctx_tokens.shape
    need = int(load().switchsd_labels_workspace_bytes(B, cap))
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=ctx_tokens.device)
    code = load().switchsd_copy_labels(
        _dev(ctx_tokens, torch.int32, "ctx_tokens"), _dev(ctx_lens, torch.int32, "ctx_lens", (B,)), B, cap, n,
        _dev(out_labels, torch.uint8, "out_labels", (B, cap)), _dev(workspace, torch.uint8, "workspace"),
        workspace.numel(), _stream_ptr(stream))
    _check(code, "switchsd_copy_labels")
