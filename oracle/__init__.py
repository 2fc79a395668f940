"""CPU oracle of the SwitchSD per-step controller -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg may import this
package.  The product path (``paper_2609_20186_gb300``) never imports it and shares no code with it.

The arithmetic lives in ``switchsd_oracle.c`` (plain C, double precision); this module compiles it with
gcc into ``oracle/_build/liboracle.so`` and wraps it with numpy-friendly functions.  Each C function
cites the passage of the paper it follows:

- ``longest_suffix_match``: the kappa-gram gate and recency ranking of §3.3;
- ``probe_linear``: Eq. 3 (logit of the linear probe, no bias);
- ``probe_mlp``: two-layer probe extension (no counterpart in the paper, used by one workload);
- ``switch``: Fig. 1's three cases with Eq. 4's threshold;
- ``verify_row``: greedy verification and append, §3.3 at temperature 0 (App. A).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "switchsd_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")

MODE_NO_REP = 0
MODE_COPY = 1
MODE_REP_NO_COPY = 2
ROW_OK = 0
ROW_CAPACITY = 1

_lock = threading.Lock()
_lib = None

_i32p = ctypes.POINTER(ctypes.c_int32)
_u16p = ctypes.POINTER(ctypes.c_uint16)
_f32p = ctypes.POINTER(ctypes.c_float)
_f64p = ctypes.POINTER(ctypes.c_double)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain -O2, no machine-specific flags)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    stale = (not os.path.exists(_LIB_PATH)) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC],
                       check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def compile_library(src: str, out: str) -> str:
    """Compiles an oracle source file (this one, or a copy under test) into a shared library."""
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", out, src], check=True)
    return out


def configure(lib):
    """Declares the C signatures on a loaded oracle library; returns it."""
    lib.oracle_longest_suffix_match.argtypes = [_i32p, ctypes.c_int32, ctypes.c_int32,
                                                ctypes.c_int32, _i32p, _i32p]
    lib.oracle_longest_suffix_match.restype = ctypes.c_int
    lib.oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
    lib.oracle_bf16_to_double.restype = ctypes.c_double
    lib.oracle_probe_linear.argtypes = [_u16p, _u16p, ctypes.c_int32]
    lib.oracle_probe_linear.restype = ctypes.c_double
    lib.oracle_probe_mlp.argtypes = [_u16p, _u16p, _f32p, _u16p, ctypes.c_float,
                                     ctypes.c_int32, ctypes.c_int32]
    lib.oracle_probe_mlp.restype = ctypes.c_double
    lib.oracle_switch.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                  ctypes.c_double, ctypes.c_float, ctypes.c_int32,
                                  ctypes.c_int32, _i32p, ctypes.c_int32, _i32p, _i32p]
    lib.oracle_switch.restype = ctypes.c_int32
    lib.oracle_verify_row.argtypes = [_i32p, _i32p, ctypes.c_int32, _i32p, ctypes.c_int32,
                                      _i32p, _i32p]
    lib.oracle_verify_row.restype = ctypes.c_int32
    lib.oracle_step_rows.argtypes = [
        _i32p, _i32p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,  # ctx lens b0 b1 cap
        _u16p, ctypes.c_int32, _u16p, ctypes.c_int32,                   # hidden d probe_w kind
        ctypes.c_int32, _f32p, ctypes.c_float,                          # H1 b1 b2
        ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,  # k n_min n_max kappa
        ctypes.c_float,                                                 # logit_tau
        _i32p, _i32p, _i32p, _f64p, _i32p, _i32p]
    lib.oracle_step_rows.restype = None
    lib.oracle_verify_rows.argtypes = [_i32p, _i32p, ctypes.c_int32, ctypes.c_int32,
                                       ctypes.c_int32, ctypes.c_int32, _i32p, _i32p, _i32p,
                                       _i32p, _i32p]
    lib.oracle_verify_rows.restype = None
    lib.oracle_verify_sampled_row.argtypes = [_i32p, _i32p, ctypes.c_int32, _i32p, ctypes.c_int32,
                                              _f32p, _f32p, _f32p, _i32p, _i32p]
    lib.oracle_verify_sampled_row.restype = ctypes.c_int32
    lib.oracle_verify_sampled_rows.argtypes = [_i32p, _i32p, ctypes.c_int32, ctypes.c_int32,
                                               ctypes.c_int32, ctypes.c_int32, _i32p, _i32p, _f32p,
                                               _f32p, _f32p, _i32p, _i32p, _i32p]
    lib.oracle_verify_sampled_rows.restype = None
    lib.oracle_window_repeats.argtypes = [_i32p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]
    lib.oracle_window_repeats.restype = ctypes.c_int32
    lib.oracle_copy_labels.argtypes = [_i32p, ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(ctypes.c_uint8)]
    lib.oracle_copy_labels.restype = None
    lib.oracle_candidates.argtypes = [_i32p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                      ctypes.c_double, ctypes.c_float, ctypes.c_int32, ctypes.c_int32, _i32p,
                                      _i32p, _i32p, _i32p]
    lib.oracle_candidates.restype = ctypes.c_int32
    lib.oracle_verify_candidates_row.argtypes = [_i32p, _i32p, ctypes.c_int32, _i32p, _i32p, ctypes.c_int32,
                                                 ctypes.c_int32, _i32p, _i32p, _i32p]
    lib.oracle_verify_candidates_row.restype = ctypes.c_int32
    lib.oracle_step_candidates_rows.argtypes = [
        _i32p, _i32p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
        _u16p, ctypes.c_int32, _u16p, ctypes.c_int32, ctypes.c_int32, _f32p, ctypes.c_float,
        ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_float,
        _i32p, _i32p, _i32p, _i32p, _f64p, _i32p, _i32p, _i32p]
    lib.oracle_step_candidates_rows.restype = None
    lib.oracle_verify_candidates_rows.argtypes = [_i32p, _i32p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                                  ctypes.c_int32, ctypes.c_int32, _i32p, _i32p, _i32p, _i32p,
                                                  _i32p, _i32p, _i32p]
    lib.oracle_verify_candidates_rows.restype = None
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = configure(ctypes.CDLL(build()))
        return _lib


def use_library(lib):
    """Routes this module's functions to `lib` (a configured oracle library); returns the previous
    one.  Used by the tests that plant mistakes in a copy of the oracle."""
    global _lib
    with _lock:
        old, _lib = _lib, lib
        return old


def _ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(ctype)


def _c(a, dtype) -> np.ndarray:
    a = np.ascontiguousarray(a, dtype=dtype)
    return a


# ---------------------------------------------------------------------------------------------
# Single-row functions (used by the pins)
# ---------------------------------------------------------------------------------------------

def longest_suffix_match(x, n_min: int, n_max: int, L: int | None = None):
    """(n*, e*) of the longest, then most recent, earlier occurrence of the context's suffix
    (§3.3), or (0, -1) if no n in [n_min, n_max] has one."""
    lib = _load()
    x = _c(x, np.int32)
    if L is None:
        L = x.shape[0]
    n = ctypes.c_int32()
    e = ctypes.c_int32()
    lib.oracle_longest_suffix_match(_ptr(x, _i32p), L, n_min, n_max, ctypes.byref(n),
                                    ctypes.byref(e))
    return n.value, e.value


def bf16_to_double(v: int) -> float:
    return _load().oracle_bf16_to_double(v)


def probe_linear(h_bits, w_bits) -> float:
    """Logit of Eq. 3's linear probe (no bias), summed in double."""
    h = _c(h_bits, np.uint16)
    w = _c(w_bits, np.uint16)
    assert h.shape == w.shape
    return _load().oracle_probe_linear(_ptr(h, _u16p), _ptr(w, _u16p), h.shape[0])


def probe_mlp(h_bits, W1_bits, w2_bits, b1=None, b2: float = 0.0) -> float:
    """Logit of the two-layer probe w2 . ReLU(W1 h + b1) + b2, in double."""
    h = _c(h_bits, np.uint16)
    W1 = _c(W1_bits, np.uint16)
    w2 = _c(w2_bits, np.uint16)
    H1, d = W1.shape
    assert h.shape == (d,) and w2.shape == (H1,)
    b1p = None
    if b1 is not None:
        b1a = _c(b1, np.float32)
        b1p = _ptr(b1a, _f32p)
    return _load().oracle_probe_mlp(_ptr(h, _u16p), _ptr(W1, _u16p), b1p, _ptr(w2, _u16p),
                                    float(b2), d, H1)


def switch(has_match: bool, n_star: int, e_star: int, z: float, logit_tau: float, kappa: int,
           k: int, x, L: int | None = None):
    """Fig. 1 / Eq. 4: returns (mode, draft list)."""
    x = _c(x, np.int32)
    if L is None:
        L = x.shape[0]
    draft = np.zeros(max(k, 1), np.int32)
    ln = ctypes.c_int32()
    mode = _load().oracle_switch(int(has_match), n_star, e_star, float(z), float(logit_tau), kappa,
                                 k, _ptr(x, _i32p), L, _ptr(draft, _i32p), ctypes.byref(ln))
    return mode, draft[: ln.value].tolist()


def verify_row(row: np.ndarray, L: int, cap: int, draft, target):
    """Greedy verify + append on one row buffer (modified in place).
    Returns (new_L, accept, status)."""
    assert row.dtype == np.int32 and row.flags.c_contiguous and row.shape[0] >= cap
    d = _c(draft, np.int32)
    t = _c(target, np.int32)
    assert t.shape[0] >= d.shape[0] + 1
    Lc = ctypes.c_int32(L)
    acc = ctypes.c_int32()
    st = _load().oracle_verify_row(_ptr(row, _i32p), ctypes.byref(Lc), cap, _ptr(d, _i32p),
                                   d.shape[0], _ptr(t, _i32p), ctypes.byref(acc))
    return Lc.value, acc.value, st


def verify_sampled_row(row: np.ndarray, L: int, cap: int, draft, p, u, resample, q=None):
    """Verification at T > 0 (App. A) + append on one row buffer (modified in place): draft token i
    is accepted iff float32(u[i] * q[i]) < p[i] (q = None: a copy draft, q = 1); resample has
    len(draft) + 1 entries.  Returns (new_L, accept, status)."""
    assert row.dtype == np.int32 and row.flags.c_contiguous and row.shape[0] >= cap
    d = _c(draft, np.int32)
    n = d.shape[0]
    pa, ua = _c(p, np.float32), _c(u, np.float32)
    qa = None if q is None else _c(q, np.float32)
    r = _c(resample, np.int32)
    assert pa.shape[0] >= n and ua.shape[0] >= n and r.shape[0] >= n + 1
    assert qa is None or qa.shape[0] >= n
    Lc = ctypes.c_int32(L)
    acc = ctypes.c_int32()
    st = _load().oracle_verify_sampled_row(_ptr(row, _i32p), ctypes.byref(Lc), cap, _ptr(d, _i32p), n,
                                           _ptr(pa, _f32p), None if qa is None else _ptr(qa, _f32p),
                                           _ptr(ua, _f32p), _ptr(r, _i32p), ctypes.byref(acc))
    return Lc.value, acc.value, st


# ---------------------------------------------------------------------------------------------
# Batched functions (ABI layouts), used by the parity tests and the CPU baseline
# ---------------------------------------------------------------------------------------------

def step(ctx: np.ndarray, lens: np.ndarray, hidden_bits: np.ndarray, probe_w_bits: np.ndarray, *,
         k: int, n_min: int, n_max: int, kappa: int = 0, logit_tau: float = 0.0,
         probe_kind: int = 0, probe_hidden: int = 0, b1=None, b2: float = 0.0,
         rows: tuple[int, int] | None = None) -> dict:
    """One controller step on the rows [b0, b1) of a batch (all rows by default).

    ctx int32 [B, cap]; lens int32 [B]; hidden bf16 bits uint16 [B, d]; probe_w bf16 bits (w[d], or
    W1[H1, d] followed by w2[H1] for the two-layer probe).  Returns numpy arrays over all B rows
    (rows outside the range are zero): draft [B, k], len, mode, score (float64 logit), match_n,
    match_end.
    """
    lib = _load()
    assert ctx.dtype == np.int32 and ctx.flags.c_contiguous
    B, cap = ctx.shape
    lens = _c(lens, np.int32)
    hidden = _c(hidden_bits, np.uint16)
    assert hidden.ndim == 2 and hidden.shape[0] == B
    d = hidden.shape[1]
    pw = _c(probe_w_bits, np.uint16).reshape(-1)
    b1a = None if b1 is None else _c(b1, np.float32)
    b0, bend = rows if rows is not None else (0, B)
    out = {
        "draft": np.zeros((B, k), np.int32),
        "len": np.zeros(B, np.int32),
        "mode": np.zeros(B, np.int32),
        "score": np.zeros(B, np.float64),
        "match_n": np.zeros(B, np.int32),
        "match_end": np.full(B, -1, np.int32),
    }
    lib.oracle_step_rows(_ptr(ctx, _i32p), _ptr(lens, _i32p), b0, bend, cap, _ptr(hidden, _u16p), d,
                         _ptr(pw, _u16p), probe_kind, probe_hidden,
                         None if b1a is None else _ptr(b1a, _f32p), float(b2), k, n_min, n_max,
                         kappa, float(logit_tau), _ptr(out["draft"], _i32p), _ptr(out["len"], _i32p),
                         _ptr(out["mode"], _i32p), _ptr(out["score"], _f64p),
                         _ptr(out["match_n"], _i32p), _ptr(out["match_end"], _i32p))
    return out


def verify(ctx: np.ndarray, lens: np.ndarray, draft: np.ndarray, draft_len: np.ndarray,
           target: np.ndarray, rows: tuple[int, int] | None = None):
    """Greedy verify + append on rows [b0, b1) (all by default); ctx and lens are updated in place.
    Returns (accept [B], status [B])."""
    lib = _load()
    assert ctx.dtype == np.int32 and ctx.flags.c_contiguous
    assert lens.dtype == np.int32 and lens.flags.c_contiguous
    B, cap = ctx.shape
    draft = _c(draft, np.int32)
    k = draft.shape[1]
    draft_len = _c(draft_len, np.int32)
    target = _c(target, np.int32)
    assert target.shape == (B, k + 1)
    acc = np.zeros(B, np.int32)
    st = np.zeros(B, np.int32)
    b0, bend = rows if rows is not None else (0, B)
    lib.oracle_verify_rows(_ptr(ctx, _i32p), _ptr(lens, _i32p), b0, bend, cap, k,
                           _ptr(draft, _i32p), _ptr(draft_len, _i32p), _ptr(target, _i32p),
                           _ptr(acc, _i32p), _ptr(st, _i32p))
    return acc, st


def verify_sampled(ctx: np.ndarray, lens: np.ndarray, draft: np.ndarray, draft_len: np.ndarray,
                   p: np.ndarray, u: np.ndarray, resample: np.ndarray, q: np.ndarray | None = None,
                   rows: tuple[int, int] | None = None):
    """Verification at T > 0 + append on rows [b0, b1) (all by default); ctx and lens are updated in
    place.  p, u, q float32 [B, k] (q None: every draft is a copy draft), resample int32 [B, k + 1].
    Returns (accept [B], status [B])."""
    lib = _load()
    assert ctx.dtype == np.int32 and ctx.flags.c_contiguous
    assert lens.dtype == np.int32 and lens.flags.c_contiguous
    B, cap = ctx.shape
    draft = _c(draft, np.int32)
    k = draft.shape[1]
    draft_len = _c(draft_len, np.int32)
    p, u = _c(p, np.float32), _c(u, np.float32)
    assert p.shape == (B, k) and u.shape == (B, k)
    qa = None if q is None else _c(q, np.float32)
    assert qa is None or qa.shape == (B, k)
    resample = _c(resample, np.int32)
    assert resample.shape == (B, k + 1)
    acc = np.zeros(B, np.int32)
    st = np.zeros(B, np.int32)
    b0, bend = rows if rows is not None else (0, B)
    lib.oracle_verify_sampled_rows(_ptr(ctx, _i32p), _ptr(lens, _i32p), b0, bend, cap, k,
                                   _ptr(draft, _i32p), _ptr(draft_len, _i32p), _ptr(p, _f32p),
                                   None if qa is None else _ptr(qa, _f32p), _ptr(u, _f32p),
                                   _ptr(resample, _i32p), _ptr(acc, _i32p), _ptr(st, _i32p))
    return acc, st


def window_repeats(x, n: int, s: int) -> bool:
    """Whether the n-token window of x starting at s also starts at an earlier position (§3.2)."""
    xa = _c(x, np.int32)
    return bool(_load().oracle_window_repeats(_ptr(xa, _i32p), xa.shape[0], n, s))


def copy_labels(x, n: int = 5) -> np.ndarray:
    """Copy-mode labels (§3.2) of the sequence x: uint8 [len(x)], 1 where the position lies in an
    n-token window that also occurs starting earlier."""
    xa = _c(x, np.int32)
    y = np.zeros(xa.shape[0], np.uint8)
    _load().oracle_copy_labels(_ptr(xa, _i32p), xa.shape[0], n, y.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)))
    return y


def candidates(x, *, n_min: int, n_max: int, kappa: int, z: float, logit_tau: float, W: int, D: int):
    """Copy candidates of one context (§3.3): returns (mode, [candidate token lists], [candidate ends])
    -- ends only for a copy row."""
    xa = _c(x, np.int32)
    L = xa.shape[0]
    cand = np.zeros((W, D), np.int32)
    clen = np.zeros(W, np.int32)
    ends = np.zeros(max(W, 1), np.int32)
    nc = ctypes.c_int32()
    mode = _load().oracle_candidates(_ptr(xa, _i32p), L, n_min, n_max, kappa, float(z), float(logit_tau), W, D,
                                     _ptr(cand, _i32p), _ptr(clen, _i32p), ctypes.byref(nc), _ptr(ends, _i32p))
    n = nc.value
    return mode, [cand[w, : clen[w]].tolist() for w in range(n)], ends[:n].tolist()


def verify_candidates_row(row: np.ndarray, L: int, cap: int, cands, target):
    """Verification of W candidates (§3.3) on one row buffer (modified in place): cands a list of token
    lists (empty list = no candidate), target [W][D+1] (D = the longest candidate slot).
    Returns (new_L, accept, choice, status)."""
    W = max(len(cands), 1)
    D = max([len(c) for c in cands] + [np.asarray(target).shape[1] - 1])
    cand = np.zeros((W, D), np.int32)
    clen = np.zeros(W, np.int32)
    for w, c in enumerate(cands):
        cand[w, : len(c)] = c
        clen[w] = len(c)
    t = np.zeros((W, D + 1), np.int32)
    ta = np.asarray(target, np.int32)
    t[: ta.shape[0], : ta.shape[1]] = ta
    Lc, acc, ch = ctypes.c_int32(L), ctypes.c_int32(), ctypes.c_int32()
    st = _load().oracle_verify_candidates_row(_ptr(row, _i32p), ctypes.byref(Lc), cap, _ptr(cand, _i32p),
                                              _ptr(clen, _i32p), len(cands), D, _ptr(t, _i32p), ctypes.byref(acc),
                                              ctypes.byref(ch))
    return Lc.value, acc.value, ch.value, st


def step_candidates(ctx: np.ndarray, lens: np.ndarray, hidden_bits: np.ndarray, probe_w_bits: np.ndarray, *,
                    W: int, D: int, n_min: int, n_max: int, kappa: int = 0, logit_tau: float = 0.0,
                    probe_kind: int = 0, probe_hidden: int = 0, b1=None, b2: float = 0.0,
                    rows: tuple[int, int] | None = None) -> dict:
    """The candidate step on rows [b0, b1): cand [B, W, D], cand_len [B, W], ncand, mode, score, match_n,
    match_end (numpy, rows outside the range zero)."""
    lib = _load()
    B, cap = ctx.shape
    lens = _c(lens, np.int32)
    hidden = _c(hidden_bits, np.uint16)
    d = hidden.shape[1]
    pw = _c(probe_w_bits, np.uint16).reshape(-1)
    b1a = None if b1 is None else _c(b1, np.float32)
    b0, bend = rows if rows is not None else (0, B)
    out = {"cand": np.zeros((B, W, D), np.int32), "cand_len": np.zeros((B, W), np.int32),
           "ncand": np.zeros(B, np.int32), "mode": np.zeros(B, np.int32), "score": np.zeros(B, np.float64),
           "match_n": np.zeros(B, np.int32), "match_end": np.full(B, -1, np.int32)}
    scratch = np.zeros(max(W, 1), np.int32)
    lib.oracle_step_candidates_rows(_ptr(ctx, _i32p), _ptr(lens, _i32p), b0, bend, cap, _ptr(hidden, _u16p), d,
                                    _ptr(pw, _u16p), probe_kind, probe_hidden,
                                    None if b1a is None else _ptr(b1a, _f32p), float(b2), W, D, n_min, n_max,
                                    kappa, float(logit_tau), _ptr(out["cand"], _i32p), _ptr(out["cand_len"], _i32p),
                                    _ptr(out["ncand"], _i32p), _ptr(out["mode"], _i32p), _ptr(out["score"], _f64p),
                                    _ptr(out["match_n"], _i32p), _ptr(out["match_end"], _i32p),
                                    _ptr(scratch, _i32p))
    return out


def verify_candidates(ctx: np.ndarray, lens: np.ndarray, cand: np.ndarray, cand_len: np.ndarray,
                      ncand: np.ndarray, target: np.ndarray, rows: tuple[int, int] | None = None):
    """Verification of the candidates on rows [b0, b1); ctx / lens updated in place.  cand [B, W, D],
    cand_len [B, W], ncand [B], target [B, W, D+1].  Returns (accept, choice, status) [B]."""
    lib = _load()
    B, cap = ctx.shape
    cand = _c(cand, np.int32)
    W, D = cand.shape[1], cand.shape[2]
    cand_len, ncand, target = _c(cand_len, np.int32), _c(ncand, np.int32), _c(target, np.int32)
    assert target.shape == (B, W, D + 1)
    acc, ch, st = np.zeros(B, np.int32), np.zeros(B, np.int32), np.zeros(B, np.int32)
    b0, bend = rows if rows is not None else (0, B)
    lib.oracle_verify_candidates_rows(_ptr(ctx, _i32p), _ptr(lens, _i32p), b0, bend, cap, W, D, _ptr(cand, _i32p),
                                      _ptr(cand_len, _i32p), _ptr(ncand, _i32p), _ptr(target, _i32p),
                                      _ptr(acc, _i32p), _ptr(ch, _i32p), _ptr(st, _i32p))
    return acc, ch, st
