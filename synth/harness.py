"""Stand-in for the neural drafter and the target model's verification forward (host side).

Greedy verification (temperature 0) keeps the context equal to the target model's own greedy
sequence.  The target model is out of scope, so each row's greedy continuation is a seeded token
stream ``future`` (Workload.future: the row's token law plus planted copies of earlier spans with
occasional edits).  Then, for a row of current length L:

- the target's greedy token after draft prefix i is future[L + i] whenever that prefix is the
  target's own (the only prefixes verification can accept), so target[i] = future[L + i - L0] for
  i = 0..k;
- rows whose mode is not COPY get a neural draft of ``gamma`` tokens: draft[i] = future[L + i - L0]
  with probability ``p_neural`` (a seeded coin), else a seeded token different from it.

Randomness comes from ``harness_key(seed, row, step, 4 * i + slot)`` (slot 0: the neural coin, low
32 bits; slot 1: the replacement token, a token being (word >> 32) mod V).  The CUDA harness kernel
implements the same chain, so both sides produce identical drafts and targets for identical inputs.
No controller arithmetic happens here.
"""
from __future__ import annotations

import numpy as np

from .rng import harness_key

MODE_COPY = 1  # the documented ABI value of the copy mode


def _token(r: np.ndarray, V: int) -> np.ndarray:
    return ((r >> np.uint64(32)) % np.uint64(V)).astype(np.int64)


def harness_targets(params: dict, step: int, ctx_lens: np.ndarray, mode: np.ndarray,
                    draft: np.ndarray, draft_len: np.ndarray, future: np.ndarray,
                    rows=None):
    """Returns (vdraft [B, k], vlen [B], target [B, k+1]) as int32 arrays; rows outside ``rows``
    (default: all) are left zero.  Each row's result depends only on its own inputs."""
    B, k = draft.shape
    V = params["V"]
    L0 = params["L0"]
    gamma = params["gamma"]
    thr = np.uint64(params["thr_neural"])
    seed = params["seed"]
    nfut = future.shape[1]
    vdraft = np.zeros((B, k), np.int32)
    vlen = np.zeros(B, np.int32)
    target = np.zeros((B, k + 1), np.int32)
    idx = range(B) if rows is None else rows
    i = np.arange(k + 1, dtype=np.int64)
    for b in idx:
        b = int(b)
        L = int(ctx_lens[b])
        pos = L - L0 + i
        ok = (pos >= 0) & (pos < nfut)
        g = np.where(ok, future[b, np.clip(pos, 0, max(nfut - 1, 0))] if nfut else 0, 0)
        target[b] = g.astype(np.int32)
        if int(mode[b]) == MODE_COPY:
            ln = int(draft_len[b])
            vdraft[b, :ln] = draft[b, :ln]
        else:
            ln = gamma
            slots = 4 * np.arange(ln, dtype=np.uint64)
            coin = harness_key(seed, b, step, slots) & np.uint64(0xFFFFFFFF)
            alt = _token(harness_key(seed, b, step, slots + np.uint64(1)), V)
            gg = g[:ln].astype(np.int64)
            alt = np.where(alt == gg, (alt + 1) % V, alt)
            vdraft[b, :ln] = np.where(coin < thr, gg, alt).astype(np.int32)
        vlen[b] = ln
    return vdraft, vlen, target
