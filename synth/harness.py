"""Stand-in for the neural drafter and the target model's verification forward (host side).

The controller's verification input is the target model's greedy token after each draft prefix
(``target_argmax``, k+1 entries per row).  The target model is out of scope, so this harness
synthesises it from the draft with a seeded per-token agreement law:

- rows whose mode is not COPY get a neural draft of k seeded tokens (the drafter is out of scope);
- for each draft index i < len: the target agrees with draft[i] with probability ``p_in`` if the
  absolute position L + i lies inside a future span (``labels``), else ``p_out``, and never at
  i >= ``agree_cap``; a disagreeing target token is a seeded id different from draft[i];
- target[i] for i >= len (the bonus token and unused slots) is a seeded id.

All randomness comes from ``harness_key(seed, row, step, 4 * i + slot)`` with slots
``TOKEN_STREAMS``; the CUDA harness kernel implements the same chain, so both sides see identical
targets for identical drafts.  No controller arithmetic happens here.
"""
from __future__ import annotations

import numpy as np

from .rng import harness_key

TOKEN_STREAMS = {"agree": 0, "alt": 1, "neural": 2, "bonus": 3}
MODE_COPY = 1  # the documented ABI value of the copy mode


def _token(r: np.ndarray, V: int) -> np.ndarray:
    return ((r >> np.uint64(32)) % np.uint64(V)).astype(np.int64)


def harness_targets(params: dict, step: int, ctx_lens: np.ndarray, mode: np.ndarray,
                    draft: np.ndarray, draft_len: np.ndarray, labels: np.ndarray,
                    rows: np.ndarray | None = None):
    """Returns (vdraft [B, k], vlen [B], target [B, k+1]) as int32 arrays.

    ``rows`` (optional) restricts the work to those row indices (others are left zero); each row's
    result depends only on its own inputs.
    """
    B, k = draft.shape
    V = params["V"]
    L0 = params["L0"]
    thr_in = np.uint64(params["thr_in"])
    thr_out = np.uint64(params["thr_out"])
    agree_cap = params["agree_cap"]
    seed = params["seed"]
    vdraft = np.zeros((B, k), np.int32)
    vlen = np.zeros(B, np.int32)
    target = np.zeros((B, k + 1), np.int32)
    idx = np.arange(B) if rows is None else np.asarray(rows)
    i = np.arange(k + 1, dtype=np.uint64)
    nlab = labels.shape[1]
    for b in idx:
        b = int(b)
        L = int(ctx_lens[b])
        r_agree = harness_key(seed, b, step, 4 * i + 0)
        r_alt = harness_key(seed, b, step, 4 * i + 1)
        r_neural = harness_key(seed, b, step, 4 * i + 2)
        r_bonus = harness_key(seed, b, step, 4 * i + 3)
        if int(mode[b]) == MODE_COPY:
            ln = int(draft_len[b])
            d = np.zeros(k, np.int64)
            d[:ln] = draft[b, :ln]
        else:
            ln = k
            d = _token(r_neural[:k], V)
        vdraft[b, :ln] = d[:ln]
        vlen[b] = ln
        t = _token(r_bonus, V)
        for j in range(ln):
            p = L + j - L0
            lab = labels[b, p] if 0 <= p < nlab else 0
            thr = thr_in if lab else thr_out
            agree = (j < agree_cap) and ((r_agree[j] & np.uint64(0xFFFFFFFF)) < thr)
            if agree:
                t[j] = d[j]
            else:
                alt = int(_token(r_alt[j: j + 1], V)[0])
                if alt == int(d[j]):
                    alt = (alt + 1) % V
                t[j] = alt
        target[b] = t.astype(np.int32)
    return vdraft, vlen, target
