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
32 bits; slot 1: the replacement token, a token being (word >> 32) mod V; slots 2 and 3 feed the
sampled stand-in below).  The CUDA harness kernel
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


def harness_sampled(params: dict, step: int, ctx_lens: np.ndarray, mode: np.ndarray,
                    draft: np.ndarray, draft_len: np.ndarray, future: np.ndarray, rows=None):
    """The stand-in at temperature T > 0 (the inputs of the sampled verification).  Returns
    (vdraft [B, k], vlen [B], p [B, k], q [B, k], u [B, k], resample [B, k+1]); with g = the target
    stream at the draft positions:

    - p[i] = p_hit where vdraft[i] == g[i], else p_miss (i < vlen; 0 beyond);
    - q[i] = 1 for a copy row, q_neural for a neural row (i < vlen; 1 beyond);
    - u[i] = (key(4 i + 2) >> 40) * 2^-24 for every i < k (exact in binary32);
    - resample[i] = g[i] for i < vlen, except where g[i] == vdraft[i]: then the token of key(4 i + 3),
      plus one mod V if that equals vdraft[i] (the residual excludes the rejected token);
      resample[vlen] = g[vlen]; 0 beyond.
    """
    B, k = draft.shape
    V = params["V"]
    seed = params["seed"]
    p_hit, p_miss = np.float32(params["p_hit"]), np.float32(params["p_miss"])
    q_neural = np.float32(params["q_neural"])
    vdraft, vlen, g = harness_targets(params, step, ctx_lens, mode, draft, draft_len, future, rows)
    p = np.zeros((B, k), np.float32)
    q = np.ones((B, k), np.float32)
    u = np.zeros((B, k), np.float32)
    resample = np.zeros((B, k + 1), np.int32)
    idx = range(B) if rows is None else rows
    slots = 4 * np.arange(k, dtype=np.uint64)
    for b in idx:
        b = int(b)
        ln = int(vlen[b])
        d = vdraft[b, :ln].astype(np.int64)
        gg = g[b, :ln].astype(np.int64)
        p[b, :ln] = np.where(d == gg, p_hit, p_miss)
        if int(mode[b]) != MODE_COPY:
            q[b, :ln] = q_neural
        word = harness_key(seed, b, step, slots + np.uint64(2))
        u[b] = ((word >> np.uint64(40)).astype(np.float64) * 2.0 ** -24).astype(np.float32)
        alt = _token(harness_key(seed, b, step, slots[:ln] + np.uint64(3)), V)
        alt = np.where(alt == d, (alt + 1) % V, alt)
        resample[b, :ln] = np.where(gg == d, alt, gg).astype(np.int32)
        resample[b, ln] = g[b, ln]
    return vdraft, vlen, p, q, u, resample


def harness_candidates(params: dict, step: int, ctx_lens: np.ndarray, mode: np.ndarray, cand: np.ndarray,
                       cand_len: np.ndarray, ncand: np.ndarray, future: np.ndarray, rows=None):
    """The stand-in for the verification of W copy candidates.  Returns (vcand [B, W, D], vlen [B, W],
    vn [B], target [B, W, D+1]): a copy row passes its candidates on; any other row gets
    min(gamma, D) neural tokens (the law of harness_targets) as its one candidate; target[b][w] is the
    target stream at the row's next D+1 positions for every kept candidate (the target's greedy token
    after any prefix the verification can accept), 0 for unused slots."""
    B, W, D = cand.shape
    V, L0, seed = params["V"], params["L0"], params["seed"]
    gamma = min(params["gamma"], D)
    thr = np.uint64(params["thr_neural"])
    nfut = future.shape[1]
    vcand = np.zeros((B, W, D), np.int32)
    vlen = np.zeros((B, W), np.int32)
    vn = np.zeros(B, np.int32)
    target = np.zeros((B, W, D + 1), np.int32)
    idx = range(B) if rows is None else rows
    i = np.arange(D + 1, dtype=np.int64)
    for b in idx:
        b = int(b)
        pos = int(ctx_lens[b]) - L0 + i
        ok = (pos >= 0) & (pos < nfut)
        g = np.where(ok, future[b, np.clip(pos, 0, max(nfut - 1, 0))] if nfut else 0, 0).astype(np.int64)
        if int(mode[b]) == MODE_COPY:
            n = min(max(int(ncand[b]), 0), W)
            for w in range(n):
                ln = int(cand_len[b, w])
                vcand[b, w, :ln] = cand[b, w, :ln]
                vlen[b, w] = ln
        else:
            n = 1
            slots = 4 * np.arange(gamma, dtype=np.uint64)
            coin = harness_key(seed, b, step, slots) & np.uint64(0xFFFFFFFF)
            alt = _token(harness_key(seed, b, step, slots + np.uint64(1)), V)
            gg = g[:gamma]
            alt = np.where(alt == gg, (alt + 1) % V, alt)
            vcand[b, 0, :gamma] = np.where(coin < thr, gg, alt).astype(np.int32)
            vlen[b, 0] = gamma
        vn[b] = n
        target[b, :n] = g.astype(np.int32)
    return vcand, vlen, vn, target
