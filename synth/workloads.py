"""The five seeded synthetic workloads and their generators.

The paper measures on HumanEval, Math500, CNN/DailyMail and MT-Bench with real models (§4).  None of
those is used or reproduced here: every context is synthetic, built to have the structure those
workloads give the controller -- long generations with planted verbatim copies of earlier spans
(copy intent) and short accidental n-gram repeats (§3.1).  Token ids are int32 in [0, V).

Recipes (one seed per workload):

- ``planted``  (B=1, 2,048 tokens): uniform ids; two planted copies of 64-token earlier spans, the
  second ending at the context's end; 20 accidental 3-gram repeats.  Three variants fix the expected
  switch case: ``copy`` (probe logit > 0 by construction), ``nocopy`` (logit < 0), ``norep`` (the
  final token occurs nowhere else).
- ``uniform_spans`` (B=64, 8,192): uniform ids; 10 % of positions inside planted copies of length
  32 + Geom(1/64) - 1, at most 512; accidental 3- or 4-gram repeats at rate 1/200.
- ``zipf_spans`` (B=64, 32,768): Zipf(1.1) ids (rank -> id by a seeded permutation), which repeat
  short n-grams densely by themselves; 5 % planted copy coverage with the same length law.
- ``code`` (B=256, 16,384): eight seeded 200-token blocks per row, tiled in seeded order with 1-3
  random token edits per instance, after a uniform filler of the remainder.
- ``mixed`` (B=16, 131,072): first half Zipf(1.1) prose; second half Zipf filler with 30 % planted
  copies of length 16 + Geom(1/256) - 1, at most 4,096, sourced anywhere earlier.

The target model's greedy continuation of each row (``future``) follows the row's token law with
``future_coverage`` of planted copies of earlier spans, 10 % of whose tokens are edited; the target
stand-in (synth.harness) reads it.  Hidden states are bf16 N(0, 1) per (step, row); the linear probe is w ~ N(0, 1/d) in bf16 so that the
logit is O(1); the two-layer probe is W1 ~ N(0, 1/d) [256, d], w2 ~ N(0, 1/256), no biases.
"""
from __future__ import annotations

import dataclasses
import math
from dataclasses import dataclass

import numpy as np

from .rng import bf16_bits_from_f32

# Stream ids mixed into numpy SeedSequences so that each kind of input has its own stream.
_S_CTX, _S_HIDDEN, _S_PROBE, _S_FUTURE, _S_BLOCKS, _S_PERM = 1, 2, 3, 4, 5, 9


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    L0: int
    V: int
    d: int
    k: int
    n_min: int
    n_max: int
    steps: int
    seed: int
    structure: str
    kappa: int = 0                 # 0 means kappa = n_min
    tau: float = 0.5
    probe_kind: int = 0            # 0 linear w[d]; 1 two-layer W1[H1, d] + w2[H1]
    probe_hidden: int = 0
    coverage: float = 0.0          # planted copy coverage of the initial context
    span_min: int = 32
    span_p: float = 1.0 / 64.0
    span_max: int = 512
    accidental_rate: float = 0.0   # explicit accidental short repeats per position
    future_coverage: float = 0.0   # planted-copy share of the target's future tokens
    p_in: float = 0.9              # per-token survival of a planted future copy (else an edit)
    p_neural: float = 0.75         # per-token agreement of the neural draft with the target
    gamma: int = 6                 # neural draft length (the drafter's lookahead, Table 3)
    p_hit: float = 0.9             # sampled stand-in: target probability of a draft token on the stream
    p_miss: float = 0.05           # ... and of one off it (the configs' "p=0.9 inside / 0.05 outside")
    q_neural: float = 0.8          # ... the neural drafter's probability of its own token
    variant: str = ""              # planted workload: copy | nocopy | norep

    @property
    def cap(self) -> int:
        """Row capacity: initial length plus the most the context can grow, rounded to 4 tokens."""
        need = self.L0 + self.steps * (self.k + 1)
        return (need + 3) // 4 * 4

    @property
    def logit_tau(self) -> float:
        """logit(tau) rounded to binary32: the decision threshold in logit space."""
        t = self.tau
        if t <= 0.0:
            return float("-inf")
        if t >= 1.0:
            return float("inf")
        return float(np.float32(math.log(t / (1.0 - t))))

    @property
    def kappa_eff(self) -> int:
        return self.kappa if self.kappa > 0 else self.n_min

    def scaled(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    # ------------------------------------------------------------------ generators
    def contexts(self) -> tuple[np.ndarray, np.ndarray]:
        """ctx int32 [B, cap] (zeros beyond L0) and lens int32 [B] (all L0)."""
        ctx = np.zeros((self.B, self.cap), np.int32)
        for b in range(self.B):
            ctx[b, : self.L0] = self.context_row(b)
        return ctx, np.full(self.B, self.L0, np.int32)

    def context_row(self, b: int) -> np.ndarray:
        rng = np.random.default_rng([self.seed, _S_CTX, b])
        fn = _GENERATORS[self.structure]
        x = fn(self, rng, b)
        assert x.shape == (self.L0,) and x.dtype == np.int32
        return x

    def probe_weights(self) -> np.ndarray:
        """bf16 bits: w[d] (linear) or W1[H1, d] followed by w2[H1] (two-layer), flattened."""
        rng = np.random.default_rng([self.seed, _S_PROBE])
        if self.structure == "planted":
            return _planted_probe(self)
        if self.probe_kind == 0:
            w = rng.standard_normal(self.d, dtype=np.float32) / np.float32(math.sqrt(self.d))
            return bf16_bits_from_f32(w)
        H1 = self.probe_hidden
        W1 = rng.standard_normal((H1, self.d), dtype=np.float32) / np.float32(math.sqrt(self.d))
        w2 = rng.standard_normal(H1, dtype=np.float32) / np.float32(math.sqrt(H1))
        return np.concatenate([bf16_bits_from_f32(W1).reshape(-1), bf16_bits_from_f32(w2)])

    def hidden(self, step: int) -> np.ndarray:
        """bf16 bits [B, d] for one step: N(0, 1)."""
        if self.structure == "planted":
            return _planted_hidden(self)
        rng = np.random.default_rng([self.seed, _S_HIDDEN, step])
        h = rng.standard_normal((self.B, self.d), dtype=np.float32)
        return bf16_bits_from_f32(h)

    def hidden_all(self) -> np.ndarray:
        """bf16 bits [steps, B, d]."""
        out = np.empty((self.steps, self.B, self.d), np.uint16)
        for t in range(self.steps):
            out[t] = self.hidden(t)
        return out

    def future_row(self, b: int) -> np.ndarray:
        """The target model's greedy continuation of row b: int32 tokens for absolute positions
        [L0, cap).  Drawn with the row's own token law, then ``future_coverage`` of it is
        overwritten with planted copies of earlier spans (context or earlier future), each copied
        token kept with probability ``p_in`` (else replaced: an edit)."""
        n = self.cap - self.L0
        rng = np.random.default_rng([self.seed, _S_FUTURE, b])
        if self.structure == "planted":
            return _planted_future(self, rng)
        x = self.context_row(b)
        full = np.concatenate([x, _FUTURE_BASE[self.structure](self, rng, b, n)]).astype(np.int32)
        if self.future_coverage > 0.0:
            _plant_spans(full, rng, self.future_coverage, self.span_min, self.span_p,
                         self.span_max, (self.L0, self.cap), keep=self.p_in, V=self.V)
        return full[self.L0:].copy()

    def future(self) -> np.ndarray:
        """int32 [B, cap - L0]: every row's future_row."""
        out = np.zeros((self.B, self.cap - self.L0), np.int32)
        for b in range(self.B):
            out[b] = self.future_row(b)
        return out

    def harness_params(self) -> dict:
        """Integer parameters of the target stand-in (see synth.harness)."""
        return {
            "seed": self.seed,
            "V": self.V,
            "L0": self.L0,
            "gamma": min(self.gamma, self.k),
            "thr_neural": _prob_to_thr(self.p_neural),
            "p_hit": self.p_hit,
            "p_miss": self.p_miss,
            "q_neural": self.q_neural,
        }

    def expected_planted(self) -> dict:
        """For the planted workload: the match, draft and verification the construction fixes."""
        assert self.structure == "planted"
        x = self.context_row(0)
        src = _PLANTED_SRC2
        e_star = src + 63
        out = {"match_n": self.n_max, "match_end": e_star,
               "draft": x[e_star + 1: e_star + 1 + self.k].tolist()}
        if self.variant == "norep":
            out.update(match_n=0, match_end=-1, draft=[], mode=0)
        elif self.variant == "nocopy":
            out.update(draft=[], mode=2)
        else:
            out.update(mode=1, accept=_PLANTED_AGREE)
        return out


def _prob_to_thr(p: float) -> int:
    """Probability -> threshold on a uniform 32-bit word (2**32 means always)."""
    if p >= 1.0:
        return 1 << 32
    if p <= 0.0:
        return 0
    return int(round(p * (1 << 32)))


def _span_len(rng, lo: int, p: float, hi: int) -> int:
    return int(min(lo + int(rng.geometric(p)) - 1, hi))


def _zipf_sampler(V: int, a: float, seed: int):
    ranks = np.arange(1, V + 1, dtype=np.float64)
    w = ranks ** (-a)
    cdf = np.cumsum(w)
    cdf /= cdf[-1]
    perm = np.random.default_rng([seed, _S_PERM]).permutation(V).astype(np.int32)

    def draw(rng, n):
        u = rng.random(n)
        r = np.searchsorted(cdf, u, side="right")
        r = np.minimum(r, V - 1)
        return perm[r]

    return draw


_ZIPF_CACHE: dict = {}


def _zipf(wl: Workload):
    key = (wl.V, wl.seed)
    if key not in _ZIPF_CACHE:
        _ZIPF_CACHE[key] = _zipf_sampler(wl.V, 1.1, wl.seed)
    return _ZIPF_CACHE[key]


def _plant_spans(x: np.ndarray, rng, coverage: float, lo: int, p: float, hi: int,
                 region: tuple[int, int], keep: float = 1.0, V: int = 0) -> None:
    """Overwrite ``coverage`` of positions in ``region`` with copies of earlier spans; with
    keep < 1 each copied token is replaced by a random id with probability 1 - keep."""
    r0, r1 = region
    target = int(coverage * (r1 - r0))
    used = np.zeros(x.shape[0], bool)
    spans = []
    covered = 0
    tries = 0
    while covered < target and tries < 100000:
        tries += 1
        ln = _span_len(rng, lo, p, hi)
        a = max(r0, ln)
        if a > r1 - ln:
            continue
        dst = int(rng.integers(a, r1 - ln + 1))
        if used[dst: dst + ln].any():
            continue
        src = int(rng.integers(0, dst - ln + 1))
        used[dst: dst + ln] = True
        spans.append((dst, src, ln))
        covered += ln
    for dst, src, ln in sorted(spans):
        x[dst: dst + ln] = x[src: src + ln]
        if keep < 1.0:
            edit = rng.random(ln) >= keep
            x[dst: dst + ln][edit] = rng.integers(0, V, int(edit.sum()), dtype=np.int64)


def _accidental_repeats(x: np.ndarray, rng, count: int, nlo: int, nhi: int) -> None:
    L = x.shape[0]
    for _ in range(count):
        n = int(rng.integers(nlo, nhi + 1))
        src = int(rng.integers(0, L - 2 * n))
        dst = int(rng.integers(src + n, L - n + 1))
        x[dst: dst + n] = x[src: src + n]


# ---- planted (B = 1) ------------------------------------------------------------------------
_PLANTED_SRC2 = 300     # source of the copy that ends the context
_PLANTED_SRC1 = 800
_PLANTED_DST1 = 1200


def _gen_planted(wl: Workload, rng, b: int) -> np.ndarray:
    L = wl.L0
    x = rng.integers(0, wl.V, L, dtype=np.int64).astype(np.int32)
    # accidental 3-grams: sourced from [400, 790), written into [1300, L - 100)
    for _ in range(20):
        src = int(rng.integers(400, 787))
        dst = int(rng.integers(1300, L - 103))
        x[dst: dst + 3] = x[src: src + 3]
    x[_PLANTED_DST1: _PLANTED_DST1 + 64] = x[_PLANTED_SRC1: _PLANTED_SRC1 + 64]
    x[L - 64: L] = x[_PLANTED_SRC2: _PLANTED_SRC2 + 64]
    if wl.variant == "norep":
        seen = set(x[: L - 1].tolist())
        v = int(rng.integers(0, wl.V))
        while v in seen:
            v = (v + 1) % wl.V
        x[L - 1] = v
    return x


_PLANTED_AGREE = 5      # the target follows the planted continuation for 5 tokens


def _planted_future(wl: Workload, rng) -> np.ndarray:
    """The target continues the planted copy for _PLANTED_AGREE tokens, then departs from it."""
    n = wl.cap - wl.L0
    x = wl.context_row(0)
    cont = x[_PLANTED_SRC2 + 64: _PLANTED_SRC2 + 64 + wl.k]
    g = rng.integers(0, wl.V, n, dtype=np.int64).astype(np.int32)
    g[:_PLANTED_AGREE] = cont[:_PLANTED_AGREE]
    if g[_PLANTED_AGREE] == cont[_PLANTED_AGREE]:
        g[_PLANTED_AGREE] = (g[_PLANTED_AGREE] + 1) % wl.V
    return g


def _planted_hidden(wl: Workload) -> np.ndarray:
    rng = np.random.default_rng([wl.seed, _S_HIDDEN, 0])
    h = rng.standard_normal((wl.B, wl.d), dtype=np.float32)
    return bf16_bits_from_f32(h)


def _planted_probe(wl: Workload) -> np.ndarray:
    """w_j = s * |g_j| / sqrt(d) * sign(h_j): every product w_j h_j has sign s, so the logit's sign is
    s by construction (s = -1 for the nocopy variant)."""
    from .rng import f32_from_bf16_bits
    h = f32_from_bf16_bits(_planted_hidden(wl)[0])
    rng = np.random.default_rng([wl.seed, _S_PROBE])
    g = np.abs(rng.standard_normal(wl.d, dtype=np.float32)) / np.float32(math.sqrt(wl.d))
    s = np.float32(-1.0 if wl.variant == "nocopy" else 1.0)
    w = s * g * np.sign(h).astype(np.float32)
    return bf16_bits_from_f32(w)


# ---- the others -----------------------------------------------------------------------------
def _gen_uniform_spans(wl: Workload, rng, b: int) -> np.ndarray:
    x = rng.integers(0, wl.V, wl.L0, dtype=np.int64).astype(np.int32)
    _accidental_repeats(x, rng, int(round(wl.L0 * wl.accidental_rate)), 3, 4)
    _plant_spans(x, rng, wl.coverage, wl.span_min, wl.span_p, wl.span_max, (0, wl.L0))
    return x


def _gen_zipf_spans(wl: Workload, rng, b: int) -> np.ndarray:
    x = _zipf(wl)(rng, wl.L0).astype(np.int32)
    _plant_spans(x, rng, wl.coverage, wl.span_min, wl.span_p, wl.span_max, (0, wl.L0))
    return x


def _code_blocks(wl: Workload, b: int) -> np.ndarray:
    rng = np.random.default_rng([wl.seed, _S_BLOCKS, b])
    return rng.integers(0, wl.V, (8, 200), dtype=np.int64).astype(np.int32)


def _code_instances(wl: Workload, rng, blocks: np.ndarray, n_inst: int) -> np.ndarray:
    out = np.empty(n_inst * 200, np.int32)
    for i in range(n_inst):
        inst = blocks[int(rng.integers(0, 8))].copy()
        n_edit = int(rng.integers(1, 4))
        pos = rng.integers(0, 200, n_edit)
        inst[pos] = rng.integers(0, wl.V, n_edit, dtype=np.int64)
        out[200 * i: 200 * (i + 1)] = inst
    return out


def _gen_code(wl: Workload, rng, b: int) -> np.ndarray:
    L = wl.L0
    blocks = _code_blocks(wl, b)
    n_inst = L // 200
    filler = L - n_inst * 200
    x = np.empty(L, np.int32)
    x[:filler] = rng.integers(0, wl.V, filler, dtype=np.int64)
    x[filler:] = _code_instances(wl, rng, blocks, n_inst)
    return x


def _gen_mixed(wl: Workload, rng, b: int) -> np.ndarray:
    L = wl.L0
    x = _zipf(wl)(rng, L).astype(np.int32)
    _plant_spans(x, rng, wl.coverage, wl.span_min, wl.span_p, wl.span_max, (L // 2, L))
    return x


def _fut_uniform(wl, rng, b, n):
    return rng.integers(0, wl.V, n, dtype=np.int64).astype(np.int32)


def _fut_zipf(wl, rng, b, n):
    return _zipf(wl)(rng, n).astype(np.int32)


def _fut_code(wl, rng, b, n):
    """The code rows keep tiling their eight blocks (with 1-3 edits per instance)."""
    inst = _code_instances(wl, rng, _code_blocks(wl, b), (n + 199) // 200)
    return inst[:n]


_FUTURE_BASE = {"uniform_spans": _fut_uniform, "zipf_spans": _fut_zipf, "code": _fut_code,
                "mixed": _fut_zipf}


_GENERATORS = {
    "planted": _gen_planted,
    "uniform_spans": _gen_uniform_spans,
    "zipf_spans": _gen_zipf_spans,
    "code": _gen_code,
    "mixed": _gen_mixed,
}


def _planted(variant: str) -> Workload:
    return Workload(name=f"planted_{variant}", B=1, L0=2048, V=128256, d=4096, k=8, n_min=3,
                    n_max=8, steps=1, seed=1001, structure="planted", variant=variant)


WORKLOADS: dict[str, Workload] = {
    "planted_copy": _planted("copy"),
    "planted_nocopy": _planted("nocopy"),
    "planted_norep": _planted("norep"),
    "uniform_8k": Workload(name="uniform_8k", B=64, L0=8192, V=128256, d=4096, k=8, n_min=3,
                           n_max=8, steps=256, seed=1002, structure="uniform_spans", coverage=0.10,
                           accidental_rate=1.0 / 200.0, future_coverage=0.10),
    "zipf_32k": Workload(name="zipf_32k", B=64, L0=32768, V=128256, d=4096, k=16, n_min=3,
                         n_max=8, steps=512, seed=1003, structure="zipf_spans", coverage=0.05,
                         future_coverage=0.05),
    "code_16k": Workload(name="code_16k", B=256, L0=16384, V=152064, d=5120, k=8, n_min=3,
                         n_max=8, steps=256, seed=1004, structure="code", probe_kind=1,
                         probe_hidden=256, future_coverage=0.80),
    "mixed_128k": Workload(name="mixed_128k", B=16, L0=131072, V=152064, d=5120, k=32, n_min=2,
                           n_max=12, steps=128, seed=1005, structure="mixed", coverage=0.30,
                           span_min=16, span_p=1.0 / 256.0, span_max=4096, future_coverage=0.30),
}


def get_workload(name: str) -> Workload:
    return WORKLOADS[name]
