"""The oracle's pins catch plausible mistakes.

Each mutant plants one mistake in a copy of oracle/switchsd_oracle.c (an off-by-one, a reversed loop,
a wrong comparison, a dropped term, a missing step), is compiled on the CPU and routed under the
oracle's Python functions; the battery below -- drawn from the pins of test_oracle_*.py -- must fail
for every mutant and pass for the real oracle.  Nothing here touches the CUDA path.
"""
import ctypes
import itertools
import math
import os

import numpy as np
import pytest
import torch

import oracle
import synth

SRC = os.path.join(os.path.dirname(oracle.__file__), "switchsd_oracle.c")

MUTANTS = {
    "search: skips the earliest end": ("for (int32_t e = L - 2; e >= n - 1; --e)",
                                       "for (int32_t e = L - 2; e >= n; --e)"),
    "search: counts the suffix itself": ("for (int32_t e = L - 2; e >= n - 1; --e)",
                                         "for (int32_t e = L - 1; e >= n - 1; --e)"),
    "search: shortest n first": ("for (int32_t n = n_max; n >= n_min; --n)",
                                 "for (int32_t n = n_min; n <= n_max; ++n)"),
    "search: oldest occurrence first": ("for (int32_t e = L - 2; e >= n - 1; --e)",
                                        "for (int32_t e = n - 1; e <= L - 2; ++e)"),
    "search: compares a shifted suffix": ("x[e - i] == x[L - 1 - i]", "x[e - i] == x[L - 2 - i]"),
    "search: needs one token less": ("while (i < n && x[e - i]", "while (i < n - 1 && x[e - i]"),
    "probe: drops the last term": ("for (int32_t j = 0; j < d; ++j)\n        z +=",
                                   "for (int32_t j = 0; j < d - 1; ++j)\n        z +="),
    "probe: squares the weight": ("z += oracle_bf16_to_double(w[j]) * oracle_bf16_to_double(h[j]);",
                                  "z += oracle_bf16_to_double(w[j]) * oracle_bf16_to_double(w[j]);"),
    "bf16: wrong shift": ("((uint32_t)v) << 16", "((uint32_t)v) << 15"),
    "mlp: no ReLU": ("if (a < 0.0) a = 0.0;", ""),
    "mlp: ignores b1": ("double a = (b1 != NULL) ? (double)b1[u] : 0.0;", "double a = 0.0;"),
    "mlp: transposed W1": ("W1[(int64_t)u * d + j]", "W1[(int64_t)j * H1 + u]"),
    "switch: strict threshold": ("(float)z >= logit_tau", "(float)z > logit_tau"),
    "switch: strict kappa": ("n_star >= kappa", "n_star > kappa"),
    "switch: draft not clipped": ("int32_t n = avail < k ? avail : k;", "int32_t n = k;"),
    "switch: draft off by one": ("draft[i] = x[e_star + 1 + i];", "draft[i] = x[e_star + i];"),
    "verify: no bonus token": ("row[*L + a] = target[a];\n    *L += a + 1;", "*L += a;"),
    "verify: capacity off by one": ("if (*L + a + 1 > cap) {", "if (*L + a + 1 >= cap) {"),
    "verify: accepts one past the mismatch": ("while (a < len && draft[a] == target[a]) ++a;",
                                              "while (a < len && draft[a] == target[a]) ++a;\n"
                                              "    if (a < len) ++a;"),
    "sampled: accepts a tie": ("if (!(prod < p[a])) break;", "if (!(prod <= p[a])) break;"),
    "sampled: ignores q": ("float qa = (q != NULL) ? q[a] : 1.0f;", "float qa = 1.0f;"),
    "sampled: inverts the ratio": ("float prod = u[a] * qa;\n        if (!(prod < p[a])) break;",
                                   "float prod = u[a] * p[a];\n        if (!(prod < qa)) break;"),
    "sampled: wrong resample": ("row[*L + a] = resample[a];", "row[*L + a] = resample[a > 0 ? a - 1 : 0];"),
    "labels: counts the window itself": ("for (int32_t s2 = 0; s2 < s; ++s2) {", "for (int32_t s2 = 0; s2 <= s; ++s2) {"),
    "labels: labels the window start only": ("for (int32_t j = s; j < s + n; ++j) y[j] = 1;", "y[s] = 1;"),
    "labels: last window skipped": ("for (int32_t s = 0; s + n <= L; ++s)", "for (int32_t s = 0; s + n < L; ++s)"),
    "labels: one token short": ("while (i < n && x[s2 + i] == x[s + i]) ++i;", "while (i < n - 1 && x[s2 + i] == x[s + i]) ++i;"),
    "candidates: oldest first": ("    for (int32_t e = L - 2; e >= 0; --e) {\n        /* common suffix",
                                 "    for (int32_t e = 0; e <= L - 2; ++e) {\n        /* common suffix"),
    "candidates: n_min gate": ("if (m >= kappa && n < W) cand_end[n++] = e;", "if (m >= n_min && n < W) cand_end[n++] = e;"),
    "candidates: latest on a tie": ("        if (a > a_best) {", "        if (a >= a_best) {"),
    "candidates: first candidate's bonus": ("row[*L + a_best] = target[(int64_t)best * (D + 1) + a_best];",
                                            "row[*L + a_best] = target[a_best];"),
}


def _brute(x, n_min, n_max):
    L = len(x)
    hits = [(n, e) for n in range(n_min, n_max + 1) if n <= L
            for e in range(0, L - 1) if e - n + 1 >= 0 and tuple(x[e - n + 1: e + 1]) == tuple(x[L - n:])]
    return min(hits, key=lambda t: (-t[0], -t[1])) if hits else (0, -1)


def _tb(bits):
    return torch.from_numpy(np.ascontiguousarray(bits, np.uint16).view(np.int16)).view(torch.bfloat16)


def battery() -> list:
    """Returns the names of the checks that fail for the oracle currently routed."""
    failed = []

    def check(name, ok):
        if not ok:
            failed.append(name)

    # search vs brute force (ternary contexts up to length 7, three n ranges)
    ok = True
    for n_min, n_max in ((1, 3), (2, 4), (3, 8)):
        for L in range(1, 8):
            for x in itertools.product(range(3), repeat=L):
                if oracle.longest_suffix_match(np.array(x, np.int32), n_min, n_max) != \
                        _brute(list(x), n_min, n_max):
                    ok = False
                    break
            if not ok:
                break
    check("search brute force", ok)
    # probe vs torch float64
    rng = np.random.default_rng(0)
    d = 96
    h = synth.bf16_bits_from_f32(rng.standard_normal(d).astype(np.float32))
    w = synth.bf16_bits_from_f32(rng.standard_normal(d).astype(np.float32) / 8)
    ref = torch.dot(_tb(w).double(), _tb(h).double()).item()
    check("probe vs torch", abs(oracle.probe_linear(h, w) - ref) <= 1e-12 * max(1, abs(ref)))
    H1 = 12
    W1 = synth.bf16_bits_from_f32(rng.standard_normal((H1, d)).astype(np.float32) / 8)
    w2 = synth.bf16_bits_from_f32(rng.standard_normal(H1).astype(np.float32))
    b1 = rng.standard_normal(H1).astype(np.float32)
    refm = (torch.relu(_tb(W1).double() @ _tb(h).double() + torch.from_numpy(b1).double())
            @ _tb(w2).double() + 0.5).item()
    check("mlp vs torch", abs(oracle.probe_mlp(h, W1, w2, b1=b1, b2=0.5) - refm) <= 1e-9)
    # switch hand cases
    x = np.array([10, 11, 12, 13, 14, 99, 11, 12, 13], np.int32)
    check("switch copy", oracle.switch(True, 3, 3, 0.7, 0.0, 2, 3, x) == (1, [14, 99, 11]))
    check("switch tie", oracle.switch(True, 3, 3, 0.0, 0.0, 2, 3, x)[0] == 1)
    check("switch kappa", oracle.switch(True, 3, 3, 1.0, 0.0, 3, 3, x)[0] == 1)
    y = np.array([8, 9, 1, 2, 8, 9], np.int32)
    check("switch clip", oracle.switch(True, 2, 1, 1.0, 0.0, 2, 16, y) == (1, [1, 2, 8, 9]))
    # verify hand cases
    row = np.zeros(16, np.int32)
    row[:3] = [1, 2, 3]
    check("verify partial", oracle.verify_row(row, 3, 16, [4, 5, 6], [4, 5, 0, 1]) == (6, 2, 0)
          and row[:6].tolist() == [1, 2, 3, 4, 5, 0])
    row = np.zeros(6, np.int32)
    row[:4] = [1, 2, 3, 4]
    check("verify fits exactly", oracle.verify_row(row, 4, 6, [5, 9], [5, 6, 7]) == (6, 1, 0))
    # sampled verification hand cases (test_oracle_sampled.py)
    row = np.zeros(16, np.int32)
    row[:3] = [1, 2, 3]
    check("sampled partial", oracle.verify_sampled_row(row, 3, 16, [4, 5, 6], [0.6, 0.4, 0.9], [0.5] * 3,
                                                       [7, 8, 9, 10]) == (5, 1, 0) and row[4] == 8)
    row = np.zeros(8, np.int32)
    check("sampled tie", oracle.verify_sampled_row(row, 1, 8, [4], [0.5], [0.5], [7, 9])[1] == 0)
    row = np.zeros(8, np.int32)
    check("sampled q", oracle.verify_sampled_row(row, 1, 8, [4, 5], [0.3, 0.3], [0.5, 0.7], [7, 8, 9],
                                                 q=[0.5, 0.5])[1] == 1)
    row = np.zeros(8, np.int32)
    check("sampled low p", oracle.verify_sampled_row(row, 1, 8, [4], [0.2], [0.5], [7, 9], q=[1.0])[1] == 0)
    # copy-mode labels (test_oracle_labels.py)
    check("labels repeat", oracle.copy_labels([1, 2, 3, 4, 5, 9, 1, 2, 3, 4, 5], 5).tolist() == [0] * 6 + [1] * 5)
    check("labels unique", oracle.copy_labels([1, 2, 3, 4, 5, 6], 5).sum() == 0)
    check("labels short", oracle.copy_labels([1, 2, 3, 4, 8, 1, 2, 3, 4], 5).sum() == 0)
    # candidates (test_oracle_candidates.py)
    x = np.array([1, 2, 3, 9, 1, 2, 3, 8, 1, 2, 3], np.int32)
    check("candidates order", oracle.candidates(x, n_min=2, n_max=4, kappa=3, z=1.0, logit_tau=0.0, W=4, D=3)
          == (1, [[8, 1, 2], [9, 1, 2]], [6, 2]))
    y = np.array([5, 2, 3, 9, 1, 2, 3], np.int32)
    check("candidates gate", oracle.candidates(y, n_min=2, n_max=4, kappa=3, z=1.0, logit_tau=0.0, W=4, D=3)[0] == 2)
    row = np.zeros(32, np.int32)
    check("candidates choose", oracle.verify_candidates_row(row, 1, 32, [[4, 5], [4, 6]], [[4, 9, 0], [4, 8, 0]])
          == (3, 1, 0, 0))
    row = np.zeros(32, np.int32)
    row[:3] = [1, 2, 3]
    check("candidates bonus", oracle.verify_candidates_row(row, 3, 32, [[4, 5, 6], [4, 7, 8, 9]],
                                                           [[4, 0, 0, 0, 0], [4, 7, 8, 1, 0]]) == (7, 3, 1, 0)
          and row[6] == 1)
    return failed


def _compile_mutant(tmp_path, name, old, new):
    text = open(SRC).read()
    assert text.count(old) >= 1, f"mutation site of {name!r} not found"
    src = tmp_path / "mutant.c"
    src.write_text(text.replace(old, new))
    lib = tmp_path / "libmutant.so"
    oracle.compile_library(str(src), str(lib))
    return oracle.configure(ctypes.CDLL(str(lib)))


def test_real_oracle_passes_battery():
    assert battery() == []


@pytest.mark.parametrize("name", list(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    lib = _compile_mutant(tmp_path, name, old, new)
    previous = oracle.use_library(lib)
    try:
        failed = battery()
    finally:
        oracle.use_library(previous)
    assert failed, f"mutant {name!r} passed every pin"
