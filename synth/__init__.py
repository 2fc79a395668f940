"""Seeded synthetic inputs for the SwitchSD controller.

This package is the only code that serves both the CUDA path and the CPU oracle.  It generates inputs
(contexts, hidden states, probe weights, the target's future tokens) and, in ``harness``, the stand-in for the
out-of-scope neural drafter and target model.  It contains none of the controller's arithmetic: no
n-gram search, no probe evaluation, no switch and no verification.
"""
from .rng import splitmix64, harness_key, bf16_bits_from_f32, f32_from_bf16_bits  # noqa: F401
from .workloads import WORKLOADS, Workload, get_workload  # noqa: F401
from .harness import harness_targets, harness_sampled, harness_candidates  # noqa: F401
