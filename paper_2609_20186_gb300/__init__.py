"""GB300-native (sm_103a) SwitchSD per-step controller.

The controller (paper: "To Copy or Not to Copy: Controlling Speculative Decoding via Intrinsic Model
Signals", §3.3, Fig. 1) runs in hand-written CUDA kernels behind the C ABI of ``include/switchsd.h``
(``libswitchsd.so``).  This package holds the kernels (``csrc/``), their build (``build.py``), the
ctypes binding (``binding.py``, same names as the C functions) and a device-resident session helper
(``session.py``).  Importing the package does not load the library; the first call does, and fails
loudly if it was not built.
"""
from .binding import (  # noqa: F401
    switchsd_step, switchsd_verify, switchsd_verify_step, switchsd_harness_target, switchsd_params,
    switchsd_verify_params, switchsd_harness_params, NgramIndex, load, strerror, abi_version,
    MODE_NO_REP, MODE_COPY, MODE_REP_NO_COPY, PROBE_LINEAR, PROBE_MLP,
)
from .session import HostPlan, Session, bf16_tensor  # noqa: F401
