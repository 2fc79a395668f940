"""The bounded-wait failure path on the GPU, made to fire without any fault.

Every wait of the kernels is bounded; when one runs out the kernel records SWITCHSD_ROW_TIMEOUT in the
row's status word, gives every copy or message still addressed to its shared memory a second bounded
wait, and returns, so the context stays usable.  A child process sets
SWITCHSD_DIAG_MESSAGE_WAIT_POLLS=0: the rescan kernel's leader then gives up on the row's messages at
once, without waiting for them at all.  The test checks that every row reports the timeout with no copy
draft and an unchanged search result, that the verification's append in the same launch still happened,
and that the process goes on launching (a second fused step, a synchronize) without an error.  A process
without the variable gets status 0 on the same inputs.
"""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import json, sys
sys.path.insert(0, sys.argv[1])
import numpy as np, torch
import synth
from paper_2609_20186_gb300 import Session, bf16_tensor

wl = synth.get_workload("zipf_32k").scaled(name="timeout", B=8, L0=5000, steps=3)
ctx, lens = wl.contexts()
sess = Session(ctx, lens, wl.probe_weights(), k=wl.k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
               logit_tau=wl.logit_tau, future=wl.future(), harness=wl.harness_params(), d=wl.d)
sess.step(bf16_tensor(wl.hidden(0), sess.device))
first = sess.step_outputs()
sess.harness(0)
lens0 = sess.lens.cpu().numpy().copy()
sess.verify_step(bf16_tensor(wl.hidden(1), sess.device))
second = sess.step_outputs()
torch.cuda.synchronize()
print(json.dumps({"first": {k: first[k].tolist() for k in ("status", "mode", "len")},
                  "second": {k: second[k].tolist() for k in ("status", "mode", "len")},
                  "grew": (sess.lens.cpu().numpy() - lens0).tolist(),
                  "accept": sess.accept.cpu().numpy().tolist()}))
"""


def _child(env_extra):
    env = dict(os.environ)
    env.pop("SWITCHSD_DIAG_MESSAGE_WAIT_POLLS", None)
    env.update(env_extra)
    r = subprocess.run([sys.executable, "-c", CHILD, ROOT], env=env, capture_output=True, text=True,
                       timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    return json.loads(r.stdout.strip().splitlines()[-1])


def test_message_wait_runs_out_and_reports_timeout():
    out = _child({"SWITCHSD_DIAG_MESSAGE_WAIT_POLLS": "0"})
    for leg in ("first", "second"):
        assert all(s == 3 for s in out[leg]["status"]), out[leg]        # SWITCHSD_ROW_TIMEOUT
        assert all(m == 0 for m in out[leg]["mode"])                     # no repetition, no copy draft
        assert all(n == 0 for n in out[leg]["len"])
    # the verification inside the second launch appended a + 1 tokens to every row all the same
    assert all(a >= 0 for a in out["accept"])
    assert [g for g in out["grew"]] == [a + 1 for a in out["accept"]]


def test_without_the_diagnostic_no_row_times_out():
    out = _child({})
    for leg in ("first", "second"):
        assert all(s == 0 for s in out[leg]["status"]), out[leg]
