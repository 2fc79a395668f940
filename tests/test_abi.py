"""The C ABI library without a GPU: it loads, exports every function include/*.h declares, and its
host-side validation returns the documented codes before any CUDA call is made."""
import ctypes
import math
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
INCLUDE = os.path.join(ROOT, "include")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_20186_gb300 import build, binding
    build.build()
    return binding.load()


def declared_functions():
    names = set()
    for f in os.listdir(INCLUDE):
        if not f.endswith(".h"):
            continue
        text = open(os.path.join(INCLUDE, f)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"\b(switchsd_\w+)\s*\(", text):
            names.add(m.group(1))
    return sorted(names)


def test_headers_declare_the_boundary():
    names = declared_functions()
    for must in ("switchsd_step", "switchsd_verify", "switchsd_strerror", "switchsd_abi_version",
                 "switchsd_harness_target"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2609_20186_gb300 import build
    out = subprocess.run(["nm", "-D", "--defined-only", build.LIB], capture_output=True, text=True,
                         check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if line.strip()}
    for name in declared_functions():
        assert name in exported, name
        assert hasattr(lib, name)


def test_binding_declares_every_function():
    """Every function of include/*.h has a ctypes signature in the binding (an undeclared one would
    pass 64-bit device pointers through ctypes' default int conversion)."""
    from paper_2609_20186_gb300 import binding as bd
    missing = sorted(set(declared_functions()) - set(bd._SIGNATURES))
    assert missing == []


def test_abi_version_and_strerror(lib):
    from paper_2609_20186_gb300 import binding as bd
    assert bd.abi_version() == 8
    for code in (0, -1, -2, -3, 1, 2, 3):
        assert bd.strerror(code) != "unknown code"
    assert bd.strerror(12345) == "unknown code"


def _params(**kw):
    from paper_2609_20186_gb300 import binding as bd
    p = bd.switchsd_params()
    p.B, p.cap, p.d, p.k, p.n_min, p.n_max = 4, 64, 16, 8, 3, 8
    p.logit_tau = 0.0
    for key, v in kw.items():
        setattr(p, key, v)
    return p


FAKE = 0x10000  # a 16-byte-aligned non-NULL address; never dereferenced by host validation


def _step(lib, p, ctx=FAKE, hidden=FAKE, probe=FAKE, lens=FAKE):
    return lib.switchsd_step(ctx, lens, hidden, probe, ctypes.byref(p) if p is not None else None,
                             FAKE, FAKE, FAKE, FAKE)


def test_step_validation(lib):
    from paper_2609_20186_gb300 import binding as bd
    assert _step(lib, None) == bd.ERR_ARG
    assert _step(lib, _params(), ctx=0) == bd.ERR_ARG
    assert _step(lib, _params(), ctx=FAKE + 4) == bd.ERR_ARG          # misaligned rows
    assert _step(lib, _params(), hidden=FAKE + 2) == bd.ERR_ARG
    assert _step(lib, _params(probe_kind=7)) == bd.ERR_ARG
    assert _step(lib, _params(B=0)) == bd.ERR_SHAPE
    assert _step(lib, _params(cap=66)) == bd.ERR_SHAPE                 # cap % 4 != 0
    assert _step(lib, _params(d=12)) == bd.ERR_SHAPE                   # d % 8 != 0
    assert _step(lib, _params(k=0)) == bd.ERR_SHAPE
    assert _step(lib, _params(k=65)) == bd.ERR_SHAPE
    assert _step(lib, _params(n_min=0)) == bd.ERR_SHAPE
    assert _step(lib, _params(n_min=5, n_max=4)) == bd.ERR_SHAPE
    assert _step(lib, _params(n_max=33)) == bd.ERR_SHAPE
    assert _step(lib, _params(split=3)) == bd.ERR_SHAPE
    assert _step(lib, _params(prefetch=4)) == bd.ERR_ARG
    assert _step(lib, _params(hidden_rows=9)) == bd.ERR_ARG   # k + 1 rows only with a verification
    assert _step(lib, _params(len_bound=65)) == bd.ERR_ARG    # above cap
    assert _step(lib, _params(len_bound=-1)) == bd.ERR_ARG
    assert _step(lib, _params(prefetch=-1)) == bd.ERR_ARG
    assert _step(lib, _params(probe_kind=1, probe_hidden=0)) == bd.ERR_SHAPE
    # the two-layer probe needs its workspace
    assert _step(lib, _params(probe_kind=1, probe_hidden=256)) == bd.ERR_ARG
    need = bd.switchsd_workspace_bytes(4, 1, 256)
    assert need >= 4 * 4 * 4 and need % 256 == 0
    assert bd.switchsd_workspace_bytes(4, 0, 0) == 0
    assert _step(lib, _params(probe_kind=1, probe_hidden=256, workspace=FAKE,
                              workspace_bytes=need - 1)) == bd.ERR_ARG
    assert _step(lib, _params(probe_kind=1, probe_hidden=256, d=8200)) == bd.ERR_SHAPE
    # hidden_rows = k + 1 with the two-layer probe: the workspace also holds B x d gathered bf16 states
    grown = bd.switchsd_workspace_bytes(4, 1, 256, 16, hidden_rows=9)
    assert grown == bd.switchsd_workspace_bytes(4, 1, 256, 16) + 256
    assert bd.switchsd_workspace_bytes(4, 0, 0, 16, hidden_rows=9) == 0
    f = FAKE
    q = _params(probe_kind=1, probe_hidden=256, hidden_rows=9, workspace=FAKE, workspace_bytes=grown - 1)
    assert lib.switchsd_verify_step(f, f, f, f, f, f, f, f, ctypes.byref(q), f, f, f, f) == bd.ERR_ARG


def test_verify_validation(lib):
    from paper_2609_20186_gb300 import binding as bd
    vp = bd.switchsd_verify_params()
    vp.B, vp.cap, vp.k = 4, 64, 8
    vp.draft_len = vp.ctx_tokens = vp.ctx_lens = FAKE
    assert lib.switchsd_verify(FAKE, FAKE, FAKE, None) == bd.ERR_ARG
    assert lib.switchsd_verify(0, FAKE, FAKE, ctypes.byref(vp)) == bd.ERR_ARG
    vp.k = 0
    assert lib.switchsd_verify(FAKE, FAKE, FAKE, ctypes.byref(vp)) == bd.ERR_SHAPE
    vp.k, vp.cap = 8, 63
    assert lib.switchsd_verify(FAKE, FAKE, FAKE, ctypes.byref(vp)) == bd.ERR_SHAPE
    vp.cap, vp.ctx_lens = 64, None
    assert lib.switchsd_verify(FAKE, FAKE, FAKE, ctypes.byref(vp)) == bd.ERR_ARG


def test_verify_sampled_validation(lib):
    from paper_2609_20186_gb300 import binding as bd
    vp = bd.switchsd_verify_params()
    vp.B, vp.cap, vp.k = 4, 64, 8
    vp.draft_len = vp.ctx_tokens = vp.ctx_lens = FAKE
    f = FAKE
    assert lib.switchsd_verify_sampled(f, f, None, f, f, f, None) == bd.ERR_ARG
    assert lib.switchsd_verify_sampled(f, None, None, f, f, f, ctypes.byref(vp)) == bd.ERR_ARG  # no p
    assert lib.switchsd_verify_sampled(f, f, None, None, f, f, ctypes.byref(vp)) == bd.ERR_ARG  # no u
    vp.k = 65
    assert lib.switchsd_verify_sampled(f, f, None, f, f, f, ctypes.byref(vp)) == bd.ERR_SHAPE
    hp = bd.switchsd_harness_params()
    hp.B, hp.k, hp.V, hp.gamma = 4, 8, 100, 6
    assert lib.switchsd_harness_sampled(f, f, f, f, None, f, f, None, f, f, f, ctypes.byref(hp)) == bd.ERR_ARG
    hp.gamma = 9
    assert lib.switchsd_harness_sampled(f, f, f, f, None, f, f, f, f, f, f, ctypes.byref(hp)) == bd.ERR_SHAPE


def test_labels_validation(lib):
    from paper_2609_20186_gb300 import binding as bd
    need = lib.switchsd_labels_workspace_bytes(4, 1000)
    assert need >= 4 * 2000 * 4                          # a table of >= 2 cap slots per row
    assert lib.switchsd_labels_workspace_bytes(0, 1000) == 0
    f = FAKE
    assert lib.switchsd_copy_labels(None, f, 4, 1000, 5, f, f, need, None) == bd.ERR_ARG
    assert lib.switchsd_copy_labels(f, f, 4, 1000, 5, f, None, need, None) == bd.ERR_ARG
    assert lib.switchsd_copy_labels(f, f, 4, 1000, 5, f, f + 2, need, None) == bd.ERR_ARG   # misaligned
    assert lib.switchsd_copy_labels(f, f, 4, 1000, 5, f, f, need - 1, None) == bd.ERR_ARG  # too small
    assert lib.switchsd_copy_labels(f, f, 4, 1000, 0, f, f, need, None) == bd.ERR_SHAPE
    assert lib.switchsd_copy_labels(f, f, 4, 1000, 33, f, f, need, None) == bd.ERR_SHAPE
    assert lib.switchsd_copy_labels(f, f, 0, 1000, 5, f, f, need, None) == bd.ERR_SHAPE


def test_host_staged_validation(lib):
    """switchsd_step_host / switchsd_verify_step_host reject a bad io before any copy, and pass a bad
    step on unchanged (no byte counts: nothing is queued before the step's own validation)."""
    from paper_2609_20186_gb300 import binding as bd
    f = FAKE
    io = bd.switchsd_host_io()
    p = _params()
    assert lib.switchsd_step_host(None, f, f, f, f, ctypes.byref(p), f, f, f, f) == bd.ERR_ARG
    assert lib.switchsd_step_host(ctypes.byref(io), f, f, f, f, None, f, f, f, f) == bd.ERR_ARG
    io.in_bytes = 64                                     # a copy with no buffers
    assert lib.switchsd_step_host(ctypes.byref(io), f, f, f, f, ctypes.byref(p), f, f, f, f) == bd.ERR_ARG
    io.in_bytes, io.out_bytes = 0, 64
    assert lib.switchsd_verify_step_host(ctypes.byref(io), f, f, f, f, f, f, f, f, ctypes.byref(p),
                                         f, f, f, f) == bd.ERR_ARG
    io.out_bytes = 0
    bad = _params(B=0)
    assert lib.switchsd_step_host(ctypes.byref(io), f, f, f, f, ctypes.byref(bad), f, f, f, f) == bd.ERR_SHAPE
    assert lib.switchsd_verify_step_host(ctypes.byref(io), f, f, f, f, f, f, f, f, ctypes.byref(bad),
                                         f, f, f, f) == bd.ERR_SHAPE
    assert lib.switchsd_verify_sampled_step_host(None, f, f, None, f, f, f, f, f, f, f, f, ctypes.byref(p),
                                                 f, f, f, f) == bd.ERR_ARG
    assert lib.switchsd_verify_sampled_step_host(ctypes.byref(io), f, f, None, f, f, f, f, f, f, f, f,
                                                 ctypes.byref(bad), f, f, f, f) == bd.ERR_SHAPE


def test_plan_validation(lib):
    """switchsd_plan_create / _run / _destroy reject bad arguments before any CUDA call."""
    from paper_2609_20186_gb300 import binding as bd
    f = FAKE
    io = bd.switchsd_host_io()
    p = _params()
    a = bd.switchsd_step_args()
    a.ctx_tokens = a.ctx_lens = a.hidden = a.probe_w = f
    a.out_draft = a.out_len = a.out_mode = a.out_score = f
    a.params = ctypes.pointer(p)
    h = ctypes.c_void_p(12345)
    assert lib.switchsd_plan_create(ctypes.byref(a), ctypes.byref(io), None) == bd.ERR_ARG
    assert lib.switchsd_plan_create(None, ctypes.byref(io), ctypes.byref(h)) == bd.ERR_ARG
    assert h.value is None                               # *out is cleared on failure
    assert lib.switchsd_plan_create(ctypes.byref(a), None, ctypes.byref(h)) == bd.ERR_ARG
    a.draft = f                                          # a partial set of verification buffers
    assert lib.switchsd_plan_create(ctypes.byref(a), ctypes.byref(io), ctypes.byref(h)) == bd.ERR_ARG
    a.draft = None
    io.in_bytes = 16                                     # a copy without buffers
    assert lib.switchsd_plan_create(ctypes.byref(a), ctypes.byref(io), ctypes.byref(h)) == bd.ERR_ARG
    a.p_draft = f                                        # sampled arguments without a verification
    assert lib.switchsd_plan_create(ctypes.byref(a), ctypes.byref(io), ctypes.byref(h)) == bd.ERR_ARG
    a.draft = a.target_argmax = a.draft_len = a.out_accept = f   # ... or without the uniforms
    assert lib.switchsd_plan_create(ctypes.byref(a), ctypes.byref(io), ctypes.byref(h)) == bd.ERR_ARG
    a.p_draft = a.draft = a.target_argmax = a.draft_len = a.out_accept = None
    a.params = None
    io.in_bytes = 0
    assert lib.switchsd_plan_create(ctypes.byref(a), ctypes.byref(io), ctypes.byref(h)) == bd.ERR_ARG
    assert lib.switchsd_plan_run(None, None, None, 1) == bd.ERR_ARG
    lib.switchsd_plan_destroy(None)


def test_read_ceiling_validation(lib):
    from paper_2609_20186_gb300 import binding as bd
    f = FAKE
    assert lib.switchsd_harness_read(None, f, 4, 64, f, 16, 8, 1, f, None) == bd.ERR_ARG
    assert lib.switchsd_harness_read(f + 4, f, 4, 64, f, 16, 8, 1, f, None) == bd.ERR_ARG   # misaligned
    assert lib.switchsd_harness_read(f, f, 4, 64, f + 2, 16, 8, 1, f, None) == bd.ERR_ARG
    assert lib.switchsd_harness_read(f, f, 4, 66, f, 16, 8, 1, f, None) == bd.ERR_SHAPE     # cap % 4
    assert lib.switchsd_harness_read(f, f, 4, 64, f, 12, 8, 1, f, None) == bd.ERR_SHAPE     # d % 8
    assert lib.switchsd_harness_read(f, f, 4, 64, f, 16, 0, 1, f, None) == bd.ERR_SHAPE     # split
    assert lib.switchsd_harness_read(f, f, 0, 64, f, 16, 8, 1, f, None) == bd.ERR_SHAPE


def test_candidates_index_static_validation(lib):
    """The candidate, index and static-workspace entry points reject bad arguments before any CUDA call."""
    from paper_2609_20186_gb300 import binding as bd
    f = FAKE
    p = _params()
    # switchsd_step_candidates: W in 1..WMAX, D in 1..KMAX, every output given
    cand = lambda W, D, outs=(f, f, f): lib.switchsd_step_candidates(f, f, f, f, ctypes.byref(p), W, D, *outs, f, f)
    assert cand(0, 20) == bd.ERR_SHAPE
    assert cand(17, 20) == bd.ERR_SHAPE                  # W above SWITCHSD_WMAX (16)
    assert cand(10, 0) == bd.ERR_SHAPE
    assert cand(10, 65) == bd.ERR_SHAPE
    assert cand(10, 20, (None, f, f)) == bd.ERR_ARG
    assert cand(10, 20, (f, f, None)) == bd.ERR_ARG
    # the fused candidate verification needs its verification buffers
    assert lib.switchsd_verify_candidates_step(None, f, f, f, f, f, f, f, f, f, ctypes.byref(p), 10, 20,
                                               f, f, f, f, f) == bd.ERR_ARG
    assert lib.switchsd_verify_candidates_step(f, f, f, f, f, None, f, f, f, f, ctypes.byref(p), 10, 20,
                                               f, f, f, f, f) == bd.ERR_ARG
    # switchsd_verify_candidates: pointers, then shapes
    vp = bd.switchsd_candidates_verify_params()
    vp.B, vp.cap, vp.W, vp.D = 4, 64, 10, 20
    vp.cand_len = vp.ncand = vp.ctx_tokens = vp.ctx_lens = f
    assert lib.switchsd_verify_candidates(f, f, f, f, None) == bd.ERR_ARG
    assert lib.switchsd_verify_candidates(f, f, f, None, ctypes.byref(vp)) == bd.ERR_ARG
    vp.W = 17
    assert lib.switchsd_verify_candidates(f, f, f, f, ctypes.byref(vp)) == bd.ERR_SHAPE
    vp.W, vp.cap = 10, 66
    assert lib.switchsd_verify_candidates(f, f, f, f, ctypes.byref(vp)) == bd.ERR_SHAPE
    # the fused verification needs its buffers too
    assert lib.switchsd_verify_step(None, f, f, f, f, f, f, f, ctypes.byref(p), f, f, f, f) == bd.ERR_ARG
    assert lib.switchsd_verify_step(f, f, f, None, f, f, f, f, ctypes.byref(p), f, f, f, f) == bd.ERR_ARG
    # switchsd_index_create: shapes before any allocation
    h = ctypes.c_void_p()
    assert lib.switchsd_index_create(None, ctypes.byref(h)) == bd.ERR_ARG
    for kw in (dict(B=0), dict(cap=66), dict(n_min=0), dict(n_min=5, n_max=4), dict(n_max=33)):
        q = _params(**kw)
        assert lib.switchsd_index_create(ctypes.byref(q), ctypes.byref(h)) == bd.ERR_SHAPE, kw
        assert h.value is None
    # switchsd_step_static_workspace: no params; a two-layer probe whose scratch exceeds the 16 MiB array
    assert lib.switchsd_step_static_workspace(f, f, f, f, None, f, f, f, f) == bd.ERR_ARG
    big = _params(probe_kind=1, probe_hidden=1024, d=8192, B=4096)
    assert bd.switchsd_workspace_bytes(4096, 1, 1024, 8192) > 16 << 20
    assert lib.switchsd_step_static_workspace(f, f, f, f, ctypes.byref(big), f, f, f, f) == bd.ERR_SHAPE


def test_binding_rejects_cpu_tensors(lib):
    import torch
    from paper_2609_20186_gb300 import binding as bd
    t = torch.zeros(2, 8, dtype=torch.int32)
    with pytest.raises(TypeError):
        bd.switchsd_verify(t, torch.zeros(2, 9, dtype=torch.int32), torch.zeros(2, dtype=torch.int32),
                           draft_len=torch.zeros(2, dtype=torch.int32), ctx_tokens=t,
                           ctx_lens=torch.zeros(2, dtype=torch.int32))


def test_params_layout_matches_the_header(tmp_path):
    """The binding's ctypes structures have the C header's layout (size and every field's offset): a
    program compiled against include/switchsd.h prints them."""
    import ctypes
    import shutil
    import subprocess
    from paper_2609_20186_gb300 import binding as bd

    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    structs = {"switchsd_params": bd.switchsd_params, "switchsd_verify_params": bd.switchsd_verify_params,
               "switchsd_candidates_verify_params": bd.switchsd_candidates_verify_params}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "switchsd.h"', "int main(void) {"]
    for name, st in structs.items():
        lines.append(f'  printf("{name} size %zu\\n", sizeof({name}));')
        for field, _ in st._fields_:
            lines.append(f'  printf("{name} {field} %zu\\n", offsetof({name}, {field}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    subprocess.run([cc, "-std=c99", "-I", os.path.join(root, "include"), str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines()
    got = {tuple(line.split()[:2]): int(line.split()[2]) for line in out}
    for name, st in structs.items():
        assert got[(name, "size")] == ctypes.sizeof(st), name
        for field, _ in st._fields_:
            assert got[(name, field)] == getattr(st, field).offset, (name, field)
