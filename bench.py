#!/usr/bin/env python3
"""Benchmark of the SwitchSD per-step controller on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload zipf_32k] [--impl ours|reference]

The controller iteration of a batch: verification and append of the previous draft, then search,
probe, switch and copy draft (switchsd_verify_step); between iterations the target stand-in
(switchsd_harness_target) replaces the out-of-scope drafter and target forward.  The default workload
is B=64 sequences of 32,768-token contexts (Zipf(1.1) tokens, 5 % planted copy spans, d=4096 linear
probe, n 3..8, k=16).

A step is one launch of switchsd_verify_step (verification of the batch's previous draft, then the
next step) on one batch.  Inputs larger than L2: the run keeps R independent batches of B rows whose
contexts together exceed 2.2x L2, and launch i of the loop works on batch i mod R, so each launch reads
its batch's context from HBM (one batch alone, ~10.6 MB, would stay in the 126 MB L2).  The K launches
and one target stand-in launch per round of R are captured in one CUDA graph; the graph is replayed
once untimed and once between CUDA events on its stream.  ``value`` = B x K / that time.  The
roofline uses the algorithmic bytes of each launch (its contexts, hidden states, probe weights,
verification reads and writes, outputs) over the average launch duration (timed region / K).  Also
reported: the latency of single cold launches (L2 flushed, event-bracketed), and ``e2e``, the loop on
one batch through host buffers (pinned H2D of each step's hidden states, D2H of the modes, draft
lengths, drafts and accepted lengths).

--impl reference times the CPU oracle (tests-only reference implementation) on the host cores.
Multi-GPU: the controller has no cross-row exchange, so N GPUs run N independent replicas (weak
scaling, no collective on the data path); rank 0 prints the aggregate.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "controller steps/sec (seq×step) at B=64, 32K ctx; achieved HBM GB/s vs peak"
UNIT = "seq*steps/s"
PROFILE_SUMMARY = os.path.join(ROOT, "profiles", "rescan_kernel_zipf_32k.txt")
SPIN_CYCLES = 600_000  # ~0.3 ms at 2 GHz: longer than the host needs to enqueue one step


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=512)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--workload", default="zipf_32k", choices=sorted(synth.WORKLOADS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--split", type=int, default=0, help="CTAs per row (0 = library choice)")
    ap.add_argument("--search", default="scan", choices=["scan", "index"],
                    help="rescan the contexts every step, or keep the incremental n-gram index")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="budget of the CPU-baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-per-config", action="store_true",
                    help="time the selected workload only (by default the 32K headline also times the "
                         "suite's other workloads into the same line)")
    ap.add_argument("--candidates", type=int, default=0,
                    help="W > 0: the step with W copy candidates (§3.3, App. D; the paper's W = 10)")
    ap.add_argument("--cand-len", type=int, default=20, help="D, the candidate length (the paper's 20)")
    ap.add_argument("--task", default="step", choices=["step", "labels"],
                    help="step: the controller step (the headline); labels: copy-mode labels (§3.2)")
    ap.add_argument("--verify", default="greedy", choices=["greedy", "sampled"],
                    help="verification at temperature 0 (greedy) or T > 0 (sampled: App. A)")
    ap.add_argument("--no-prefetch", action="store_true",
                    help="read nothing before the preceding kernel is done (params.prefetch = 0)")
    return ap.parse_args(argv)


# ------------------------------------------------------------------------------------------------
# distributed plumbing (replicas only)
# ------------------------------------------------------------------------------------------------
def dist_init(n_gpus: int):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def reduce_max(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(units_per_rank: float, seconds_per_rank: float, world: int) -> float:
    """Whole-job throughput of `world` replicas: all units over the slowest rank's time."""
    return units_per_rank * world / reduce_max(seconds_per_rank, world)


# ------------------------------------------------------------------------------------------------
# clocks during the timed region
# ------------------------------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str | None):
        self.proc = None
        self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
               "-lms", "20"]
        if gpu_id:
            cmd.insert(1, f"--id={gpu_id}")
        try:
            self.proc = subprocess.Popen(cmd, stdout=self.file, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self) -> dict | None:
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        sm, smax, power = [], [], []
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = set()
        for line in self.file.read().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
                power.append(float(parts[2]))
            except ValueError:
                continue
            for name, v in zip(names, parts[3:7]):
                if v.lower() == "active":
                    reasons.add(name)
        os.unlink(self.file.name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": sorted(reasons), "samples": 0}
        busy = [s for s in sm if s > 0.5 * max(sm)]
        return {"sm_mhz": statistics.median(busy), "sm_max_mhz": max(smax),
                "reasons": sorted(reasons), "samples": len(sm),
                "power_w_max": max(power) if power else None}


def measured_peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "source": "fallback"}


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_20186_gb300", "csrc")
    for f in ("common.cuh", "step.cuh", "rescan.cu"):  # the headline kernel's sources
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str) -> float | None:
    """DRAM bytes per launch of the step kernel from the committed ncu summary, if it was taken on
    the current kernel source (the summary records the source hash) and this workload."""
    try:
        text = open(PROFILE_SUMMARY).read()
    except OSError:
        return None
    fields = {}
    for line in text.splitlines():
        if ":" in line and line.startswith("bench_"):
            k, v = line.split(":", 1)
            fields[k.strip()] = v.strip()
    if fields.get("bench_kernel_hash") != kernel_source_hash():
        return None
    if fields.get("bench_workload") != workload:
        return None
    try:
        return float(fields["bench_dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


# ------------------------------------------------------------------------------------------------
# CPU oracle timing (baseline and reference arm)
# ------------------------------------------------------------------------------------------------
def host_threads() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return max(1, os.cpu_count() or 1)


def time_oracle(wl: synth.Workload, budget_s: float, max_steps: int, rows: int | None = None,
                warmup: int = 0, sampled: bool = False, cand: tuple[int, int] | None = None,
                threads: int = 1, state: dict | None = None):
    """Runs the oracle loop (oracle step, host target stand-in, oracle verify) on rows [0, R):
    ``warmup`` untimed steps, then up to max_steps timed steps or until budget_s of oracle time is
    spent.  Returns (seq*steps, seconds, timed_steps, R).  Only the oracle's calls are timed.

    threads > 1 runs each oracle call as that many concurrent calls on contiguous ranges of rows (rows
    are independent; the oracle's C calls release the interpreter lock), the oracle itself unchanged.
    state: if given, receives the final contexts and lengths."""
    import oracle
    from concurrent.futures import ThreadPoolExecutor
    R = wl.B if rows is None else min(rows, wl.B)
    ctx, lens = wl.contexts()
    future = wl.future()
    pw = wl.probe_weights()
    hp = wl.harness_params()
    nt = max(1, min(threads, R))
    chunks = [(R * i // nt, R * (i + 1) // nt) for i in range(nt)]
    pool = ThreadPoolExecutor(nt) if nt > 1 else None

    def over_rows(fn):
        """fn(b0, b1) -> dict or tuple of [B] arrays filled on rows [b0, b1); merged over the chunks."""
        if pool is None:
            return fn(0, R)
        parts = list(pool.map(lambda c: fn(*c), chunks))
        first = parts[0]
        if isinstance(first, dict):
            for (b0, b1), part in zip(chunks[1:], parts[1:]):
                for key in first:
                    first[key][b0:b1] = part[key][b0:b1]
            return first
        for (b0, b1), part in zip(chunks[1:], parts[1:]):
            for x, y in zip(first, part):
                x[b0:b1] = y[b0:b1]
        return first

    spent = 0.0
    done = 0
    try:
        for t in range(warmup + max_steps):
            h = wl.hidden(t)
            if cand is not None:
                Wc, Dc = cand
                t0 = time.perf_counter()
                out = over_rows(lambda b0, b1: oracle.step_candidates(
                    ctx, lens, h, pw, W=Wc, D=Dc, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                    logit_tau=wl.logit_tau, probe_kind=wl.probe_kind, probe_hidden=wl.probe_hidden,
                    rows=(b0, b1)))
                dt = time.perf_counter() - t0
                vc, vl, vn, tg = synth.harness_candidates(hp, t, lens, out["mode"], out["cand"],
                                                          out["cand_len"], out["ncand"], future, rows=range(R))
                t0 = time.perf_counter()
                over_rows(lambda b0, b1: oracle.verify_candidates(ctx, lens, vc, vl, vn, tg, rows=(b0, b1)))
                dt += time.perf_counter() - t0
            else:
                t0 = time.perf_counter()
                out = over_rows(lambda b0, b1: oracle.step(
                    ctx, lens, h, pw, k=wl.k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                    logit_tau=wl.logit_tau, probe_kind=wl.probe_kind, probe_hidden=wl.probe_hidden,
                    rows=(b0, b1)))
                dt = time.perf_counter() - t0
                if sampled:
                    vd, vl, pp, qq, uu, rs = synth.harness_sampled(hp, t, lens, out["mode"], out["draft"],
                                                                   out["len"], future, rows=range(R))
                    t0 = time.perf_counter()
                    over_rows(lambda b0, b1: oracle.verify_sampled(ctx, lens, vd, vl, pp, uu, rs, q=qq,
                                                                   rows=(b0, b1)))
                else:
                    vd, vl, tg = synth.harness_targets(hp, t, lens, out["mode"], out["draft"], out["len"],
                                                       future, rows=range(R))
                    t0 = time.perf_counter()
                    over_rows(lambda b0, b1: oracle.verify(ctx, lens, vd, vl, tg, rows=(b0, b1)))
                dt += time.perf_counter() - t0
            if t < warmup:
                continue
            spent += dt
            done += 1
            if spent >= budget_s:
                break
    finally:
        if pool is not None:
            pool.shutdown()
    if state is not None:
        state.update(ctx=ctx, lens=lens)
    return R * done, spent, done, R


def cpu_baseline(wl: synth.Workload, budget_s: float, sampled: bool = False, cand=None) -> dict:
    """The oracle on all host cores (rows split over threads), with a single-thread run beside it."""
    nt = host_threads()
    units, secs, steps, R = time_oracle(wl, budget_s, wl.steps, sampled=sampled, cand=cand, threads=nt)
    u1, s1, steps1, _ = time_oracle(wl, budget_s / 3, wl.steps, sampled=sampled, cand=cand, threads=1)
    return {"value": units / secs, "unit": UNIT, "cores": min(nt, R), "kind": "oracle",
            "single_thread_value": u1 / s1,
            "sample": f"{wl.name}: rows 0..{R - 1}, first {steps} controller steps (oracle step + "
                      f"verify timed over {min(nt, R)} threads, each a contiguous range of rows; the host "
                      f"target stand-in is not timed); single thread: first {steps1} steps"}


def config_of(wl: synth.Workload, world: int, split: int, search: str = "scan",
              prefetch: bool = True, verify: str = "greedy", candidates: int = 0, cand_len: int = 0) -> dict:
    return {"workload": wl.name, "search": search, "verify": verify,
            "candidates": ({"W": candidates, "D": cand_len} if candidates > 0 else None),
            "prefetch": bool(prefetch), "B": wl.B, "L0": wl.L0, "V": wl.V, "d": wl.d, "k": wl.k,
            "n_min": wl.n_min, "n_max": wl.n_max, "kappa": wl.kappa_eff, "tau": wl.tau,
            "probe": "linear" if wl.probe_kind == 0 else f"mlp{wl.d}x{wl.probe_hidden}",
            "global_batch": wl.B * world, "seq_len": wl.L0, "parallelism": f"replicas{world}",
            "split": split,
            "l2": "cold: every timed launch reads contexts that are not in L2"}


def run_reference(args, world, rank):
    """The reference arm: the CPU oracle on this host's cores, W untimed + K timed steps of the workload
    on a bounded sample of rows (all rows when B <= 64, else the first 16)."""
    if rank != 0:
        return
    import oracle
    oracle.build()
    base = synth.get_workload(args.workload)
    wl = base.scaled(steps=args.warmup + args.steps)
    R = wl.B if wl.B <= 64 else 16
    nt = host_threads()
    units, secs, steps, R = time_oracle(wl, float("inf"), args.steps, rows=R, warmup=args.warmup,
                                        sampled=args.verify == "sampled",
                                        cand=(args.candidates, args.cand_len) if args.candidates > 0 else None,
                                        threads=nt)
    value = units / secs
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": secs / steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int32 (search/verify), f64 (probe)", "data": "synthetic",
            "impl": "reference",
            "config": config_of(base, world, args.split, args.search, not args.no_prefetch, args.verify,
                                 args.candidates, args.cand_len),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": min(nt, R), "kind": "oracle",
                             "sample": f"{wl.name}: rows 0..{R - 1}, {args.warmup} untimed + "
                                       f"{steps} timed steps, rows split over {min(nt, R)} threads"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------------------
# GPU run
# ------------------------------------------------------------------------------------------------
def choose_replicas(batch_bytes: int, l2_bytes: int, K: int, min_cover: int = 64, max_r: int = 1024) -> int:
    """Replica batches of the timed loop: the smallest power of two R such that the other R - 1 batches'
    contexts cover 2.2x L2 (a batch read again R launches later has been pushed out of L2 in between),
    and R >= min(K, min_cover), so that a timed region of up to min_cover launches reads each batch once
    (the target stand-in then runs outside it); at most max_r (workloads far below L2 stay L2-resident)."""
    r = 2
    while r < max_r and ((r - 1) * batch_bytes < 2.2 * l2_bytes or r < min(K, min_cover)):
        r *= 2
    return r


class ReplicaLoop:
    """R independent batches of B rows stored as one [R*B, cap] state.  Launch i of a round runs
    switchsd_verify_step on batch i (its rows only); then one target stand-in covers all R*B rows."""

    def __init__(self, wl, R, cap, ctx1, lens1, pw, future1, hidden, split, dev, stream,
                 search="scan", prefetch=True, sampled=False, cand_w=0, cand_d=20):
        import ctypes
        import torch
        from paper_2609_20186_gb300 import binding as bd, bf16_tensor

        self.bd, self.ct = bd, ctypes
        self.lib = bd.load()
        self.R, self.B, self.k, self.cap = R, wl.B, wl.k, cap
        self.sampled = sampled  # verification at T > 0 (the sampled stand-in and rule)
        self.cw, self.cd = cand_w, cand_d  # W copy candidates of D tokens (0: the single-draft step)
        B, k = wl.B, wl.k
        ctx = np.zeros((B, cap), np.int32)
        ctx[:, : ctx1.shape[1]] = ctx1[:, : min(cap, ctx1.shape[1])]
        self.ctx = torch.from_numpy(ctx).to(dev).repeat(R, 1).contiguous()
        self.lens = torch.from_numpy(np.ascontiguousarray(lens1, np.int32)).to(dev).repeat(R).contiguous()
        self.probe_w = bf16_tensor(pw.reshape(-1), dev)
        fut = torch.from_numpy(np.ascontiguousarray(future1, np.int32)).to(dev)
        self.future = fut.repeat(R, 1).contiguous()
        i32 = dict(dtype=torch.int32, device=dev)
        N = R * B
        self.draft = torch.zeros(N, k, **i32)
        self.len = torch.zeros(N, **i32)
        self.mode = torch.zeros(N, **i32)
        self.score = torch.zeros(N, dtype=torch.float32, device=dev)
        self.vdraft = torch.zeros(N, k, **i32)
        self.vlen = torch.zeros(N, **i32)
        self.target = torch.zeros(N, k + 1, **i32)
        self.accept = torch.zeros(N, **i32)
        self.hidden = hidden                     # bf16 [nh, B, d]: launch i reads block i mod nh
        sp = stream.cuda_stream
        p = bd.switchsd_params()
        p.B, p.cap, p.d, p.k = B, cap, wl.d, k
        p.n_min, p.n_max, p.kappa, p.logit_tau = wl.n_min, wl.n_max, wl.kappa, wl.logit_tau
        p.probe_kind, p.probe_hidden, p.b1, p.b2, p.split = wl.probe_kind, wl.probe_hidden, None, 0.0, split
        p.out_match_n = p.out_match_end = p.status = None
        p.stream = sp
        # The kernel before each launch is another batch's launch, the target stand-in or a copy:
        # none writes this batch's rows or hidden states (generated once, never written), so their
        # copies may start before it finishes.
        p.prefetch = (bd.PREFETCH_CONTEXT | bd.PREFETCH_PROBE) if prefetch else 0
        # params.len_bound (split on a bound, copies before the length read) measured no faster here
        p.len_bound = 0
        # one workspace per batch, so consecutive launches never share one
        probe = bd.switchsd_params()
        probe.B, probe.d, probe.probe_kind, probe.probe_hidden = B, wl.d, wl.probe_kind, wl.probe_hidden
        ws = max(256, int(self.lib.switchsd_workspace_bytes(ctypes.byref(probe))))
        self.workspace = torch.empty(R, ws, dtype=torch.uint8, device=dev)
        self.params = []
        # one incremental n-gram index per batch (search = index), built from its initial contexts
        self.indexes = []
        for r in range(R):
            q = bd.switchsd_params.from_buffer_copy(p)
            q.workspace, q.workspace_bytes = self.workspace[r].data_ptr(), ws
            if search == "index":
                idx = bd.NgramIndex(B, cap, wl.n_min, wl.n_max)
                code = self.lib.switchsd_index_build(idx.handle, self.ctx.data_ptr() + r * B * cap * 4,
                                                     self.lens.data_ptr() + r * B * 4, sp)
                if code != 0:
                    raise RuntimeError(f"index build failed: {code}")
                self.indexes.append(idx)
                q.index = idx.handle
            self.params.append(q)
        self.p = p
        hp = bd.switchsd_harness_params()
        h = wl.harness_params()
        hp.B, hp.k, hp.V, hp.L0 = N, k, h["V"], h["L0"]
        hp.n_future = self.future.shape[1]
        hp.gamma, hp.step, hp.seed, hp.thr_neural = h["gamma"], 0, h["seed"], h["thr_neural"]
        hp.p_hit, hp.p_miss, hp.q_neural = h["p_hit"], h["p_miss"], h["q_neural"]
        hp.stream = sp
        self.hp = hp
        e32, e16 = 4, 2
        Wc, Dc = max(cand_w, 1), cand_d
        self.cand, self.clen = torch.zeros(N, Wc, Dc, **i32), torch.zeros(N, Wc, **i32)
        self.ncand = torch.zeros(N, **i32)
        self.vcand, self.vclen = torch.zeros(N, Wc, Dc, **i32), torch.zeros(N, Wc, **i32)
        self.vn, self.ctarget = torch.zeros(N, **i32), torch.zeros(N, Wc, Dc + 1, **i32)
        self.choice = torch.zeros(N, **i32)
        self.cvps = []
        for r in range(R):
            v = bd.switchsd_candidates_verify_params()
            v.B, v.cap, v.W, v.D = B, cap, Wc, Dc
            v.cand_len = self.vclen.data_ptr() + r * B * Wc * 4
            v.ncand = self.vn.data_ptr() + r * B * 4
            v.ctx_tokens = self.ctx.data_ptr() + r * B * cap * 4
            v.ctx_lens = self.lens.data_ptr() + r * B * 4
            v.status, v.stream = None, sp
            v.index = self.indexes[r].handle if self.indexes else None
            self.cvps.append(v)
        f32 = dict(dtype=torch.float32, device=dev)
        self.vp = torch.zeros(N, k, **f32)
        self.vq = torch.ones(N, k, **f32)
        self.vu = torch.zeros(N, k, **f32)
        self.rows = []
        for r in range(R):
            o = r * B
            self.rows.append(dict(
                vp=self.vp.data_ptr() + o * k * e32, vq=self.vq.data_ptr() + o * k * e32,
                vu=self.vu.data_ptr() + o * k * e32,
                vdraft=self.vdraft.data_ptr() + o * k * e32, target=self.target.data_ptr() + o * (k + 1) * e32,
                vlen=self.vlen.data_ptr() + o * e32, accept=self.accept.data_ptr() + o * e32,
                ctx=self.ctx.data_ptr() + o * cap * e32, lens=self.lens.data_ptr() + o * e32,
                draft=self.draft.data_ptr() + o * k * e32, len=self.len.data_ptr() + o * e32,
                mode=self.mode.data_ptr() + o * e32, score=self.score.data_ptr() + o * e32))
        self.hstride = B * wl.d * e16

    def launch(self, r: int, step_index: int, first: bool):
        c = self.rows[r]
        hid = self.hidden.data_ptr() + (step_index % self.hidden.shape[0]) * self.hstride
        if self.cw > 0:
            B, Wc, Dc, o = self.B, self.cw, self.cd, r * self.B
            outs = (self.cand.data_ptr() + o * Wc * Dc * 4, self.clen.data_ptr() + o * Wc * 4,
                    self.ncand.data_ptr() + o * 4, c["mode"], c["score"])
            if first:
                code = self.lib.switchsd_step_candidates(c["ctx"], c["lens"], hid, self.probe_w.data_ptr(),
                                                         self.ct.byref(self.params[r]), Wc, Dc, *outs)
            else:  # verification of the previous candidates and the next step, fused
                code = self.lib.switchsd_verify_candidates_step(
                    self.vcand.data_ptr() + o * Wc * Dc * 4, self.ctarget.data_ptr() + o * Wc * (Dc + 1) * 4,
                    self.vclen.data_ptr() + o * Wc * 4, self.vn.data_ptr() + o * 4, c["accept"],
                    self.choice.data_ptr() + o * 4, c["ctx"], c["lens"], hid, self.probe_w.data_ptr(),
                    self.ct.byref(self.params[r]), Wc, Dc, *outs)
        elif first:
            code = self.lib.switchsd_step(c["ctx"], c["lens"], hid, self.probe_w.data_ptr(),
                                          self.ct.byref(self.params[r]), c["draft"], c["len"], c["mode"],
                                          c["score"])
        elif self.sampled:
            code = self.lib.switchsd_verify_sampled_step(
                c["vdraft"], c["vp"], c["vq"], c["vu"], c["target"], c["vlen"], c["accept"], c["ctx"], c["lens"],
                hid, self.probe_w.data_ptr(), self.ct.byref(self.params[r]), c["draft"], c["len"], c["mode"],
                c["score"])
        else:
            code = self.lib.switchsd_verify_step(c["vdraft"], c["target"], c["vlen"], c["accept"], c["ctx"],
                                                 c["lens"], hid, self.probe_w.data_ptr(),
                                                 self.ct.byref(self.params[r]), c["draft"], c["len"],
                                                 c["mode"], c["score"])
        if code != 0:
            raise RuntimeError(f"launch failed: {code} ({self.bd.strerror(code)})")

    def harness(self, q: int):
        self.hp.step = q
        if self.cw > 0:
            code = self.lib.switchsd_harness_candidates(
                self.lens.data_ptr(), self.mode.data_ptr(), self.cand.data_ptr(), self.clen.data_ptr(),
                self.ncand.data_ptr(), self.future.data_ptr(), self.cw, self.cd, self.vcand.data_ptr(),
                self.vclen.data_ptr(), self.vn.data_ptr(), self.ctarget.data_ptr(), self.ct.byref(self.hp))
        elif self.sampled:
            code = self.lib.switchsd_harness_sampled(
                self.lens.data_ptr(), self.mode.data_ptr(), self.draft.data_ptr(), self.len.data_ptr(),
                self.future.data_ptr(), self.vdraft.data_ptr(), self.vlen.data_ptr(), self.vp.data_ptr(),
                self.vq.data_ptr(), self.vu.data_ptr(), self.target.data_ptr(), self.ct.byref(self.hp))
        else:
            code = self.lib.switchsd_harness_target(
                self.lens.data_ptr(), self.mode.data_ptr(), self.draft.data_ptr(), self.len.data_ptr(),
                self.future.data_ptr(), self.vdraft.data_ptr(), self.vlen.data_ptr(), self.target.data_ptr(),
                self.ct.byref(self.hp))
        if code != 0:
            raise RuntimeError(f"harness failed: {code}")

    def round(self, q: int, first_round: bool, step_base: int):
        for r in range(self.R):
            self.launch(r, step_base + r, first_round)
        self.harness(q)


def nvtx_range(name: str):
    """An NVTX range around a phase of the run (visible in a profiler timeline); a no-op without NVTX."""
    import contextlib
    import torch
    try:
        torch.cuda.nvtx.range_push(name)
    except Exception:
        return contextlib.nullcontext()

    @contextlib.contextmanager
    def _pop():
        try:
            yield
        finally:
            try:
                torch.cuda.nvtx.range_pop()
            except Exception:
                pass
    return _pop()


def l2_flush(buf):
    """Writes a buffer of 2x L2 so that nothing the next launches read is left in L2."""
    buf.fill_(1.0)


def measure_loop(base, args, dev, cs, l2, W, K, split, search, prefetch, sampled, cand_w, cand_d, world,
                 headline=False, flush=None):
    """Times K fused controller launches (switchsd_verify_step, or its sampled / candidate / index form)
    of workload `base` captured in one CUDA graph, launch i on replica batch i mod R (see
    choose_replicas), after at least W untimed launches and an L2 flush.  Returns the measurement as a
    dict; the headline also gets the clock record, the L2-resident leg and the cold single launches."""
    import torch
    from paper_2609_20186_gb300 import bf16_tensor

    B, d, k = base.B, base.d, base.k
    batch_bytes = B * (base.L0 + 1024) * 4
    R = choose_replicas(batch_bytes, l2, K, max_r=(32 if search == "index" else 1024))
    rounds = -(-K // R)
    warm_rounds = max(1, -(-W // R))
    per_row_steps = warm_rounds + 2 * rounds + (COLD_STEPS if headline else 0) + 1
    wl = base.scaled(steps=per_row_steps)
    cap = wl.cap
    ctx1, lens1 = wl.contexts()
    future1 = wl.future()
    pw = wl.probe_weights()
    n_hidden = min((warm_rounds + rounds) * R, 64)        # distinct hidden blocks, cycled over launches
    hidden_host = np.empty((n_hidden, B, d), np.uint16)
    for i in range(n_hidden):
        hidden_host[i] = wl.hidden(i)
    hidden = bf16_tensor(hidden_host, dev)
    loop = ReplicaLoop(wl, R, cap, ctx1, lens1, pw, future1, hidden, split, dev, cs, search=search,
                       prefetch=prefetch, sampled=sampled, cand_w=cand_w, cand_d=cand_d)
    if flush is None:
        flush = torch.empty(2 * l2 // 4, dtype=torch.float32, device=dev)

    with torch.cuda.stream(cs):
        for q in range(warm_rounds):                       # eager warm-up rounds (every batch once per round)
            loop.round(q, q == 0, q * R)
        # length snapshots at round boundaries: outside the timed graph, except between its own rounds
        lens_hist = torch.zeros(rounds + 1, R * B, dtype=torch.int32, device=dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cs):
            for j in range(rounds):
                q = warm_rounds + j
                if j > 0:
                    loop.harness(q - 1)                    # the target's tokens for the round just run
                    lens_hist[j].copy_(loop.lens)
                for r in range(min(R, K - j * R)):
                    loop.launch(r, q * R + r, False)
        snap = [(t, t.clone()) for t in (loop.lens, loop.vdraft, loop.vlen, loop.target, loop.mode,
                                         loop.draft, loop.len, loop.score, loop.accept, loop.vp, loop.vq,
                                         loop.vu, loop.vcand, loop.vclen, loop.vn, loop.ctarget)]

        def restore():
            for dst, src in snap:
                dst.copy_(src)
        lens_hist[0].copy_(loop.lens)
        g.replay()                                         # first replay: graph upload + warm-up
        cs.synchronize()
    # A replay from the restored state repeats the same launches on the same inputs (tokens past a
    # restored length are never read), so identical untimed replays can surround the timed one while the
    # clocks are sampled.  The index keeps its inserts across replays: its leg is replayed once only.
    replayable = search != "index"
    barrier(world)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(_gpu_uuid(torch.cuda.get_device_properties(dev))) if headline else None

    def surround():
        if sampler is None or not replayable:
            return
        t_end = time.perf_counter() + CLOCK_WINDOW_S
        while time.perf_counter() < t_end:
            restore()
            l2_flush(flush)
            torch.cuda._sleep(SPIN_CYCLES)
            g.replay()
            cs.synchronize()

    with torch.cuda.stream(cs):
        surround()
        if replayable:
            restore()
        elif True:
            # the index's leg: its state after the first replay is the start of the timed one
            lens_hist[0].copy_(loop.lens)
        l2_flush(flush)
        # a GPU spin long enough for the host to submit the graph, so the region starts with work queued
        torch.cuda._sleep(SPIN_CYCLES)
        with nvtx_range(f"timed {base.name} {search} x{K}"):
            ev0.record(cs)
            g.replay()
            ev1.record(cs)
            ev1.synchronize()
        lens_hist[rounds].copy_(loop.lens)
        cs.synchronize()
        surround()
    clocks = sampler.stop() if sampler is not None else None
    if clocks is not None:
        clocks["window"] = (f"sampled over {2 * CLOCK_WINDOW_S:.1f} s of identical replays of the timed "
                            "graph surrounding the timed replay")
    region_s = ev0.elapsed_time(ev1) / 1e3
    barrier(world)

    # algorithmic bytes of every fused launch in the timed replay (lens after each round's append)
    Lh = lens_hist.cpu().numpy().astype(np.int64).reshape(rounds + 1, R, B)
    probe_bytes = 2 * B * d + (2 * d if wl.probe_kind == 0 else 2 * (wl.probe_hidden * d + wl.probe_hidden))
    launch_bytes = []
    for j in range(rounds):
        n_this = min(R, K - j * R)
        grow = (Lh[j + 1] - Lh[j])[:n_this]                # a + 1 per row
        if np.any(grow <= 0):
            raise SystemExit(f"timed graph round {j}: rows did not grow; the launches did not run")
        ctx_read = 4 * Lh[j + 1][:n_this].sum(axis=1)
        verify_rw = 8 * B + (28 if sampled else 16) * grow.sum(axis=1)
        outputs = 12 * B + 4 * B * k                       # mode, len, score, draft (bound)
        if cand_w > 0:
            verify_rw = 8 * B + 4 * B * cand_w * (2 * cand_d + 2) + 4 * grow.sum(axis=1)
            outputs = 12 * B + 4 * B * cand_w * (cand_d + 1)
        if search == "index":
            nn = wl.n_max - wl.n_min + 1
            ctx_read = np.full(n_this, 4 * B * (32 + nn * (4 + 4 * wl.n_max)), np.int64) + \
                12 * nn * grow.sum(axis=1)
        launch_bytes.extend((ctx_read + probe_bytes + verify_rw + outputs).tolist())
    launch_bytes = np.array(launch_bytes, dtype=np.float64)
    per_launch_s = region_s / K
    out = {"R": R, "cap": cap, "rounds": rounds, "region_s": region_s, "per_launch_s": per_launch_s,
           "launch_bytes": float(launch_bytes.mean()), "clocks": clocks,
           "mean_context_tokens": float(Lh[1:].mean()),
           "scan_equivalent_gbs": float(4 * Lh[1:].sum(axis=2).mean() / per_launch_s / 1e9),
           "ctx_bytes_all": R * B * cap * 4, "launches_per_step": 1 if wl.probe_kind == 0 else 2,
           "harness_in_region": rounds - 1,
           "value": replica_throughput(B * K, region_s, world),
           "ms_per_step": reduce_max(region_s, world) / K * 1e3}

    if headline and replayable:
        # the controller's per-mode tallies of the timed launches (switchsd_params.counters): the same
        # launches replayed from the restored state with the counters on, outside the timed region
        from paper_2609_20186_gb300 import binding as bdm
        ctr = torch.zeros(bdm.COUNTERS, dtype=torch.int64, device=dev)
        saved = loop.params
        loop.params = []
        for q in saved:
            q2 = bdm.switchsd_params.from_buffer_copy(q)
            q2.counters = ctr.data_ptr()
            loop.params.append(q2)
        with torch.cuda.stream(cs):
            restore()
            gc = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gc, stream=cs):
                for j in range(rounds):
                    q = warm_rounds + j
                    if j > 0:
                        loop.harness(q - 1)
                    for r in range(min(R, K - j * R)):
                        loop.launch(r, q * R + r, False)
            restore()
            ctr.zero_()
            gc.replay()
            cs.synchronize()
            restore()
        loop.params = saved
        c = ctr.cpu().numpy()
        steps_all = int(c[0] + c[1] + c[2])
        out["modes"] = {
            "steps": steps_all, "no_rep": int(c[0]), "copy": int(c[1]), "rep_no_copy": int(c[2]),
            "copy_share": float(c[1]) / max(steps_all, 1),
            "copy_drafts_verified": int(c[3]),
            "mean_accept_copy": float(c[4]) / max(int(c[3]), 1),
            "neural_drafts_verified": int(c[5]),
            "mean_accept_neural": float(c[6]) / max(int(c[5]), 1),
            "note": "device counters (switchsd_params.counters) over the timed launches, replayed from the "
                    "same state: rows per mode chosen, and per drafter (the previous step's mode) the drafts "
                    "verified and their mean accepted length; neural drafts are the target stand-in's"}
    if headline and R >= 2 and search == "scan":
        # warm L2, reported separately: K launches alternating between two batches only
        with torch.cuda.stream(cs):
            restore()
            g2 = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g2, stream=cs):
                for i in range(K):
                    loop.launch(i % 2, warm_rounds * R + i, False)
            g2.replay()
            cs.synchronize()
            restore()
            e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e2.record(cs)
            g2.replay()
            e3.record(cs)
            e3.synchronize()
            restore()
        us = e2.elapsed_time(e3) * 1e3 / K
        out["l2_resident"] = {"launch_us": us, "value": B / (us * 1e-6), "unit": UNIT,
                              "note": "L2-resident: K launches alternating between two batches "
                                      f"({2 * B * cap * 4 / 2**20:.0f} MiB of contexts, inside L2); not the headline"}
    if headline:
        out["cold"] = cold_latency(loop, dev, cs, warm_rounds + rounds, l2)
    if search == "scan" and cand_w == 0:
        out["ceiling"] = read_ceiling(loop, d, K, warm_rounds * R, prefetch, cs, flush)
    out["loop"] = loop
    return out


def roofline_of(m: dict, peaks: dict, kernel: str, traffic) -> dict:
    achieved = m["launch_bytes"] / m["per_launch_s"] / 1e9
    r = {"kernel": kernel, "bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
         "frac": achieved / peaks["hbm_gbs"], "traffic": traffic,
         "algorithmic_bytes_per_launch": m["launch_bytes"], "launch_us": m["per_launch_s"] * 1e6,
         "duration": "timed region / K launches (CUDA events on the launching stream around one graph "
                     "replay of the K launches)",
         "peak_source": peaks["source"] + " hbm_gbs (copy)", "frac_nominal": achieved / NOMINAL_HBM_GBS}
    c = m.get("ceiling")
    if c is not None:
        c = dict(c)
        c["frac"] = c["achieved"] / peaks["hbm_gbs"]
        c["step_time_ratio"] = c["launch_us"] / (m["per_launch_s"] * 1e6)
        r["size_matched_ceiling"] = c
    return r


def l2_note(m: dict, B: int, l2: int) -> str:
    if (m["R"] - 1) * B * m["cap"] * 4 < 2.2 * l2:
        return (f"L2-resident: the whole workload ({m['R']} batches, {m['ctx_bytes_all'] / 2**20:.1f} MiB of "
                "contexts) is below L2")
    return (f"inputs larger than L2: {m['R']} independent batches of B={B} ({m['ctx_bytes_all'] / 2**20:.0f} MiB "
            f"of contexts vs {l2 / 2**20:.0f} MiB L2), launch i reads batch i mod {m['R']}, L2 flushed before "
            "the timed replay")


PER_CONFIG = (("planted_copy", "scan"), ("uniform_8k", "scan"), ("code_16k", "scan"), ("mixed_128k", "scan"),
              ("mixed_128k", "index"))


def run_ours(args, world, rank, local):
    import torch
    from paper_2609_20186_gb300 import binding

    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA device (the controller has no CPU path)")
    if args.candidates > 0 and args.verify == "sampled":
        raise SystemExit("--candidates runs with greedy verification")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    binding.load()
    base = synth.get_workload(args.workload)
    W, K = args.warmup, args.steps
    B, d, k = base.B, base.d, base.k
    props = torch.cuda.get_device_properties(dev)
    l2 = int(getattr(props, "L2_cache_size", 128 << 20))

    # CPU baseline first (rank 0, N = 1): the oracle runs before any CUDA work of the timed run
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        cpu = cpu_baseline(base, args.cpu_seconds, sampled=args.verify == "sampled",
                           cand=(args.candidates, args.cand_len) if args.candidates > 0 else None)

    cs = torch.cuda.Stream(dev)
    flush = torch.empty(2 * l2 // 4, dtype=torch.float32, device=dev)
    prefetch = not args.no_prefetch
    sampled = args.verify == "sampled"
    m = measure_loop(base, args, dev, cs, l2, W, K, args.split, args.search, prefetch, sampled,
                     args.candidates, args.cand_len, world, headline=True, flush=flush)
    peaks = measured_peaks()
    # the committed summary profiles the greedy single-draft rescan instance: other modes get no traffic
    profiled_mode = args.search == "scan" and args.candidates == 0 and args.verify == "greedy" and prefetch
    traffic = profiled_traffic(base.name) if profiled_mode else None
    roof = roofline_of(m, peaks, "switchsd_verify_step" + (" (index)" if args.search == "index" else ""),
                       traffic)

    e2e = None
    if not args.no_e2e and args.candidates == 0:  # the public-API loop covers the single-draft step
        with nvtx_range("e2e"):
            e2e = run_e2e(base, dev, W, K, args.split, world, prefetch=prefetch, sampled=sampled)

    head = m
    loops = [head.pop("loop")]
    # The other workloads of the suite, each measured the same way (same K and W), in the same line.
    per_config = None
    if not args.no_per_config and args.workload == "zipf_32k" and args.candidates == 0 and not sampled:
        per_config = {}
        for name, search in PER_CONFIG:
            loops.clear()
            torch.cuda.synchronize()
            torch.cuda.empty_cache()
            wb = synth.get_workload(name)
            mc = measure_loop(wb, args, dev, cs, l2, W, K, args.split, search, prefetch, False, 0, 20, world,
                              flush=flush)
            mc.pop("loop")
            entry = {"value": mc["value"], "unit": UNIT, "ms_per_step": mc["ms_per_step"],
                     "B": wb.B, "L0": wb.L0, "k": wb.k, "d": wb.d, "n_min": wb.n_min, "n_max": wb.n_max,
                     "probe": "linear" if wb.probe_kind == 0 else f"mlp{wb.d}x{wb.probe_hidden}",
                     "search": search, "launches_per_step": mc["launches_per_step"],
                     "l2": l2_note(mc, wb.B, l2)}
            if search == "index":
                entry["scan_equivalent_gbs"] = mc["scan_equivalent_gbs"]
                entry["launch_us"] = mc["per_launch_s"] * 1e6
                entry["roofline"] = None
                entry["note"] = ("the index reads the context tail and its hash tables, not the context: its "
                                 "bytes are not the scan's, so it has no HBM roofline; scan_equivalent_gbs = "
                                 "the context bytes a rescan would read over the same time (effective, not "
                                 "achieved)")
            else:
                entry["roofline"] = roofline_of(mc, peaks, "switchsd_verify_step" +
                                                (" + two-layer probe kernel" if wb.probe_kind else ""), None)
            if not args.no_e2e and search == "scan":
                entry["e2e"] = run_e2e(wb, dev, W, K, args.split, world, prefetch=prefetch)
            per_config[name + ("_index" if search == "index" else "")] = entry
    loops.clear()

    if rank != 0:
        return
    line = {
        "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": head["ms_per_step"], "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int32 (search/verify), bf16 in / fp32 accumulate (probe)",
        "data": "synthetic",
        "config": config_of(base, world, args.split, args.search, prefetch, args.verify,
                            args.candidates, args.cand_len),
        "roofline": roof,
        "controller": {"protocol": l2_note(head, B, l2), "replicas": head["R"],
                       "cold_single_launch_us": head.get("cold"), "l2_resident": head.get("l2_resident"),
                       "search": args.search, "scan_equivalent_gbs": head["scan_equivalent_gbs"],
                       "mean_context_tokens": head["mean_context_tokens"],
                       "launches_per_step": head["launches_per_step"],
                       "target_standin_launches_in_timed_region": head["harness_in_region"],
                       "modes": head.get("modes")},
        "gpu_launches": K * head["launches_per_step"] + 2 * head["harness_in_region"],
        "gpu_launches_note": "fused controller launches (switchsd_verify_step; plus the two-layer probe kernel "
                             "when used) in one CUDA graph, and, when K exceeds the replica count, one target "
                             "stand-in launch and one length snapshot per extra round",
        "clocks": head["clocks"],
        "e2e": e2e,
        "cpu_baseline": cpu,
        "per_config": per_config,
    }
    print(json.dumps(line), flush=True)


COLD_STEPS = 32
NOMINAL_HBM_GBS = 7900.0  # HBM3e nominal of this GPU
CLOCK_WINDOW_S = 0.4


def _gpu_uuid(props):
    try:
        return "GPU-" + str(props.uuid)
    except Exception:
        return None


def cold_latency(loop, dev, cs, step_base, l2) -> dict:
    """Event-bracketed single fused launches on batch 0 with L2 flushed before each (write then read
    2x L2 of unrelated buffers, then a GPU spin so the host has queued the launch)."""
    import torch
    flush_w = torch.empty(2 * l2 // 4, dtype=torch.float32, device=dev)
    flush_r = torch.ones(2 * l2 // 4, dtype=torch.float32, device=dev)
    sink = torch.zeros(1, dtype=torch.float32, device=dev)
    ts = []
    with torch.cuda.stream(cs):
        for i in range(COLD_STEPS):
            flush_w.fill_(1.0)
            sink.add_(flush_r.sum())
            torch.cuda._sleep(SPIN_CYCLES)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(cs)
            loop.launch(0, (step_base + i) % loop.hidden.shape[0], False)
            e1.record(cs)
            loop.harness(step_base + i)
            ts.append((e0, e1))
        cs.synchronize()
    us = sorted(a.elapsed_time(b) * 1e3 for a, b in ts)
    return {"median_us": us[len(us) // 2], "min_us": us[0], "launches": len(us),
            "note": "includes the ~2.2 us event-pair and ~2.2 us stream launch overhead of this GPU"}


def read_ceiling(loop, d: int, K: int, step_base: int, prefetch: bool, cs, flush) -> dict:
    """The size-matched ceiling: switchsd_harness_read -- a plain read of each launch's contexts and
    hidden states and nothing else -- in the timed graph's launch order (K launches, launch i on batch
    i mod R, programmatic dependent launch, L2 flushed before the timed replay), best of a few CTA splits
    per row."""
    import torch
    R, B, cap = loop.R, loop.B, loop.cap
    nh = loop.hidden.shape[0]
    out = torch.empty(R, B * 32, dtype=torch.int32, device=loop.lens.device)
    L = loop.lens.cpu().numpy().astype(np.int64).reshape(R, B)
    per_batch = 16 * ((L + 3) // 4).sum(axis=1) + 2 * B * d
    nbytes = float(np.mean([per_batch[i % R] for i in range(K)]))

    def enqueue(split):
        for i in range(K):
            r = i % R
            code = loop.lib.switchsd_harness_read(
                loop.rows[r]["ctx"], loop.rows[r]["lens"], B, cap,
                loop.hidden.data_ptr() + ((step_base + i) % nh) * loop.hstride, d, split, int(prefetch),
                out[r].data_ptr(), cs.cuda_stream)
            if code != 0:
                raise RuntimeError(f"switchsd_harness_read failed: {code}")

    best = None
    for split in (2, 4, 8, 16):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(cs):
            enqueue(split)                                  # eager warm-up
            with torch.cuda.graph(g, stream=cs):
                enqueue(split)
            g.replay()
            l2_flush(flush)
            torch.cuda._sleep(SPIN_CYCLES)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(cs)
            g.replay()
            e1.record(cs)
            e1.synchronize()
        us = e0.elapsed_time(e1) * 1e3 / K
        if best is None or us < best[0]:
            best = (us, split)
    us, split = best
    return {"kernel": "switchsd_harness_read", "launch_us": us, "achieved": nbytes / us / 1e3,
            "bytes_per_launch": nbytes, "split": split, "prefetch": bool(prefetch),
            "note": "bulk copies of every launch's context tokens and hidden states into shared memory, "
                    "folded, and nothing else; same graph, launch order, replica batches and L2 flush; "
                    "best of splits 2, 4, 8, 16"}


def run_e2e(base, dev, W, K, split, world, prefetch=True, sampled=False):
    """The same loop through the public API with host buffers, one batch.  Per step: the target
    stand-in for the previous draft, then one replay of a switchsd_plan of switchsd_verify_step_host
    (or switchsd_verify_sampled_step_host) -- pinned H2D of this step's hidden states, the fused launch,
    one D2H of mode / draft length / accepted length / draft -- and a host sync."""
    import torch
    from paper_2609_20186_gb300 import Session, binding

    wl = base.scaled(steps=W + K)
    B, d, k = wl.B, wl.d, wl.k
    ctx, lens = wl.contexts()
    sess = Session(ctx, lens, wl.probe_weights(), k=k, n_min=wl.n_min, n_max=wl.n_max,
                   kappa=wl.kappa, logit_tau=wl.logit_tau, probe_kind=wl.probe_kind,
                   probe_hidden=wl.probe_hidden, future=wl.future(), harness=wl.harness_params(),
                   split=split, d=d, device=dev,  # an H2D copy precedes each call
                   prefetch=(binding.PREFETCH_CONTEXT | binding.PREFETCH_PROBE) if prefetch else 0,
                   counters=True)
    host_h = torch.empty(W + K, B, d, dtype=torch.int16).pin_memory()
    for t in range(W + K):
        host_h[t].copy_(torch.from_numpy(wl.hidden(t).view(np.int16)))
    dev_h = torch.empty(B, d, dtype=torch.bfloat16, device=dev)
    host_out = torch.empty(B * (k + 3), dtype=torch.int32).pin_memory()  # mode, len, accept, draft
    stream = torch.cuda.current_stream()
    # switchsd_plan: the host-staged fused step (switchsd_verify_step_host, or the sampled one) recorded
    # once as a graph
    plan = sess.host_plan(host_h[1], dev_h, host_out, verify=not sampled, sampled=sampled)

    def one(t):
        if t == 0:
            sess.step_host(host_h[0], dev_h, host_out)
            return
        if sampled:
            sess.harness_sampled(t - 1)  # the target's probabilities, uniforms and resample tokens
        else:
            sess.harness(t - 1)          # the target's tokens for the previous draft
        plan.run(host_h[t])              # H2D of this step's hidden states, the fused launch, D2H, sync

    for t in range(W):
        one(t)
    torch.cuda.synchronize()
    barrier(world)
    t0 = time.perf_counter()
    for i in range(K):
        one(W + i)
    secs = time.perf_counter() - t0
    value = replica_throughput(B * K, secs, world)
    c = sess.counters.cpu().numpy()
    steps_all = int(c[0] + c[1] + c[2])
    modes = {"steps": steps_all, "no_rep": int(c[0]), "copy": int(c[1]), "rep_no_copy": int(c[2]),
             "copy_share": float(c[1]) / max(steps_all, 1),
             "copy_drafts_verified": int(c[3]), "mean_accept_copy": float(c[4]) / max(int(c[3]), 1),
             "neural_drafts_verified": int(c[5]), "mean_accept_neural": float(c[6]) / max(int(c[5]), 1),
             "note": f"device counters (switchsd_params.counters) over the {W + K} steps of this loop on one "
                     "batch: rows per mode chosen, and per drafter (the previous step's mode) the drafts "
                     "verified and their mean accepted length; neural drafts are the target stand-in's"}
    return {"value": value, "unit": UNIT, "h2d_bytes_per_step": B * d * 2, "modes": modes,
            "d2h_bytes_per_step": B * (k + 3) * 4,
            "note": ("one batch; per step: target stand-in, then one switchsd_plan_run call replaying "
                     + ("switchsd_verify_sampled_step_host" if sampled else "switchsd_verify_step_host")
                     + " recorded as a CUDA graph (pinned H2D of hidden, fused launch, one D2H of "
                       "mode/len/accept/draft), host sync; L2 not flushed")}


LABEL_METRIC = "copy-mode labels/sec (positions, §3.2, n_train=5); achieved HBM GB/s vs peak"
LABEL_UNIT = "positions/s"


def label_cpu_baseline(wl: synth.Workload, budget_s: float) -> dict:
    """The oracle's labels (plain O(L^2 n) definition) on whole rows of the workload until budget_s."""
    import oracle
    oracle.build()
    ctx, lens = wl.contexts()
    done, spent = 0, 0.0
    for b in range(wl.B):
        t0 = time.perf_counter()
        oracle.copy_labels(ctx[b, : int(lens[b])], 5)
        spent += time.perf_counter() - t0
        done += int(lens[b])
        if spent >= budget_s:
            break
    return {"value": done / spent, "unit": LABEL_UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{wl.name}: oracle copy_labels on whole rows, {done} positions (single thread)"}


def run_labels(args, world, rank, local):
    """--task labels: switchsd_copy_labels over R replica batches of the workload's contexts (inputs
    larger than L2), K calls in a CUDA graph; value = labelled positions per second."""
    import torch
    from paper_2609_20186_gb300 import binding as bd

    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA device (the controller has no CPU path)")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    lib = bd.load()
    wl = synth.get_workload(args.workload)
    W, K = args.warmup, args.steps
    props = torch.cuda.get_device_properties(dev)
    l2 = int(getattr(props, "L2_cache_size", 128 << 20))
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = label_cpu_baseline(wl, args.cpu_seconds)
    ctx1, lens1 = wl.contexts()
    B, cap = ctx1.shape
    R = choose_replicas(B * cap * 4, l2, max(K, 1))
    ctx = torch.from_numpy(np.tile(ctx1, (R, 1))).to(dev)
    lens = torch.from_numpy(np.tile(lens1, R)).to(dev)
    labels = torch.zeros(R * B, cap, dtype=torch.uint8, device=dev)
    ws_bytes = int(lib.switchsd_labels_workspace_bytes(B, cap))
    ws = torch.empty(R, ws_bytes, dtype=torch.uint8, device=dev)
    cs = torch.cuda.Stream(dev)
    sp = cs.cuda_stream

    def call(i):
        r = i % R
        code = lib.switchsd_copy_labels(ctx.data_ptr() + r * B * cap * 4, lens.data_ptr() + r * B * 4, B, cap, 5,
                                        labels.data_ptr() + r * B * cap, ws[r].data_ptr(), ws_bytes, sp)
        if code != 0:
            raise RuntimeError(f"switchsd_copy_labels failed: {code}")

    with torch.cuda.stream(cs):
        for i in range(max(W, 3)):
            call(i)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cs):
            for i in range(K):
                call(i)
        g.replay()
        cs.synchronize()
        barrier(world)
        sampler = ClockSampler(_gpu_uuid(props))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(cs)
        g.replay()
        e1.record(cs)
        e1.synchronize()
        torch.cuda.synchronize()
        clocks = sampler.stop()
    ms = e0.elapsed_time(e1)
    secs = reduce_max(ms / 1e3, world)
    positions = float(lens1.sum()) * K
    value = replica_throughput(positions, secs, world)
    bytes_per_call = float(lens1.sum()) * 4 + B * cap                # context read, labels written
    achieved = bytes_per_call / (secs / K) / 1e9
    peaks = measured_peaks()
    if rank == 0:
        line = {"metric": LABEL_METRIC, "value": value, "unit": LABEL_UNIT, "n_gpus": world, "steps": K,
                "warmup": W, "ms_per_step": secs * 1e3 / K, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "int32 tokens, uint8 labels", "data": "synthetic",
                "config": {"workload": wl.name, "task": "labels", "B": B, "cap": cap, "n_train": 5,
                           "global_batch": B * world, "seq_len": wl.L0, "parallelism": f"replicas{world}",
                           "replicas": R,
                           "l2": f"inputs larger than L2: {R} batches of B={B} ({R * B * cap * 4 >> 20} MiB)"},
                "roofline": {"kernel": "switchsd_copy_labels", "bound": "hbm", "achieved": achieved,
                             "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
                             "traffic": None, "algorithmic_bytes_per_launch": bytes_per_call,
                             "peak_source": f"{peaks['source']} hbm_gbs (copy)"},
                "gpu_launches": 2 * K, "clocks": clocks, "cpu_baseline": cpu}
        print(json.dumps(line), flush=True)


def main(argv=None):
    args = parse_args(argv)
    world, rank, local = dist_init(args.gpus)
    try:
        if args.impl == "reference":
            run_reference(args, world, rank)
        elif args.task == "labels":
            run_labels(args, world, rank, local)
        else:
            run_ours(args, world, rank, local)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
