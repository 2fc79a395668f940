#!/usr/bin/env python3
"""Benchmark of the SwitchSD per-step controller on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload zipf_32k] [--impl ours|reference]

A step is one controller iteration over a batch: switchsd_step (search, probe, switch, copy draft),
the target stand-in (switchsd_harness_target, not timed: it replaces the out-of-scope target forward)
and switchsd_verify (greedy verification + append).  The default workload is B=64 sequences of
32,768-token contexts (Zipf(1.1) tokens, 5 % planted copy spans, d=4096 linear probe, n 3..8, k=16).

Timing: before every timed step an unrelated buffer of 2x L2 is written and then a second one is read,
so the step finds its inputs in HBM, not in L2 (the contexts total ~10.6 MB, which L2 would
otherwise hold).  CUDA events on the launching stream bracket switchsd_step and switchsd_verify;
``value`` = B x steps / the summed controller time.  The dominant kernel's roofline uses the
algorithmic bytes of each launch (the row contexts scanned, the hidden states and probe weights read,
the outputs written) over its event-timed duration.  ``e2e`` repeats the loop through host buffers:
each step copies the step's hidden states from pinned host memory and reads back the modes, draft
lengths, drafts and accepted lengths.

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
PROFILE_SUMMARY = os.path.join(ROOT, "profiles", "step_kernel_zipf_32k.txt")


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=512)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--workload", default="zipf_32k", choices=sorted(synth.WORKLOADS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--split", type=int, default=0, help="CTAs per row (0 = library choice)")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="budget of the CPU-baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
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
    for f in ("common.cuh", "step.cu"):
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
def time_oracle(wl: synth.Workload, budget_s: float, max_steps: int, rows: int | None = None,
                warmup: int = 0):
    """Runs the oracle loop (oracle step, host target stand-in, oracle verify) on rows [0, R):
    ``warmup`` untimed steps, then up to max_steps timed steps or until budget_s of oracle time is
    spent.  Returns (seq*steps, seconds, timed_steps, R).  Only the oracle's calls are timed."""
    import oracle
    R = wl.B if rows is None else min(rows, wl.B)
    ctx, lens = wl.contexts()
    labels = wl.labels()
    pw = wl.probe_weights()
    hp = wl.harness_params()
    spent = 0.0
    done = 0
    for t in range(warmup + max_steps):
        h = wl.hidden(t)
        t0 = time.perf_counter()
        out = oracle.step(ctx, lens, h, pw, k=wl.k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                          logit_tau=wl.logit_tau, probe_kind=wl.probe_kind,
                          probe_hidden=wl.probe_hidden, rows=(0, R))
        dt = time.perf_counter() - t0
        vd, vl, tg = synth.harness_targets(hp, t, lens, out["mode"], out["draft"], out["len"],
                                           labels, rows=range(R))
        t0 = time.perf_counter()
        oracle.verify(ctx, lens, vd, vl, tg, rows=(0, R))
        dt += time.perf_counter() - t0
        if t < warmup:
            continue
        spent += dt
        done += 1
        if spent >= budget_s:
            break
    return R * done, spent, done, R


def cpu_baseline(wl: synth.Workload, budget_s: float) -> dict:
    units, secs, steps, R = time_oracle(wl, budget_s, wl.steps)
    return {"value": units / secs, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{wl.name}: rows 0..{R - 1}, first {steps} controller steps (oracle step + "
                      f"verify timed, single thread; the host target stand-in is not timed)"}


def config_of(wl: synth.Workload, world: int, split: int) -> dict:
    return {"workload": wl.name, "B": wl.B, "L0": wl.L0, "V": wl.V, "d": wl.d, "k": wl.k,
            "n_min": wl.n_min, "n_max": wl.n_max, "kappa": wl.kappa_eff, "tau": wl.tau,
            "probe": "linear" if wl.probe_kind == 0 else f"mlp{wl.d}x{wl.probe_hidden}",
            "global_batch": wl.B * world, "seq_len": wl.L0, "parallelism": f"replicas{world}",
            "split": split,
            "l2": "flushed before every timed step (write 2x L2, then read another 2x L2 buffer)"}


def run_reference(args, world, rank):
    """The reference arm: the CPU oracle on this host, W untimed + K timed steps of the workload on
    a bounded sample of rows (all rows when B <= 64, else the first 16)."""
    if rank != 0:
        return
    import oracle
    oracle.build()
    base = synth.get_workload(args.workload)
    wl = base.scaled(steps=args.warmup + args.steps)
    R = wl.B if wl.B <= 64 else 16
    units, secs, steps, R = time_oracle(wl, float("inf"), args.steps, rows=R, warmup=args.warmup)
    value = units / secs
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": secs / steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int32 (search/verify), f64 (probe)", "data": "synthetic",
            "impl": "reference",
            "config": config_of(base, world, args.split),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": f"{wl.name}: rows 0..{R - 1}, {args.warmup} untimed + "
                                       f"{steps} timed steps, single thread"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------------------
# GPU run
# ------------------------------------------------------------------------------------------------
def run_ours(args, world, rank, local):
    import torch
    from paper_2609_20186_gb300 import Session, bf16_tensor, binding

    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA device (the controller has no CPU path)")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    binding.load()
    base = synth.get_workload(args.workload)
    W, K = args.warmup, args.steps
    wl = base.scaled(steps=W + K)     # same per-step law; capacity sized for W + K iterations
    B, d, k = wl.B, wl.d, wl.k

    # CPU baseline first (rank 0, N = 1): the oracle runs before any CUDA work of the timed run
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        cpu = cpu_baseline(base, args.cpu_seconds)

    ctx, lens = wl.contexts()
    labels = wl.labels()
    pw = wl.probe_weights()
    hidden_host = wl.hidden_all()                    # [W+K, B, d] bf16 bits
    hidden = bf16_tensor(hidden_host, dev)
    sess = Session(ctx, lens, pw, k=k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                   logit_tau=wl.logit_tau, probe_kind=wl.probe_kind,
                   probe_hidden=wl.probe_hidden, labels=labels, harness=wl.harness_params(),
                   split=args.split, device=dev)
    props = torch.cuda.get_device_properties(dev)
    l2 = int(getattr(props, "L2_cache_size", 128 << 20))
    flush_w = torch.empty(2 * l2 // 4, dtype=torch.float32, device=dev)
    flush_r = torch.ones(2 * l2 // 4, dtype=torch.float32, device=dev)
    sink = torch.zeros(1, dtype=torch.float32, device=dev)

    def flush():
        flush_w.fill_(1.0)
        sink.add_(flush_r.sum())

    for t in range(W):
        flush()
        sess.iterate(hidden[t], t, debug=False)
    torch.cuda.synchronize()

    lens_hist = torch.zeros(K, B, dtype=torch.int32, device=dev)
    len_hist = torch.zeros(K, B, dtype=torch.int32, device=dev)
    acc_hist = torch.zeros(K, B, dtype=torch.int32, device=dev)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
    uuid = None
    try:
        uuid = "GPU-" + str(props.uuid)
    except Exception:
        pass
    barrier(world)
    torch.cuda.synchronize()
    sampler = ClockSampler(uuid)
    time.sleep(0.05)
    wall0 = time.perf_counter()
    for i in range(K):
        t = W + i
        flush()
        lens_hist[i].copy_(sess.lens)
        ev[i][0].record()
        sess.step(hidden[t], debug=False)
        ev[i][1].record()
        sess.harness(t)
        ev[i][2].record()
        sess.verify(debug=False)
        ev[i][3].record()
        len_hist[i].copy_(sess.len)
        acc_hist[i].copy_(sess.accept)
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    barrier(world)
    clocks = sampler.stop()

    step_ms = np.array([e[0].elapsed_time(e[1]) for e in ev])
    verify_ms = np.array([e[2].elapsed_time(e[3]) for e in ev])
    ctrl_s = float((step_ms.sum() + verify_ms.sum()) / 1e3)
    value = replica_throughput(B * K, ctrl_s, world)
    ms_per_step = reduce_max(ctrl_s, world) / K * 1e3

    Lh = lens_hist.cpu().numpy().astype(np.int64)
    lh = len_hist.cpu().numpy().astype(np.int64)
    ah = acc_hist.cpu().numpy().astype(np.int64)
    if wl.probe_kind == 0:
        probe_bytes = 2 * B * d + 2 * d
    else:
        probe_bytes = 2 * B * d + 2 * (wl.probe_hidden * d + wl.probe_hidden)
    step_bytes = 4 * Lh.sum(axis=1) + probe_bytes + 4 * lh.sum(axis=1) + 12 * B
    verify_bytes = 20 * B + 12 * (np.maximum(ah, 0) + 1).sum(axis=1)
    peaks = measured_peaks()
    step_gbs = float(step_bytes.mean() / (step_ms.mean() / 1e3) / 1e9)
    verify_gbs = float(verify_bytes.mean() / (verify_ms.mean() / 1e3) / 1e9)
    ctrl_gbs = float((step_bytes.sum() + verify_bytes.sum()) / ctrl_s / 1e9)
    traffic = profiled_traffic(base.name)
    launches_per_step = (2 if wl.probe_kind == 0 else 3)

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(wl, ctx, lens, pw, labels, hidden_host, W, K, args.split, dev, world)

    if rank != 0:
        return
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int32 (search/verify), bf16 in / fp32 accumulate (probe)",
        "data": "synthetic", "config": config_of(base, world, args.split),
        "roofline": {"kernel": "switchsd_step", "bound": "hbm", "achieved": step_gbs,
                     "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": step_gbs / peaks["hbm_gbs"],
                     "traffic": traffic,
                     "algorithmic_bytes_per_launch": float(step_bytes.mean()),
                     "launch_us": float(step_ms.mean() * 1e3),
                     "peak_source": peaks["source"] + " (hbm_gbs, copy)"},
        "controller": {"step_us": float(step_ms.mean() * 1e3),
                       "verify_us": float(verify_ms.mean() * 1e3),
                       "verify_gbs": verify_gbs, "step_plus_verify_gbs": ctrl_gbs,
                       "step_plus_verify_frac": ctrl_gbs / peaks["hbm_gbs"],
                       "loop_wall_ms_per_step_incl_flush_and_harness": wall / K * 1e3,
                       "mean_context_tokens": float(Lh.mean()),
                       "mean_copy_draft": float(lh.mean()),
                       "mean_accept": float(np.maximum(ah, 0).mean())},
        "gpu_launches": K * launches_per_step,
        "gpu_launches_note": f"{launches_per_step} controller kernels per step inside the event "
                             f"brackets; plus {K} target stand-in launches between them",
        "clocks": clocks,
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    print(json.dumps(line), flush=True)


def run_e2e(wl, ctx, lens, pw, labels, hidden_host, W, K, split, dev, world):
    """The same loop through the public API with host buffers: per step, H2D of the hidden states
    from pinned memory, the three calls, D2H of mode / draft length / draft / accepted length."""
    import torch
    from paper_2609_20186_gb300 import Session

    B, d, k = wl.B, wl.d, wl.k
    sess = Session(ctx, lens, pw, k=k, n_min=wl.n_min, n_max=wl.n_max, kappa=wl.kappa,
                   logit_tau=wl.logit_tau, probe_kind=wl.probe_kind, probe_hidden=wl.probe_hidden,
                   labels=labels, harness=wl.harness_params(), split=split, device=dev)
    host_h = torch.from_numpy(hidden_host.view(np.int16)).pin_memory()
    dev_h = torch.empty(B, d, dtype=torch.bfloat16, device=dev)
    out_mode = torch.empty(B, dtype=torch.int32).pin_memory()
    out_len = torch.empty(B, dtype=torch.int32).pin_memory()
    out_draft = torch.empty(B, k, dtype=torch.int32).pin_memory()
    out_acc = torch.empty(B, dtype=torch.int32).pin_memory()
    stream = torch.cuda.current_stream()

    def one(t):
        dev_h.view(torch.int16).copy_(host_h[t], non_blocking=True)
        sess.iterate(dev_h, t, debug=False)
        out_mode.copy_(sess.mode, non_blocking=True)
        out_len.copy_(sess.len, non_blocking=True)
        out_draft.copy_(sess.draft, non_blocking=True)
        out_acc.copy_(sess.accept, non_blocking=True)
        stream.synchronize()

    for t in range(W):
        one(t)
    barrier(world)
    t0 = time.perf_counter()
    for i in range(K):
        one(W + i)
    secs = time.perf_counter() - t0
    value = replica_throughput(B * K, secs, world)
    return {"value": value, "unit": UNIT, "h2d_bytes_per_step": B * d * 2,
            "d2h_bytes_per_step": B * (k + 3) * 4,
            "note": "per step: pinned H2D of hidden, step + target stand-in + verify, D2H of "
                    "mode/len/draft/accept, host sync; L2 not flushed"}


def main(argv=None):
    args = parse_args(argv)
    world, rank, local = dist_init(args.gpus)
    try:
        if args.impl == "reference":
            run_reference(args, world, rank)
        else:
            run_ours(args, world, rank, local)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
