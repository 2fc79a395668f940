"""Host-side logic of bench.py: replica throughput over ranks (gloo, world size 2, CPU), replica
count for the inputs-larger-than-L2 protocol, the CPU baseline's split of rows over threads, and the
reference arm's JSON line."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    secs = [0.5, 2.0][rank]                     # rank 1 is the slow one
    out[rank] = (bench.replica_throughput(100.0, secs, world), bench.reduce_max(secs, world))
    dist.barrier()
    dist.destroy_process_group()


def test_replica_throughput_gloo_world2():
    ctx = mp.get_context("spawn")
    manager = ctx.Manager()
    out = manager.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    # whole-job throughput: all units of both replicas over the slowest rank's time
    for r in range(2):
        value, tmax = out[r]
        assert tmax == 2.0
        assert value == pytest.approx(200.0 / 2.0)


def test_choose_replicas():
    """The replica count keeps every timed launch's batch out of L2 whatever the step count: the other
    R - 1 batches cover 2.2x L2, and a region of up to 64 launches reads each batch once."""
    sys.path.insert(0, ROOT)
    import bench
    l2 = 126 << 20
    batch = 10 << 20
    for K in (1, 3, 20, 64, 512):
        r = bench.choose_replicas(batch, l2, K)
        assert r & (r - 1) == 0 and (r - 1) * batch >= 2.2 * l2
        assert r >= min(K, 64)
        assert r == 2 or ((r // 2 - 1) * batch < 2.2 * l2 or r // 2 < min(K, 64))  # the smallest such
    assert bench.choose_replicas(1 << 30, l2, 20) == 32      # huge batches: 20 distinct batches still
    assert bench.choose_replicas(1 << 30, l2, 1) == 2
    assert bench.choose_replicas(8 << 10, l2, 20, max_r=1024) == 1024  # far below L2: capped


def test_reference_arm_line():
    """--impl reference times the CPU oracle and prints one JSON line with the contract's keys."""
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "3", "--warmup", "1", "--workload", "uniform_8k"],
                       capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["steps"] == 3 and line["warmup"] == 1
    assert line["value"] > 0 and line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]
    assert line["config"]["workload"] == "uniform_8k"


@pytest.mark.parametrize("mode", ["greedy", "sampled", "candidates"])
def test_threaded_oracle_timing_computes_the_same(mode):
    """The CPU baseline runs the oracle on contiguous row ranges in threads: the loop must leave the same
    contexts and lengths as one thread (rows are independent)."""
    sys.path.insert(0, ROOT)
    import bench
    import synth
    wl = synth.get_workload("zipf_32k").scaled(B=12, L0=3001, steps=6)
    kw = dict(sampled=mode == "sampled", cand=(4, 8) if mode == "candidates" else None)
    one, many = {}, {}
    u1, _, s1, _ = bench.time_oracle(wl, 1e9, 6, threads=1, state=one, **kw)
    u4, _, s4, _ = bench.time_oracle(wl, 1e9, 6, threads=4, state=many, **kw)
    assert (u1, s1) == (u4, s4) == (12 * 6, 6)
    assert (one["lens"] > wl.L0).all()
    assert (one["lens"] == many["lens"]).all() and (one["ctx"] == many["ctx"]).all()
