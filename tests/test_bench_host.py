"""CPU checks of bench.py's host logic: the replica (N > 1) timing reduction over gloo ranks,
its action-availability-latency arithmetic against the oracle's control clock, and the time
bound of the reference arm."""
import multiprocessing as mp
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank), UAD_BENCH_BACKEND="gloo")
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist
    w, r, _ = bench.dist_setup()
    bench.barrier(w)
    t = bench.max_over_ranks(100.0 + 7.0 * r, w)
    q.put((r, w, t))
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_replica_timing_takes_max_over_ranks(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    assert [g[0] for g in got] == list(range(world))
    assert all(g[1] == world for g in got)
    assert all(g[2] == 100.0 + 7.0 * (world - 1) for g in got)


def test_bench_aal_matches_oracle_clock():
    sys.path.insert(0, ROOT)
    import bench
    from oracle.clock import aal
    rng = np.random.default_rng(0)
    for _ in range(50):
        H = int(rng.integers(2, 60))
        ready = np.sort(rng.uniform(0, 30, size=H)).tolist()
        ready = [r if rng.random() < 0.7 else ready[0] for r in ready]
        t_act = float(rng.uniform(0.5, 20))
        S = int(rng.integers(1, H + 1))
        assert bench.aal_ms(ready, t_act, S) == pytest.approx(aal(ready, t_act, S), rel=1e-12, abs=1e-12)


def test_tail_blocking_under_the_clock():
    """First tail action (index U) waits max(0, ready_U - request_U), request_U = start of the
    urgent actions' execution + U * T_act (App. C.1 latency model with one release group)."""
    import bench
    ready = [5.0, 5.0] + [30.0] * 8
    assert bench.tail_blocking_ms(ready, 12.5, 2) == 0.0          # 5 + 2 * 12.5 = 30: just in time
    assert bench.tail_blocking_ms(ready, 10.0, 2) == 5.0          # 5 + 2 * 10 = 25 < 30
    assert bench.tail_blocking_ms([4.0] + [20.0] * 9, 10.0, 1) == 6.0
    # the model's closed form: blocking = max((N* - K) T_D - U T_act, 0) with ready times K T_D, N* T_D
    t_d, k, ns, t_act = 1.3, 1, 10, 2.0
    for u in range(1, 9):
        r = [k * t_d] * u + [ns * t_d] * (10 - u)
        assert abs(bench.tail_blocking_ms(r, t_act, u) - max((ns - k) * t_d - u * t_act, 0.0)) < 1e-12


def test_bootstrap_interval():
    import bench
    lo, hi = bench.bootstrap_ci([2.0] * 7)
    assert lo == hi == 2.0
    v = np.random.default_rng(3).normal(10.0, 1.0, 200)
    lo, hi = bench.bootstrap_ci(v)
    se = v.std(ddof=1) / np.sqrt(v.size)
    assert lo < v.mean() < hi
    assert abs((hi - lo) - 2 * 1.96 * se) < 0.25 * (2 * 1.96 * se)   # normal-theory width within 25%


def test_reference_arm_is_bounded_in_time(monkeypatch, capsys):
    """The reference arm (the CPU oracle) stops once its time bound is spent, whatever K is, and
    still reports at least one timed chunk; its line carries the fields the driver reads."""
    import argparse
    import json
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setattr(bench, "REF_SECONDS", 0.0)
    args = argparse.Namespace(gpus=1, steps=1000, warmup=3)
    assert bench.run_reference(args, bench.WORKLOADS["tiny"], 1, 0) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0 and line["steps"] == 1000
    assert line["cpu_baseline"]["value"] == line["value"]
    assert line["cpu_baseline"]["sample"].startswith("1 full chunk(s) of robot 0 timed after 0 warm-up")
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}


def test_roofline_bound_follows_the_ridge_point():
    """The dominant kernel is held to HBM below the ridge point of the peaks and to the bf16
    tensor rate above it; achieved = its work per launch over its average launch time."""
    sys.path.insert(0, ROOT)
    import bench
    pk = (6000.0, 2000.0, 1500.0, "measured")   # GB/s, burst TFLOP/s, sustained TFLOP/s
    # latency-bound evaluation kernel: 600 MB and 36 GFLOP per launch (60 flop/B < 250 ridge)
    prof = [{"name": "step", "launches": 10, "total_ms": 8.0, "bytes": 6.0e9, "flops": 3.6e11},
            {"name": "euler", "launches": 10, "total_ms": 0.1, "bytes": 1.0e6, "flops": 1.0e6}]
    r = bench.roofline_object(prof, 10, 0.81, pk, None)
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["kernel"] == "step"
    assert abs(r["achieved"] - 6.0e9 / 8e-3 / 1e9) < 1e-6 and abs(r["frac"] - 750.0 / 6000.0) < 1e-9
    assert r["peak_source"].startswith("measured hbm_gbs")
    # a large-batch GEMM: 50 MB and 54 GFLOP per launch (1080 flop/B > ridge), 180 launches
    prof = [{"name": "gate_up", "launches": 180, "total_ms": 13.5, "bytes": 9.0e9, "flops": 9.72e12},
            {"name": "attention", "launches": 180, "total_ms": 9.0, "bytes": 3.6e9, "flops": 6.1e12}]
    r = bench.roofline_object(prof, 10, 3.9, pk, None)
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s" and r["peak"] == 1500.0
    assert abs(r["achieved"] - 9.72e12 / 13.5e-3 / 1e12) < 1e-6
    assert abs(r["flops_per_launch"] - 5.4e10) < 1.0 and r["peak_source"].startswith("measured bf16_tflops_sustained")
    assert abs(r["step"]["tensor_frac"] - (15.82e12 / 10) / 3.9e-3 / 1e12 / 1500.0) < 1e-9


def test_oracle_thread_count_is_what_the_process_may_use():
    import bench
    n = bench.oracle_threads()
    assert 1 <= n <= (os.cpu_count() or n)


def test_gpus_flag_starts_the_ranks_itself():
    """`bench.py --gpus 2` without an outside launcher re-runs itself as two ranks under
    torch.distributed.run (gloo here, no GPU); rank 0 alone prints the reference arm's line."""
    import subprocess
    env = dict(os.environ, UAD_BENCH_BACKEND="gloo")
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK", "MASTER_ADDR", "MASTER_PORT"):
        env.pop(k, None)
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                        "--workload", "tiny", "--steps", "1", "--warmup", "0"],
                       capture_output=True, text=True, timeout=600, env=env, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    import json
    lines = [json.loads(x) for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1 and lines[0]["impl"] == "reference", r.stdout
    assert lines[0]["n_gpus"] == 2


def test_rank_count_must_match_gpus_flag():
    import subprocess
    env = dict(os.environ, WORLD_SIZE="3", RANK="0", LOCAL_RANK="0")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                        "--workload", "tiny", "--steps", "1", "--warmup", "0"],
                       capture_output=True, text=True, timeout=120, env=env, cwd=ROOT)
    assert r.returncode == 2 and "refusing" in r.stderr
    assert not [x for x in r.stdout.splitlines() if x.startswith("{")]
