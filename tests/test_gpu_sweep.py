"""Schedule sweep on the pi0-like expert at batch 1 (the measured side of App. A "Latency", App. B
and App. C.1 "Parameter Configuration"), from device release times of the CUDA path:

* Trajectory Reconciliation adds no evaluation, so a chunk takes N* evaluations whatever the
  schedule: chunk time is flat across the sweep grid (first-group budget x size, rest at 10);
* an action released after k steps is available after k evaluations: first-action time is
  k times the evaluation time;
* the U selection at K = 1 (smallest U whose tail blocking is under 0.2 ms) picks the same U
  from the oracle's control clock (oracle/clock.py) as from bench.py's, and both agree with the
  closed form of Eq. 12 at the measured evaluation time.
"""
import os
import statistics
import sys

import numpy as np
import pytest
import torch

import paper_2609_37772_gb300 as uad
from oracle.clock import action_waits, latency_model_uaer
from uad_inputs import ARCHS, group_budgets, make_noise, make_prefix_kv, make_weights, sweep_grid

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402

pytestmark = pytest.mark.gpu
N_STAR, REPS = 10, 4


@pytest.fixture(scope="module")
def pi0():
    a = ARCHS["pi0"]
    ex = uad.Expert(a, make_weights(a), max_batch=1)
    ex.set_prefix(0, *make_prefix_kv(a))
    ex.prepare_times(N_STAR)
    noise = torch.from_numpy(make_noise(a, 1)).cuda()
    yield a, ex, noise
    ex.close()


def run(ex, noise, bud, reps=REPS, warm=2):
    """Device release times of every action (ms from the chunk's first kernel), per chunk."""
    for _ in range(warm):
        ex.denoise(noise, bud)
        ex.finish(timeout_us=60_000_000)
    rows, evals = [], set()
    for _ in range(reps):
        ex.denoise(noise, bud)
        r = ex.finish(timeout_us=60_000_000)
        evals.add(r["evals"])
        st = ex.step_times()
        rows.append([float(st[int(b) - 1]) for b in bud[0]])
    return rows, evals, st


def test_chunk_time_flat_and_first_action_linear_in_k(pi0):
    a, ex, noise = pi0
    chunk, per_eval = {}, {}
    for k, u in sweep_grid():
        bud = group_budgets(a.chunk_len, [(0, u - 1, k), (u, a.chunk_len - 1, N_STAR)])[None]
        rows, evals, st = run(ex, noise, bud)
        assert evals == {N_STAR}                       # TR: no evaluation beyond N*
        chunk[(k, u)] = statistics.median(max(r) for r in rows)
        t_eval = chunk[(k, u)] / N_STAR
        first = statistics.median(r[0] for r in rows)
        per_eval[(k, u)] = t_eval
        # released after k evaluations (the chunk's start-up is a few microseconds)
        assert abs(first - k * t_eval) <= 0.05 * k * t_eval + 0.02, (k, u, first, t_eval)
    lo, hi = min(chunk.values()), max(chunk.values())
    print(f"chunk ms over the sweep grid: {lo:.3f} .. {hi:.3f}; per evaluation "
          f"{min(per_eval.values()):.4f} .. {max(per_eval.values()):.4f} ms")
    assert hi <= 1.05 * lo, chunk


def test_u_selection_matches_the_oracle_clock(pi0):
    a, ex, noise = pi0
    S, t_evals = 10, []
    for t_act in (12.5, 50.0, 0.5):
        sel_bench, sel_oracle = None, None
        for u in range(1, S):
            bud = group_budgets(a.chunk_len, [(0, u - 1, 1), (u, a.chunk_len - 1, N_STAR)])[None]
            rows, evals, _ = run(ex, noise, bud, reps=2, warm=1)
            assert evals == {N_STAR}
            ready = rows[-1][:S]
            b_bench = bench.tail_blocking_ms(ready, t_act, u)
            b_oracle = action_waits(ready, t_act)[u]
            assert b_bench == pytest.approx(b_oracle, abs=1e-12)
            # Eq. 12's blocking term at the measured evaluation time (no VLM here)
            t_d = ready[u] / N_STAR
            t_evals.append(t_d)
            model = max((N_STAR - 1) * t_d - u * t_act, 0.0)
            assert abs(b_oracle - model) <= 0.05 * N_STAR * t_d + 0.02, (u, t_act, b_oracle, model)
            if sel_bench is None and b_bench < 0.2:
                sel_bench = u
            if sel_oracle is None and b_oracle < 0.2:
                sel_oracle = u
        assert sel_bench == sel_oracle, (t_act, sel_bench, sel_oracle)
        print(f"T_act {t_act} ms: selected U = {sel_bench}")
    # with a 0.5 ms action the tail cannot keep up for small U: blocking at U = 1 is positive
    assert latency_model_uaer(0.0, statistics.mean(t_evals), N_STAR, 1, 1, 0.5, S) > 0


def test_chunk_time_linear_in_uniform_n(pi0):
    """App. B: with every action at the same budget N, a chunk is N evaluations, so its time is
    linear in N (a small constant for the chunk's start-up and the time table aside)."""
    a, ex, noise = pi0
    ns = [1, 2, 4, 6, 8, 10]
    t = []
    for n in ns:
        bud = group_budgets(a.chunk_len, [(0, a.chunk_len - 1, n)])[None]
        rows, evals, _ = run(ex, noise, bud, reps=3, warm=1)
        assert evals == {n}
        t.append(statistics.median(max(r) for r in rows))
    slope, icpt = np.polyfit(ns, t, 1)
    resid = max(abs(ti - (slope * n + icpt)) for n, ti in zip(ns, t))
    print(f"chunk ms = {icpt:.3f} + {slope:.4f} N (largest residual {resid:.4f} ms)")
    assert resid <= 0.02 * max(t)
    assert abs(icpt) <= 0.25 * slope
