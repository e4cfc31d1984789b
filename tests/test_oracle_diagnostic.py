"""The relative-L2 diagnostic of Trajectory Reconciliation (Sec. 4.3, Fig. 3) on the oracle:
properties the paper states (exact recovery at K = 1) and the structure of the variants."""
import numpy as np
import pytest

import bench
from oracle.model import build_model
from oracle.uad import denoise
from uad_inputs import ARCHS, group_budgets, make_noise, make_prefix_kv, make_weights


@pytest.fixture(scope="module")
def tiny():
    a = ARCHS["tiny"]
    return a, build_model(a, make_weights(a, seed=4), make_prefix_kv(a, robot=0, seed=4))


def run(tiny, bud, **kw):
    a, m = tiny
    noise = make_noise(a, seed=21)[0]
    van = denoise(m.velocity, noise, [3] * a.chunk_len, tr=True, gac=False)["final"]
    r = denoise(m.velocity, noise, bud, **kw)
    return bench.diagnostic_errors(r["final"], r["ghost"], van, bud, kw.get("tr", True)), r


def test_k1_with_tr_recovers_vanilla_exactly(tiny):
    """K = 1: the first evaluation equals vanilla's, re-integrating it at 1/N* gives vanilla's
    state, so tail and ghost actions match vanilla exactly before GAC (Sec. 4.3)."""
    a, _ = tiny
    bud = group_budgets(a.chunk_len, [(0, 4, 1), (5, a.chunk_len - 1, 3)])
    e, _ = run(tiny, bud, tr=True, gac=False)
    assert e["tail"] == 0.0 and e["ghost"] == 0.0
    assert e["released"] > 1e-3          # one Euler step of size 1 is not three of size 1/3


def test_uniform_schedule_has_no_error(tiny):
    a, _ = tiny
    e, _ = run(tiny, [3] * a.chunk_len, tr=True, gac=True)
    assert e == {"tail": 0.0}


def test_early_release_without_tr_perturbs_the_tail(tiny):
    """Naive early release changes the joint context of the tail (Sec. 4.3): nonzero tail error
    at K = 1 without TR, where TR makes it exactly zero."""
    a, _ = tiny
    bud = group_budgets(a.chunk_len, [(0, 4, 1), (5, a.chunk_len - 1, 3)])
    e, _ = run(tiny, bud, tr=False, gac=False)
    assert e["tail"] > 1e-6 and "ghost" not in e


@pytest.mark.parametrize("k", [1, 2])
def test_variants_share_what_they_must(tiny, k):
    """Released actions are fixed at step K whatever happens later; GAC changes only the tail."""
    a, _ = tiny
    bud = group_budgets(a.chunk_len, [(0, 3, k), (4, a.chunk_len - 1, 3)])
    e0, r0 = run(tiny, bud, tr=False, gac=False)
    e1, r1 = run(tiny, bud, tr=True, gac=False)
    e2, r2 = run(tiny, bud, tr=True, gac=True)
    early = np.asarray(bud) < 3
    assert np.array_equal(r0["final"][early], r1["final"][early])
    assert np.array_equal(r1["final"][early], r2["final"][early])
    assert np.array_equal(r1["ghost"], r2["ghost"])
    assert e1["released"] == e0["released"] == e2["released"] and e1["ghost"] == e2["ghost"]
    # GAC moves the tail by exactly E / |tail| per row on every additive dimension (Eq. 9)
    tail = r2["tail"]
    assert np.allclose(r2["final"][tail] - r1["final"][tail], r2["E"] / len(tail), rtol=0, atol=1e-12)


def test_relative_l2_definition():
    ref = np.array([[3.0, 4.0], [0.0, 0.0]])
    assert bench.rel_l2(ref, ref) == 0.0
    assert abs(bench.rel_l2(ref * 1.1, ref) - 0.1) < 1e-12
    assert bench.rel_l2(np.ones(3), np.zeros(3)) == pytest.approx(np.sqrt(3))
