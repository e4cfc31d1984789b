"""CPU checks of the C ABI: the library loads, exports every symbol include/uad.h declares,
and its host-side urgency planner matches the oracle's plan exactly (no GPU needed)."""
import os
import re
from fractions import Fraction

import numpy as np
import pytest

import paper_2609_37772_gb300 as uad
from oracle import plan as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(uad_[a-z0-9_]+)\s*\(", src))
    return sorted(names)


def test_library_exports_every_declared_symbol():
    names = declared_symbols()
    assert len(names) >= 12
    for n in names:
        assert hasattr(uad._lib, n), n
    assert set(uad.EXPORTS) <= set(names)
    assert b"sm_103a" in uad.uad_version()


def _oracle_flags(ts):
    return (1 if ts.active else 0) | (2 if ts.ghost and not ts.tau == 1 else 0)


SCHEDULES = [
    [4] * 10 + [7] * 15 + [10] * 25,
    [1] * 4 + [10] * 12,
    [5] * 4 + [10] * 12,
    [3, 1, 4, 1, 5, 9, 2, 6],
    [2] * 16,
    [8, 16, 16, 16],
    [1] * 5,                       # N* = 1: one step, nothing released early
    [64, 1, 33, 64, 2],            # the largest budget the library accepts
]


@pytest.mark.parametrize("budgets", SCHEDULES)
@pytest.mark.parametrize("tr", [True, False])
def test_host_plan_matches_oracle(budgets, tr):
    ns = P.n_star(budgets)
    for k in range(1, ns + 1):
        got_ns, flags, num, den = uad.plan_step(budgets, k, tr)
        assert got_ns == ns
        for i, ts in enumerate(P.step_plan(budgets, k, tr)):
            assert bool(flags[i] & 1) == ts.active
            assert bool(flags[i] & 2) == (ts.ghost and tr)
            assert bool(flags[i] & 16) == (ts.ghost and not tr)
            assert bool(flags[i] & 4) == ts.release
            assert bool(flags[i] & 8) == (int(budgets[i]) < ns)
            assert Fraction(int(num[i]), int(den[i])) == ts.tau
            assert np.gcd(num[i], den[i]) == 1


def test_brute_force_plans():
    """Every budget assignment with H = 3 and budgets 1..4."""
    import itertools
    for b in itertools.product(range(1, 5), repeat=3):
        ns = max(b)
        for k in range(1, ns + 1):
            _, flags, num, den = uad.plan_step(list(b), k, True)
            for i, ts in enumerate(P.step_plan(list(b), k, True)):
                assert Fraction(int(num[i]), int(den[i])) == ts.tau
                assert bool(flags[i] & 4) == ts.release


def test_plan_rejects_bad_budgets():
    with pytest.raises(uad.UADError):
        uad.plan_step([0, 3], 1)
    with pytest.raises(uad.UADError):
        uad.plan_step([65], 1)
