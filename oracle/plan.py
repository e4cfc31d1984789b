"""Per-token step plan of Urgency-Aware Denoising -- oracle (test infrastructure).

Sec. 4.2, Eq. 4: every action i carries its own step budget N_i; the vanilla policy is the
uniform case N_i = N* (Sec. 3, Eq. 2). The integration interval is the same for every
action, so action i advances with Euler step 1/N_i (Eq. 5) and sits at flow time
(k-1)/N_i when step k evaluates it. An action whose budget is spent before N* (an urgent
action, "early" below) is released at step N_i (Sec. 4.2, UAER). With Trajectory
Reconciliation its internal state is re-integrated with the canonical step 1/N* (Eq. 6) and
continues as a ghost state with step 1/N* (Eq. 7, second case), i.e. at flow time (k-1)/N*.

Readings where the paper is silent (recorded with the other readings of the build):
  * several release groups: every budget below N* is an early-release group; each is
    released at its own step and reconciled to 1/N*;
  * flow time fed to the time embedding is the fraction of the interval already covered,
    tau = (k-1)/N_i in [0, 1), 0 at the noise end;
  * without TR (UAER-only ablation) a released action is fed back frozen at its released
    value with tau = 1.

Times are kept as exact fractions so that the CUDA path's integer plan can be compared
bit-exactly.
"""
from __future__ import annotations

from dataclasses import dataclass
from fractions import Fraction

import numpy as np


@dataclass
class TokenStep:
    active: bool      # k <= N_i: the action's own Euler update runs this step
    ghost: bool       # early action past its release: ghost state (TR) or frozen (no TR)
    tau: Fraction     # flow time fed to the velocity network
    release: bool     # k == N_i < N*: released after this step's update


def n_star(budgets) -> int:
    return int(np.max(budgets))


def step_plan(budgets, k: int, tr: bool = True):
    """Plan of step k (1-based) for every token of one robot."""
    ns = n_star(budgets)
    out = []
    for n_i in (int(b) for b in budgets):
        if n_i < 1:
            raise ValueError("step budgets must be >= 1")
        if k <= n_i:
            out.append(TokenStep(True, False, Fraction(k - 1, n_i), k == n_i and n_i < ns))
        elif tr:
            out.append(TokenStep(False, True, Fraction(k - 1, ns), False))
        else:
            out.append(TokenStep(False, True, Fraction(1), False))
    return out


def executable_tail(budgets, n_exec: int):
    """Tail actions that GAC corrects: full budget and index < S (Eq. 9, i = U..S-1)."""
    ns = n_star(budgets)
    return [i for i, n_i in enumerate(budgets) if int(n_i) == ns and i < n_exec]


def early_tokens(budgets):
    """Actions released before N* (the urgent set U of Eq. 3, one or more groups)."""
    ns = n_star(budgets)
    return [i for i, n_i in enumerate(budgets) if int(n_i) < ns]


def distinct_times(budgets, tr: bool = True):
    """Every flow time the schedule feeds to the network (the time-conditioning set)."""
    ns = n_star(budgets)
    return sorted({ts.tau for k in range(1, ns + 1) for ts in step_plan(budgets, k, tr)})
