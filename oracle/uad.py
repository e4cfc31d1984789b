"""The UAD denoising loop in fp64 -- oracle (test infrastructure).

Follows, in the paper's order:
  Sec. 3, Eqs. 1-2   x_0 ~ N(0, I); v_k = F(x_{k-1}); x_k = x_{k-1} + v_k / N.
  Sec. 4.2, Eqs. 4-5 per-action budgets N_i and steps x_k^i = x_{k-1}^i + v_k^i / N_i;
                     UAER: after N_i < N* steps, a^i = x_{N_i}^i is released.
  Sec. 4.3, Eq. 6    TR: x'^i_K = x_0^i + (1/N*) sum_{k<=K} v_k^i for released actions (kept
                     here as a running sum started at x_0, added to every step, which is the
                     same sum in the same order as Eq. 6).
  Sec. 4.3, Eq. 7    reconciled (ghost) states are fed to later evaluations and continue with
                     step 1/N*; tail actions continue with 1/N*.
  Sec. 4.3           ghost actions a'^i = x'^i_{N*}.
  Sec. 4.4, Eq. 8    E = sum over released actions of (a'^i - a^i).
  Sec. 4.4, Eq. 9    a^i = x^i_{N*} + E / |executable tail| on additive dimensions; other
                     dimensions (rotations, gripper) are left unchanged; skipped for
                     chunk-relative actions (Sec. 4.4, last paragraph; App. C.4).

The velocity network is passed in as ``velocity(u, tau) -> v`` so that the loop can be
checked with closed-form fields as well as with the synthetic transformer.
"""
from __future__ import annotations

import numpy as np

from . import so3
from .plan import early_tokens, executable_tail, n_star, step_plan


def denoise(velocity, x0, budgets, n_exec=None, tr=True, gac=True, gac_mask=None,
            chunk_relative=False, rot_dim=None):
    """Run one action chunk.

    velocity   callable (u [H, D], tau [H]) -> v [H, D]
    x0         initial noise [H, D]
    budgets    per-action step budgets N_i [H] (ints >= 1); N* = max N_i
    n_exec     S, actions executed before replanning (default H)
    tr, gac    Trajectory Reconciliation / Ghost Action Correction on or off
    gac_mask   [D] bool, True for additive dimensions (default: all additive)
    rot_dim    first of three dimensions holding a rotation vector, corrected by composition
               on SO(3) (so3.py; never additive whatever gac_mask says); None: no rotation

    Returns a dict with
      final         [H, D]  actions as handed to the controller: released actions for early
                            tokens, x_{N*} (+ GAC) for the rest
      released      [H, D]  a^i for early tokens (NaN elsewhere)
      ghost         [H, D]  reconciled end states: x'_{N*} for early tokens, x_{N*} elsewhere;
                            without TR there is no reconciled state (ghosts exist through
                            TR, Sec. 4.3), so early rows hold the frozen action fed back
      release_step  [H]     N_i for early tokens, N* for the others (when they are available)
      E             [D]     Eq. 8 estimate (zeros when GAC does not run); on the rotation
                            dimensions the rotation vector of the accumulated error e_R
      evals         int     evaluations of the velocity network (N*)
      tail          list    indices that GAC corrected
    """
    x0 = np.asarray(x0, dtype=np.float64)
    budgets = [int(b) for b in budgets]
    H, D = x0.shape
    if len(budgets) != H:
        raise ValueError("one budget per action")
    if gac and not tr and not chunk_relative:
        raise ValueError("GAC needs the ghost actions that TR produces")
    S = H if n_exec is None else int(n_exec)
    ns = n_star(budgets)
    early = early_tokens(budgets)
    x = x0.copy()
    g = x0.copy()                      # ghost / reconciled state (only early rows are used)
    released = np.full((H, D), np.nan)
    release_step = np.full(H, ns, dtype=np.int64)
    evals = 0
    for k in range(1, ns + 1):
        plan = step_plan(budgets, k, tr)
        u = np.empty_like(x)
        tau = np.empty(H)
        for i, ts in enumerate(plan):
            if ts.active:
                u[i] = x[i]
            elif tr:
                u[i] = g[i]
            else:
                u[i] = released[i]
            tau[i] = float(ts.tau)
        v = np.asarray(velocity(u, tau), dtype=np.float64)
        evals += 1
        for i, ts in enumerate(plan):
            if ts.active:
                x[i] = x[i] + v[i] / budgets[i]
            if budgets[i] < ns and tr:
                g[i] = g[i] + v[i] / ns
            if ts.release:
                released[i] = x[i]
                release_step[i] = k
    final = x.copy()
    ghost = x.copy()
    ghost[early] = g[early] if tr else released[early]
    E = np.zeros(D)
    tail = []
    if gac and not chunk_relative and early:
        tail = executable_tail(budgets, S)
        if tail:
            E = np.sum(g[early] - released[early], axis=0)
            mask = np.ones(D, dtype=bool) if gac_mask is None else np.asarray(gac_mask, dtype=bool).copy()
            if rot_dim is not None:
                rd = slice(rot_dim, rot_dim + 3)
                mask[rd] = False
                E[rd], final[tail, rd] = so3.gac_rotation(released[early][:, rd], g[early][:, rd],
                                                          final[tail][:, rd])
            final[np.ix_(tail, np.nonzero(mask)[0])] += E[mask] / len(tail)
    return dict(final=final, released=released, ghost=ghost, release_step=release_step,
                E=E, evals=evals, tail=tail, n_star=ns)


def denoise_batch(models, x0, budgets, **kw):
    """Independent robots: one chunk per (model, noise, budgets) row."""
    return [denoise(m.velocity, x0[b], budgets[b], **kw) for b, m in enumerate(models)]
