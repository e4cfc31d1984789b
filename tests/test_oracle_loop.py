"""Pins of the oracle's denoising loop (Eqs. 1-9) against closed forms and invariants.

Nothing here compares the oracle with itself: every expected value comes from a closed form
of the paper's equations (hand-derived rationals in tests/golden/tau_field.txt, matrix
powers, the ODE solution within the Euler error bound) or from an invariant the paper
states (uniform schedule = vanilla, exact recovery at K = 1, GAC preserves the total
displacement, zero extra evaluations).
"""
import os
from fractions import Fraction

import numpy as np
import pytest
import scipy.linalg

from oracle import plan as P
from oracle.uad import denoise

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "tau_field.txt")


def _tau_rows():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if line and not line.startswith("#"):
            ns, k, rel, gh, tail = line.split()
            rows.append((int(ns), int(k), Fraction(rel), Fraction(gh), Fraction(tail)))
    return rows


def tau_field(w, b):
    return lambda u, tau: np.asarray(tau)[:, None] * w[None, :] + b[None, :]


@pytest.mark.parametrize("row", _tau_rows(), ids=lambda r: f"N{r[0]}K{r[1]}")
def test_tau_field_golden(row):
    ns, K, c_rel, c_gh, c_tail = row
    H, U, D = 6, 2, 3
    rng = np.random.default_rng(ns * 100 + K)
    w, b = rng.normal(size=D), rng.normal(size=D)
    x0 = rng.normal(size=(H, D))
    budgets = [K] * U + [ns] * (H - U)
    S = 5
    out = denoise(tau_field(w, b), x0, budgets, n_exec=S, tr=True, gac=True)
    early, tail = [0, 1], [2, 3, 4]
    exp_rel = x0[early] + b + w * float(c_rel)
    exp_gh = x0[early] + b + w * float(c_gh)
    E = U * w * float(c_gh - c_rel)
    exp_tail = x0[tail] + b + w * float(c_tail) + E / len(tail)
    np.testing.assert_allclose(out["released"][early], exp_rel, rtol=0, atol=1e-12)
    np.testing.assert_allclose(out["final"][early], exp_rel, rtol=0, atol=1e-12)
    np.testing.assert_allclose(out["ghost"][early], exp_gh, rtol=0, atol=1e-12)
    np.testing.assert_allclose(out["E"], E, rtol=0, atol=1e-12)
    np.testing.assert_allclose(out["final"][tail], exp_tail, rtol=0, atol=1e-12)
    # the non-executable action (index >= S) is not corrected
    np.testing.assert_allclose(out["final"][5], x0[5] + b + w * float(c_tail), rtol=0, atol=1e-12)
    assert out["evals"] == ns
    assert list(out["release_step"]) == [K, K] + [ns] * (H - U)
    assert out["tail"] == tail


def _matrix_power_chunk(A, c, x0, n, steps=None):
    """Euler with v = A x + c and step 1/n for `steps` steps, as a closed form:
    x_s = B^s x0 + (sum_{j<s} B^j) c / n,  B = I + A/n."""
    steps = n if steps is None else steps
    B = np.eye(len(x0)) + A / n
    acc = sum(np.linalg.matrix_power(B, j) for j in range(steps))
    return np.linalg.matrix_power(B, steps) @ x0 + acc @ c / n


@pytest.mark.parametrize("ns,K", [(10, 4), (7, 1), (3, 2), (4, 3)])
def test_linear_field_closed_form(ns, K):
    """Per-token linear field v_i = A_i x_i + c_i (tokens decoupled)."""
    H, D, U = 4, 3, 2
    rng = np.random.default_rng(7)
    A = rng.normal(scale=0.7, size=(H, D, D))
    c = rng.normal(size=(H, D))
    x0 = rng.normal(size=(H, D))

    def vel(u, tau):
        return np.einsum("hij,hj->hi", A, u) + c

    budgets = [K] * U + [ns] * (H - U)
    out = denoise(vel, x0, budgets, tr=True, gac=True)
    for i in range(H):
        if i < U:
            a = _matrix_power_chunk(A[i], c[i], x0[i], K)
            np.testing.assert_allclose(out["released"][i], a, rtol=1e-12, atol=1e-12)
            # Eq. 5 gives sum_{k<=K} v_k = K (x_K - x_0), so Eq. 6 is the interpolation
            # x'_K = x_0 + (K/N*)(a - x_0); the ghost then runs N* - K steps of 1/N*.
            gK = x0[i] + K / ns * (a - x0[i])
            g = _matrix_power_chunk(A[i], c[i], gK, ns, ns - K)
            np.testing.assert_allclose(out["ghost"][i], g, rtol=1e-12, atol=1e-12)
        else:
            np.testing.assert_allclose(out["ghost"][i], _matrix_power_chunk(A[i], c[i], x0[i], ns),
                                       rtol=1e-12, atol=1e-12)


def test_coupled_linear_field_k1_recovers_vanilla():
    """Sec. 4.3 'Exact Recovery for K=1', with tokens coupled (like attention): the chunk
    evolves as X_N = (I + M/N)^N X_0 + ..., and UAD with K = 1 must give the same tail and
    ghost states."""
    H, D, ns, U = 5, 2, 6, 3
    rng = np.random.default_rng(3)
    M = rng.normal(scale=0.3, size=(H * D, H * D))
    c = rng.normal(size=H * D)
    x0 = rng.normal(size=(H, D))

    def vel(u, tau):
        return (M @ u.reshape(-1) + c).reshape(H, D)

    vanilla = _matrix_power_chunk(M, c, x0.reshape(-1), ns).reshape(H, D)
    uni = denoise(vel, x0, [ns] * H)
    np.testing.assert_allclose(uni["final"], vanilla, rtol=1e-12, atol=1e-12)
    out = denoise(vel, x0, [1] * U + [ns] * (H - U), gac=False)
    np.testing.assert_allclose(out["ghost"], vanilla, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(out["final"][U:], vanilla[U:], rtol=1e-12, atol=1e-12)
    # the released actions took one full Euler step from the shared noise
    np.testing.assert_allclose(out["released"][:U], x0[:U] + vel(x0, None)[:U], rtol=1e-12)


@pytest.mark.parametrize("n", [8, 16, 32, 64])
def test_vanilla_converges_to_ode_solution(n):
    """Eqs. 1-2 integrate dx/dt = A x + c on [0, 1]; Euler's global error is O(1/n)."""
    D = 3
    rng = np.random.default_rng(11)
    A = rng.normal(scale=0.5, size=(D, D))
    c = rng.normal(size=D)
    x0 = rng.normal(size=(1, D))
    out = denoise(lambda u, tau: u @ A.T + c, x0, [n])
    eA = scipy.linalg.expm(A)
    exact = eA @ x0[0] + np.linalg.solve(A, (eA - np.eye(D)) @ c)
    err = np.abs(out["final"][0] - exact).max()
    # first-order bound: |err| <= C / n with C from the n=8 case scaled (checked loosely)
    assert err < 2.0 / n
    assert err > 0.02 / n   # it really is a first-order method, not the exact solution


def test_gac_invariants_and_mask():
    rng = np.random.default_rng(5)
    H, D, S = 8, 4, 6
    x0 = rng.normal(size=(H, D))
    A = rng.normal(scale=0.2, size=(H * D, H * D))

    def vel(u, tau):
        return (A @ u.reshape(-1)).reshape(H, D) + np.asarray(tau)[:, None]

    budgets = [2, 2, 5, 5, 5, 5, 5, 5]
    mask = np.array([True, False, True, False])
    on = denoise(vel, x0, budgets, n_exec=S, gac=True, gac_mask=mask)
    off = denoise(vel, x0, budgets, n_exec=S, gac=False)
    tail = on["tail"]
    assert tail == [2, 3, 4, 5]
    E = (off["ghost"][:2] - off["released"][:2]).sum(axis=0)   # Eq. 8
    np.testing.assert_allclose(on["E"], E, atol=1e-13)
    delta = on["final"] - off["final"]
    # Eq. 9 preserves the total compensating displacement on additive dims...
    np.testing.assert_allclose(delta[tail].sum(axis=0)[mask], E[mask], atol=1e-13)
    # ...spread uniformly, leaves masked dims, released and non-executable actions alone
    np.testing.assert_allclose(delta[tail][:, mask], np.tile(E[mask] / 4, (4, 1)), atol=1e-13)
    assert np.all(delta[:, ~mask] == 0)
    assert np.all(delta[[0, 1, 6, 7]] == 0)
    # chunk-relative actions: GAC is skipped entirely (Sec. 4.4, App. C.4)
    rel = denoise(vel, x0, budgets, n_exec=S, gac=True, chunk_relative=True)
    assert np.array_equal(rel["final"], off["final"])


def test_released_actions_are_the_early_states():
    """UAER releases x_K (Sec. 4.2); later steps and GAC never modify them (Sec. 4.4)."""
    rng = np.random.default_rng(9)
    H, D = 5, 2
    x0 = rng.normal(size=(H, D))
    M = rng.normal(scale=0.4, size=(H * D, H * D))
    vel = lambda u, tau: (M @ u.reshape(-1)).reshape(H, D)
    budgets = [2, 3, 6, 6, 6]
    out = denoise(vel, x0, budgets, gac=True)
    # rerun truncated at the release step: the budget-2 action's state after step 2 is a^0
    snap = {}

    def spy(u, tau):
        v = vel(u, tau)
        snap.setdefault(len(snap) + 1, (u.copy(), v.copy()))
        return v

    denoise(spy, x0, budgets, gac=True)
    u1, v1 = snap[1]
    u2, v2 = snap[2]
    a0 = x0[0] + v1[0] / 2 + v2[0] / 2
    np.testing.assert_allclose(out["released"][0], a0, atol=1e-14)
    np.testing.assert_allclose(out["final"][0], a0, atol=0)
    np.testing.assert_allclose(out["final"][1], out["released"][1], atol=0)
    # evaluation count: N* = 6 evaluations, TR adds none (Sec. 4.3)
    assert out["evals"] == 6 and len(snap) == 6


def test_uniform_schedule_is_vanilla_bitwise():
    """With N_i = N* for all actions, nothing is early: no ghost, no GAC, and every state
    follows Eq. 2 (the same arithmetic as a K = N* 'urgent' group that is not early)."""
    rng = np.random.default_rng(1)
    H, D = 4, 3
    x0 = rng.normal(size=(H, D))
    M = rng.normal(scale=0.4, size=(H * D, H * D))
    vel = lambda u, tau: (M @ u.reshape(-1)).reshape(H, D) * (1 + np.asarray(tau))[:, None]
    out = denoise(vel, x0, [5] * H, gac=True)
    assert out["tail"] == [] and np.all(out["E"] == 0)
    assert np.array_equal(out["final"], out["ghost"])
    assert np.isnan(out["released"]).all()
    x = x0.copy()
    for k in range(1, 6):
        x = x + vel(x, np.full(H, (k - 1) / 5)) / 5
    assert np.array_equal(out["final"], x)


def test_tr_off_freezes_released_inputs():
    """UAER-only ablation: after release the action is fed back unchanged at tau = 1."""
    H, D = 3, 1
    seen = []

    def vel(u, tau):
        seen.append((u.copy(), np.asarray(tau).copy()))
        return np.ones((H, D))

    x0 = np.zeros((H, D))
    out = denoise(vel, x0, [1, 3, 3], tr=False, gac=False)
    assert [float(t[0]) for _, t in seen] == [0.0, 1.0, 1.0]
    assert [float(u[0, 0]) for u, _ in seen] == [0.0, 1.0, 1.0]
    assert out["released"][0, 0] == 1.0
    assert out["ghost"][0, 0] == 1.0          # no reconciled state: the frozen action
    with pytest.raises(ValueError):
        denoise(vel, x0, [1, 3, 3], tr=False, gac=True)


def test_plan_times_and_sets():
    b = [4] * 10 + [7] * 15 + [10] * 25
    assert P.n_star(b) == 10
    s5 = P.step_plan(b, 5)
    assert s5[0].ghost and s5[0].tau == Fraction(4, 10)
    assert s5[10].active and s5[10].tau == Fraction(4, 7)
    assert s5[30].tau == Fraction(4, 10)
    s4 = P.step_plan(b, 4)
    assert s4[0].release and not s4[10].release and not s4[30].release
    assert P.step_plan(b, 7)[12].release
    assert not any(t.release for t in P.step_plan(b, 10))
    assert P.executable_tail(b, 50) == list(range(25, 50))
    assert P.executable_tail(b, 30) == list(range(25, 30))
    assert P.early_tokens(b) == list(range(25))
    times = P.distinct_times(b)
    expect = sorted({Fraction(j, n) for n in (4, 7, 10) for j in range(n)})
    assert times == expect
    with pytest.raises(ValueError):
        P.step_plan([0, 3], 1)


def _random_schedules(rng, n):
    for _ in range(n):
        H = int(rng.integers(3, 13))
        groups = int(rng.integers(1, 4))
        levels = sorted(set(int(x) for x in rng.integers(1, 9, size=groups)))
        b = np.array(levels, dtype=int)[rng.integers(0, len(levels), size=H)]
        yield H, [int(x) for x in b]


@pytest.mark.parametrize("tr", [True, False])
def test_inputs_times_and_outputs_follow_eqs_5_to_9_on_random_schedules(tr):
    """Record every call of a coupled nonlinear field and rebuild, from the recorded velocities
    alone, what Eqs. 5-9 say the loop must have fed and returned: each action's flow time and
    input at every step (own step 1/N_i while active; after release the reconciled state
    x_0 + (1/N*) sum_j v_j with TR, the frozen released value at flow time 1 without), the
    released, ghost and tail states, and E with its uniform spread over the executable tail."""
    rng = np.random.default_rng(11 + tr)
    for H, budgets in _random_schedules(rng, 40):
        D = 3
        ns = max(budgets)
        S = int(rng.integers(1, H + 1))
        x0 = rng.normal(size=(H, D))
        A = rng.normal(scale=0.4, size=(H * D, H * D))
        c = rng.normal(size=D)
        tape = []

        def vel(u, tau):
            v = np.tanh((A @ u.reshape(-1)).reshape(H, D)) + np.asarray(tau)[:, None] * c
            tape.append((u.copy(), np.asarray(tau, float).copy(), v.copy()))
            return v

        out = denoise(vel, x0, budgets, n_exec=S, tr=tr, gac=tr)
        assert len(tape) == ns == out["evals"]
        V = np.stack([t[2] for t in tape])                        # [N*, H, D]
        for i, n_i in enumerate(budgets):
            own = x0[i] + np.cumsum(V[:n_i, i] / n_i, axis=0)      # x_k under Eq. 5, k = 1..N_i
            canon = x0[i] + np.cumsum(V[:, i] / ns, axis=0)       # Eqs. 6-7: step 1/N* from x_0
            for k in range(1, ns + 1):
                u, tau, _ = tape[k - 1]
                if k <= n_i:
                    want_u = x0[i] if k == 1 else own[k - 2]
                    assert tau[i] == float(Fraction(k - 1, n_i))
                elif tr:
                    want_u = canon[k - 2]
                    assert tau[i] == float(Fraction(k - 1, ns))
                else:
                    want_u = own[-1]
                    assert tau[i] == 1
                np.testing.assert_allclose(u[i], want_u, rtol=0, atol=1e-12)
            assert out["release_step"][i] == n_i
            if n_i < ns:
                np.testing.assert_allclose(out["released"][i], own[-1], rtol=0, atol=1e-12)
                np.testing.assert_array_equal(out["final"][i], out["released"][i])
                if tr:
                    np.testing.assert_allclose(out["ghost"][i], canon[-1], rtol=0, atol=1e-12)
                else:                                             # no reconciled state without TR
                    np.testing.assert_array_equal(out["ghost"][i], out["released"][i])
        early = [i for i, n in enumerate(budgets) if n < ns]
        tail = [i for i, n in enumerate(budgets) if n == ns and i < S]
        assert out["tail"] == (tail if tr and early else [])        # the actions GAC corrected
        x_end = {i: x0[i] + np.cumsum(V[:, i] / ns, axis=0)[-1] for i in range(H) if budgets[i] == ns}
        if tr and early and tail:
            E = sum(out["ghost"][i] - out["released"][i] for i in early)
            np.testing.assert_allclose(out["E"], E, rtol=0, atol=1e-12)
            for i in tail:
                np.testing.assert_allclose(out["final"][i], x_end[i] + E / len(tail), rtol=0, atol=1e-12)
        else:
            for i in tail:
                np.testing.assert_allclose(out["final"][i], x_end[i], rtol=0, atol=1e-12)
        for i, n in enumerate(budgets):
            if n == ns and i >= S:
                np.testing.assert_allclose(out["final"][i], x_end[i], rtol=0, atol=1e-12)
