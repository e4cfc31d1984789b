"""Action availability latency under the control clock -- oracle (test infrastructure).

Sec. 5.1 (Metrics) defines AAL as the wait from requesting an action until it is available,
averaged over executed actions; App. C.3 (Control-Time Alignment) gives every executed
action a fixed duration T_act, so the controller requests action i+1 one T_act after action
i started executing. App. B gives the closed forms this clock must reproduce under the
model's assumptions (Eqs. 11-12).
"""
from __future__ import annotations


def action_waits(ready, t_act):
    """ready[i] = time action i becomes available (request of action 0 at t = 0)."""
    waits, request = [], 0.0
    for i, r in enumerate(ready):
        if i > 0:
            request = start + t_act
        start = max(request, r)
        waits.append(max(0.0, r - request))
    return waits


def aal(ready, t_act, n_exec):
    w = action_waits(list(ready)[:n_exec], t_act)
    return sum(w) / n_exec


def latency_model_vanilla(t_vlm, t_d, n_star, n_exec):
    """App. B, Eq. 11."""
    return (t_vlm + n_star * t_d) / n_exec


def latency_model_uaer(t_vlm, t_d, n_star, k, u, t_act, n_exec):
    """App. B, Eq. 12."""
    return (t_vlm + k * t_d + max((n_star - k) * t_d - u * t_act, 0.0)) / n_exec
