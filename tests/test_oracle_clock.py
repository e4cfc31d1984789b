"""Pins of the control clock against the paper's latency model (App. B, Eqs. 11-12)."""
import pytest

from oracle.clock import aal, action_waits, latency_model_uaer, latency_model_vanilla


@pytest.mark.parametrize("t_vlm,t_d,ns,S", [(8.0, 17.0, 7, 10), (0.0, 0.1, 10, 50), (5, 2.5, 3, 10)])
def test_clock_reproduces_vanilla_model(t_vlm, t_d, ns, S):
    ready = [t_vlm + ns * t_d] * S            # all actions available together
    assert aal(ready, 12.5, S) == pytest.approx(latency_model_vanilla(t_vlm, t_d, ns, S))


@pytest.mark.parametrize("t_act", [1.0, 10.0, 50.0])
@pytest.mark.parametrize("K,U", [(1, 2), (1, 5), (2, 3), (4, 1)])
def test_clock_reproduces_uaer_model(K, U, t_act):
    t_vlm, t_d, ns, S = 6.0, 17.0, 7, 10
    ready = [t_vlm + K * t_d] * U + [t_vlm + ns * t_d] * (S - U)
    assert aal(ready, t_act, S) == pytest.approx(
        latency_model_uaer(t_vlm, t_d, ns, K, U, t_act, S))


def test_waits_chain():
    # action 1 arrives late: the controller idles, later requests shift accordingly
    w = action_waits([1.0, 30.0, 30.0, 45.0], 10.0)
    assert w == [1.0, 19.0, 0.0, 0.0]
