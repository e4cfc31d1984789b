"""The persistent evaluation kernel's bounded waits, made to run out without any GPU fault: the
first completion count of every evaluation is told to wait for one arrival more than the kernel
ever makes, with a 1 ms limit. Every wait gives up, records its code and lets the launch wind
down; uad_finish reports the error; the same context then runs a correct chunk."""
import numpy as np
import pytest

import paper_2609_37772_gb300 as uad
from oracle.model import build_model
from oracle.uad import denoise
from uad_inputs import ARCHS, group_budgets, make_noise, make_prefix_kv, make_weights

pytestmark = pytest.mark.gpu


def test_expired_wait_is_reported_and_the_context_recovers():
    a = ARCHS["pi0_small"]
    blob = make_weights(a, seed=21)
    kv = make_prefix_kv(a, seed=21)
    noise = make_noise(a, seed=21)
    bud = group_budgets(a.chunk_len, [(0, 9, 3), (10, a.chunk_len - 1, 6)])
    ex = uad.Expert(a, blob)
    try:
        ex.set_prefix(0, *kv)
        names = {r["name"] for r in ex.profile(noise, bud[None])}
        assert names == {"begin", "step_kernel"}, names   # the persistent kernel serves this chunk
        ex.set_wait_limit(wait_ns=1_000_000, unreachable=1)
        ex.denoise(noise, bud[None])
        r = ex.finish(timeout_us=60_000_000, check=False)
        assert r["rc"] == uad.UAD_ECUDA, r["rc"]
        # whichever bounded wait ran out first recorded its code (51: a completion count; the
        # issuer's operand wait, 42, can expire first with a 1 ms limit)
        msg = uad.uad_last_error(ex.h).decode()
        assert "timed out (code" in msg, msg
        # released actions were never flagged: nothing reached the controller
        rc, _, ready, _ = ex.poll(0, min_ready=1, timeout_us=0)
        assert rc in (uad.UAD_ETIMEDOUT, uad.UAD_ESTATE) or not ready.any()
        ex.set_wait_limit()   # back to the 2 s default, counts reachable again
        ex.denoise(noise, bud[None])
        ok = ex.finish(timeout_us=60_000_000)
        ref = denoise(build_model(a, blob, kv).velocity, noise[0], bud)
        err = np.abs(ok["final"][0] - ref["final"]).max() / np.abs(ref["final"]).max()
        print(f"after recovery: max rel err {err:.2e}")
        assert ok["rc"] == 0 and err <= 2e-2 and ok["evals"] == 6
    finally:
        ex.close()


def test_expired_wait_falls_back_to_per_operation_kernels():
    """After a wait of the persistent kernel ran out (as it would if its CTAs were not all
    resident), the context runs later chunks on the per-operation kernels, correctly, until the
    wait limit is set again."""
    a = ARCHS["pi0_small"]
    blob = make_weights(a, seed=22)
    kv = make_prefix_kv(a, seed=22)
    noise = make_noise(a, seed=22)
    bud = group_budgets(a.chunk_len, [(0, 9, 3), (10, a.chunk_len - 1, 6)])
    ex = uad.Expert(a, blob)
    try:
        ex.set_prefix(0, *kv)
        ex.set_wait_limit(wait_ns=1_000_000, unreachable=1)
        ex.denoise(noise, bud[None])
        r = ex.finish(timeout_us=60_000_000, check=False)
        assert r["rc"] == uad.UAD_ECUDA, r["rc"]
        msg = uad.uad_last_error(ex.h).decode()
        assert "per-operation kernels" in msg, msg
        names = {r["name"] for r in ex.profile(noise, bud[None])}
        assert "step_kernel" not in names and "qkv_proj" in names, names
        ex.denoise(noise, bud[None])
        ok = ex.finish(timeout_us=60_000_000)
        ref = denoise(build_model(a, blob, kv).velocity, noise[0], bud)
        err = np.abs(ok["final"][0] - ref["final"]).max() / np.abs(ref["final"]).max()
        print(f"per-operation fall-back: max rel err {err:.2e}")
        assert ok["rc"] == 0 and err <= 2e-2 and ok["evals"] == 6
        ex.set_wait_limit()
        names = {r["name"] for r in ex.profile(noise, bud[None])}
        assert names == {"begin", "step_kernel"}, names
    finally:
        ex.close()
