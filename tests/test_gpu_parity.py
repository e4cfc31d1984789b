"""GPU parity: the CUDA path through the C ABI against the fp64 oracle on the same seeded
inputs. Tolerance (stated in the spec of the path): max |a_gpu - a_oracle| / max |a_oracle|
over each output set <= 1e-4 in fp32 mode and <= 2e-2 in bf16 mode; release steps and the
evaluation count are compared exactly."""
import itertools

import numpy as np
import pytest
import torch

import paper_2609_37772_gb300 as uad
from oracle.model import build_model
from oracle.uad import denoise
from uad_inputs import (ARCHS, draw_sweep_schedules, group_budgets, make_noise, make_prefix_kv,
                        make_prefix_tokens, make_weights, round_to_bf16)

pytestmark = pytest.mark.gpu
TOL = {"f32": 1e-4, "bf16": 2e-2}
TIMEOUT = 120_000_000


def rel_err(got, ref):
    return float(np.abs(np.asarray(got, np.float64) - ref).max() / max(1e-6, np.abs(ref).max()))


def prefixes(a, B, seed=0):
    if a.kind == "dit":
        return [make_prefix_tokens(a, robot=b, seed=seed) for b in range(B)]
    return [make_prefix_kv(a, robot=b, seed=seed) for b in range(B)]


class Case:
    def __init__(self, arch, B=1, seed=0, blob=None):
        self.a, self.B = arch, B
        self.blob = make_weights(arch, seed=seed) if blob is None else blob
        self.pre = prefixes(arch, B, seed)
        self.ex = uad.Expert(arch, self.blob, max_batch=B)
        for b, p in enumerate(self.pre):
            if arch.kind == "dit":
                self.ex.set_prefix(b, p)
            else:
                self.ex.set_prefix(b, *p)
        self._models = None

    def models(self):
        if self._models is None:
            self._models = [build_model(self.a, self.blob, p) for p in self.pre]
        return self._models

    def gpu(self, noise, budgets, poll=True, **kw):
        budgets = np.asarray(budgets, np.int32).reshape(self.B, -1)
        self.ex.denoise(noise, budgets, **kw)
        polled = []
        if poll:
            for b in range(self.B):
                rc, out, ready, step = self.ex.poll(b, min_ready=self.a.chunk_len, timeout_us=TIMEOUT)
                assert rc == self.a.chunk_len, rc
                polled.append((out.copy(), step.copy()))
        res = self.ex.finish(timeout_us=TIMEOUT)
        res["polled"] = polled
        return res

    def oracle(self, noise, budgets, **kw):
        budgets = np.asarray(budgets, np.int32).reshape(self.B, -1)
        kw = {("n_exec" if k == "n_exec" else k): v for k, v in kw.items()}
        if kw.get("n_exec", 0) == 0:
            kw.pop("n_exec", None)
        return [denoise(m.velocity, noise[b], budgets[b], **kw) for b, m in enumerate(self.models())]

    def close(self):
        self.ex.close()


def check(case, res, refs, budgets, tol):
    """Final and ghost actions within `tol` of the action scale (reading C13). E of Eq. 8 sums
    (ghost - released) over the U early actions, so its error is bounded by the sum of those
    actions' errors: |dE| <= U * tol * (max|ghost| + max|final|) of the oracle. Prints the errors
    reached (shown with pytest -s)."""
    budgets = np.asarray(budgets).reshape(case.B, -1)
    worst = {"final": 0.0, "ghost": 0.0, "E/bound": 0.0}
    for b, ref in enumerate(refs):
        ef, eg = rel_err(res["final"][b], ref["final"]), rel_err(res["ghost"][b], ref["ghost"])
        worst["final"], worst["ghost"] = max(worst["final"], ef), max(worst["ghost"], eg)
        assert ef <= tol, ("final", b, ef)
        assert eg <= tol, ("ghost", b, eg)
        if np.abs(ref["E"]).max() > 0:
            U = int((budgets[b] < budgets[b].max()).sum())
            bound = U * tol * (np.abs(ref["ghost"]).max() + np.abs(ref["final"]).max())
            dE = float(np.abs(res["E"][b] - ref["E"]).max())
            worst["E/bound"] = max(worst["E/bound"], dE / bound)
            assert dE <= bound, ("E", b, dE, bound)
        else:
            assert np.all(res["E"][b] == 0)
        if res["polled"]:
            out, step = res["polled"][b]
            assert np.array_equal(step, ref["release_step"].astype(np.int32))
            # what the controller received is exactly what finish reports
            assert np.array_equal(out, res["final"][b])
    assert res["evals"] == max(r["evals"] for r in refs) and res["tr_extra_evals"] == 0
    print(f"[{case.a.name} B={case.B}] max rel err final {worst['final']:.2e} ghost {worst['ghost']:.2e} "
          f"(tolerance {tol:g}); E error / bound {worst['E/bound']:.2e}")


# ---------------------------------------------------------------------------------------------
@pytest.fixture(scope="module")
def tiny():
    c = Case(ARCHS["tiny"])
    yield c
    c.close()


def test_tiny_fp32_urgent4_at5(tiny):
    a = tiny.a
    noise = make_noise(a)
    bud = group_budgets(a.chunk_len, [(0, 3, 5), (4, a.chunk_len - 1, 10)])
    res = tiny.gpu(noise, bud)
    check(tiny, res, tiny.oracle(noise, bud), bud, TOL["f32"])


@pytest.mark.parametrize("kw", [dict(tr=False, gac=False), dict(gac=False), dict(chunk_relative=True),
                                dict(n_exec=10), dict(gac_mask=[1, 1, 1, 0, 0, 0, 0])])
def test_tiny_variants(tiny, kw):
    a = tiny.a
    noise = make_noise(a, seed=3)
    bud = group_budgets(a.chunk_len, [(0, 1, 2), (2, 5, 6), (6, a.chunk_len - 1, 8)])
    res = tiny.gpu(noise, bud, **kw)
    check(tiny, res, tiny.oracle(noise, bud, **kw), bud, TOL["f32"])


def test_k1_exact_recovery_bitwise(tiny):
    """Sec. 4.3: with K = 1, tail and ghost actions equal vanilla inference exactly."""
    a = tiny.a
    noise = make_noise(a, seed=5)
    van = tiny.gpu(noise, np.full(a.chunk_len, 10), poll=False)
    uadr = tiny.gpu(noise, group_budgets(a.chunk_len, [(0, 4, 1), (5, a.chunk_len - 1, 10)]), gac=False, poll=False)
    assert np.array_equal(uadr["ghost"], van["final"])
    assert np.array_equal(uadr["final"][:, 5:], van["final"][:, 5:])


def test_uniform_schedule_is_vanilla(tiny):
    a = tiny.a
    noise = make_noise(a, seed=6)
    bud = np.full(a.chunk_len, 7)
    res = tiny.gpu(noise, bud)
    assert np.array_equal(res["final"], res["ghost"]) and np.all(res["E"] == 0)
    check(tiny, res, tiny.oracle(noise, bud), bud, TOL["f32"])


def test_deterministic(tiny):
    a = tiny.a
    noise = make_noise(a, seed=8)
    bud = group_budgets(a.chunk_len, [(0, 3, 3), (4, a.chunk_len - 1, 9)])
    r1 = tiny.gpu(noise, bud, poll=False)
    r2 = tiny.gpu(noise, bud, poll=False)
    for k in ("final", "ghost", "E"):
        assert np.array_equal(r1[k], r2[k])


def test_released_actions_never_change(tiny):
    """Poll the urgent group as soon as it is released, then compare with finish."""
    a = tiny.a
    noise = make_noise(a, seed=9)
    bud = group_budgets(a.chunk_len, [(0, 3, 2), (4, a.chunk_len - 1, 10)])
    tiny.ex.denoise(noise, bud[None])
    rc, out, ready, step = tiny.ex.poll(0, min_ready=4, timeout_us=TIMEOUT)
    assert rc >= 4 and ready[:4].all() and (step[:4] == 2).all()
    snap = out[:4].copy()
    res = tiny.ex.finish(timeout_us=TIMEOUT)
    assert np.array_equal(res["final"][0, :4], snap)
    rc2, out2, ready2, _ = tiny.ex.poll(0, min_ready=a.chunk_len, timeout_us=TIMEOUT)
    assert rc2 == a.chunk_len and np.array_equal(out2[:4], snap)


def test_device_buffers(tiny):
    a = tiny.a
    noise = make_noise(a, seed=10)
    bud = group_budgets(a.chunk_len, [(0, 3, 5), (4, a.chunk_len - 1, 10)])
    host = tiny.gpu(noise, bud, poll=False)
    dn = torch.from_numpy(noise).cuda()
    tiny.ex.denoise(dn, bud[None], stream=torch.cuda.current_stream())
    f = torch.zeros_like(dn)
    g = torch.zeros_like(dn)
    e = torch.zeros(1, a.action_dim, device="cuda")
    tiny.ex.finish(timeout_us=TIMEOUT, final=f, ghost=g, gac_error=e)
    assert np.array_equal(f.cpu().numpy(), host["final"]) and np.array_equal(g.cpu().numpy(), host["ghost"])


def test_errors_are_reported(tiny):
    a = tiny.a
    noise = make_noise(a)
    with pytest.raises(uad.UADError) as ei:
        tiny.ex.finish()
    assert ei.value.code == uad.UAD_ESTATE
    with pytest.raises(uad.UADError) as ei:
        tiny.ex.denoise(noise, np.zeros(a.chunk_len))
    assert ei.value.code == uad.UAD_EINVAL
    with pytest.raises(uad.UADError) as ei:
        tiny.ex.denoise(noise, np.full(a.chunk_len, 3), tr=False, gac=True)
    assert ei.value.code == uad.UAD_EINVAL
    with pytest.raises(uad.UADError):
        tiny.ex.denoise(noise, np.full(a.chunk_len, 3), n_star=4)
    tiny.ex.denoise(noise, np.full(a.chunk_len, 3)[None])
    with pytest.raises(uad.UADError) as ei:
        tiny.ex.denoise(noise, np.full(a.chunk_len, 3)[None])
    assert ei.value.code == uad.UAD_ESTATE
    tiny.ex.finish(timeout_us=TIMEOUT)


def test_timeouts_leave_the_chunk_in_flight(tiny):
    """A delayed chunk (the caller's stream is held by a bounded sleep kernel before the library's
    work may start): poll and finish with short deadlines return UAD_ETIMEDOUT without waiting and
    leave the chunk in flight, a new observation is refused while it is in flight, and a later
    finish returns the complete chunk."""
    a = tiny.a
    noise = make_noise(a)
    bud = group_budgets(a.chunk_len, [(0, 3, 5), (4, a.chunk_len - 1, 10)])
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        torch.cuda._sleep(400_000_000)        # ~0.2 s of GPU time on the caller's stream
    tiny.ex.denoise(noise, bud[None], stream=stream)
    rc, _, ready, _ = tiny.ex.poll(0, min_ready=1, timeout_us=1000)
    assert rc == uad.UAD_ETIMEDOUT and not ready.any()
    res = tiny.ex.finish(timeout_us=1000, check=False)
    assert res["rc"] == uad.UAD_ETIMEDOUT
    with pytest.raises(uad.UADError) as ei:
        tiny.ex.set_prefix(0, *make_prefix_kv(a))
    assert ei.value.code == uad.UAD_ESTATE
    res = tiny.ex.finish(timeout_us=TIMEOUT)
    assert res["rc"] == uad.UAD_OK and res["evals"] == 10
    torch.cuda.synchronize()


def test_nonfinite_is_reported(tiny):
    a = tiny.a
    noise = make_noise(a)
    noise[0, 2, 1] = np.nan
    tiny.ex.denoise(noise, np.full(a.chunk_len, 2)[None])
    res = tiny.ex.finish(timeout_us=TIMEOUT, check=False)
    assert res["rc"] == uad.UAD_ENONFINITE and res["nonfinite"] > 0


def test_brute_force_small_chunks():
    """All 4^3 budget assignments on a 3-action chunk with 2-dim actions (fp32)."""
    a = ARCHS["tiny"].replace(chunk_len=3, action_dim=2, n_layers=1)
    c = Case(a, seed=4)
    noise = make_noise(a, seed=4)
    try:
        for bud in itertools.product(range(1, 5), repeat=3):
            res = c.gpu(noise, bud)
            check(c, res, c.oracle(noise, bud), bud, TOL["f32"])
    finally:
        c.close()


def test_fp32_rope_gqa_arch():
    a = ARCHS["tiny_f32_rope"]
    c = Case(a, seed=2)
    try:
        noise = make_noise(a, seed=2)
        bud = group_budgets(a.chunk_len, [(0, 3, 4), (4, 9, 7), (10, a.chunk_len - 1, 10)])
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["f32"])
    finally:
        c.close()


@pytest.mark.parametrize("name", ["pi0_small", "dit_small"])
def test_bf16_small_archs(name):
    a = ARCHS[name]
    c = Case(a, seed=1)
    try:
        noise = make_noise(a, seed=1)
        H = a.chunk_len
        bud = group_budgets(H, [(0, 3, 4), (4, H // 2, 7), (H // 2 + 1, H - 1, 10)])
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["bf16"])
    finally:
        c.close()


@pytest.mark.parametrize("B", [1, 4])
def test_bf16_expert_without_rope(B):
    """A bf16 joint-attention expert without rotary embedding: q and k leave the QKV projection's
    epilogue as computed. B = 1 runs the persistent kernel, B = 4 the per-operation tensor-core
    projection and attention."""
    a = ARCHS["pi0_small"].replace(name="pi0_small_norope", rope=False)
    c = Case(a, B=B, seed=21)
    try:
        noise = make_noise(a, batch=B, seed=21)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=21)
        names = kernel_names(c, noise, bud)
        assert ("step_kernel" in names) == (B == 1) and (B == 1 or "qkv_proj" in names), names
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["bf16"])
    finally:
        c.close()


def test_batched_robots_own_schedules():
    a = ARCHS["pi0_small"]
    B = 4
    c = Case(a, B=B, seed=7)
    try:
        noise = make_noise(a, batch=B, seed=7)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=7)
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["bf16"])
    finally:
        c.close()


@pytest.mark.parametrize("name", ["tiny_concat", "concat_small"])
def test_time_concatenating_expert(name):
    """SmolVLA-style per-action time conditioning (App. C.1: each token's time embedding joins its
    action embedding before the action MLP), fp32 on CUDA cores and bf16 on the tensor cores."""
    a = ARCHS[name]
    c = Case(a, seed=16)
    try:
        noise = make_noise(a, seed=16)
        H = a.chunk_len
        bud = group_budgets(H, [(0, 3, 4), (4, H // 2, 7), (H // 2 + 1, H - 1, 10)])
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL[a.dtype])
    finally:
        c.close()


# ---- full-size workloads -----------------------------------------------------------------------
def test_pi0_full_three_groups():
    """pi0-like bf16 expert, B = 1, groups 0-9 @ 4, 10-24 @ 7, 25-49 @ 10 (all outputs)."""
    a = ARCHS["pi0"]
    c = Case(a)
    try:
        noise = make_noise(a)
        bud = group_budgets(50, [(0, 9, 4), (10, 24, 7), (25, 49, 10)])
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["bf16"])
    finally:
        c.close()


@pytest.mark.parametrize("ns", [4, 16])
def test_dit_full(ns):
    a = ARCHS["dit"]
    c = Case(a)
    try:
        noise = make_noise(a)
        bud = group_budgets(16, [(0, 3, ns // 2), (4, 15, ns)])
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["bf16"])
    finally:
        c.close()


@pytest.mark.parametrize("name,B", [("dit", 4), ("dit_small", 6)])
def test_dit_batched(name, B):
    """The DiT head for several robots, each with its own prefix tokens and schedule: at 4 robots
    (64 tokens, one token tile: every projection takes the extra K splits) and at 6 (96 tokens,
    two token tiles); every robot vs the oracle."""
    a = ARCHS[name]
    c = Case(a, B=B, seed=4)
    try:
        noise = make_noise(a, batch=B, seed=4)
        if name == "dit":   # N* = 4 keeps the fp64 oracle of the full head short
            bud = np.stack([group_budgets(a.chunk_len, [(0, 1 + b, 2), (2 + b, a.chunk_len - 1, 4)]) for b in range(B)])
        else:
            bud = draw_sweep_schedules(a.chunk_len, B, seed=4)
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["bf16"])
    finally:
        c.close()


def test_tensor_core_gemm_matches_cuda_core_gemm(monkeypatch):
    """The tcgen05 projection path against the CUDA-core GEMM on the same bf16 operands."""
    a = ARCHS["pi0_small"]
    blob = make_weights(a, seed=11)
    noise = make_noise(a, seed=11)
    bud = group_budgets(a.chunk_len, [(0, 9, 3), (10, a.chunk_len - 1, 6)])
    outs = []
    for mode in ("simt", "tc"):
        monkeypatch.setenv("UAD_GEMM", mode)
        c = Case(a, seed=11, blob=blob)
        try:
            outs.append(c.gpu(noise, bud, poll=False))
        finally:
            c.close()
    for k in ("final", "ghost"):
        assert rel_err(outs[1][k], outs[0][k].astype(np.float64)) <= 5e-3, k


def test_step_kernel_matches_per_operation_kernels(monkeypatch):
    """The persistent evaluation kernel (one launch per step, few tokens) against
    the per-operation kernels on the same bf16 operands, and both against the oracle."""
    a = ARCHS["pi0_small"]
    blob = make_weights(a, seed=12)
    noise = make_noise(a, seed=12)
    bud = group_budgets(a.chunk_len, [(0, 9, 3), (10, 29, 5), (30, a.chunk_len - 1, 8)])
    outs, launches = [], []
    for mode in ("0", "1"):
        monkeypatch.setenv("UAD_STEP", mode)
        c = Case(a, seed=12, blob=blob)
        try:
            launches.append(c.ex.launches_per_chunk(1, 8))
            outs.append(c.gpu(noise, bud))
            if mode == "1":
                check(c, outs[-1], c.oracle(noise, bud), bud, TOL["bf16"])
        finally:
            c.close()
    assert launches[1] == 1 + 8 < launches[0]   # one launch per step: evaluation + step epilogue
    for k in ("final", "ghost"):
        assert rel_err(outs[1][k], outs[0][k].astype(np.float64)) <= 5e-3, k
    assert np.array_equal(outs[1]["polled"][0][1], outs[0]["polled"][0][1])


def kernel_names(c, noise, bud):
    return {r["name"] for r in c.ex.profile(noise, bud)}


def test_step_kernel_batched_robots():
    """Three robots of 16 tokens, each with its own prefix and schedule, on the persistent kernel
    (48 token rows plus one projection row per distinct flow time of a step)."""
    a = ARCHS["pi0_small"].replace(name="pi0_small_h16", chunk_len=16)
    B = 3
    c = Case(a, B=B, seed=13)
    try:
        assert c.ex.launches_per_chunk(B, 10) == 1 + 10
        noise = make_noise(a, batch=B, seed=13)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=13)
        assert "step_kernel" in kernel_names(c, noise, bud)
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["bf16"])
    finally:
        c.close()


def test_step_kernel_many_attention_items():
    """Eight KV heads over a 1900-token prefix: 240 attention items leave too few idle CTAs to merge
    the key chunks inside the attention step, so the persistent kernel merges them in a step of its
    own and separates every phase by a grid barrier."""
    a = ARCHS["pi0_small"].replace(name="mha_long_prefix", width=512, n_heads=8, n_kv_heads=8, head_dim=64,
                                   mlp_dim=1024, chunk_len=16, prefix_len=1900)
    c = Case(a, seed=15)
    try:
        noise = make_noise(a, seed=15)
        bud = group_budgets(a.chunk_len, [(0, 3, 3), (4, 9, 5), (10, 15, 8)])
        assert "step_kernel" in kernel_names(c, noise, bud[None])
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["bf16"])
    finally:
        c.close()


def test_full_rows_fall_back_to_per_operation_kernels():
    """Four robots of 16 tokens fill all 64 rows of the persistent kernel, leaving no room for
    the per-flow-time rows: the chunk runs on the per-operation kernels, with the same results."""
    a = ARCHS["pi0_small"].replace(name="pi0_small_h16", chunk_len=16)
    B = 4
    c = Case(a, B=B, seed=14)
    try:
        noise = make_noise(a, batch=B, seed=14)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=14)
        names = kernel_names(c, noise, bud)
        assert "step_kernel" not in names and "qkv_proj" in names
        check(c, c.gpu(noise, bud), c.oracle(noise, bud), bud, TOL["bf16"])
    finally:
        c.close()


def test_pi0_full_batched_16_robots_sampled():
    """16 robots (M = 800 tokens: wide 128 x 256 projection tiles), each with its own prefix and
    a schedule from the sweep grid; robots 0, 7 and 15 are checked against the oracle."""
    a = ARCHS["pi0"]
    B = 16
    blob = make_weights(a, seed=3)
    ex = uad.Expert(a, blob, max_batch=B)
    try:
        pre = [make_prefix_kv(a, robot=b, seed=3) for b in range(B)]
        for b in range(B):
            ex.set_prefix(b, *pre[b])
        noise = make_noise(a, batch=B, seed=3)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=3)
        ex.denoise(noise, bud)
        res = ex.finish(timeout_us=TIMEOUT)
        worst = 0.0
        for b in (0, 7, 15):
            ref = denoise(build_model(a, blob, pre[b]).velocity, noise[b], bud[b])
            ef, eg = rel_err(res["final"][b], ref["final"]), rel_err(res["ghost"][b], ref["ghost"])
            worst = max(worst, ef, eg)
            assert ef <= TOL["bf16"] and eg <= TOL["bf16"], (b, ef, eg)
        assert res["evals"] == 10
        print(f"[pi0 B={B}, robots (0, 7, 15)] max rel err {worst:.2e} (tolerance {TOL['bf16']:g})")
    finally:
        ex.close()


@pytest.mark.parametrize("B", [8, 24])
def test_pi0_full_batched_between_sampled(B):
    """Batch sizes between the serving configurations: 8 robots (400 tokens: the qkv and gate/up
    projections on the persistent wide form, o and down on narrow split-K tiles with partial
    planes, the split-KV attention) and 24 (1200 tokens: every projection wide, the many-tile
    attention on 96 query tiles without the head-dim split); first, middle and last robot vs the
    oracle."""
    a = ARCHS["pi0"]
    blob = make_weights(a, seed=9)
    ex = uad.Expert(a, blob, max_batch=B)
    try:
        pre = [make_prefix_kv(a, robot=b, seed=9) for b in range(B)]
        for b in range(B):
            ex.set_prefix(b, *pre[b])
        noise = make_noise(a, batch=B, seed=9)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=9)
        ex.denoise(noise, bud)
        res = ex.finish(timeout_us=TIMEOUT)
        worst = 0.0
        for b in (0, B // 2, B - 1):
            ref = denoise(build_model(a, blob, pre[b]).velocity, noise[b], bud[b])
            ef, eg = rel_err(res["final"][b], ref["final"]), rel_err(res["ghost"][b], ref["ghost"])
            worst = max(worst, ef, eg)
            assert ef <= TOL["bf16"] and eg <= TOL["bf16"], (b, ef, eg)
        assert res["evals"] == 10
        print(f"[pi0 B={B}, robots (0, {B // 2}, {B - 1})] max rel err {worst:.2e} (tolerance {TOL['bf16']:g})")
    finally:
        ex.close()


def test_pi0_full_batched_64_robots_sampled():
    """64 robots (M = 3200 tokens), the batched serving configuration: every projection on wide
    tensor-core tiles (the o and down projections with the partial-plane epilogue), attention on
    the many-tile path, the residual norm one warp per row; robots 0, 31 and 63 vs the oracle."""
    a = ARCHS["pi0"]
    B = 64
    blob = make_weights(a, seed=5)
    ex = uad.Expert(a, blob, max_batch=B)
    try:
        pre = [make_prefix_kv(a, robot=b, seed=5) for b in range(B)]
        for b in range(B):
            ex.set_prefix(b, *pre[b])
        noise = make_noise(a, batch=B, seed=5)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=5)
        ex.denoise(noise, bud)
        res = ex.finish(timeout_us=TIMEOUT)
        worst = 0.0
        for b in (0, 31, 63):
            ref = denoise(build_model(a, blob, pre[b]).velocity, noise[b], bud[b])
            ef, eg = rel_err(res["final"][b], ref["final"]), rel_err(res["ghost"][b], ref["ghost"])
            worst = max(worst, ef, eg)
            assert ef <= TOL["bf16"] and eg <= TOL["bf16"], (b, ef, eg)
        assert res["evals"] == 10
        print(f"[pi0 B={B}, robots (0, 31, 63)] max rel err {worst:.2e} (tolerance {TOL['bf16']:g})")
    finally:
        ex.close()


@pytest.mark.parametrize("B", [32, 40])
def test_one_pass_attention_many_tiles(B):
    """32 or 40 robots x 2 query tiles on the small bf16 expert: the attention takes its path for
    many query tiles (one pass over 128-key chunks, O in tensor memory rescaled only when a row
    maximum grows past 2^8); with 64 tiles (at most half as many as the SMs) each tile runs on two
    CTAs, one per half of the head dims, with 80 on one; sampled robots vs the oracle."""
    a = ARCHS["pi0_small"]
    blob = make_weights(a, seed=12)
    ex = uad.Expert(a, blob, max_batch=B)
    try:
        pre = [make_prefix_kv(a, robot=b, seed=12) for b in range(B)]
        for b in range(B):
            ex.set_prefix(b, *pre[b])
        noise = make_noise(a, batch=B, seed=12)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=12)
        ex.denoise(noise, bud)
        res = ex.finish(timeout_us=TIMEOUT)
        for b in (0, 13, B - 1):
            ref = denoise(build_model(a, blob, pre[b]).velocity, noise[b], bud[b])
            assert rel_err(res["final"][b], ref["final"]) <= TOL["bf16"]
            assert rel_err(res["ghost"][b], ref["ghost"]) <= TOL["bf16"]
    finally:
        ex.close()


@pytest.mark.parametrize("prefix,B", [(78, 32), (206, 32), (206, 40)])
def test_one_pass_attention_key_counts(prefix, B):
    """The many-tile attention at the key-count edges: 128 keys (one chunk, no later chunk to load
    ahead) and 256 keys (two full chunks, no masked keys), split over head-dim halves (64 tiles)
    and not (80 tiles); sampled robots vs the oracle."""
    a = ARCHS["pi0_small"].replace(name=f"pi0_small_p{prefix}", prefix_len=prefix)
    blob = make_weights(a, seed=15)
    ex = uad.Expert(a, blob, max_batch=B)
    try:
        pre = [make_prefix_kv(a, robot=b, seed=15) for b in range(B)]
        for b in range(B):
            ex.set_prefix(b, *pre[b])
        noise = make_noise(a, batch=B, seed=15)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=15)
        ex.denoise(noise, bud)
        res = ex.finish(timeout_us=TIMEOUT)
        for b in (0, B // 2, B - 1):
            ref = denoise(build_model(a, blob, pre[b]).velocity, noise[b], bud[b])
            assert rel_err(res["final"][b], ref["final"]) <= TOL["bf16"]
            assert rel_err(res["ghost"][b], ref["ghost"]) <= TOL["bf16"]
    finally:
        ex.close()


def test_one_pass_attention_rescales_when_the_maximum_grows():
    """The many-tile attention path with prefix keys past the first 128-key chunk scaled by 16
    (a power of two: still exact in bf16), so that every query row's maximum score jumps far
    past 2^8 in the exponent at the second chunk and the running O rows and sums are rescaled in
    tensor memory; sampled robots vs the oracle on the same keys."""
    a = ARCHS["pi0_small"]
    B = 32
    blob = make_weights(a, seed=14)
    ex = uad.Expert(a, blob, max_batch=B)
    try:
        pre = []
        for b in range(B):
            k, v = make_prefix_kv(a, robot=b, seed=14)
            k = k.copy()
            k[:, 128:] *= 16.0
            pre.append((k, v))
            ex.set_prefix(b, k, v)
        noise = make_noise(a, batch=B, seed=14)
        bud = draw_sweep_schedules(a.chunk_len, B, seed=14)
        ex.denoise(noise, bud)
        res = ex.finish(timeout_us=TIMEOUT)
        for b in (0, 17, 31):
            ref = denoise(build_model(a, blob, pre[b]).velocity, noise[b], bud[b])
            assert rel_err(res["final"][b], ref["final"]) <= TOL["bf16"]
            assert rel_err(res["ghost"][b], ref["ghost"]) <= TOL["bf16"]
    finally:
        ex.close()


def test_relative_l2_diagnostic_matches_oracle(tiny):
    """The Fig. 3 diagnostic (relative L2 error to vanilla inference of released, ghost and tail
    actions, per variant) computed from the CUDA path equals the oracle's; with K = 1 and TR the
    tail and ghost errors vanish on both (exact recovery)."""
    import bench
    a = tiny.a
    noise = make_noise(a, seed=31)
    van_g = tiny.gpu(noise, np.full(a.chunk_len, 3), poll=False)["final"][0]
    van_o = tiny.oracle(noise, np.full(a.chunk_len, 3), gac=False)[0]["final"]
    for k, u in ((1, 4), (2, 6)):
        bud = group_budgets(a.chunk_len, [(0, u - 1, k), (u, a.chunk_len - 1, 3)])
        for name, kw in bench.DIAG_VARIANTS.items():
            rg = tiny.gpu(noise, bud, poll=False, **kw)
            ro = tiny.oracle(noise, bud, **kw)[0]
            eg = bench.diagnostic_errors(rg["final"][0], rg["ghost"][0], van_g, bud, kw["tr"])
            eo = bench.diagnostic_errors(ro["final"], ro["ghost"], van_o, bud, kw["tr"])
            assert eg.keys() == eo.keys()
            for key in eg:
                assert abs(eg[key] - eo[key]) <= 1e-4 * max(1.0, eo[key]), (k, u, name, key, eg[key], eo[key])
            if k == 1 and name == "uaer+tr":
                assert eg["tail"] == 0.0 and eg["ghost"] == 0.0


@pytest.mark.parametrize("bud_groups", [[(0, 3, 2), (4, 15, 6)], [(0, 0, 1), (1, 5, 3), (6, 15, 7)]])
def test_gac_on_so3_matches_oracle(tiny, bud_groups):
    """D = 7 actions: dimensions 0-2 additive, 3-5 a rotation vector corrected by composition
    on SO(3) (App. C.1), 6 (gripper) masked; fp32 against the fp64 oracle."""
    a = tiny.a
    noise = make_noise(a, seed=41)
    bud = group_budgets(a.chunk_len, bud_groups)
    mask = np.array([1, 1, 1, 0, 0, 0, 0], np.uint8)
    res = tiny.gpu(noise, bud, gac_mask=mask, rot_dim=3)
    ref = tiny.oracle(noise, bud, gac_mask=mask.astype(bool), rot_dim=3)
    check(tiny, res, ref, bud, TOL["f32"])
    assert np.abs(res["E"][0] - ref[0]["E"]).max() <= 1e-4 * max(1.0, np.abs(ref[0]["E"]).max())
    # the rotation dimensions moved, the gripper did not
    plain = tiny.oracle(noise, bud, gac_mask=mask.astype(bool))[0]
    tail = ref[0]["tail"]
    assert np.abs(ref[0]["final"][tail][:, 3:6] - plain["final"][tail][:, 3:6]).max() > 1e-4
    assert np.array_equal(res["final"][0][:, 6], tiny.gpu(noise, bud, gac_mask=mask, poll=False)["final"][0][:, 6])


def test_rot_dim_is_validated(tiny):
    a = tiny.a
    bud = group_budgets(a.chunk_len, [(0, 3, 2), (4, a.chunk_len - 1, 4)])
    with pytest.raises(uad.UADError):
        tiny.ex.denoise(make_noise(a, seed=1), bud[None], rot_dim=a.action_dim - 2)


@pytest.mark.parametrize("name", ["tiny", "pi0_small", "dit_small"])
def test_prefix_given_in_bf16(name):
    """uad_set_prefix_kv takes the prefix in fp32 or bf16, from host or device memory: the same
    bf16-exact prefix given as fp32, as bf16 bit patterns on the host and as a bf16 device tensor
    gives a chunk within tolerance of the oracle every time."""
    a = ARCHS[name]
    blob = make_weights(a, seed=21)
    pre = prefixes(a, 1, seed=21)[0]
    exact = [round_to_bf16(p) for p in ((pre,) if a.kind == "dit" else pre)]
    model = build_model(a, blob, exact[0] if a.kind == "dit" else tuple(exact))
    noise = make_noise(a, seed=21)
    bud = group_budgets(a.chunk_len, [(0, 3, 2), (4, a.chunk_len - 1, 5)])
    ref = denoise(model.velocity, noise[0], bud)
    tol = TOL[a.dtype]
    forms = [(exact, "f32"),
             ([(e.view(np.uint32) >> 16).astype(np.uint16) for e in exact], "bf16"),
             ([torch.from_numpy(e).to(torch.bfloat16).cuda() for e in exact], "bf16")]
    ex = uad.Expert(a, blob)
    try:
        for p, dt in forms:
            ex.set_prefix(0, *p, dtype=dt)
            ex.denoise(noise, bud[None])
            res = ex.finish(timeout_us=TIMEOUT)
            assert rel_err(res["final"][0], ref["final"]) <= tol, (dt, rel_err(res["final"][0], ref["final"]))
            assert rel_err(res["ghost"][0], ref["ghost"]) <= tol
            assert res["evals"] == ref["evals"]
    finally:
        ex.close()
