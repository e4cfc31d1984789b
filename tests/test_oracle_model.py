"""Pins of the oracle's synthetic action expert (the velocity network of Eq. 1).

The paper fixes no layer-level architecture, so the network's composition is this
project's stated design and parity for it is unpinned beyond what is checked here: each
building block against an independent library routine (torch fp64), and structural
invariants of the whole network (grouped-query heads equal expanded multi-head attention,
token-permutation equivariance without position information, RoPE scores depending only
on relative position, per-action time conditioning being per token), and special cases in
which a block collapses to a closed form (a zero gate makes a layer the identity; a scale of
-1 replaces the normalised stream by the shift), which pin the order of the modulation
vectors and of the weights in the blob.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as Fnn

from oracle import model as M
from oracle.model import Model
from uad_inputs import ARCHS, make_noise, make_prefix_kv, make_prefix_tokens, make_weights, split_blob, blob_from_weights

T = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))


def test_norms_and_activations_match_torch():
    rng = np.random.default_rng(0)
    h = rng.normal(size=(7, 96)) * 3 + 0.5
    np.testing.assert_allclose(M.rms_norm(h), Fnn.rms_norm(T(h), (96,), eps=M.EPS).numpy(), rtol=1e-13)
    np.testing.assert_allclose(M.layer_norm(h), Fnn.layer_norm(T(h), (96,), eps=M.EPS).numpy(),
                               rtol=1e-12, atol=1e-12)
    x = rng.normal(size=1000) * 4
    np.testing.assert_allclose(M.gelu_tanh(x), Fnn.gelu(T(x), approximate="tanh").numpy(), rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(M.silu(x), Fnn.silu(T(x)).numpy(), rtol=1e-13, atol=1e-15)


@pytest.mark.parametrize("hq,hkv", [(8, 1), (4, 4), (6, 2)])
def test_attention_matches_sdpa(hq, hkv):
    rng = np.random.default_rng(hq)
    q = rng.normal(size=(11, hq, 32))
    k = rng.normal(size=(37, hkv, 32))
    v = rng.normal(size=(37, hkv, 32))
    ours = M.attention(q, k, v)
    rep = hq // hkv
    ref = Fnn.scaled_dot_product_attention(
        T(q).transpose(0, 1), T(np.repeat(k, rep, axis=1)).transpose(0, 1),
        T(np.repeat(v, rep, axis=1)).transpose(0, 1)).transpose(0, 1).numpy()
    np.testing.assert_allclose(ours, ref, rtol=1e-12, atol=1e-13)


def test_rope_is_complex_rotation():
    rng = np.random.default_rng(2)
    x = rng.normal(size=(5, 3, 16))
    pos = np.array([0, 1, 7, 100, 865])
    got = M.rope(x, pos)
    z = x[..., :8] + 1j * x[..., 8:]
    inv = M.ROPE_THETA ** (-np.arange(8) * 2.0 / 16)
    z = z * np.exp(1j * pos[:, None, None] * inv[None, None, :])
    np.testing.assert_allclose(got, np.concatenate([z.real, z.imag], axis=-1), rtol=1e-12, atol=1e-12)


def test_rope_scores_depend_on_relative_position():
    rng = np.random.default_rng(4)
    q, k = rng.normal(size=(1, 1, 64)), rng.normal(size=(1, 1, 64))
    s1 = (M.rope(q, [50]) * M.rope(k, [20])).sum()
    s2 = (M.rope(q, [850]) * M.rope(k, [820])).sum()
    s3 = (M.rope(q, [851]) * M.rope(k, [820])).sum()
    assert s1 == pytest.approx(s2, rel=1e-10)
    assert abs(s1 - s3) > 1e-6


def test_sinusoid_values():
    e = M.sinusoid([0.0, np.pi / 2000.0], 8, M.TIME_SCALE)
    np.testing.assert_allclose(e[0], [0, 0, 0, 0, 1, 1, 1, 1], atol=0)
    assert e[1, 0] == pytest.approx(1.0, abs=1e-15)          # f_0 = 1: sin(pi/2)
    assert e[1, 4] == pytest.approx(0.0, abs=1e-15)
    np.testing.assert_allclose(e[:, :4] ** 2 + e[:, 4:] ** 2, 1.0, rtol=1e-14)
    # f_j = 1e4^(-j/half): j = 2 of half = 4 -> 1e-2
    e2 = M.sinusoid([1.0], 8, 1.0)
    assert e2[0, 2] == pytest.approx(np.sin(1e-2), rel=1e-14)


def _tiny(**kw):
    return ARCHS["tiny"].replace(n_layers=1, width=64, n_heads=4, n_kv_heads=1, head_dim=16,
                                 mlp_dim=96, action_dim=3, chunk_len=6, prefix_len=9, **kw)


def test_gqa_equals_expanded_mha():
    """Hkv = 1 with 4 query heads equals Hkv = 4 with the K/V projections and the prefix
    replicated per head: catches a wrong query-head -> KV-head mapping."""
    a1 = _tiny(rope=True)
    a4 = a1.replace(n_kv_heads=4)
    w1 = split_blob(a1, make_weights(a1, seed=3))
    w4 = dict(w1)
    for p in ("l0.wk", "l0.wv"):
        w4[p] = np.tile(w1[p], (1, 4))
    k, v = make_prefix_kv(a1, seed=3)
    m1 = Model(a1, blob_from_weights(a1, w1)); m1.set_prefix_kv(k, v)
    m4 = Model(a4, blob_from_weights(a4, w4)); m4.set_prefix_kv(np.repeat(k, 4, 2), np.repeat(v, 4, 2))
    u = make_noise(a1, seed=3)[0]
    tau = np.linspace(0, 0.9, 6)
    np.testing.assert_allclose(m1.velocity(u, tau), m4.velocity(u, tau), rtol=1e-12, atol=1e-12)


def test_permutation_equivariance_without_rope():
    """No position information in the attention-prefix arch without RoPE: permuting the
    chunk's tokens (state and flow time together) permutes the velocities -- catches a
    stray mask or a token-index mix-up."""
    a = _tiny(rope=False)
    m = Model(a, make_weights(a, seed=5)); m.set_prefix_kv(*make_prefix_kv(a, seed=5))
    u = make_noise(a, seed=5)[0]
    tau = np.array([0.0, 0.1, 0.5, 0.25, 0.9, 0.7])
    perm = np.array([3, 0, 5, 1, 4, 2])
    np.testing.assert_allclose(m.velocity(u, tau)[perm], m.velocity(u[perm], tau[perm]), rtol=1e-11, atol=1e-12)


def test_per_token_time_conditioning_is_local():
    """Changing one token's flow time changes its conditioning only (App. C.1): with the
    modulation weights zeroed except the final norm's, v_j depends on tau_j alone."""
    a = _tiny(rope=False)
    w = split_blob(a, make_weights(a, seed=6))
    for n in ("l0.mod1_w", "l0.mod1_b", "l0.mod2_w", "l0.mod2_b"):
        w[n] = np.zeros_like(w[n])
    w["l0.mod1_b"] = np.concatenate([np.zeros(128), np.ones(64)])   # gate = 1, scale = shift = 0
    w["l0.mod2_b"] = w["l0.mod1_b"].copy()
    m = Model(a, blob_from_weights(a, w)); m.set_prefix_kv(*make_prefix_kv(a, seed=6))
    u = make_noise(a, seed=6)[0]
    t1 = np.array([0.0, 0.1, 0.2, 0.3, 0.4, 0.5])
    t2 = t1.copy(); t2[2] = 0.95
    v1, v2 = m.velocity(u, t1), m.velocity(u, t2)
    assert np.abs(v1[2] - v2[2]).max() > 1e-4
    np.testing.assert_array_equal(np.delete(v1, 2, 0), np.delete(v2, 2, 0))


def test_dit_prefix_projection_and_cross_attention():
    """DiT arch: cross-attention K/V are the prefix tokens times Wkc/Wvc (projected once)."""
    a = ARCHS["dit_small"].replace(n_layers=1)
    blob = make_weights(a, seed=8)
    w = split_blob(a, blob)
    toks = make_prefix_tokens(a, seed=8)
    m = Model(a, blob); m.set_prefix_tokens(toks)
    np.testing.assert_allclose(m.kpre[0].reshape(a.prefix_len, -1), toks.astype(np.float64) @ w["l0.wkc"], rtol=1e-12)
    v = m.velocity(make_noise(a, seed=8)[0], np.zeros(a.chunk_len))
    assert v.shape == (a.chunk_len, a.action_dim) and np.isfinite(v).all()


def test_k1_exact_recovery_with_the_network():
    """Sec. 4.3: with K = 1 the first evaluation equals vanilla's and TR re-integrates it with
    1/N*, so tail and ghost actions equal vanilla inference exactly -- here bit for bit."""
    from oracle.uad import denoise
    a = ARCHS["tiny"]
    m = Model(a, make_weights(a)); m.set_prefix_kv(*make_prefix_kv(a))
    x0 = make_noise(a)[0]
    ns = 10
    van = denoise(m.velocity, x0, [ns] * a.chunk_len)
    uad = denoise(m.velocity, x0, [1] * 4 + [ns] * (a.chunk_len - 4), gac=False)
    assert np.array_equal(uad["ghost"], van["final"])
    assert np.array_equal(uad["final"][4:], van["final"][4:])
    assert not np.array_equal(uad["final"][:4], van["final"][:4])
    assert uad["evals"] == van["evals"] == ns


# ---- SmolVLA-style time conditioning: the time embedding joins the action MLP (App. C.1) --------
def _concat0():
    return ARCHS["tiny_concat"].replace(n_layers=0, chunk_len=5)


def test_concat_input_mlp_closed_form():
    """Zero layers, identity MLP weights and a constant action embedding: v = RMSNorm(SiLU(a0 +
    e(tau))) Wout + bout with e(tau)_j = sin(1000 tau 10^(-4 j / (W/2))) for j < W/2 and the
    matching cos above; e is written out here from its definition."""
    a = _concat0()
    W, D = a.width, a.action_dim
    rng = np.random.default_rng(11)
    a0 = rng.normal(size=W)
    w = {"in_w": np.zeros((D, W)), "in_b": a0, "ti_wa": np.eye(W), "ti_wt": np.eye(W), "ti_b": np.zeros(W),
         "to_w": np.eye(W), "to_b": np.zeros(W), "out_w": rng.normal(size=(W, D)) * 0.1, "out_b": rng.normal(size=D)}
    m = Model(a, blob_from_weights(a, w))
    tau = np.array([0.0, 0.1, 0.25, 0.5, 0.9])
    v = m.velocity(rng.normal(size=(a.chunk_len, D)), tau)
    half = W // 2
    for i, t in enumerate(tau):
        e = np.array([np.sin(1000.0 * t * 10000.0 ** (-j / half)) for j in range(half)] +
                     [np.cos(1000.0 * t * 10000.0 ** (-j / half)) for j in range(half)])
        x = a0.astype(np.float32).astype(np.float64) + e
        g = x / (1.0 + np.exp(-x))
        y = g / np.sqrt(np.mean(g * g) + 1e-6)
        ref = y @ w["out_w"].astype(np.float32).astype(np.float64) + w["out_b"].astype(np.float32)
        np.testing.assert_allclose(v[i], ref, rtol=1e-6, atol=1e-7)


def test_concat_time_conditioning_is_per_token():
    """Without layers a token's velocity depends on its own state and flow time only."""
    a = _concat0()
    m = Model(a, make_weights(a, seed=12))
    u = make_noise(a, seed=12)[0]
    t1 = np.array([0.0, 0.2, 0.4, 0.6, 0.8])
    t2 = t1.copy(); t2[2] = 0.95
    v1, v2 = m.velocity(u, t1), m.velocity(u, t2)
    assert np.abs(v1[2] - v2[2]).max() > 1e-4
    np.testing.assert_array_equal(np.delete(v1, 2, 0), np.delete(v2, 2, 0))


def test_concat_layer_is_the_adarms_layer_without_modulation():
    """A "concat" layer equals an "adarms" layer whose modulation is scale = shift = 0 and
    gate = 1 for every token (plain RMSNorm, ungated residuals)."""
    ac = ARCHS["tiny_concat"].replace(n_layers=1, rope=True, n_kv_heads=2)
    aa = ARCHS["tiny"].replace(n_layers=1, rope=True, n_kv_heads=2)
    wc = split_blob(ac, make_weights(ac, seed=13))
    wa = split_blob(aa, make_weights(aa, seed=13))
    W = aa.width
    for n in ("wq", "wk", "wv", "wo", "wg", "wu", "wd"):
        wa["l0." + n] = wc["l0." + n]
    for n in ("l0.mod1", "l0.mod2"):
        wa[n + "_w"] = np.zeros_like(wa[n + "_w"])
        wa[n + "_b"] = np.concatenate([np.zeros(2 * W), np.ones(W)])
    kv = make_prefix_kv(ac, seed=13)
    mc = Model(ac, blob_from_weights(ac, wc)); mc.set_prefix_kv(*kv)
    ma = Model(aa, blob_from_weights(aa, wa)); ma.set_prefix_kv(*kv)
    h = np.random.default_rng(13).normal(size=(ac.chunk_len, W))
    tau = np.linspace(0.0, 0.9, ac.chunk_len)
    np.testing.assert_allclose(mc._layer(0, h, mc.time_cond(tau)), ma._layer(0, h, ma.time_cond(tau)),
                               rtol=1e-12, atol=1e-12)


def test_k1_exact_recovery_with_the_concat_network():
    """Sec. 4.3 with the SmolVLA-style expert: K = 1 tail and ghosts equal vanilla bit for bit."""
    from oracle.uad import denoise
    a = ARCHS["tiny_concat"]
    m = Model(a, make_weights(a)); m.set_prefix_kv(*make_prefix_kv(a))
    x0 = make_noise(a)[0]
    van = denoise(m.velocity, x0, [10] * a.chunk_len)
    uad = denoise(m.velocity, x0, [1] * 4 + [10] * (a.chunk_len - 4), gac=False)
    assert np.array_equal(uad["ghost"], van["final"]) and np.array_equal(uad["final"][4:], van["final"][4:])


def _with_prefix(a, blob, seed):
    m = Model(a, blob)
    if a.n_layers:
        if a.kind == "dit":
            m.set_prefix_tokens(make_prefix_tokens(a, seed=seed))
        else:
            m.set_prefix_kv(*make_prefix_kv(a, seed=seed))
    return m


def _gates_zeroed(a, w):
    """Copy of the weights with every gate of every layer zero: for adaRMS the third W-slice of
    both modulations (scale, shift, gate); for DiT gate1 and gate2 of (shift1, scale1, gate1,
    shift2, scale2, gate2), and the ungated cross-attention's output projection."""
    W = a.width
    w = {k: v.copy() for k, v in w.items()}
    for l in range(a.n_layers):
        p = f"l{l}."
        if a.kind == "adarms":
            for mod in ("mod1", "mod2"):
                w[p + mod + "_w"][:, 2 * W:] = 0
                w[p + mod + "_b"][2 * W:] = 0
        else:
            for g in (2, 5):
                w[p + "mod_w"][:, g * W:(g + 1) * W] = 0
                w[p + "mod_b"][g * W:(g + 1) * W] = 0
            w[p + "woc"][:] = 0
    return w


@pytest.mark.parametrize("name", ["tiny", "dit_small"])
def test_layers_with_zero_gates_are_the_identity(name):
    """Every residual branch is scaled by its gate (DiT's cross-attention, ungated, by its output
    projection), so with those zero the network equals the same network without layers: pins
    where the gates sit in the modulation vectors."""
    from uad_inputs import weight_specs
    a = ARCHS[name]
    w = _gates_zeroed(a, split_blob(a, make_weights(a, seed=30)))
    m = _with_prefix(a, blob_from_weights(a, w), 30)
    a0 = a.replace(n_layers=0)
    m0 = Model(a0, blob_from_weights(a0, {n: w[n] for n, _ in weight_specs(a0)}))
    u = make_noise(a, seed=30)[0]
    tau = np.linspace(0.0, 0.9, a.chunk_len)
    np.testing.assert_allclose(m.velocity(u, tau), m0.velocity(u, tau), rtol=1e-12, atol=1e-12)
    full = _with_prefix(a, make_weights(a, seed=30), 30)
    assert not np.allclose(full.velocity(u, tau), m0.velocity(u, tau))


@pytest.mark.parametrize("name", ["tiny", "dit_small"])
def test_final_modulation_order(name):
    """The final norm's modulation is (scale, shift) for adaRMS and (shift, scale) for DiT: with
    scale = -1 the normalised stream drops out and v = shift W_out + b_out for every token."""
    a = ARCHS[name]
    W = a.width
    w = {k: v.copy() for k, v in split_blob(a, make_weights(a, seed=31)).items()}
    s = np.random.default_rng(31).normal(size=W).astype(np.float32)
    minus = -np.ones(W, np.float32)
    w["modf_w"][:] = 0
    w["modf_b"][:] = np.concatenate([minus, s] if a.kind == "adarms" else [s, minus])
    m = _with_prefix(a, blob_from_weights(a, w), 31)
    v = m.velocity(make_noise(a, seed=31)[0], np.linspace(0.0, 0.9, a.chunk_len))
    want = s.astype(np.float64) @ w["out_w"].astype(np.float64) + w["out_b"]
    np.testing.assert_allclose(v, np.tile(want, (a.chunk_len, 1)), rtol=1e-12, atol=1e-12)


def test_dit_tokens_are_told_apart_by_position():
    """The DiT head adds a sinusoidal code of the token index to its input (its attention has no
    other position information): tokens with equal states and flow times get different
    velocities, where the attention-prefix expert without RoPE gives them equal ones."""
    a = ARCHS["dit_small"]
    m = _with_prefix(a, make_weights(a, seed=32), 32)
    u = np.tile(make_noise(a, seed=32)[0][:1], (a.chunk_len, 1))
    tau = np.full(a.chunk_len, 0.3)
    v = m.velocity(u, tau)
    d = np.abs(v[:, None, :] - v[None, :, :]).max(axis=-1) + np.eye(a.chunk_len)
    assert d.min() > 1e-4
    b = _tiny(rope=False)
    mb = _with_prefix(b, make_weights(b, seed=32), 32)
    ub = np.tile(make_noise(b, seed=32)[0][:1], (b.chunk_len, 1))
    vb = mb.velocity(ub, np.full(b.chunk_len, 0.3))
    np.testing.assert_allclose(vb, np.tile(vb[:1], (b.chunk_len, 1)), rtol=1e-12, atol=1e-12)


def test_dit_cross_attention_reads_the_stream_through_its_norm():
    """The DiT cross-attention's queries come from the unmodulated LayerNorm of the stream, so with
    the gated branches off a layer's update is unchanged when every row of the stream is scaled
    and shifted (up to the norm's epsilon)."""
    a = ARCHS["dit_small"].replace(n_layers=1)
    W = a.width
    w = {k: v.copy() for k, v in split_blob(a, make_weights(a, seed=33)).items()}
    for g in (2, 5):
        w["l0.mod_w"][:, g * W:(g + 1) * W] = 0
        w["l0.mod_b"][g * W:(g + 1) * W] = 0
    m = _with_prefix(a, blob_from_weights(a, w), 33)
    c = m.time_cond(np.linspace(0.0, 0.9, a.chunk_len))
    h = np.random.default_rng(33).normal(size=(a.chunk_len, W))
    h2 = 3.0 * h + 0.5
    d1 = m._layer(0, h, c) - h
    d2 = m._layer(0, h2, c) - h2
    assert np.abs(d1).max() > 1e-3
    np.testing.assert_allclose(d2, d1, rtol=0, atol=1e-5 * np.abs(d1).max())


def _dit_layer_with_constant_modulation(seed, mod_b, woc_zero=True):
    a = ARCHS["dit_small"].replace(n_layers=1)
    w = {k: v.copy() for k, v in split_blob(a, make_weights(a, seed=seed)).items()}
    w["l0.mod_w"][:] = 0
    w["l0.mod_b"][:] = np.concatenate(mod_b).astype(np.float32)
    if woc_zero:
        w["l0.woc"][:] = 0
    m = _with_prefix(a, blob_from_weights(a, w), seed)
    h = np.random.default_rng(seed).normal(size=(a.chunk_len, a.width)) * 2 + 0.3
    c = m.time_cond(np.linspace(0.0, 0.9, a.chunk_len))
    return a, {k: v.astype(np.float64) for k, v in w.items()}, m._layer(0, h, c) - h


def test_dit_self_attention_modulation_order():
    """DiT layer modulation (shift1, scale1, gate1, ...): with scale1 = -1 every token enters the
    self-attention as shift1, whose uniform attention returns its own value row, so the update is
    gate1 * (shift1 Wv Wo) whatever the stream (MLP gate and cross-attention output off)."""
    W = ARCHS["dit_small"].width
    rng = np.random.default_rng(34)
    sh1, g1, sh2, sc2 = (rng.normal(size=W) for _ in range(4))
    a, w, d = _dit_layer_with_constant_modulation(34, [sh1, -np.ones(W), g1, sh2, sc2, np.zeros(W)])
    sh1, g1 = (x.astype(np.float32).astype(np.float64) for x in (sh1, g1))
    want = g1 * ((sh1 @ w["l0.wv"]) @ w["l0.wo"])
    np.testing.assert_allclose(d, np.tile(want, (a.chunk_len, 1)), rtol=1e-11, atol=1e-12)


def test_dit_mlp_modulation_order():
    """With scale2 = -1 the MLP sees shift2 on every token: the update is
    gate2 * (gelu_tanh(shift2 W1 + b1) W2 + b2) (self-attention gate and cross-attention output
    off); the activation here is torch's."""
    W = ARCHS["dit_small"].width
    rng = np.random.default_rng(35)
    sh1, sc1, sh2, g2 = (rng.normal(size=W) for _ in range(4))
    a, w, d = _dit_layer_with_constant_modulation(35, [sh1, sc1, np.zeros(W), sh2, -np.ones(W), g2])
    sh2, g2 = (x.astype(np.float32).astype(np.float64) for x in (sh2, g2))
    act = Fnn.gelu(T(sh2 @ w["l0.w1"] + w["l0.b1"]), approximate="tanh").numpy()
    want = g2 * (act @ w["l0.w2"] + w["l0.b2"])
    np.testing.assert_allclose(d, np.tile(want, (a.chunk_len, 1)), rtol=1e-11, atol=1e-12)


def test_time_mlp_has_two_silus():
    """c = SiLU(SiLU(e W1 + b1) W2 + b2): with W2 = 0, c = SiLU(b2) for every flow time; with
    W1 = 0, c = SiLU(SiLU(b1) W2 + b2) (torch's SiLU)."""
    a = _tiny(rope=False)
    m = Model(a, make_weights(a, seed=36))
    tau = np.array([0.0, 0.25, 0.5, 0.9])
    w2 = m.w["t_w2"].copy()
    m.w["t_w2"][:] = 0
    np.testing.assert_allclose(m.time_cond(tau), np.tile(Fnn.silu(T(m.w["t_b2"])).numpy(), (4, 1)), rtol=1e-13)
    m.w["t_w2"][:] = w2
    m.w["t_w1"][:] = 0
    inner = Fnn.silu(T(m.w["t_b1"])).numpy()
    want = Fnn.silu(T(inner @ w2 + m.w["t_b2"])).numpy()
    np.testing.assert_allclose(m.time_cond(tau), np.tile(want, (4, 1)), rtol=1e-12, atol=1e-14)


def test_concat_input_mlp_weights_read_what_they_are_named_for():
    """SmolVLA-style input MLP: ti_wa multiplies the action embedding and ti_wt the time
    embedding. With ti_wt = 0 the network no longer sees the flow time (its layers are
    unmodulated); with ti_wa = 0 it no longer sees the action state."""
    a = ARCHS["tiny_concat"]
    u1, u2 = make_noise(a, seed=37)[0], make_noise(a, seed=38)[0]
    t1, t2 = np.linspace(0.0, 0.9, a.chunk_len), np.linspace(0.9, 0.0, a.chunk_len)
    m = _with_prefix(a, make_weights(a, seed=37), 37)
    assert not np.allclose(m.velocity(u1, t1), m.velocity(u1, t2))
    assert not np.allclose(m.velocity(u1, t1), m.velocity(u2, t1))
    wt = m.w["ti_wt"].copy()
    m.w["ti_wt"][:] = 0
    np.testing.assert_allclose(m.velocity(u1, t1), m.velocity(u1, t2), rtol=1e-12, atol=1e-13)
    m.w["ti_wt"][:] = wt
    m.w["ti_wa"][:] = 0
    np.testing.assert_allclose(m.velocity(u1, t1), m.velocity(u2, t1), rtol=1e-12, atol=1e-13)
