"""Pins of the oracle's synthetic action expert (the velocity network of Eq. 1).

The paper fixes no layer-level architecture, so the network's composition is this
project's stated design and parity for it is unpinned beyond what is checked here: each
building block against an independent library routine (torch fp64), and structural
invariants of the whole network (grouped-query heads equal expanded multi-head attention,
token-permutation equivariance without position information, RoPE scores depending only
on relative position, per-action time conditioning being per token).
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
