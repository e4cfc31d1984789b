"""Synthetic action expert F_theta(x, tau, prefix) in fp64 -- oracle (test infrastructure).

The paper evaluates a velocity network v_k = F_theta(x_{k-1}, o, L) (Sec. 3, Eq. 1) whose
action tokens attend to each other and to the vision-language context through shared
attention (Sec. 4.3: tokens are coupled by attention), and extends it with one flow time per
action token, which for pi0.5 conditions the adaptive normalisation layers of the action
expert (App. C.1, "Per-Action Time Conditioning"). The paper gives no layer-level
definition, so the composition below is this project's stated architecture:

  time conditioning (per token):  e = [sin(1000 tau f_j), cos(1000 tau f_j)],
        f_j = 10000^(-j/(W/2)),  c = SiLU(SiLU(e W1 + b1) W2 + b2)
  "adarms" layer (pi0-like / tiny):
        (scale, shift, gate) = c Wm + bm
        y  = RMSNorm(h) * (1 + scale) + shift           (RMSNorm: h / sqrt(mean h^2 + 1e-6))
        q, k, v = y Wq, y Wk, y Wv ; RoPE(theta=1e4, rotate-half) at positions P + i if enabled
        o  = softmax(q [Kpre; k]^T / sqrt(dh)) [Vpre; v]   (GQA, bidirectional, no mask)
        h += gate * (o Wo)
        (scale2, shift2, gate2) = c Wm2 + bm2 ; y = RMSNorm(h)(1+scale2)+shift2
        h += gate2 * ((gelu_tanh(y Wg) * (y Wu)) Wd)
  "dit" layer (adaLN-zero style):
        (shift1, scale1, gate1, shift2, scale2, gate2) = c Wm + bm
        y = LN(h)(1+scale1)+shift1 ; h += gate1 * SelfAttn(y over the H chunk tokens) Wo
        h += CrossAttn(LN(h) Wqc ; prefix Wkc, prefix Wvc) Woc
        y = LN(h)(1+scale2)+shift2 ; h += gate2 * (gelu_tanh(y W1 + b1) W2 + b2)
        (LN: no affine, eps 1e-6; the DiT input adds a sinusoidal position code of index i)
  input / output: h = x Win + bin ; v = Norm_final(h)(1+scale_f)+shift_f) Wout + bout
  "concat" (SmolVLA-style: the token's time embedding is given to it before the action MLP,
  App. C.1): e = sinusoid(tau) as above (no time MLP), a = x Win + bin,
        h = SiLU(a Wia + e Wit + bi) Wo_in + bo_in  (the MLP over [a ; e]),
        layers as "adarms" with RMSNorm unmodulated and ungated residuals,
        v = RMSNorm(h) Wout + bout

Everything here is fp64 on the (bf16-exact, for bf16 archs) weights. Library primitives
used as steps: numpy matmul, exp, sin, cos, tanh.
"""
from __future__ import annotations

import numpy as np

from uad_inputs import Arch, split_blob

EPS = 1e-6
TIME_SCALE = 1000.0
MAX_PERIOD = 10000.0
ROPE_THETA = 10000.0


def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x):
    return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))


def sinusoid(values, width, scale):
    """[n] -> [n, width]: first half sin(scale*v*f_j), second half cos, f_j = 1e4^(-j/half)."""
    half = width // 2
    f = np.exp(-np.log(MAX_PERIOD) * np.arange(half, dtype=np.float64) / half)
    arg = scale * np.asarray(values, dtype=np.float64)[:, None] * f[None, :]
    return np.concatenate([np.sin(arg), np.cos(arg)], axis=1)


def rms_norm(h):
    return h / np.sqrt(np.mean(h * h, axis=-1, keepdims=True) + EPS)


def layer_norm(h):
    mu = np.mean(h, axis=-1, keepdims=True)
    var = np.mean((h - mu) ** 2, axis=-1, keepdims=True)
    return (h - mu) / np.sqrt(var + EPS)


def rope(x, positions):
    """Rotate-half RoPE. x [n, heads, dh], positions [n]."""
    dh = x.shape[-1]
    half = dh // 2
    inv = ROPE_THETA ** (-np.arange(half, dtype=np.float64) * 2.0 / dh)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv[None, :]
    cos, sin = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def attention(q, k, v):
    """softmax(q k^T / sqrt(dh)) v with grouped heads.

    q [n, Hq, dh], k/v [m, Hkv, dh]; query head j reads key/value head j // (Hq / Hkv).
    """
    n, hq, dh = q.shape
    hkv = k.shape[1]
    group = hq // hkv
    out = np.empty_like(q)
    for j in range(hq):
        g = j // group
        s = q[:, j, :] @ k[:, g, :].T / np.sqrt(dh)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[:, j, :] = p @ v[:, g, :]
    return out


class Model:
    """fp64 F_theta for one robot's prefix. ``velocity(u, tau)`` is Eq. 1 with per-token tau."""

    def __init__(self, arch: Arch, blob: np.ndarray):
        self.a = arch
        self.w = {k: np.asarray(v, dtype=np.float64) for k, v in split_blob(arch, blob).items()}
        self.kpre = self.vpre = None
        self.evals = 0

    # -- observation context ---------------------------------------------------------------
    def set_prefix_kv(self, k, v):
        """Attention-prefix archs: per-layer prefix keys/values [L, P, Hkv, dh]."""
        self.kpre = np.asarray(k, dtype=np.float64)
        self.vpre = np.asarray(v, dtype=np.float64)

    def set_prefix_tokens(self, tokens):
        """DiT arch: cross-attention keys/values are projected once per observation."""
        a, w = self.a, self.w
        t = np.asarray(tokens, dtype=np.float64)
        shp = (t.shape[0], a.n_heads, a.head_dim)
        self.kpre = np.stack([(t @ w[f"l{l}.wkc"]).reshape(shp) for l in range(a.n_layers)])
        self.vpre = np.stack([(t @ w[f"l{l}.wvc"]).reshape(shp) for l in range(a.n_layers)])

    # -- per-action time conditioning (App. C.1) ---------------------------------------------
    def time_cond(self, tau):
        w = self.w
        e = sinusoid(tau, self.a.width, TIME_SCALE)
        if self.a.kind == "concat":
            return e
        return silu(silu(e @ w["t_w1"] + w["t_b1"]) @ w["t_w2"] + w["t_b2"])

    # -- the velocity field --------------------------------------------------------------------
    def velocity(self, u, tau):
        """u [H, D] model-input states, tau [H] per-token flow times -> v [H, D]."""
        a, w = self.a, self.w
        self.evals += 1
        u = np.asarray(u, dtype=np.float64)
        H, W = u.shape[0], a.width
        c = self.time_cond(tau)
        h = u @ w["in_w"] + w["in_b"]
        if a.kind == "concat":
            # the action MLP over the token's action embedding and its own time embedding
            h = silu(h @ w["ti_wa"] + c @ w["ti_wt"] + w["ti_b"]) @ w["to_w"] + w["to_b"]
            for l in range(a.n_layers):
                h = self._layer(l, h, c)
            return rms_norm(h) @ w["out_w"] + w["out_b"]
        if a.kind == "dit":
            h = h + sinusoid(np.arange(H), W, 1.0)
        for l in range(a.n_layers):
            h = self._layer(l, h, c)
        mf = c @ w["modf_w"] + w["modf_b"]
        if a.kind == "adarms":
            scale, shift = mf[:, :W], mf[:, W:]
            y = rms_norm(h) * (1.0 + scale) + shift
        else:
            shift, scale = mf[:, :W], mf[:, W:]
            y = layer_norm(h) * (1.0 + scale) + shift
        return y @ w["out_w"] + w["out_b"]

    def _layer(self, l, h, c):
        a, w, p = self.a, self.w, f"l{l}."
        H, W, hq, hkv, dh = h.shape[0], a.width, a.n_heads, a.n_kv_heads, a.head_dim
        if a.kind == "concat":
            y = rms_norm(h)
            q = (y @ w[p + "wq"]).reshape(H, hq, dh)
            k = (y @ w[p + "wk"]).reshape(H, hkv, dh)
            v = (y @ w[p + "wv"]).reshape(H, hkv, dh)
            if a.rope:
                pos = a.prefix_len + np.arange(H)
                q, k = rope(q, pos), rope(k, pos)
            o = attention(q, np.concatenate([self.kpre[l], k]), np.concatenate([self.vpre[l], v]))
            h = h + o.reshape(H, hq * dh) @ w[p + "wo"]
            y = rms_norm(h)
            return h + (gelu_tanh(y @ w[p + "wg"]) * (y @ w[p + "wu"])) @ w[p + "wd"]
        if a.kind == "adarms":
            m = c @ w[p + "mod1_w"] + w[p + "mod1_b"]
            scale, shift, gate = m[:, :W], m[:, W:2 * W], m[:, 2 * W:]
            y = rms_norm(h) * (1.0 + scale) + shift
            q = (y @ w[p + "wq"]).reshape(H, hq, dh)
            k = (y @ w[p + "wk"]).reshape(H, hkv, dh)
            v = (y @ w[p + "wv"]).reshape(H, hkv, dh)
            if a.rope:
                pos = a.prefix_len + np.arange(H)
                q, k = rope(q, pos), rope(k, pos)
            o = attention(q, np.concatenate([self.kpre[l], k]), np.concatenate([self.vpre[l], v]))
            h = h + gate * (o.reshape(H, hq * dh) @ w[p + "wo"])
            m = c @ w[p + "mod2_w"] + w[p + "mod2_b"]
            scale, shift, gate = m[:, :W], m[:, W:2 * W], m[:, 2 * W:]
            y = rms_norm(h) * (1.0 + scale) + shift
            act = gelu_tanh(y @ w[p + "wg"]) * (y @ w[p + "wu"])
            return h + gate * (act @ w[p + "wd"])
        # dit
        m = c @ w[p + "mod_w"] + w[p + "mod_b"]
        sh1, sc1, g1, sh2, sc2, g2 = (m[:, i * W:(i + 1) * W] for i in range(6))
        y = layer_norm(h) * (1.0 + sc1) + sh1
        q = (y @ w[p + "wq"]).reshape(H, hq, dh)
        k = (y @ w[p + "wk"]).reshape(H, hq, dh)
        v = (y @ w[p + "wv"]).reshape(H, hq, dh)
        h = h + g1 * (attention(q, k, v).reshape(H, hq * dh) @ w[p + "wo"])
        qc = (layer_norm(h) @ w[p + "wqc"]).reshape(H, hq, dh)
        h = h + attention(qc, self.kpre[l], self.vpre[l]).reshape(H, hq * dh) @ w[p + "woc"]
        y = layer_norm(h) * (1.0 + sc2) + sh2
        return h + g2 * (gelu_tanh(y @ w[p + "w1"] + w[p + "b1"]) @ w[p + "w2"] + w[p + "b2"])


def build_model(arch: Arch, blob, robot_prefix):
    """Convenience: a Model bound to one robot's prefix (K/V pair or DiT tokens)."""
    m = Model(arch, blob)
    if arch.kind == "dit":
        m.set_prefix_tokens(robot_prefix)
    else:
        m.set_prefix_kv(*robot_prefix)
    return m
