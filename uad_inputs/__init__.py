"""Seeded synthetic inputs shared by the CUDA path's tests/benchmarks and the CPU oracle.

This module holds *no arithmetic of the method*: it only knows the shapes of the synthetic
action experts, the order of tensors in the flat weight blob (the checkpoint format that
``uad_init`` consumes), and how to draw seeded random numbers for weights, prefix KV,
prefix tokens, initial noise and urgency schedules.

Recipe (stands in for the paper's pretrained SmolVLA / pi0.5 checkpoints and the
LIBERO / Meta-World observations, which are not available):

* weights and biases ~ N(0, 0.02), drawn in blob order in blocks of 4 Mi values, each
  block from its own numpy PCG64 stream keyed (seed, 1, block);
  for bf16 architectures every value is rounded to the nearest bf16 (ties to even), so
  the fp32 blob holds exactly representable bf16 values;
* prefix K/V (attention-prefix architectures) ~ N(0, 1) per layer, [L, P, Hkv, dh],
  rounded to bf16 for bf16 architectures; prefix tokens (cross-attention architecture)
  ~ N(0, 1), [P, prefix_width];
* initial noise x_0 ~ N(0, 1) in fp32, [B, H, D] (Sec. 3, the policy's initial state);
* every stream is keyed by (seed, purpose, robot) so that the same robot gets the
  same prefix whatever the batch size.
"""
from __future__ import annotations

import dataclasses
import numpy as np

__all__ = [
    "Arch", "ARCHS", "weight_specs", "weight_count", "make_weights", "make_prefix_kv",
    "make_prefix_tokens", "make_noise", "round_to_bf16", "group_budgets",
    "sweep_grid", "draw_sweep_schedules", "blob_from_weights",
]


@dataclasses.dataclass(frozen=True)
class Arch:
    """Shape of a synthetic action expert (the velocity network of Eq. 1)."""
    name: str
    kind: str            # "adarms": joint attention over prefix KV + chunk, adaptive RMSNorm
                         # "dit":    chunk self-attention + cross-attention, adaLN-zero
                         # "concat": joint attention, plain RMSNorm; each token's time embedding
                         #           joins its action embedding in the input MLP (SmolVLA-style)
    dtype: str           # "f32" or "bf16" (weights / GEMM operands)
    n_layers: int
    width: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    mlp_dim: int
    action_dim: int
    chunk_len: int       # H
    prefix_len: int      # P
    prefix_width: int = 0  # DiT cross-attention prefix token width
    rope: bool = False

    def replace(self, **kw) -> "Arch":
        return dataclasses.replace(self, **kw)


ARCHS = {
    # 2 layers, width 256, 4 heads x 64, MLP 1024, fp32, H=16, D=7, 64 prefix tokens.
    "tiny": Arch("tiny", "adarms", "f32", 2, 256, 4, 4, 64, 1024, 7, 16, 64),
    # pi0-like: 18 layers, width 1024, GeGLU 4096, 8 query heads / 1 KV head of 256,
    # 816 prefix tokens, H=50, D=32, RoPE on the chunk tokens.
    "pi0": Arch("pi0", "adarms", "bf16", 18, 1024, 8, 1, 256, 4096, 32, 50, 816, rope=True),
    # DiT-style head: 16 layers, width 1536, 24 heads x 64, MLP 6144, cross-attention to
    # 300 prefix tokens of width 2048, H=16, D=32.
    "dit": Arch("dit", "dit", "bf16", 16, 1536, 24, 24, 64, 6144, 32, 16, 300, prefix_width=2048),
    # Small variants for parity tests that still span several tiles and ragged tails.
    "pi0_small": Arch("pi0_small", "adarms", "bf16", 2, 512, 4, 1, 128, 1536, 32, 50, 200, rope=True),
    "dit_small": Arch("dit_small", "dit", "bf16", 2, 384, 6, 6, 64, 1536, 32, 16, 72, prefix_width=256),
    "tiny_f32_rope": Arch("tiny_f32_rope", "adarms", "f32", 2, 256, 4, 2, 64, 1024, 7, 16, 64, rope=True),
    # Time embedding concatenated with the action embedding before the input MLP (App. C.1's
    # SmolVLA variant): fp32 tiny and a bf16 small expert with GQA and RoPE.
    "tiny_concat": Arch("tiny_concat", "concat", "f32", 2, 256, 4, 4, 64, 1024, 7, 16, 64),
    "concat_small": Arch("concat_small", "concat", "bf16", 2, 512, 8, 2, 64, 1536, 32, 50, 120, rope=True),
}


def weight_specs(a: Arch):
    """Ordered (name, shape) list of the flat fp32 weight blob.

    Linear weights are stored [in, out] (y = x W + b). Modulation vectors are packed in the
    order (scale, shift, gate) for "adarms" and (shift1, scale1, gate1, shift2, scale2,
    gate2) for "dit"; the final norm's modulation is (scale, shift) / (shift, scale).
    The gate/up and q/k/v projections are separate tensors here; the library re-lays them
    out internally. "concat" has no time MLP and no modulation: its input MLP takes the action
    embedding (ti_wa) and the sinusoidal time embedding (ti_wt) side by side, then to_w.
    """
    W, D, F = a.width, a.action_dim, a.mlp_dim
    q, kv = a.n_heads * a.head_dim, a.n_kv_heads * a.head_dim
    if a.kind == "concat":
        s = [("in_w", (D, W)), ("in_b", (W,)), ("ti_wa", (W, W)), ("ti_wt", (W, W)), ("ti_b", (W,)),
             ("to_w", (W, W)), ("to_b", (W,))]
        for l in range(a.n_layers):
            p = f"l{l}."
            s += [(p + "wq", (W, q)), (p + "wk", (W, kv)), (p + "wv", (W, kv)), (p + "wo", (q, W)),
                  (p + "wg", (W, F)), (p + "wu", (W, F)), (p + "wd", (F, W))]
        return s + [("out_w", (W, D)), ("out_b", (D,))]
    s = [("t_w1", (W, W)), ("t_b1", (W,)), ("t_w2", (W, W)), ("t_b2", (W,)),
         ("in_w", (D, W)), ("in_b", (W,))]
    for l in range(a.n_layers):
        p = f"l{l}."
        if a.kind == "adarms":
            s += [(p + "mod1_w", (W, 3 * W)), (p + "mod1_b", (3 * W,)),
                  (p + "wq", (W, q)), (p + "wk", (W, kv)), (p + "wv", (W, kv)), (p + "wo", (q, W)),
                  (p + "mod2_w", (W, 3 * W)), (p + "mod2_b", (3 * W,)),
                  (p + "wg", (W, F)), (p + "wu", (W, F)), (p + "wd", (F, W))]
        elif a.kind == "dit":
            Pw = a.prefix_width
            s += [(p + "mod_w", (W, 6 * W)), (p + "mod_b", (6 * W,)),
                  (p + "wq", (W, q)), (p + "wk", (W, q)), (p + "wv", (W, q)), (p + "wo", (q, W)),
                  (p + "wqc", (W, q)), (p + "wkc", (Pw, q)), (p + "wvc", (Pw, q)), (p + "woc", (q, W)),
                  (p + "w1", (W, F)), (p + "b1", (F,)), (p + "w2", (F, W)), (p + "b2", (W,))]
        else:
            raise ValueError(a.kind)
    s += [("modf_w", (W, 2 * W)), ("modf_b", (2 * W,)), ("out_w", (W, D)), ("out_b", (D,))]
    return s


def weight_count(a: Arch) -> int:
    return int(sum(int(np.prod(sh)) for _, sh in weight_specs(a)))


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bfloat16 (ties to even); returns fp32 values."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) & np.uint32(0xFFFF0000)
    return r.view(np.float32)


def _rng(seed: int, *key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, *key])))


_BLOCK = 1 << 22


def _normal_blocks(n: int, seed: int, tag: int, std: float, bf16: bool) -> np.ndarray:
    """n values ~ N(0, std^2), drawn in blocks of 4 Mi values, block j from its own PCG64
    stream keyed (seed, tag, j): the result does not depend on how many threads fill it."""
    import concurrent.futures as cf
    import os
    out = np.empty(n, dtype=np.float32)

    def fill(j):
        lo, hi = j * _BLOCK, min(n, (j + 1) * _BLOCK)
        blk = _rng(seed, tag, j).standard_normal(hi - lo, dtype=np.float32)
        blk *= np.float32(std)
        out[lo:hi] = round_to_bf16(blk) if bf16 else blk

    nblk = (n + _BLOCK - 1) // _BLOCK
    with cf.ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
        list(ex.map(fill, range(nblk)))
    return out


def make_weights(a: Arch, seed: int = 0, std: float = 0.02) -> np.ndarray:
    """Flat fp32 weight blob in weight_specs order, N(0, std), bf16-exact for bf16 archs."""
    return _normal_blocks(weight_count(a), seed, 1, std, a.dtype == "bf16")


def blob_from_weights(a: Arch, weights: dict) -> np.ndarray:
    """Pack a name -> array dict (e.g. a hand-built test model) into blob order."""
    parts = []
    for name, shape in weight_specs(a):
        w = np.asarray(weights[name], dtype=np.float32)
        assert w.shape == tuple(shape), (name, w.shape, shape)
        parts.append(w.reshape(-1))
    return np.concatenate(parts)


def split_blob(a: Arch, blob: np.ndarray) -> dict:
    """Name -> view of the blob (shapes per weight_specs)."""
    out, off = {}, 0
    for name, shape in weight_specs(a):
        n = int(np.prod(shape))
        out[name] = blob[off:off + n].reshape(shape)
        off += n
    assert off == blob.size
    return out


def make_prefix_kv(a: Arch, robot: int = 0, seed: int = 0):
    """Per-layer prefix keys and values [L, P, Hkv, dh] ~ N(0, 1) (attention-prefix archs)."""
    g = _rng(seed, 2, robot)
    shape = (a.n_layers, a.prefix_len, a.n_kv_heads, a.head_dim)
    k = g.standard_normal(shape, dtype=np.float32)
    v = g.standard_normal(shape, dtype=np.float32)
    if a.dtype == "bf16":
        k, v = round_to_bf16(k), round_to_bf16(v)
    return k, v


def make_prefix_tokens(a: Arch, robot: int = 0, seed: int = 0) -> np.ndarray:
    """Cross-attention prefix tokens [P, prefix_width] ~ N(0, 1) (DiT arch)."""
    g = _rng(seed, 3, robot)
    t = g.standard_normal((a.prefix_len, a.prefix_width), dtype=np.float32)
    if a.dtype == "bf16":
        t = round_to_bf16(t)
    return t


def make_noise(a: Arch, batch: int = 1, seed: int = 0) -> np.ndarray:
    """Initial chunk noise x_0 ~ N(0, I), fp32 [B, H, D]."""
    g = _rng(seed, 4)
    return g.standard_normal((batch, a.chunk_len, a.action_dim), dtype=np.float32)


def group_budgets(H: int, groups) -> np.ndarray:
    """Per-token step budgets from [(first, last_inclusive, budget), ...]; int32 [H]."""
    b = np.zeros(H, dtype=np.int32)
    for lo, hi, n in groups:
        b[lo:hi + 1] = n
    assert (b > 0).all(), "every token needs a budget"
    return b


def sweep_grid():
    """First-group release budgets x first-group sizes of the schedule sweep (rest at 10)."""
    return [(k, u) for k in (2, 3, 4, 6) for u in (5, 10, 20)]


def draw_sweep_schedules(H: int, batch: int, seed: int = 0, n_star: int = 10) -> np.ndarray:
    """One schedule per robot drawn uniformly from sweep_grid(); int32 [B, H]."""
    g = _rng(seed, 5)
    grid = sweep_grid()
    out = np.empty((batch, H), dtype=np.int32)
    for b in range(batch):
        k, u = grid[int(g.integers(len(grid)))]
        out[b] = group_budgets(H, [(0, u - 1, k), (u, H - 1, n_star)])
    return out
