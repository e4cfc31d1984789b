"""The seeded input generators shared by the CUDA path's tests and the oracle.

They hold none of the method's arithmetic, but every parity case rests on them: the same seed
must give the same inputs on any machine and thread count, bf16 experts must get values that
bf16 holds exactly (so that the oracle and the kernels start from identical operands), and a
robot's prefix and noise must not depend on how many robots share the batch.
"""
import numpy as np
import pytest
import torch

import uad_inputs
from uad_inputs import (ARCHS, blob_from_weights, draw_sweep_schedules, group_budgets,
                        make_noise, make_prefix_kv, make_prefix_tokens, make_weights,
                        round_to_bf16, split_blob, sweep_grid, weight_count, weight_specs)


def _low_bits_zero(x):
    return bool(((np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
                  & np.uint32(0xFFFF)) == 0).all())


def test_round_to_bf16_matches_torch_round_to_nearest_even():
    g = np.random.default_rng(0)
    x = np.concatenate([
        g.standard_normal(100_000).astype(np.float32),
        (g.standard_normal(10_000) * 1e30).astype(np.float32),
        (g.standard_normal(10_000) * 1e-38).astype(np.float32),   # subnormals
        np.array([0.0, -0.0, np.inf, -np.inf, np.finfo(np.float32).max,
                  -np.finfo(np.float32).max, np.finfo(np.float32).tiny], dtype=np.float32),
    ])
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    np.testing.assert_array_equal(round_to_bf16(x).view(np.uint32), want.view(np.uint32))


def test_round_to_bf16_breaks_ties_to_even():
    # 1 + 2^-8 lies halfway between bf16 neighbours 1 and 1 + 2^-7: the even one (1) wins;
    # 1 + 3 * 2^-8 lies halfway between 1 + 2^-7 and 1 + 2^-6: again the even one wins.
    x = np.array([1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, -(1 + 2.0 ** -8), 1 + 2.0 ** -8 + 2.0 ** -20],
                 dtype=np.float32)
    np.testing.assert_array_equal(round_to_bf16(x),
                                  np.array([1.0, 1 + 2.0 ** -6, -1.0, 1 + 2.0 ** -7], np.float32))
    nan = round_to_bf16(np.array([np.nan], np.float32))
    assert np.isnan(nan).all()


@pytest.mark.parametrize("name", ["tiny", "pi0_small", "dit_small", "tiny_concat", "concat_small"])
def test_weights_are_seeded_and_exact_in_the_arch_dtype(name):
    a = ARCHS[name]
    w = make_weights(a, seed=7)
    assert w.dtype == np.float32 and w.size == weight_count(a)
    np.testing.assert_array_equal(w, make_weights(a, seed=7))
    assert not np.array_equal(w, make_weights(a, seed=8))
    if a.dtype == "bf16":
        assert _low_bits_zero(w)
    else:
        assert not _low_bits_zero(w)            # fp32 experts keep full fp32 values
    assert abs(float(w.std()) - 0.02) < 0.002 and abs(float(w.mean())) < 0.002


def test_weight_blocks_do_not_depend_on_the_total_length():
    # Each 4 Mi-value block comes from its own stream, so a longer blob begins with the
    # values of a shorter one, whatever the thread count that filled it.
    n = uad_inputs._BLOCK + 1000
    long = uad_inputs._normal_blocks(n, 3, 1, 1.0, False)
    short = uad_inputs._normal_blocks(1000, 3, 1, 1.0, False)
    np.testing.assert_array_equal(long[:1000], short)
    tail = uad_inputs._rng(3, 1, 1).standard_normal(1000, dtype=np.float32)
    np.testing.assert_array_equal(long[uad_inputs._BLOCK:], tail)


@pytest.mark.parametrize("name", ["tiny", "pi0_small", "dit_small", "concat_small"])
def test_blob_layout_is_contiguous_and_round_trips(name):
    a = ARCHS[name]
    specs = weight_specs(a)
    names = [n for n, _ in specs]
    assert len(set(names)) == len(names)
    n = weight_count(a)
    assert n < (1 << 24)                       # arange stays exact in fp32
    blob = np.arange(n, dtype=np.float32)
    parts = split_blob(a, blob)
    off = 0
    for nm, shape in specs:                    # views tile the blob in order, no gaps
        assert parts[nm].shape == tuple(shape)
        assert np.shares_memory(parts[nm], blob)
        assert parts[nm].reshape(-1)[0] == off
        off += int(np.prod(shape))
    assert off == n
    np.testing.assert_array_equal(blob_from_weights(a, parts), blob)


def test_pi0_like_expert_size():
    # 18 layers of width 1024, GeGLU 4096, 8 x 256 query heads, one 256-wide KV head, plus
    # time MLP, input/output projections and the per-layer adaptive-norm modulations.
    a = ARCHS["pi0"]
    W, F, q, kv = 1024, 4096, 2048, 256
    per_layer = 2 * (W * 3 * W + 3 * W) + W * q + 2 * W * kv + q * W + 3 * W * F
    total = 2 * (W * W + W) + 32 * W + W + 18 * per_layer + W * 2 * W + 2 * W + W * 32 + 32
    assert weight_count(a) == total


@pytest.mark.parametrize("name", ["pi0_small", "tiny"])
def test_prefix_kv_is_keyed_by_robot(name):
    a = ARCHS[name]
    k0, v0 = make_prefix_kv(a, robot=0, seed=2)
    k1, v1 = make_prefix_kv(a, robot=1, seed=2)
    shape = (a.n_layers, a.prefix_len, a.n_kv_heads, a.head_dim)
    assert k0.shape == v0.shape == shape and k0.dtype == np.float32
    np.testing.assert_array_equal(k0, make_prefix_kv(a, robot=0, seed=2)[0])
    assert not np.array_equal(k0, k1) and not np.array_equal(v0, v1) and not np.array_equal(k0, v0)
    assert _low_bits_zero(k0) == (a.dtype == "bf16")
    assert abs(float(k0.std()) - 1.0) < 0.05


def test_prefix_tokens_are_keyed_by_robot():
    a = ARCHS["dit_small"]
    t0, t1 = make_prefix_tokens(a, 0, 4), make_prefix_tokens(a, 1, 4)
    assert t0.shape == (a.prefix_len, a.prefix_width)
    np.testing.assert_array_equal(t0, make_prefix_tokens(a, 0, 4))
    assert not np.array_equal(t0, t1) and _low_bits_zero(t0)


def test_noise_of_a_robot_does_not_depend_on_the_batch_size():
    a = ARCHS["pi0"]
    x1, x4 = make_noise(a, 1, seed=9), make_noise(a, 4, seed=9)
    assert x4.shape == (4, a.chunk_len, a.action_dim) and x4.dtype == np.float32
    np.testing.assert_array_equal(x4[:1], x1)
    assert not np.array_equal(x4[0], x4[1])


def test_group_budgets():
    b = group_budgets(50, [(0, 9, 4), (10, 24, 7), (25, 49, 10)])
    assert b.dtype == np.int32 and b.shape == (50,)
    assert (b[:10] == 4).all() and (b[10:25] == 7).all() and (b[25:] == 10).all()
    with pytest.raises(AssertionError):
        group_budgets(50, [(0, 9, 4), (11, 49, 10)])       # token 10 has no budget


def test_sweep_schedules_come_from_the_grid():
    H, n_star = 50, 10
    s = draw_sweep_schedules(H, 64, seed=1, n_star=n_star)
    assert s.shape == (64, H) and s.dtype == np.int32
    np.testing.assert_array_equal(s, draw_sweep_schedules(H, 64, seed=1, n_star=n_star))
    grid = set(sweep_grid())
    seen = set()
    for row in s:
        k = int(row[0])
        u = int(np.argmax(row != k)) if (row != k).any() else H
        assert (k, u) in grid and (row[u:] == n_star).all()
        seen.add((k, u))
    assert len(seen) > len(grid) // 2          # uniform over 12 entries: 64 draws cover most
