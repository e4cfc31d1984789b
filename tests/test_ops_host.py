"""CPU check of the host-only weight tiling against the layout include/uad.h documents."""
import numpy as np
import pytest

import paper_2609_37772_gb300 as uad
from uad_inputs import round_to_bf16


def test_tile_weight_layout_is_a_permutation_of_bf16_values():
    rng = np.random.default_rng(0)
    K, N = 192, 256
    w = rng.normal(size=(K, N)).astype(np.float32)
    t = uad.tile_weight(w)
    bits = round_to_bf16(w).view(np.uint32) >> 16
    # documented layout: block (n//128, k//64), row n%128, 16-byte group (k%64)//8 ^ (n%8)
    KC = K // 64
    for n in range(0, N, 37):
        for k in range(0, K, 11):
            blk = (n // 128) * KC + k // 64
            g = ((k % 64) // 8) ^ (n % 8)
            assert t[blk * 8192 + (n % 128) * 64 + g * 8 + k % 8] == bits[k, n]
    assert np.array_equal(np.sort(t), np.sort(bits.reshape(-1).astype(np.uint16)))


def test_tile_weight_rejects_bad_shapes():
    with pytest.raises(uad.UADError):
        uad.tile_weight(np.zeros((64, 100), np.float32))
    with pytest.raises(uad.UADError):
        uad.tile_weight(np.zeros((48, 128), np.float32))
