"""CPU checks of the Python binding's argument marshalling.

The C ABI takes bare pointers, so it cannot see how large a caller's buffer is: the binding
refuses a buffer of the wrong element type, size, layout or memory space before the call. Here
the binding runs against a null library context: a well-formed call reaches the library, which
answers UAD_EINVAL for the null context without touching a GPU, while a malformed one stops in
the binding with ValueError.
"""
import numpy as np
import pytest
import torch

import paper_2609_37772_gb300 as uad
from uad_inputs import ARCHS, group_budgets


def _detached(name, B=1):
    a = ARCHS[name]
    ex = uad.Expert.__new__(uad.Expert)
    ex.arch = uad.arch_struct(a, B)
    ex.H, ex.D = a.chunk_len, a.action_dim
    ex.h, ex._keep, ex._B = None, None, B
    return a, ex


def _reaches_library(call):
    with pytest.raises(uad.UADError) as ei:
        call()
    assert ei.value.code == uad.UAD_EINVAL


def test_noise_must_match_the_schedule():
    a, ex = _detached("tiny", B=2)
    bud = np.stack([group_budgets(a.chunk_len, [(0, a.chunk_len - 1, 4)])] * 2)
    good = np.zeros((2, a.chunk_len, a.action_dim), np.float32)
    _reaches_library(lambda: ex.denoise(good, bud))
    _reaches_library(lambda: ex.denoise(torch.from_numpy(good), bud))
    with pytest.raises(ValueError, match="noise: expected"):
        ex.denoise(good[:1], bud)                                  # one robot short
    with pytest.raises(ValueError, match="float32"):
        ex.denoise(torch.zeros(2, a.chunk_len, a.action_dim, dtype=torch.float64), bud)
    with pytest.raises(ValueError, match="contiguous"):
        ex.denoise(torch.zeros(2, a.action_dim, a.chunk_len).transpose(1, 2), bud)
    with pytest.raises(ValueError, match="noise: expected"):
        ex.profile(good[:1], bud)
    # numpy noise of another float type is converted, not refused
    _reaches_library(lambda: ex.denoise(good.astype(np.float64), bud))


def test_gac_mask_has_one_entry_per_action_dimension():
    a, ex = _detached("tiny")
    bud = group_budgets(a.chunk_len, [(0, 3, 2), (4, a.chunk_len - 1, 4)])[None]
    noise = np.zeros((1, a.chunk_len, a.action_dim), np.float32)
    _reaches_library(lambda: ex.denoise(noise, bud, gac_mask=np.ones(a.action_dim)))
    with pytest.raises(ValueError, match="gac_mask"):
        ex.denoise(noise, bud, gac_mask=np.ones(a.action_dim - 1))


def test_prefix_sizes_follow_the_architecture():
    a, ex = _detached("pi0_small")
    shape = (a.n_layers, a.prefix_len, a.n_kv_heads, a.head_dim)
    k = np.zeros(shape, np.float32)
    _reaches_library(lambda: ex.set_prefix(0, k, k))
    _reaches_library(lambda: ex.set_prefix(0, k.astype(np.float64), k))       # converted
    bits = np.zeros(shape, np.uint16)
    _reaches_library(lambda: ex.set_prefix(0, bits, bits, dtype="bf16"))
    tb = torch.zeros(shape, dtype=torch.bfloat16)
    _reaches_library(lambda: ex.set_prefix(0, tb, tb, dtype="bf16"))
    with pytest.raises(ValueError, match="prefix k: expected"):
        ex.set_prefix(0, k[:, :-1], k)                             # one prefix token short
    with pytest.raises(ValueError, match="prefix v: expected"):
        ex.set_prefix(0, k, k[:1])
    with pytest.raises(ValueError, match="bfloat16"):
        ex.set_prefix(0, torch.zeros(shape), torch.zeros(shape), dtype="bf16")

    d, exd = _detached("dit_small")
    tok = np.zeros((d.prefix_len, d.prefix_width), np.float32)
    _reaches_library(lambda: exd.set_prefix(0, tok))
    with pytest.raises(ValueError, match="prefix k: expected"):
        exd.set_prefix(0, tok[:, :-8])


def test_outputs_must_hold_the_whole_chunk():
    a, ex = _detached("tiny", B=3)
    H, D = a.chunk_len, a.action_dim
    _reaches_library(lambda: ex.finish(final=np.zeros((3, H, D), np.float32)))
    _reaches_library(lambda: ex.finish())                          # binding allocates them
    with pytest.raises(ValueError, match="final: expected"):
        ex.finish(final=np.zeros((1, H, D), np.float32))
    with pytest.raises(ValueError, match="ghost: expected"):
        ex.finish(ghost=torch.zeros(3, H, D - 1))
    with pytest.raises(ValueError, match="gac_error: expected"):
        ex.finish(gac_error=np.zeros((1, D), np.float32))
    with pytest.raises(ValueError, match="float32"):
        ex.finish(final=np.zeros((3, H, D), np.float64))
    # poll writes host memory: an [H][D] fp32 host buffer
    _reaches_library(lambda: ex.poll(0, out=np.zeros((H, D), np.float32)))
    with pytest.raises(ValueError, match="out: expected"):
        ex.poll(0, out=np.zeros((H - 1, D), np.float32))
    if torch.cuda.is_available():                                  # pragma: no cover
        with pytest.raises(ValueError, match="host memory"):
            ex.poll(0, out=torch.zeros(H, D, device="cuda"))
