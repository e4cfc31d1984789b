"""GPU parity of the kernel-level projection op (uad_linear) against an fp64 reference of the
same bf16 operands (tolerance: fp32 accumulation, 1e-5 of the output scale)."""
import numpy as np
import pytest
import torch

import paper_2609_37772_gb300 as uad
from uad_inputs import round_to_bf16

pytestmark = pytest.mark.gpu


def run_linear(x, w, bias, fn=None):
    fn = fn or uad.uad_linear
    M, K = x.shape
    N = w.shape[1]
    xd = torch.from_numpy(round_to_bf16(x)).to(torch.bfloat16).cuda()
    wd = torch.from_numpy(uad.tile_weight(w).view(np.int16)).cuda()
    bd = None if bias is None else torch.from_numpy(bias).cuda()
    out = torch.full((M, N), float("nan"), device="cuda")
    rc = fn(xd.data_ptr(), wd.data_ptr(), None if bd is None else bd.data_ptr(), out.data_ptr(), M, N, K,
            torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return rc, out.cpu().numpy()


def reference(x, w, bias):
    r = round_to_bf16(x).astype(np.float64) @ round_to_bf16(w).astype(np.float64)
    return r + (0 if bias is None else bias.astype(np.float64))


@pytest.mark.parametrize("M,N,K", [(50, 1024, 2048), (50, 2560, 1024), (64, 8192, 1024), (1, 128, 64),
                                   (130, 384, 4096), (50, 1024, 4096)])
def test_linear_matches_reference(M, N, K):
    rng = np.random.default_rng(M * 7 + N + K)
    x = rng.normal(size=(M, K)).astype(np.float32)
    w = (rng.normal(size=(K, N)) * 0.02).astype(np.float32)
    bias = rng.normal(size=N).astype(np.float32)
    rc, out = run_linear(x, w, bias)
    assert rc == 0
    ref = reference(x, w, bias)
    assert np.abs(out - ref).max() <= 1e-5 * np.abs(ref).max()


# Shapes that take the persistent wide form on a 152-SM GB300, with each of its tile widths and
# ragged last token tiles (plan of the busiest CTA's work):
#   (2560, 2048, 64): 16 weight tiles x 14 tiles of 192 tokens (the last 64)
#   (3000, 1024, 128): 8 x 16 tiles of 192 tokens (the last 120)
#   (2400, 1024, 128): 8 x 19 tiles of 128 tokens (the last 96)
#   (800, 2560, 192): 20 x 7 tiles of 128 tokens (the last 32)
@pytest.mark.parametrize("M,N,K", [(2560, 2048, 64), (3000, 1024, 128), (2400, 1024, 128), (800, 2560, 192)])
def test_linear_wide_tiles_match_reference(M, N, K):
    rng = np.random.default_rng(M + N + K)
    x = rng.normal(size=(M, K)).astype(np.float32)
    w = (rng.normal(size=(K, N)) * 0.02).astype(np.float32)
    bias = rng.normal(size=N).astype(np.float32)
    rc, out = run_linear(x, w, bias)
    assert rc == 0
    ref = reference(x, w, bias)
    assert np.abs(out - ref).max() <= 1e-5 * np.abs(ref).max()


def test_linear_rejects_bad_shapes():
    assert uad.uad_linear(1, 1, None, 1, 50, 100, 64, None) == uad.UAD_EINVAL
    assert uad.uad_linear(1, 1, None, 1, 0, 128, 64, None) == uad.UAD_EINVAL
    assert uad.uad_linear(None, 1, None, 1, 50, 128, 64, None) == uad.UAD_EINVAL
