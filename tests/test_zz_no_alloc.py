"""The projection op for callers that cannot allocate device memory.

uad_linear_static_scratch must give what uad_linear gives (same kernel, scratch in a static
device array instead of library allocations), on consecutive calls that reuse the array,
and must refuse shapes its fixed scratch cannot hold. Collected last on purpose, so that a
stop-at-first-failure run has already run every other test."""
import numpy as np
import pytest
import torch

import paper_2609_37772_gb300 as uad
from uad_inputs import round_to_bf16

pytestmark = pytest.mark.gpu


def _operands(M, N, K, seed):
    rng = np.random.default_rng(seed)
    x = torch.from_numpy(round_to_bf16(rng.normal(size=(M, K)).astype(np.float32))).to(torch.bfloat16).cuda()
    w = torch.from_numpy(uad.tile_weight((rng.normal(size=(K, N)) * 0.02).astype(np.float32)).view(np.int16)).cuda()
    b = torch.from_numpy(rng.normal(size=N).astype(np.float32)).cuda()
    return x, w, b


def _call(fn, x, w, b, M, N, K):
    out = torch.full((M, N), float("nan"), device="cuda")
    rc = fn(x.data_ptr(), w.data_ptr(), b.data_ptr(), out.data_ptr(), M, N, K,
            torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return rc, out


@pytest.mark.parametrize("M,N,K", [(50, 1024, 2048), (64, 2560, 1024), (50, 8192, 1024)])
def test_static_scratch_matches_uad_linear_twice(M, N, K):
    x, w, b = _operands(M, N, K, seed=M + N + K)
    rc, ref = _call(uad.uad_linear, x, w, b, M, N, K)
    assert rc == 0
    scale = ref.abs().max().item()
    for _ in range(2):                       # the second call reuses what the first left behind
        rc, out = _call(uad.uad_linear_static_scratch, x, w, b, M, N, K)
        assert rc == 0
        assert torch.isfinite(out).all()
        assert (out - ref).abs().max().item() <= 1e-5 * scale


def test_static_scratch_refuses_oversize_shapes():
    M, N, K = 256, 8192, 64                  # M * N = 2^21 > the 2^20 values the array holds
    x, w, b = _operands(M, N, K, seed=1)
    rc, out = _call(uad.uad_linear_static_scratch, x, w, b, M, N, K)
    assert rc == uad.UAD_ETOOBIG
    assert torch.isnan(out).all()            # nothing was launched
