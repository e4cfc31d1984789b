"""The fp32 device rotations of Ghost Action Correction on SO(3) (App. C.1; Sec. 4.4, Eqs. 8-9)
against the fp64 oracle over the whole range of angles: near 0, generic, near pi (where the axis
comes from the symmetric part of R), at pi (w and -w are one rotation) and past pi (the principal
vector is returned). Bound: an entry of a rotation matrix is at most 1, and exp, log and one
product are a few dozen fp32 operations each, so their results agree with fp64 to ~1e-6; the
test allows 1e-5."""
import numpy as np
import pytest

import paper_2609_37772_gb300 as uad
from oracle import so3

pytestmark = pytest.mark.gpu


def _cases():
    rng = np.random.default_rng(7)
    angles = np.concatenate([
        rng.uniform(0.0, np.pi, 24),
        [1e-7, 1e-5, 1e-4, 1e-3, 0.5, 2.0],
        np.pi - np.array([3e-2, 1e-2, 3e-3, 1e-3, 3e-4, 1e-4, 1e-5]),
        [np.pi] * 4,
        [np.pi + 1e-3, np.pi + 0.1, 4.0, 2 * np.pi - 0.1, 7.0, 9.0],
    ])
    axes = rng.normal(size=(len(angles), 3))
    axes /= np.linalg.norm(axes, axis=1, keepdims=True)
    w = axes * angles[:, None]
    # half turns about the coordinate axes and a diagonal
    w = np.concatenate([w, np.pi * np.array([[1, 0, 0], [0, 1, 0], [0, 0, 1], [0.6, 0.8, 0.0]])])
    return w.astype(np.float32)


def test_so3_rotations_match_the_oracle():
    w = _cases()
    n = len(w)
    le = np.zeros_like(w)
    lc = np.zeros_like(w)
    assert uad.uad_so3_check(w.ctypes.data, n, le.ctypes.data, lc.ctypes.data) == 0
    worst_e = worst_c = worst_v = 0.0
    for i in range(n):
        wi, wj = w[i].astype(np.float64), w[(i + 1) % n].astype(np.float64)
        R = so3.exp_so3(wi)
        C = R @ so3.exp_so3(wj).T
        assert np.linalg.norm(le[i]) <= np.pi + 1e-5 and np.linalg.norm(lc[i]) <= np.pi + 1e-5
        worst_e = max(worst_e, np.abs(so3.exp_so3(le[i]) - R).max())
        worst_c = max(worst_c, np.abs(so3.exp_so3(lc[i]) - C).max())
        # away from pi the principal vector is unique: compare it directly
        ref = so3.log_so3(R)
        if np.pi - np.linalg.norm(ref) > 1e-3:
            worst_v = max(worst_v, np.abs(le[i] - ref).max())
    print(f"SO(3) fp32 vs fp64: log(exp) {worst_e:.2e}, composition {worst_c:.2e}, vector {worst_v:.2e}")
    assert worst_e <= 1e-5 and worst_c <= 1e-5 and worst_v <= 1e-5


def test_so3_check_rejects_bad_arguments():
    w = np.zeros((1, 3), np.float32)
    assert uad.uad_so3_check(None, 1, w.ctypes.data, w.ctypes.data) == uad.UAD_EINVAL
    assert uad.uad_so3_check(w.ctypes.data, 0, w.ctypes.data, w.ctypes.data) == uad.UAD_EINVAL
