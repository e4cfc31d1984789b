"""Pins of the oracle's SO(3) Ghost Action Correction (App. C.1: rotations corrected by
composition on SO(3)): the rotation maps against an independent library, closed-form cases of
the correction, its first-order agreement with the additive rule of Eqs. 8-9."""
import numpy as np
import pytest

from oracle import so3
from oracle.uad import denoise

Rot = pytest.importorskip("scipy.spatial.transform").Rotation


def rng(seed):
    return np.random.default_rng(seed)


def test_exp_matches_library_and_is_a_rotation():
    for w in rng(0).normal(0, 1.2, (200, 3)):
        R = so3.exp_so3(w)
        assert np.allclose(R, Rot.from_rotvec(w).as_matrix(), atol=1e-12)
        assert np.allclose(R @ R.T, np.eye(3), atol=1e-12) and abs(np.linalg.det(R) - 1) < 1e-12
    assert np.allclose(so3.exp_so3([0, 0, 1e-10]), np.eye(3), atol=1e-9)


def test_log_inverts_exp_on_the_principal_branch():
    g = rng(1)
    for w in g.normal(0, 1.0, (300, 3)):
        t = np.linalg.norm(w)
        if t >= np.pi:
            w = w / t * (np.pi - 1e-3)
        assert np.allclose(so3.log_so3(so3.exp_so3(w)), w, atol=1e-9)
    for w in g.normal(0, 1.0, (50, 3)):   # near pi and tiny angles
        n = w / np.linalg.norm(w)
        for t in (np.pi - 1e-7, np.pi - 1e-5, 1e-9, 1e-5):
            r = so3.log_so3(so3.exp_so3(n * t))
            assert np.allclose(so3.exp_so3(r), so3.exp_so3(n * t), atol=1e-9)
            assert abs(np.linalg.norm(r) - t) < 1e-7
    # against the library's principal logarithm
    for w in g.normal(0, 2.0, (100, 3)):
        assert np.allclose(so3.log_so3(so3.exp_so3(w)), Rot.from_matrix(so3.exp_so3(w)).as_rotvec(), atol=1e-9)


def test_nearest_representative():
    n = np.array([0.0, 0.0, 1.0])
    w = n * (2 * np.pi - 0.5)             # same rotation as -0.5 n
    assert np.allclose(so3.nearest_rep(so3.log_so3(so3.exp_so3(w)), w), w, atol=1e-9)
    assert np.allclose(so3.nearest_rep(n * 0.3, n * 0.25), n * 0.3)


def test_corrections_compose_to_the_accumulated_error():
    """Constructed case: every ghost is a fixed rotation Q applied to its released action, so
    E_R = Q^U, and the |tail| corrections C compose exactly to E_R."""
    g = rng(2)
    q = np.array([0.05, -0.02, 0.03])
    Q = so3.exp_so3(q)
    rel = g.normal(0, 0.5, (4, 3))
    gho = np.array([so3.log_so3(Q @ so3.exp_so3(a)) for a in rel])
    tail = g.normal(0, 0.5, (6, 3))
    e, out = so3.gac_rotation(rel, gho, tail)
    assert np.allclose(e, 4 * q, atol=1e-12)
    C = so3.exp_so3(4 * q / 6)
    for r, o in zip(tail, out):
        assert np.allclose(so3.exp_so3(o), C @ so3.exp_so3(r), atol=1e-12)
    assert np.allclose(np.linalg.matrix_power(C, 6), so3.exp_so3(e), atol=1e-12)


def test_discrepancies_compose_in_token_order():
    """Reading of App. C.1 (rotations compose; the order is not stated): the early actions'
    discrepancies F_i = R(ghost_i) R(released_i)^T are applied one after another in token order,
    E_R = F_U ... F_2 F_1. Hand-worked case: a quarter turn about x (first early action) then a
    quarter turn about y (second) is a third of a turn about (1, 1, -1)/sqrt(3); the other order
    would give the axis (1, 1, 1)/sqrt(3)."""
    rel = np.zeros((2, 3))
    gho = np.array([[np.pi / 2, 0.0, 0.0], [0.0, np.pi / 2, 0.0]])
    e, _ = so3.gac_rotation(rel, gho, np.zeros((1, 3)))
    np.testing.assert_allclose(e, (2 * np.pi / 3) * np.array([1.0, 1.0, -1.0]) / np.sqrt(3), atol=1e-12)


def test_no_discrepancy_changes_nothing():
    g = rng(3)
    rel = g.normal(0, 0.7, (3, 3))
    tail = g.normal(0, 0.7, (5, 3))
    e, out = so3.gac_rotation(rel, rel.copy(), tail)
    assert np.allclose(e, 0, atol=1e-14) and np.allclose(out, tail, atol=1e-12)


def test_small_rotations_reduce_to_the_additive_rule():
    """For discrepancies of size eps the SO(3) correction differs from Eqs. 8-9 by O(eps^2)
    (on small actions, where rotation vectors add to first order)."""
    g = rng(4)
    for eps in (1e-2, 1e-3):
        rel = g.normal(0, eps, (5, 3))
        gho = rel + g.normal(0, eps, (5, 3))
        tail = g.normal(0, eps, (7, 3))
        e, out = so3.gac_rotation(rel, gho, tail)
        add = tail + np.sum(gho - rel, axis=0) / 7
        assert np.abs(out - add).max() < 20 * eps * eps
        assert np.abs(e - np.sum(gho - rel, axis=0)).max() < 20 * eps * eps


def test_denoise_rotation_dims_use_composition():
    """In a full chunk the rotation dimensions follow so3.gac_rotation, the other dimensions the
    additive rule, and a masked dimension is left alone."""
    H, D = 8, 7
    c = np.linspace(-0.4, 0.4, H * D).reshape(H, D)
    vel = lambda u, tau: c + 0.3 * np.sin(u + tau[:, None])      # a smooth synthetic field
    x0 = rng(5).normal(0, 1, (H, D))
    bud = [1, 1, 1, 4, 4, 4, 4, 4]
    mask = np.array([1, 1, 1, 0, 0, 0, 0], bool)
    r = denoise(vel, x0, bud, tr=True, gac=True, gac_mask=mask, rot_dim=3)
    plain = denoise(vel, x0, bud, tr=True, gac=False)
    tail = r["tail"]
    early = [0, 1, 2]
    e, rot = so3.gac_rotation(plain["released"][early][:, 3:6], plain["ghost"][early][:, 3:6],
                              plain["final"][tail][:, 3:6])
    assert np.allclose(r["final"][tail][:, 3:6], rot, atol=1e-12) and np.allclose(r["E"][3:6], e, atol=1e-12)
    E = np.sum(plain["ghost"][early] - plain["released"][early], axis=0)
    assert np.allclose(r["final"][tail][:, :3], plain["final"][tail][:, :3] + E[:3] / len(tail), atol=1e-12)
    assert np.array_equal(r["final"][:, 6], plain["final"][:, 6])
