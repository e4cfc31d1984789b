"""Rotations for Ghost Action Correction on SO(3) -- TEST INFRASTRUCTURE ONLY (see package doc).

The paper corrects rotational action dimensions by composition on SO(3) instead of Euclidean
subtraction (App. C.1, "TR and GAC"; Sec. 4.4) but gives no formula. Reading used here (and by
the CUDA path, which implements the same mathematics separately):

  rotation part of an action  a rotation vector w (axis times angle, radians), R(w) = exp([w]x)
  discrepancy of early action i      D_i = R(a'_i) R(a_i)^T    (ghost relative to released)
  accumulated error (Eq. 8 on SO(3)) E_R = D_{i_m} ... D_{i_2} D_{i_1}, tokens in index order
                                     (later ones multiply on the left), e_R = log(E_R)
  correction of each tail action (Eq. 9 on SO(3))
                                     R(a_j) <- C R(a_j),  C = exp(e_R / |tail|),
                                     so that the corrections over the tail compose to E_R;
                                     the new rotation vector is the representative of
                                     log(C R(a_j)) closest to a_j (w + 2 pi m w/|w|, m in -1..1)
To first order in the discrepancies this is the additive rule of Eqs. 8-9.

exp: Rodrigues' formula; log: angle from atan2(|axial part|, (trace - 1) / 2), with the axis
from the symmetric part near pi. Plain fp64 numpy, one rotation at a time.
"""
import numpy as np

PI = np.pi


def hat(w):
    x, y, z = w
    return np.array([[0.0, -z, y], [z, 0.0, -x], [-y, x, 0.0]])


def exp_so3(w):
    """R = I + sin(t)/t K + (1 - cos(t))/t^2 K^2 with K = [w]x, t = |w| (Rodrigues)."""
    w = np.asarray(w, np.float64)
    t = np.linalg.norm(w)
    K = hat(w)
    if t < 1e-8:
        a, b = 1.0 - t * t / 6.0, 0.5 - t * t / 24.0
    else:
        a, b = np.sin(t) / t, (1.0 - np.cos(t)) / (t * t)
    return np.eye(3) + a * K + b * (K @ K)


def log_so3(R):
    """Principal rotation vector of R (angle in [0, pi])."""
    R = np.asarray(R, np.float64)
    v = 0.5 * np.array([R[2, 1] - R[1, 2], R[0, 2] - R[2, 0], R[1, 0] - R[0, 1]])   # sin(t) n
    c = 0.5 * (np.trace(R) - 1.0)                                                   # cos(t)
    s = np.linalg.norm(v)
    t = np.arctan2(s, c)
    if t < 1e-8:
        return v * (1.0 + t * t / 6.0)
    if PI - t > 1e-4:
        return v * (t / s)
    # near pi: n n^T = (R + R^T)/2 - cos(t) I) / (1 - cos(t)); axis from the largest diagonal
    B = (0.5 * (R + R.T) - c * np.eye(3)) / (1.0 - c)
    k = int(np.argmax(np.diag(B)))
    n = B[:, k] / np.sqrt(max(B[k, k], 1e-300))
    if np.dot(n, v) < 0:   # sign from the (small) axial part
        n = -n
    return n * t


def nearest_rep(w, ref):
    """Among w + 2 pi m w/|w| (m = -1, 0, 1) the rotation vector closest to ref."""
    w = np.asarray(w, np.float64)
    t = np.linalg.norm(w)
    if t < 1e-12:
        return w
    n = w / t
    cands = [w + 2.0 * PI * m * n for m in (-1, 0, 1)]
    return min(cands, key=lambda c: np.linalg.norm(c - ref))


def gac_rotation(released, ghost, tail_rows):
    """Eqs. 8-9 on SO(3) for one chunk. released, ghost: [U, 3] rotation vectors of the early
    actions in token order; tail_rows: [T, 3] rotation vectors of the executable tail.
    The discrepancies F_i = R(ghost_i) R(released_i)^T are applied in token order, each after the
    previous ones: E_R = F_U ... F_2 F_1. Returns (e_R, corrected tail rows [T, 3])."""
    E = np.eye(3)
    for a, g in zip(released, ghost):
        E = exp_so3(g) @ exp_so3(a).T @ E
    e = log_so3(E)
    C = exp_so3(e / len(tail_rows))
    out = np.array([nearest_rep(log_so3(C @ exp_so3(r)), r) for r in tail_rows])
    return e, out
