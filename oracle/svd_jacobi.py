"""One-sided Jacobi SVD in pure Python/numpy fp64 (oracle; test infrastructure only).

An implementation of the singular value decomposition that shares nothing
with LAPACK, used as a brute-force second opinion on tiny matrices (a few
rows and columns): Hestenes' one-sided Jacobi method orthogonalises the
columns of W by plane rotations until every pair is orthogonal; the column
norms are then the singular values.
"""

from __future__ import annotations

import math

import numpy as np


def jacobi_svd(W, tol: float = 1e-15, max_sweeps: int = 100):
    """Return (U, s, Vt) with W = U diag(s) Vt, s sorted descending.

    W is m x n with m >= n (transpose the input otherwise)."""
    A = np.array(W, dtype=np.float64, copy=True)
    m, n = A.shape
    if m < n:
        U, s, Vt = jacobi_svd(A.T, tol, max_sweeps)
        return Vt.T, s, U.T
    V = np.eye(n)
    for _ in range(max_sweeps):
        rotated = False
        for i in range(n - 1):
            for j in range(i + 1, n):
                alpha = float(A[:, i] @ A[:, i])
                beta = float(A[:, j] @ A[:, j])
                gamma = float(A[:, i] @ A[:, j])
                if abs(gamma) <= tol * math.sqrt(alpha * beta) or gamma == 0.0:
                    continue
                rotated = True
                zeta = (beta - alpha) / (2.0 * gamma)
                t = math.copysign(1.0, zeta) / (abs(zeta) + math.sqrt(1.0 + zeta * zeta))
                c = 1.0 / math.sqrt(1.0 + t * t)
                s_ = c * t
                ai = A[:, i].copy()
                A[:, i] = c * ai - s_ * A[:, j]
                A[:, j] = s_ * ai + c * A[:, j]
                vi = V[:, i].copy()
                V[:, i] = c * vi - s_ * V[:, j]
                V[:, j] = s_ * vi + c * V[:, j]
        if not rotated:
            break
    s = np.sqrt((A * A).sum(axis=0))
    order = np.argsort(-s)
    s = s[order]
    A = A[:, order]
    V = V[:, order]
    U = np.zeros_like(A)
    for k in range(n):
        if s[k] > 0:
            U[:, k] = A[:, k] / s[k]
    return U, s, V.T
